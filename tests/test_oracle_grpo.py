"""Pins of the GRPO token-loss oracle (Sec. "GRPO Optimization", Eq. advantage and
Eq. ppo) against values fixed by the mathematics, not by re-typing its formula:
the regimes of the clipped surrogate worked out by hand, the k3 estimator's
closed forms and Taylor expansion, and invariants of the group advantage."""
import math

import numpy as np
import pytest

import oracle


def _loss(d_lp, adv, eps_low=0.2, eps_high=0.28, beta=0.0, d_ref=0.0):
    """Loss of one token whose log-ratio to the old policy is d_lp."""
    lp = np.array([[-1.0]])
    return oracle.grpo_token_loss(lp, lp - d_lp, lp + d_ref, np.array([adv]), eps_low, eps_high,
                                  beta)[0, 0]


def test_advantage_is_reward_minus_group_mean():
    r = np.array([1.0, 0.0, 0.5, 0.5, 2.0, 3.5])
    a = oracle.group_advantages(r, 3)
    assert np.allclose(a, [0.5, -0.5, 0.0, -1.5, 0.0, 1.5])
    # each group's advantages sum to zero; a group of one has zero advantage
    assert np.allclose(a.reshape(2, 3).sum(axis=1), 0.0)
    assert np.all(oracle.group_advantages(r, 1) == 0.0)
    # no variance normalisation: scaling the rewards scales the advantages
    assert np.allclose(oracle.group_advantages(3 * r, 3), 3 * a)
    with pytest.raises(ValueError):
        oracle.group_advantages(r, 4)


def test_clip_regimes_worked_by_hand():
    # rho = 1: the surrogate is A, the loss -A
    assert _loss(0.0, 2.0) == pytest.approx(-2.0, abs=1e-15)
    assert _loss(0.0, -3.0) == pytest.approx(3.0, abs=1e-15)
    # A > 0, rho = 1.5 > 1 + 0.28: clipped at 1.28 -> loss -1.28 A
    assert _loss(math.log(1.5), 2.0) == pytest.approx(-2.56, rel=1e-14)
    # A > 0, rho = 1.1 inside the band: loss -rho A
    assert _loss(math.log(1.1), 2.0) == pytest.approx(-2.2, rel=1e-14)
    # A > 0, rho = 0.5 below the band: min picks rho A (the unclipped, smaller term)
    assert _loss(math.log(0.5), 2.0) == pytest.approx(-1.0, rel=1e-14)
    # A < 0, rho = 0.5 < 1 - 0.2: min picks the clipped 0.8 A -> loss -0.8 A
    assert _loss(math.log(0.5), -2.0) == pytest.approx(1.6, rel=1e-14)
    # A < 0, rho = 1.5 above the band: min picks rho A -> loss 1.5 |A|
    assert _loss(math.log(1.5), -2.0) == pytest.approx(3.0, rel=1e-14)
    # symmetric band 0.2 / 0.2: A > 0 and rho = 1.25 clip at 1.2
    assert _loss(math.log(1.25), 1.0, eps_high=0.2) == pytest.approx(-1.2, rel=1e-14)
    # A = 0: no policy-gradient term at any ratio
    assert _loss(math.log(7.0), 0.0) == 0.0


def test_k3_estimator_closed_forms():
    assert oracle.kl_k3(np.array(-2.0), np.array(-2.0)) == 0.0
    # x = lp_ref - lp = ln 2: e^x - x - 1 = 1 - ln 2
    assert oracle.kl_k3(np.array(0.0), np.array(math.log(2.0))) == pytest.approx(1 - math.log(2.0), rel=1e-14)
    # x = -1: 1/e
    assert oracle.kl_k3(np.array(1.0), np.array(0.0)) == pytest.approx(math.exp(-1.0), rel=1e-14)
    # non-negative, and x^2 / 2 + x^3 / 6 to third order near zero
    x = np.linspace(-3, 3, 61)
    assert np.all(oracle.kl_k3(np.zeros_like(x), x) >= 0.0)
    for h in (1e-3, -1e-3):
        assert oracle.kl_k3(np.array(0.0), np.array(h)) == pytest.approx(h * h / 2 + h ** 3 / 6, rel=1e-5)


def test_kl_term_adds_beta_times_k3():
    # rho = 1, A = 0: the loss is beta * k3 alone; lp_ref - lp = ln 2
    v = _loss(0.0, 0.0, beta=0.01, d_ref=math.log(2.0))
    assert v == pytest.approx(0.01 * (1 - math.log(2.0)), rel=1e-14)


def test_token_mean_over_the_mask():
    L = np.array([[1.0, 2.0, 3.0], [4.0, 5.0, 6.0]])
    m = np.array([[1, 1, 0], [1, 0, 0]], dtype=np.uint8)
    assert oracle.grpo_loss_mean(L, m) == pytest.approx(7.0 / 3.0, rel=1e-15)
    assert oracle.grpo_loss_mean(L) == pytest.approx(3.5, rel=1e-15)
    assert oracle.grpo_loss_mean(L, np.zeros_like(m)) == 0.0


def test_gradient_free_identity_on_policy():
    """On-policy (lp = lp_old = lp_ref) the token loss is -A for every token, so the
    batch mean with a full mask is -(mean of row advantages weighted by row length)
    = 0 when every row has the same length (advantages sum to zero per group)."""
    rng = np.random.default_rng(0)
    B, T, G = 6, 5, 3
    lp = -rng.random((B, T))
    a = oracle.group_advantages(rng.random(B), G)
    L = oracle.grpo_token_loss(lp, lp, lp, a, 0.2, 0.28, 0.01)
    assert np.allclose(L, -a[:, None] * np.ones((1, T)), atol=1e-15)
    assert oracle.grpo_loss_mean(L) == pytest.approx(0.0, abs=1e-15)
