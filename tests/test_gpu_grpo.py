"""GRPO token loss on the GPU (Sec. "GRPO Optimization", Eq. advantage, Eq. ppo)
against the fp64 oracle: the standalone kernel over given log-probs (ragged T,
masks, symmetric and asymmetric clip bands, beta 0 without a reference policy,
groups of one, an empty mask), and scoring with the loss formed in its
log-prob epilogue (equal, bit for bit, to the standalone kernel applied to the
same log-probs, and to the oracle within the scoring tolerance)."""
import numpy as np
import pytest

import oracle
import synth
from _gpu import decoder, require_gpu

pytestmark = pytest.mark.gpu
RTOL, ATOL = 2e-6, 2e-6  # fp32 arithmetic on fp32 inputs vs fp64


def _inputs(B, T, seed, spread=0.6):
    rng = np.random.default_rng(seed)
    lp = -rng.gamma(2.0, 1.0, size=(B, T)).astype(np.float32)
    # log-ratios spanning the clip band and well outside it
    lp_old = (lp - rng.normal(0, spread, size=(B, T))).astype(np.float32)
    lp_ref = (lp + rng.normal(0, spread, size=(B, T))).astype(np.float32)
    rewards = rng.random(B).astype(np.float32)
    mask = (rng.random((B, T)) > 0.2).astype(np.uint8)
    return lp, lp_old, lp_ref, rewards, mask


def _gpu_loss(lp, lp_old, lp_ref, rewards, group, mask, eps_low, eps_high, beta):
    import torch
    from paper_2609_12471_gb300.runtime import grpo_token_loss
    t = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a)).cuda()
    loss, mean = grpo_token_loss(t(lp), t(lp_old), t(rewards), group, lp_ref=t(lp_ref), mask=t(mask),
                                 eps_low=eps_low, eps_high=eps_high, beta=beta)
    return loss.cpu().numpy(), float(mean.cpu().numpy()[0])


def _oracle(lp, lp_old, lp_ref, rewards, group, mask, eps_low, eps_high, beta):
    adv = oracle.group_advantages(rewards.astype(np.float64), group)
    L = oracle.grpo_token_loss(lp, lp_old, lp_ref, adv, eps_low, eps_high, beta)
    return L, oracle.grpo_loss_mean(L, mask)


@pytest.mark.parametrize("B,T,group,eps,beta,use_ref,use_mask", [
    (12, 37, 4, (0.2, 0.28), 0.01, True, True),    # multi-turn run's band, ragged T
    (8, 300, 8, (0.2, 0.2), 0.01, True, True),     # single-turn band, rows longer than a block
    (6, 5, 3, (0.2, 0.28), 0.0, False, False),     # no KL term, no reference policy, no mask
    (5, 64, 1, (0.2, 0.28), 0.05, True, True),     # groups of one: A = 0, only the KL term
])
def test_token_loss_matches_oracle(B, T, group, eps, beta, use_ref, use_mask):
    require_gpu()
    lp, lp_old, lp_ref, rewards, mask = _inputs(B, T, seed=B * 1000 + T)
    lp_ref = lp_ref if use_ref else None
    mask = mask if use_mask else None
    got, got_mean = _gpu_loss(lp, lp_old, lp_ref, rewards, group, mask, eps[0], eps[1], beta)
    ref, ref_mean = _oracle(lp, lp_old, lp_ref, rewards, group, mask, eps[0], eps[1], beta)
    np.testing.assert_allclose(got, ref, rtol=RTOL, atol=ATOL)
    assert got_mean == pytest.approx(ref_mean, rel=1e-5, abs=1e-6)


def test_empty_mask_gives_zero_mean():
    require_gpu()
    lp, lp_old, lp_ref, rewards, mask = _inputs(4, 9, seed=7)
    got, got_mean = _gpu_loss(lp, lp_old, lp_ref, rewards, 2, np.zeros_like(mask), 0.2, 0.28, 0.01)
    ref, _ = _oracle(lp, lp_old, lp_ref, rewards, 2, None, 0.2, 0.28, 0.01)
    np.testing.assert_allclose(got, ref, rtol=RTOL, atol=ATOL)
    assert got_mean == 0.0


def test_invalid_arguments_are_rejected():
    import torch
    qk = require_gpu()
    z = torch.zeros(6, 4, device="cuda")
    r = torch.zeros(6, device="cuda")
    ws = torch.empty(qk.qk_grpo_workspace_bytes(6), dtype=torch.uint8, device="cuda")
    with pytest.raises(qk.QKError):  # 6 rows are not whole groups of 4
        qk.qk_grpo_token_loss(z, z, z, 6, 4, 4, r, 4, None, 0.2, 0.28, 0.01, z, None, ws)
    with pytest.raises(qk.QKError):  # beta != 0 needs lp_ref
        qk.qk_grpo_token_loss(z, z, None, 6, 4, 4, r, 3, None, 0.2, 0.28, 0.01, z, None, ws)


@pytest.mark.parametrize("shape", ["tiny_fp32", "attn_bf16"])
def test_score_with_fused_loss(shape):
    import torch
    if shape == "tiny_fp32":
        s = synth.shape("tiny_fp32")
    else:
        s = synth.ModelShape("attn_bf16", 2, 512, 4, 2, 128, 256, 1024, "bf16")
    dec, W = decoder(s, synth.LazyWeights(s))
    B, T, group = 4, 41, 2
    toks = synth.tokens((B, T), s.vocab, stream=90)
    d = torch.tensor(toks, dtype=torch.int32, device="cuda")
    lp_plain = dec.score(d).cpu().numpy()
    rng = np.random.default_rng(3)
    lp_old = (lp_plain - rng.normal(0, 0.3, lp_plain.shape)).astype(np.float32)
    lp_ref = (lp_plain + rng.normal(0, 0.3, lp_plain.shape)).astype(np.float32)
    rewards = rng.random(B).astype(np.float32)
    mask = (rng.random(lp_plain.shape) > 0.3).astype(np.uint8)
    t = lambda a: torch.from_numpy(a).cuda()
    lp, loss, mean = dec.score_grpo(d, t(lp_old), t(rewards), group, lp_ref=t(lp_ref), mask=t(mask))
    assert dec.check_status() == 0
    lp = lp.cpu().numpy()
    loss = loss.cpu().numpy()
    # the fused epilogue computes the same log-probs as plain scoring ...
    assert np.array_equal(lp, lp_plain)
    # ... and the same token losses, bit for bit, as the standalone kernel on them
    sa, sa_mean = _gpu_loss(lp, lp_old, lp_ref, rewards, group, mask, 0.2, 0.28, 0.01)
    assert np.array_equal(loss, sa)
    assert float(mean.cpu().numpy()[0]) == sa_mean
    # end to end against the oracle's log-probs (scoring tolerance of each model)
    ref_lp = np.stack([oracle.token_logprobs(oracle.forward_logits(s, W, toks[b])[:-1], toks[b, 1:])
                       for b in range(B)])
    ref, ref_mean = _oracle(ref_lp, lp_old, lp_ref, rewards, group, mask, 0.2, 0.28, 0.01)
    lp_err = float(np.max(np.abs(lp - ref_lp)))
    # |dL/dlp| <= max(rho) |A| + beta |e^x - 1|, so the loss error follows the log-prob error
    rho = np.exp(ref_lp - lp_old)
    bound = (np.max(rho) * 1.0 + 0.01 * np.max(np.abs(np.exp(lp_ref - ref_lp) - 1)) + 1e-3) * lp_err
    assert np.max(np.abs(loss - ref)) <= 1.5 * bound + 1e-6
