"""Pins for the backward oracle (oracle/backward.py) and the GRPO token-loss derivative.

* torch.autograd through a decoder assembled here from torch library routines
  (F.rms_norm, F.scaled_dot_product_attention, F.silu, F.cross_entropy, complex
  rotation for RoPE), in float64: every gradient tensor, element by element;
* central finite differences of the loss evaluated by the forward oracle
  (forward_logits / token_logprobs, a separate code path) on sampled coordinates
  of every tensor;
* the GRPO derivative against torch.autograd of Eq. ppo written with torch ops
  and against finite differences.
A dropped term, a wrong sign or index, or a transposed operand in the backward
oracle fails at least one of them (test_oracle_mutations plants such mistakes).
"""
from dataclasses import replace

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
import synth

CFG = replace(synth.shape("tiny_fp32"), n_layers=2, hidden=32, n_q_heads=4, n_kv_heads=2,
              head_dim=8, intermediate=48, vocab=40)


def _weights(cfg, seed=7):
    # weights large enough that every branch (attention, MLP, norms) moves the loss
    rng = np.random.default_rng(seed)
    W = {}
    for nm, shp, kind, _ in synth.tensor_list(cfg):
        if kind == "g":
            W[nm] = 1.0 + 0.2 * rng.standard_normal(shp)
        else:
            W[nm] = rng.standard_normal(shp) / np.sqrt(shp[-1])
    return W


def _case(seed=11, B=2, T=9):
    rng = np.random.default_rng(seed)
    tok = rng.integers(0, CFG.vocab, (B, T))
    tok[0, 3] = tok[0, 6] = tok[1, 2]  # a token repeated within and across rows
    mask = (rng.random((B, T - 1)) < 0.75).astype(np.float64)
    mask[:, 0] = 1.0
    return tok, mask


def _torch_loss(cfg, Wt, tok, coef):
    """Loss sum coef * (-log p) of a decoder written from torch library routines."""
    d, nq, nkv = cfg.head_dim, cfg.n_q_heads, cfg.n_kv_heads
    eps = cfg.rms_eps
    total = torch.zeros((), dtype=torch.float64)
    half = d // 2
    w = torch.tensor([cfg.rope_theta ** (-2.0 * i / d) for i in range(half)], dtype=torch.float64)
    for b in range(tok.shape[0]):
        ids = torch.tensor(tok[b])
        T = ids.shape[0]
        ang = torch.arange(T, dtype=torch.float64)[:, None, None] * w
        rot = torch.polar(torch.ones_like(ang), ang)

        def rope(x):
            z = torch.complex(x[..., :half], x[..., half:]) * rot
            return torch.cat([z.real, z.imag], dim=-1)

        x = F.embedding(ids, Wt["embed"])
        for L in range(cfg.n_layers):
            p = lambda nm: Wt[f"layers.{L}.{nm}"]
            u = F.rms_norm(x, (cfg.hidden,), p("attn_norm"), eps)
            q = F.linear(u, p("wq")).view(T, nq, d)
            k = F.linear(u, p("wk")).view(T, nkv, d)
            v = F.linear(u, p("wv")).view(T, nkv, d)
            q = rope(F.rms_norm(q, (d,), p("q_norm"), eps))
            k = rope(F.rms_norm(k, (d,), p("k_norm"), eps))
            rep = nq // nkv
            o = F.scaled_dot_product_attention(q.transpose(0, 1), k.repeat_interleave(rep, 1).transpose(0, 1),
                                               v.repeat_interleave(rep, 1).transpose(0, 1), is_causal=True)
            x = x + F.linear(o.transpose(0, 1).reshape(T, nq * d), p("wo"))
            u = F.rms_norm(x, (cfg.hidden,), p("mlp_norm"), eps)
            x = x + F.linear(F.silu(F.linear(u, p("wg"))) * F.linear(u, p("wu")), p("wd"))
        z = F.linear(F.rms_norm(x, (cfg.hidden,), Wt["final_norm"], eps), Wt["lm_head"])
        nll = F.cross_entropy(z[:-1], ids[1:], reduction="none")
        total = total + (torch.tensor(coef[b]) * nll).sum()
    return total


@pytest.mark.parametrize("weighting", ["sft_mean", "signed_coef"])
def test_backward_matches_torch_autograd(weighting):
    W = _weights(CFG)
    tok, mask = _case()
    if weighting == "sft_mean":
        coef = mask / mask.sum()
        loss, grads = oracle.sft_loss_and_grads(CFG, W, tok, mask, 1.0 / mask.sum())
    else:  # coefficients of both signs, as GRPO produces
        coef = np.random.default_rng(3).standard_normal(mask.shape) * mask
        loss, grads = oracle.policy_loss_and_grads(CFG, W, tok, coef)
    Wt = {k: torch.tensor(v, requires_grad=True) for k, v in W.items()}
    ref = _torch_loss(CFG, Wt, tok, coef)
    ref.backward()
    assert loss == pytest.approx(float(ref.detach()), rel=1e-12)
    for nm in W:
        g_ref = Wt[nm].grad.numpy()
        scale = np.max(np.abs(g_ref))
        assert scale > 0, nm
        err = np.max(np.abs(grads[nm] - g_ref))
        assert err <= 1e-10 * scale, f"{nm}: max err {err:.3e} vs max |g| {scale:.3e}"


def test_backward_matches_finite_differences():
    W = _weights(CFG, seed=5)
    tok, mask = _case(seed=13)
    scale = 1.0 / mask.sum()
    _, grads = oracle.sft_loss_and_grads(CFG, W, tok, mask, scale)
    rng = np.random.default_rng(17)
    h = 1e-5
    for nm in W:
        for _ in range(3):
            idx = tuple(int(rng.integers(0, n)) for n in W[nm].shape)
            if nm == "embed":  # a row that the sequences use
                idx = (int(tok[0, 3]), idx[1])
            keep = W[nm][idx]
            W[nm][idx] = keep + h
            lp = oracle.sft_loss(CFG, W, tok, mask, scale)
            W[nm][idx] = keep - h
            lm = oracle.sft_loss(CFG, W, tok, mask, scale)
            W[nm][idx] = keep
            fd = (lp - lm) / (2 * h)
            gmax = np.max(np.abs(grads[nm]))
            assert abs(grads[nm][idx] - fd) <= 1e-6 * gmax + 1e-9, (nm, idx, grads[nm][idx], fd)


def test_backward_zero_coefficients_and_single_token_rows():
    W = _weights(CFG)
    tok, mask = _case()
    loss, grads = oracle.policy_loss_and_grads(CFG, W, tok, np.zeros(mask.shape))
    assert loss == 0.0
    assert all(np.all(g == 0.0) for g in grads.values())
    # T = 2: one scored token per row; only the embedding rows of the two tokens move
    tok2 = tok[:, :2]
    loss, grads = oracle.sft_loss_and_grads(CFG, W, tok2)
    used = set(tok2.reshape(-1).tolist())
    rows = np.nonzero(np.any(grads["embed"] != 0, axis=1))[0]
    assert set(rows.tolist()) <= used


def test_lm_head_gradient_rows_sum_to_zero_per_hidden_column():
    # d loss / d W_lm = sum_t c_t (softmax(z_t) - onehot_t) hn_t^T; each softmax row minus a
    # one-hot row sums to zero, so the gradient's columns sum to zero over the vocabulary
    W = _weights(CFG)
    tok, mask = _case()
    _, grads = oracle.sft_loss_and_grads(CFG, W, tok, mask, 1.0)
    s = grads["lm_head"].sum(axis=0)
    assert np.max(np.abs(s)) <= 1e-12 * np.max(np.abs(grads["lm_head"]))


def _grpo_inputs(seed=21):
    rng = np.random.default_rng(seed)
    B, T = 6, 5
    lp = -rng.random((B, T)) * 3
    lp_old = lp + rng.normal(0, 0.3, (B, T))  # ratios inside and outside the clip range
    lp_ref = lp + rng.normal(0, 0.3, (B, T))
    rewards = rng.integers(0, 2, B).astype(np.float64)
    rewards[0], rewards[1] = 1.0, 0.0
    adv = oracle.group_advantages(rewards, 3)
    return lp, lp_old, lp_ref, adv


@pytest.mark.parametrize("beta", [0.0, 0.04])
def test_grpo_token_grad_matches_autograd_and_finite_differences(beta):
    lp, lp_old, lp_ref, adv = _grpo_inputs()
    el, eh = 0.2, 0.28
    g = oracle.grpo_token_grad(lp, lp_old, lp_ref, adv, el, eh, beta)
    # torch autograd of Eq. ppo written with torch ops
    t = torch.tensor(lp, requires_grad=True)
    rho = torch.exp(t - torch.tensor(lp_old))
    A = torch.tensor(adv)[:, None]
    L = -torch.minimum(rho * A, torch.clamp(rho, 1 - el, 1 + eh) * A)
    x = torch.tensor(lp_ref) - t
    L = L + beta * (torch.exp(x) - x - 1)
    L.sum().backward()
    assert np.allclose(g, t.grad.numpy(), rtol=1e-12, atol=1e-14)
    # finite differences of the oracle's own token loss
    h = 1e-6
    fd = (oracle.grpo_token_loss(lp + h, lp_old, lp_ref, adv, el, eh, beta)
          - oracle.grpo_token_loss(lp - h, lp_old, lp_ref, adv, el, eh, beta)) / (2 * h)
    assert np.allclose(g, fd, rtol=1e-6, atol=1e-8)
    # both branches of the min occur, so the pin covers the clipped case
    rho_n = np.exp(lp - lp_old)
    assert np.any((rho_n > 1 + eh) | (rho_n < 1 - el)) and np.any(np.abs(g) > 0)


def test_grpo_coef_is_the_gradient_of_the_masked_mean():
    lp, lp_old, lp_ref, adv = _grpo_inputs(seed=4)
    mask = (np.random.default_rng(2).random(lp.shape) < 0.7).astype(np.float64)
    c = oracle.grpo_coef(lp, lp_old, lp_ref, adv, 0.2, 0.28, 0.04, mask)
    h = 1e-6
    rng = np.random.default_rng(9)
    for _ in range(6):
        i = (int(rng.integers(0, lp.shape[0])), int(rng.integers(0, lp.shape[1])))
        a, b = lp.copy(), lp.copy()
        a[i] += h
        b[i] -= h
        f = lambda v: oracle.grpo_loss_mean(oracle.grpo_token_loss(v, lp_old, lp_ref, adv, 0.2, 0.28, 0.04), mask)
        # d mean / d lp_i = -c_i (the coefficient multiplies -lp)
        assert -c[i] == pytest.approx((f(a) - f(b)) / (2 * h), rel=1e-6, abs=1e-10)
    assert np.all(oracle.grpo_coef(lp, lp_old, lp_ref, adv, 0.2, 0.28, 0.04, np.zeros(lp.shape)) == 0)
