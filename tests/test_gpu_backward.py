"""GPU parity of the backward pass (qk_backward_logprob) and of the GRPO gradient
coefficients (qk_grpo_coef) against the fp64 oracle (oracle/backward.py, oracle/grpo.py).

* tiny fp32 decoder (CUDA-core GEMMs, the same orchestration, epilogue and row
  kernels as the bf16 path): every gradient tensor element by element at 2e-4 of
  the tensor's largest entry, on ragged sequence lengths (37: one partial 64-tile;
  130: three tiles and a 2-row tail);
* bf16 decoders (tcgen05 GEMMs with K- and MN-major operands): a two-layer model
  (also on ragged rows of 200 positions, padded inside the call)
  and one layer at Qwen3-8B width (H 4096, 32/8 heads, I 12288; vocabulary 16384) over
  2 x 256 tokens (two causal tiles per row),
  per-tensor relative Frobenius error within the bf16 bound, and the loss;
* the GRPO coefficients element by element, and the GRPO gradient end to end.
"""
import numpy as np
import pytest

import oracle
import synth
from _gpu import decoder, require_gpu

pytestmark = pytest.mark.gpu
REL_F32 = 2e-4
# bf16 path: activations, attention probabilities and the logit / attention / residual
# gradients that feed the tensor cores are rounded to bf16 (relative 2^-9 each); a
# gradient sums such products over tokens, so its relative error is a few times 2^-9
# per rounding stage on its path (about ten stages for the first layer's tensors).
REL_BF16 = 3e-2


def _names(s):
    return [t[0] for t in synth.tensor_list(s)]


def _run(dec, tok, coef, accumulate=False, grads=None):
    import torch
    t = torch.tensor(tok, dtype=torch.int32, device="cuda")
    c = torch.tensor(coef, dtype=torch.float32, device="cuda")
    if grads is None:
        grads = dec.new_grads()
    loss = dec.backward(t, c, grads, accumulate=accumulate)
    torch.cuda.synchronize()
    assert dec.check_status() == 0
    return grads, float(loss.item())


def _coef_sft(rng, B, T):
    mask = (rng.random((B, T - 1)) < 0.8).astype(np.float64)
    mask[:, 0] = 1.0
    return mask / mask.sum()


@pytest.fixture(scope="module")
def tiny():
    s = synth.shape("tiny_fp32")
    W = synth.LazyWeights(s)
    dec, _ = decoder(s, W)
    return s, W, dec


@pytest.mark.parametrize("B,T", [(2, 37), (1, 130)])
def test_tiny_fp32_gradients_match_oracle(tiny, B, T):
    s, W, dec = tiny
    rng = np.random.default_rng(T)
    tok = synth.tokens((B, T), s.vocab, stream=40 + T)
    tok[0, 5] = tok[0, 9] = tok[-1, 2]  # repeated tokens: the embedding gradient adds them
    coef = _coef_sft(rng, B, T)
    grads, loss = _run(dec, tok, coef)
    loss_ref, ref = oracle.policy_loss_and_grads(s, W, tok, coef)
    assert loss == pytest.approx(loss_ref, rel=1e-5)
    for nm, g in zip(_names(s), grads):
        g = g.cpu().numpy().astype(np.float64)
        r = ref[nm]
        scale = float(np.max(np.abs(r)))
        assert scale > 0, nm
        err = float(np.max(np.abs(g - r)))
        assert err <= REL_F32 * scale, f"{nm}: max err {err:.3e} > {REL_F32} x {scale:.3e}"
    # accumulate = 1 adds the same gradient again
    first = [g.clone() for g in grads]
    grads, _ = _run(dec, tok, coef, accumulate=True, grads=grads)
    for nm, a, g in zip(_names(s), first, grads):
        a = a.cpu().numpy()
        assert np.allclose(g.cpu().numpy(), 2 * a, rtol=1e-6, atol=1e-7 * np.max(np.abs(a))), nm


def test_tiny_fp32_signed_coefficients_and_zero_rows(tiny):
    s, W, dec = tiny
    B, T = 3, 21
    rng = np.random.default_rng(5)
    tok = synth.tokens((B, T), s.vocab, stream=61)
    coef = rng.standard_normal((B, T - 1)) * 0.05
    coef[1] = 0.0  # a row that contributes nothing
    grads, loss = _run(dec, tok, coef)
    loss_ref, ref = oracle.policy_loss_and_grads(s, W, tok, coef)
    assert loss == pytest.approx(loss_ref, rel=1e-5, abs=1e-6)
    for nm, g in zip(_names(s), grads):
        g = g.cpu().numpy().astype(np.float64)
        scale = float(np.max(np.abs(ref[nm])))
        assert float(np.max(np.abs(g - ref[nm]))) <= REL_F32 * scale, nm


def _rel_fro(g, r):
    return float(np.linalg.norm(g - r) / np.linalg.norm(r))


def _check_bf16(s, W, dec, B, T, stream, rel=REL_BF16):
    rng = np.random.default_rng(stream)
    tok = synth.tokens((B, T), s.vocab, stream=stream)
    coef = _coef_sft(rng, B, T)
    grads, loss = _run(dec, tok, coef)
    loss_ref, ref = oracle.policy_loss_and_grads(s, W, tok, coef)
    assert loss == pytest.approx(loss_ref, rel=5e-3)
    worst = {}
    for nm, g in zip(_names(s), grads):
        g = g.cpu().numpy().astype(np.float64)
        worst[nm] = _rel_fro(g, ref[nm])
    bad = {k: v for k, v in worst.items() if not v <= rel}
    assert not bad, f"relative Frobenius error above {rel}: {bad}"
    return worst


def test_bf16_two_layer_gradients_match_oracle():
    s = synth.ModelShape("bwd_bf16", 2, 512, 4, 2, 128, 256, 1024, "bf16")
    W = synth.LazyWeights(s)
    dec, _ = decoder(s, W)
    worst = _check_bf16(s, W, dec, 2, 256, 71)
    dec.close()
    print("bf16 two-layer relative Frobenius errors:", {k: f"{v:.2e}" for k, v in worst.items()})


def test_bf16_ragged_rows_match_oracle():
    """T = 200 (one full 128-position tile and a 72-position tail): the call pads the rows to
    256 positions internally; gradients and loss are those of the unpadded rows."""
    s = synth.ModelShape("bwd_bf16", 2, 512, 4, 2, 128, 256, 1024, "bf16")
    W = synth.LazyWeights(s)
    dec, _ = decoder(s, W)
    worst = _check_bf16(s, W, dec, 2, 200, 74)
    dec.close()
    print("bf16 ragged (T 200) relative Frobenius errors:", {k: f"{v:.2e}" for k, v in worst.items()})


def test_bf16_q8b_width_layer_gradients_match_oracle():
    s = synth.ModelShape("q8b_width", 1, 4096, 32, 8, 128, 12288, 16384, "bf16")
    W = synth.LazyWeights(s)
    dec, _ = decoder(s, W)
    worst = _check_bf16(s, W, dec, 2, 256, 72)
    dec.close()
    print("bf16 8B-width layer relative Frobenius errors:", {k: f"{v:.2e}" for k, v in worst.items()})


def _grpo_case(rng, B, T):
    lp = -rng.random((B, T)) * 4
    # ratios well inside and well outside the clip band [0.8, 1.28]
    lp_old = lp + rng.choice([-0.5, -0.1, 0.1, 0.5], size=(B, T))
    lp_ref = lp + rng.normal(0, 0.3, (B, T))
    rewards = rng.integers(0, 2, B).astype(np.float64)
    mask = (rng.random((B, T)) < 0.7).astype(np.uint8)
    return lp, lp_old, lp_ref, rewards, mask


def test_grpo_coefficients_match_oracle():
    qk = require_gpu()
    import torch
    rng = np.random.default_rng(3)
    B, T, ld, G = 8, 50, 53, 4
    lp, lp_old, lp_ref, rewards, mask = _grpo_case(rng, B, T)
    pad = lambda a, dt=torch.float32: torch.tensor(np.pad(a, ((0, 0), (0, ld - T))), dtype=dt, device="cuda")
    coef = torch.zeros(B, ld, device="cuda")
    loss_tok = torch.zeros(B, ld, device="cuda")
    loss_mean = torch.zeros(1, device="cuda")
    ws = torch.empty(qk.qk_grpo_workspace_bytes(B), dtype=torch.uint8, device="cuda")
    qk.qk_grpo_coef(pad(lp), pad(lp_old), pad(lp_ref), B, T, ld, torch.tensor(rewards, dtype=torch.float32,
                    device="cuda"), G, pad(mask, torch.uint8), 0.2, 0.28, 0.04, coef, loss_tok, loss_mean, ws)
    torch.cuda.synchronize()
    adv = oracle.group_advantages(rewards, G)
    c_ref = oracle.grpo_coef(lp, lp_old, lp_ref, adv, 0.2, 0.28, 0.04, mask)
    got = coef.cpu().numpy()[:, :T]
    assert np.allclose(got, c_ref, rtol=1e-5, atol=1e-7 * np.max(np.abs(c_ref)))
    assert np.count_nonzero(c_ref) > B * T // 4  # both branches and masked tokens occur
    L = oracle.grpo_loss_mean(oracle.grpo_token_loss(lp, lp_old, lp_ref, adv, 0.2, 0.28, 0.04), mask)
    assert float(loss_mean.item()) == pytest.approx(L, rel=1e-5, abs=1e-7)


def test_grpo_gradient_end_to_end(tiny):
    """Score -> GRPO coefficients -> backward on the GPU equals the oracle's gradient of
    the GRPO loss mean (Eq. ppo through the log-probs)."""
    qk = require_gpu()
    import torch
    s, W, dec = tiny
    B, T, G = 4, 24, 2
    rng = np.random.default_rng(8)
    tok = synth.tokens((B, T), s.vocab, stream=81)
    lp_o = np.stack([oracle.token_logprobs(oracle.forward_logits(s, W, tok[b])[:-1], tok[b, 1:])
                     for b in range(B)])
    lp_old = lp_o + rng.choice([-0.5, -0.1, 0.1, 0.5], size=lp_o.shape)
    lp_ref = lp_o + rng.normal(0, 0.2, lp_o.shape)
    rewards = np.array([1.0, 0.0, 0.0, 1.0])
    dv = lambda a: torch.tensor(a, dtype=torch.float32, device="cuda")
    td = torch.tensor(tok, dtype=torch.int32, device="cuda")
    lp = dec.score(td)
    coef = torch.empty(B, T - 1, device="cuda")
    loss_tok = torch.empty(B, T - 1, device="cuda")
    ws = torch.empty(qk.qk_grpo_workspace_bytes(B), dtype=torch.uint8, device="cuda")
    qk.qk_grpo_coef(lp, dv(lp_old), dv(lp_ref), B, T - 1, T - 1, dv(rewards), G, None, 0.2, 0.28, 0.04,
                    coef, loss_tok, None, ws)
    grads = dec.new_grads()
    dec.backward(td, coef, grads)
    torch.cuda.synchronize()
    adv = oracle.group_advantages(rewards, G)
    c_ref = oracle.grpo_coef(lp_o, lp_old, lp_ref, adv, 0.2, 0.28, 0.04)
    _, ref = oracle.policy_loss_and_grads(s, W, tok, c_ref)
    for nm, g in zip(_names(s), grads):
        g = g.cpu().numpy().astype(np.float64)
        scale = float(np.max(np.abs(ref[nm])))
        assert float(np.max(np.abs(g - ref[nm]))) <= 1e-3 * scale, nm


def test_bf16_q8b_width_layer_4096_tokens_against_scoring():
    """One 8B-width layer over 1 x 4096 tokens (32 causal tiles per row, dW reductions over
    4096 tokens): the loss the backward forms equals the scoring path's mean -log p, the
    gradients are finite, and the lm_head gradient's columns sum to ~0 over the vocabulary."""
    import torch
    s = synth.ModelShape("q8b_width", 1, 4096, 32, 8, 128, 12288, 16384, "bf16")
    dec, _ = decoder(s, synth.LazyWeights(s, cache=False))
    B, T = 1, 4096
    tok = torch.tensor(synth.tokens((B, T), s.vocab, stream=73), dtype=torch.int32, device="cuda")
    coef = torch.full((B, T - 1), 1.0 / (T - 1), device="cuda")
    ref = float(-dec.score(tok).double().mean())
    grads = dec.new_grads()
    loss = float(dec.backward(tok, coef, grads).item())
    torch.cuda.synchronize()
    assert dec.check_status() == 0
    assert loss == pytest.approx(ref, abs=2e-3)
    assert all(bool(torch.isfinite(g).all()) for g in grads)
    col = grads[-1].double().sum(0).abs().max().item()
    assert col <= 1e-2 * grads[-1].double().abs().sum(0).max().item()
    dec.close()
