"""Attention parity on a small bf16 decoder with head_dim 128 (the tensor-core
attention kernels' shape): 2 layers, H 512, 4 query / 2 kv heads, I 256, V 1024.

Covers the causal prefill / scoring kernel over several 64-query tiles with a
ragged tail, chunked prefill (a second prefill starting at position 70 on top
of the cache of the first), and a decode step after prefill; logits and
log-probs against the fp64 oracle with the tolerance rule of the bf16 tests
(max(3e-2 x std, 2 x the exact-bf16-rounding floor))."""
import numpy as np
import pytest

import oracle
import synth
from _bf16_floor import forward_logits_bf16_activations
from _gpu import assert_argmax_where_gap, assert_logits_close, decoder

pytestmark = pytest.mark.gpu
SHAPE = synth.ModelShape("attn_bf16", 2, 512, 4, 2, 128, 256, 1024, "bf16")


@pytest.fixture(scope="module")
def model():
    dec, W = decoder(SHAPE, synth.LazyWeights(SHAPE))
    return dec, W


def _tol(W, toks):
    z = oracle.forward_logits(SHAPE, W, toks)
    zf = forward_logits_bf16_activations(SHAPE, W, toks)
    floor = np.abs(zf - z).max() / z.std()
    lpr = oracle.token_logprobs(z[:-1], toks[1:])
    lpf = oracle.token_logprobs(zf[:-1], toks[1:])
    return z, max(3e-2, 2 * floor), max(5e-2, 2 * np.abs(lpf - lpr).max())


def test_score_several_query_tiles_ragged_tail(model):
    import torch
    dec, W = model
    B, T = 3, 200
    toks = synth.tokens((B, T), SHAPE.vocab, stream=71)
    am = torch.empty(B, T - 1, dtype=torch.int32, device="cuda")
    lp = dec.score(torch.tensor(toks, dtype=torch.int32, device="cuda"), argmax=am).cpu().numpy()
    am = am.cpu().numpy()
    assert dec.check_status() == 0
    for b in range(B):
        z, rel, lp_tol = _tol(W, toks[b])
        lp_ref = oracle.token_logprobs(z[:-1], toks[b, 1:])
        assert np.max(np.abs(lp[b] - lp_ref)) <= lp_tol
        # a 1,024-way vocabulary: about a third of the rows clear 10 x 3e-2 x std
        assert_argmax_where_gap(am[b], z[:-1], rel * np.std(z[:-1]), min_decisive=(T - 1) // 10)


def test_chunked_prefill_then_decode(model):
    import torch
    dec, W = model
    B, T1, T2 = 2, 70, 130
    S = T1 + T2 + 1
    toks = synth.tokens((B, S), SHAPE.vocab, stream=72)
    d = torch.tensor(toks, dtype=torch.int32, device="cuda")
    kv = dec.new_kv(B, S)
    z1 = torch.empty(B, SHAPE.vocab, device="cuda")
    dec.prefill(kv, B, S, d[:, :T1].contiguous(), 0, z1)
    dec.prefill(kv, B, S, d[:, T1:T1 + T2].contiguous(), T1, z1)
    z2 = torch.empty(B, SHAPE.vocab, device="cuda")
    pos = torch.full((B,), T1 + T2, dtype=torch.int32, device="cuda")
    dec.decode_step(kv, B, S, d[:, T1 + T2].contiguous(), pos, z2)
    assert dec.check_status() == 0
    for b in range(B):
        z, rel, _ = _tol(W, toks[b])
        assert_logits_close(z1[b].cpu().numpy(), z[T1 + T2 - 1], rel)
        assert_logits_close(z2[b].cpu().numpy(), z[T1 + T2], rel)


def test_rollout_split_k_batch6_matches_oracle(model):
    """Batch 6 takes the split-K decode path (partials summed by the next norm / QK-norm /
    SwiGLU) with graph-replayed steps; compared per position with the oracle."""
    import torch
    dec, W = model
    B, P, N = 6, 20, 12
    seq = synth.tokens((B, P + N + 1), SHAPE.vocab, stream=73)
    kv = dec.new_kv(B, P + N)
    am = torch.empty(B, N + 1, dtype=torch.int32, device="cuda")
    lp = dec.rollout(kv, B, P + N, torch.tensor(seq, dtype=torch.int32, device="cuda"), P,
                     argmax=am).cpu().numpy()
    assert dec.check_status() == 0
    for b in range(B):
        z, rel, lp_tol = _tol(W, seq[b, :P + N + 1])
        lp_ref = oracle.token_logprobs(z[P - 1:P + N], seq[b, P:P + N + 1])
        assert np.max(np.abs(lp[b] - lp_ref)) <= lp_tol
    # a second call with the same buffers replays the cached step graph: same numbers
    lp2 = dec.rollout(kv, B, P + N, torch.tensor(seq, dtype=torch.int32, device="cuda"),
                      P).cpu().numpy()
    assert np.array_equal(lp, lp2)
