"""Multi-turn appends at per-row positions (Sec. "Multi-Turn On-Policy
Reflection": each rollout's feedback turn is appended to its own history, so the
rows of one batch sit at different positions).  Turn 1 prefills prompts of
different lengths (padded to a common T), a few decode steps follow at per-row
positions, turn 3 appends feedback of different lengths at each row's own
position; the logits after each row's last token are compared with the fp64
oracle's incremental decoder fed the same tokens.  A second bf16 model covers
the tensor-core prefill attention with per-row start positions."""
import numpy as np
import pytest

import oracle
import synth
from _bf16_floor import forward_logits_bf16_activations
from _gpu import assert_logits_close, decoder

pytestmark = pytest.mark.gpu


def _run(s, W, dec, rel, lens1, lens3, steps, T1, T3, seed_stream):
    import torch
    B = len(lens1)
    max_seq = max(l1 + steps + T3 for l1 in lens1) + 4
    kv = dec.new_kv(B, max_seq)
    toks1 = synth.tokens((B, T1), s.vocab, stream=seed_stream)
    dec_toks = synth.tokens((B, steps), s.vocab, stream=seed_stream + 1)
    toks3 = synth.tokens((B, T3), s.vocab, stream=seed_stream + 2)
    cu = lambda a: torch.tensor(np.ascontiguousarray(a), dtype=torch.int32, device="cuda")
    V = s.vocab
    # turn 1: prompts of different lengths, all starting at position 0
    z1 = torch.empty(B, V, device="cuda")
    dec.prefill_rows(kv, B, max_seq, cu(toks1), cu(np.zeros(B)), cu(lens1), z1)
    # turn 2: decode steps, each row at its own position
    pos = np.array(lens1)
    for j in range(steps):
        zd = torch.empty(B, V, device="cuda")
        dec.decode_step(kv, B, max_seq, cu(dec_toks[:, j]), cu(pos), zd)
        pos = pos + 1
    # turn 3: feedback of different lengths appended at each row's position
    z3 = torch.empty(B, V, device="cuda")
    dec.prefill_rows(kv, B, max_seq, cu(toks3), cu(pos), cu(lens3), z3)
    assert dec.check_status() == 0
    z1, z3 = z1.cpu().numpy(), z3.cpu().numpy()
    for b in range(B):
        seq = np.concatenate([toks1[b, :lens1[b]], dec_toks[b], toks3[b, :lens3[b]]])
        ref = oracle.forward_logits(s, W, seq)
        n1 = lens1[b]
        tol1, tol3 = rel(W, seq, n1 - 1), rel(W, seq, len(seq) - 1)
        assert_logits_close(z1[b], ref[n1 - 1], tol1)
        assert_logits_close(z3[b], ref[-1], tol3)


def test_multiturn_rows_at_different_positions_fp32():
    s = synth.shape("tiny_fp32")
    dec, W = decoder(s, synth.LazyWeights(s))
    _run(s, W, dec, lambda W, seq, i: 1e-4, lens1=[10, 17, 5], lens3=[4, 9, 6], steps=3, T1=17,
         T3=9, seed_stream=300)


def test_multiturn_rows_at_different_positions_bf16():
    s = synth.ModelShape("attn_bf16", 2, 512, 4, 2, 128, 256, 1024, "bf16")
    dec, W = decoder(s, synth.LazyWeights(s))

    def rel(W, seq, i):  # the bf16 rule of the attention tests: max(3e-2, 2 x the bf16 floor)
        z = oracle.forward_logits(s, W, seq)[i]
        zf = forward_logits_bf16_activations(s, W, seq)[i]
        return max(3e-2, 2 * float(np.abs(zf - z).max() / z.std()))

    # prompts longer than one 64-query tile, so the tensor-core prefill attention
    # runs several query tiles per row with per-row start positions
    _run(s, W, dec, rel, lens1=[70, 130, 9], lens3=[66, 3, 20], steps=2, T1=130, T3=66,
         seed_stream=310)
