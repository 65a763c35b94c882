"""Arg-max parity of the bf16 path where it can be decided: a two-layer decoder of
the Qwen3-8B layer width (H 4096, 32 / 8 heads, d 128, I 12288: the same GEMM
tiles and split-K schedules as the full model) with a 1,024-way vocabulary.

The logit tolerance is max(3e-2, 2 x F) x std, F the largest error of the
exact-bf16-rounding evaluation (about 0.03 x std here, most of it from the bf16
lm_head input), so a row is decisive when its top-2 gap exceeds about 0.65 x
std; over 512 distinct logits that holds on 8-13 % of the positions.  The exact
arg-max comparison of the bf16 decode path (fused split-K lm_head + cluster
reduce) and of the scoring path (tcgen05 lm_head + reduce) therefore has rows
to bite on, and each comparison requires at least 4 % of its rows decisive.

The lm_head repeats every even row in the odd row after it, so every logit
appears twice and every maximum is an exact tie between indices 2i and 2i + 1
(both sides compute the two logits identically).  The arg-max must then be the
lower index of the pair on every row, decisive or not: an arg-max that resolves
ties towards the higher index fails on every row.  The top-2 gap is taken over
the distinct (even) columns."""
import numpy as np
import pytest

import oracle
import synth
from _bf16_floor import forward_logits_bf16_activations
from _gpu import assert_argmax_where_gap, decoder

pytestmark = pytest.mark.gpu
SHAPE = synth.ModelShape("w8b_v1k", 2, 4096, 32, 8, 128, 12288, 1024, "bf16")
LOGIT_REL, LP_ABS = 3e-2, 5e-2
EVEN = np.arange(0, SHAPE.vocab, 2)


class PairedHead:
    """The seeded weights with lm_head row 2i + 1 replaced by row 2i."""

    def __init__(self, s):
        self.base = synth.LazyWeights(s, cache=True)
        self._lm = None

    def __getitem__(self, name):
        if name != "lm_head":
            return self.base[name]
        if self._lm is None:
            w = np.array(self.base["lm_head"])
            w[1::2] = w[0::2]
            self._lm = w
        return self._lm

    def __contains__(self, name):
        return name in self.base

    def keys(self):
        return self.base.keys()


@pytest.fixture(scope="module")
def model():
    W = PairedHead(SHAPE)
    dec, _ = decoder(SHAPE, W)
    return dec, W


def _tolerance(W, toks, decode_from):
    z = oracle.forward_logits(SHAPE, W, toks)
    zf = forward_logits_bf16_activations(SHAPE, W, toks, decode_from)
    rel = max(LOGIT_REL, 2 * np.abs(zf - z).max() / z.std())
    lpr = oracle.token_logprobs(z[:-1], toks[1:])
    lpf = oracle.token_logprobs(zf[:-1], toks[1:])
    return z, rel, max(LP_ABS, 2 * np.abs(lpf - lpr).max())


def test_oracle_ties_pairs_exactly(model):
    _, W = model
    toks = synth.tokens((6,), SHAPE.vocab, stream=90)
    z = oracle.forward_logits(SHAPE, W, toks)
    assert np.array_equal(z[:, 0::2], z[:, 1::2])
    assert np.all(oracle.argmax_lowest(z) % 2 == 0)


def test_decode_argmax_exact_where_decisive_and_ties_lowest(model):
    import torch
    dec, W = model
    B, P, N = 4, 16, 20
    seq = synth.tokens((B, P + N + 1), SHAPE.vocab, stream=91)
    kv = dec.new_kv(B, P + N)
    am = torch.empty(B, N + 1, dtype=torch.int32, device="cuda")
    lp = dec.rollout(kv, B, P + N, torch.tensor(seq, dtype=torch.int32, device="cuda"), P,
                     argmax=am).cpu().numpy()
    am = am.cpu().numpy()
    assert dec.check_status() == 0
    assert np.all(am % 2 == 0), "ties must resolve to the lowest index"
    decisive = 0
    for b in range(B):
        z, rel, lp_tol = _tolerance(W, seq[b, :P + N + 1], P)
        zr = z[P - 1:P + N]   # the prefill's last position, then the decode steps
        lp_ref = oracle.token_logprobs(zr, seq[b, P:P + N + 1])
        assert np.max(np.abs(lp[b] - lp_ref)) <= lp_tol
        decisive += assert_argmax_where_gap(am[b], zr, rel * np.std(zr), min_decisive=0,
                                            distinct=EVEN)
    assert decisive >= max(3, B * (N + 1) // 25), decisive


def test_score_argmax_exact_where_decisive_and_ties_lowest(model):
    import torch
    dec, W = model
    B, T = 3, 64
    toks = synth.tokens((B, T), SHAPE.vocab, stream=92)
    am = torch.empty(B, T - 1, dtype=torch.int32, device="cuda")
    lp = dec.score(torch.tensor(toks, dtype=torch.int32, device="cuda"), argmax=am).cpu().numpy()
    am = am.cpu().numpy()
    assert dec.check_status() == 0
    assert np.all(am % 2 == 0), "ties must resolve to the lowest index"
    decisive = 0
    for b in range(B):
        z, rel, lp_tol = _tolerance(W, toks[b], None)
        lp_ref = oracle.token_logprobs(z[:-1], toks[b, 1:])
        assert np.max(np.abs(lp[b] - lp_ref)) <= lp_tol
        decisive += assert_argmax_where_gap(am[b], z[:-1], rel * np.std(z[:-1]), min_decisive=0,
                                            distinct=EVEN)
    assert decisive >= B * (T - 1) // 25, decisive
