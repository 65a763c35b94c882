"""GPU parity on the full 36-layer Qwen3-8B-shaped bf16 model (random init).

Teacher-forced rollout and scoring at reduced lengths are compared position by
position with the fp64 oracle.  Tolerance: max |logit error| <= max(3e-2 x
std(logits), 2 x F_z) and |log-prob error| <= max(5e-2, 2 x F_lp), where F_z,
F_lp are the errors of an exact bf16-rounding evaluation of the same positions
(tests/_bf16_floor.py) that rounds where the path under test stores bf16: the
decode path's points for the rollout's decode steps, the prefill path's for its
prompt and for scoring.  On 36 random-init layers that floor is above the fixed
3e-2 x std bound (about 0.16 x std): no implementation that stores its
activations and KV cache in bf16 meets the fixed bound there, so the bound is
widened to the floor.  Arg-max is exact where the oracle's top-2 gap exceeds
10x the logit tolerance; at this tolerance over a 151,936-way vocabulary
almost no row is that decisive, so the non-vacuous bf16 arg-max check is the
narrower-vocabulary model of test_gpu_argmax.py."""
import numpy as np
import pytest

import oracle
import synth
from _bf16_floor import forward_logits_bf16_activations
from _gpu import assert_argmax_where_gap, assert_logits_close, decoder

pytestmark = pytest.mark.gpu
LOGIT_REL, LP_ABS = 3e-2, 5e-2


@pytest.fixture(scope="module")
def q8b():
    s = synth.shape("q8b")
    dec, W = decoder(s)
    return s, W, dec


@pytest.fixture(scope="module")
def short_case(q8b):
    s, W, _ = q8b
    B, P, N = 2, 24, 8
    seq = synth.tokens((B, P + N + 1), s.vocab, stream=5)
    z = np.stack([oracle.forward_logits(s, W, seq[b, :P + N]) for b in range(B)])
    lpr = np.stack([oracle.token_logprobs(z[b], seq[b, 1:]) for b in range(B)])

    def tolerances(decode_from, rows):
        """Tolerances from the floor of the path under test, over the compared rows."""
        zf = np.stack([forward_logits_bf16_activations(s, W, seq[b, :P + N], decode_from)
                       for b in range(B)])
        lpf = np.stack([oracle.token_logprobs(zf[b], seq[b, 1:]) for b in range(B)])
        floor_z = float(np.max(np.abs(zf[:, rows] - z[:, rows])))
        floor_lp = float(np.max(np.abs(lpf[:, rows] - lpr[:, rows])))
        rel = max(LOGIT_REL, 2 * floor_z / float(np.std(z[:, rows])))
        lp_abs = max(LP_ABS, 2 * floor_lp)
        print(f"bf16 floor (decode from {decode_from}): max |dz| {floor_z:.4f} "
              f"(std {np.std(z[:, rows]):.4f}), max |dlp| {floor_lp:.4f}; "
              f"tolerances {rel:.4f} x std, {lp_abs:.4f}")
        return rel, lp_abs

    roll = tolerances(P, slice(P - 1, P + N))   # prompt by prefill, then decode steps
    score = tolerances(None, slice(0, P + N))   # every position by the scoring path
    return seq, P, N, z, roll, score


def test_rollout_short_matches_oracle(q8b, short_case):
    import torch
    s, W, dec = q8b
    seq, P, N, z_all, (logit_rel, lp_abs), _ = short_case
    B = seq.shape[0]
    d = torch.tensor(seq, device="cuda", dtype=torch.int32)
    kv = dec.new_kv(B, P + N)
    logits = np.empty((B, N + 1, s.vocab))
    lp = np.empty((B, N + 1))
    am = np.empty((B, N + 1), dtype=np.int64)
    z0 = torch.empty(B, s.vocab, device="cuda")
    l0 = torch.empty(B, device="cuda")
    a0 = torch.empty(B, dtype=torch.int32, device="cuda")
    dec.prefill(kv, B, P + N, d[:, :P].contiguous(), 0, z0, d[:, P].contiguous(), l0, a0)
    logits[:, 0], lp[:, 0], am[:, 0] = z0.cpu().numpy(), l0.cpu().numpy(), a0.cpu().numpy()
    for j in range(N):
        pos = torch.full((B,), P + j, dtype=torch.int32, device="cuda")
        dec.decode_step(kv, B, P + N, d[:, P + j].contiguous(), pos, z0,
                        d[:, P + j + 1].contiguous(), l0, a0)
        logits[:, j + 1], lp[:, j + 1] = z0.cpu().numpy(), l0.cpu().numpy()
        am[:, j + 1] = a0.cpu().numpy()
    assert dec.check_status() == 0
    z_ref = z_all[:, P - 1:P + N]
    err, tol = assert_logits_close(logits, z_ref, logit_rel)
    lp_ref = np.stack([oracle.token_logprobs(z_ref[b], seq[b, P:P + N + 1]) for b in range(B)])
    assert np.max(np.abs(lp - lp_ref)) <= lp_abs
    assert_argmax_where_gap(am.reshape(-1), z_ref.reshape(-1, s.vocab), tol, min_decisive=0)
    # the rollout entry point gives the same numbers as the step-by-step calls
    kv2 = dec.new_kv(B, P + N)
    lp2 = dec.rollout(kv2, B, P + N, d, P).cpu().numpy()
    assert np.array_equal(lp2, lp.astype(np.float32))


def test_score_short_matches_oracle(q8b, short_case):
    import torch
    s, W, dec = q8b
    seq, P, N, z_all, _, (logit_rel, lp_abs) = short_case
    B, T = seq.shape[0], P + N + 1
    am = torch.empty(B, T - 1, dtype=torch.int32, device="cuda")
    lp = dec.score(torch.tensor(seq, device="cuda", dtype=torch.int32), argmax=am).cpu().numpy()
    assert dec.check_status() == 0
    lp_ref = np.stack([oracle.token_logprobs(z_all[b], seq[b, 1:]) for b in range(B)])
    assert np.max(np.abs(lp - lp_ref)) <= lp_abs
    tol = logit_rel * np.std(z_all)
    assert_argmax_where_gap(am.cpu().numpy().reshape(-1), z_all.reshape(-1, s.vocab), tol,
                            min_decisive=0)
