"""GPU parity on the tiny fp32 decoder (2 layers, H 256, 4/2 heads, d 64, I 768,
V 4096): batch 4, prompt 64, 16 teacher-forced decode steps; logits and log-probs
against the fp64 oracle at 1e-4 (the paper's fp32 checker tolerance, Sec. 3.1)."""
import numpy as np
import pytest

import oracle
import synth
from _gpu import assert_argmax_where_gap, assert_logits_close, decoder, require_gpu

pytestmark = pytest.mark.gpu
REL = 1e-4


@pytest.fixture(scope="module")
def tiny():
    s = synth.shape("tiny_fp32")
    dec, W = decoder(s, synth.LazyWeights(s))
    return s, W, dec


@pytest.fixture(scope="module")
def rollout_ref(tiny):
    s, W, _ = tiny
    B, P, N = 4, 64, 16
    seq = synth.tokens((B, P + N + 1), s.vocab)
    zs, lps = [], []
    for b in range(B):
        z, lp = oracle.rollout_teacher_forced(s, W, seq[b], P)
        zs.append(z)
        lps.append(lp)
    return seq, P, N, np.stack(zs), np.stack(lps)


def _run_steps(dec, seq, P, N):
    import torch
    B = seq.shape[0]
    V = dec.cfg.vocab
    d = torch.tensor(seq, device="cuda", dtype=torch.int32)
    kv = dec.new_kv(B, P + N)
    logits = torch.empty(B, N + 1, V, device="cuda")
    lp = torch.empty(B, N + 1, device="cuda")
    am = torch.empty(B, N + 1, dtype=torch.int32, device="cuda")
    z0 = torch.empty(B, V, device="cuda")
    l0 = torch.empty(B, device="cuda")
    a0 = torch.empty(B, dtype=torch.int32, device="cuda")
    dec.prefill(kv, B, P + N, d[:, :P].contiguous(), 0, z0, d[:, P].contiguous(), l0, a0)
    logits[:, 0], lp[:, 0], am[:, 0] = z0, l0, a0
    for j in range(N):
        pos = torch.full((B,), P + j, dtype=torch.int32, device="cuda")
        dec.decode_step(kv, B, P + N, d[:, P + j].contiguous(), pos, z0, d[:, P + j + 1].contiguous(),
                        l0, a0)
        logits[:, j + 1], lp[:, j + 1], am[:, j + 1] = z0, l0, a0
    assert dec.check_status() == 0
    return logits.cpu().numpy(), lp.cpu().numpy(), am.cpu().numpy(), kv


def test_prefill_and_decode_steps_match_oracle(tiny, rollout_ref):
    s, W, dec = tiny
    seq, P, N, z_ref, lp_ref = rollout_ref
    z, lp, am, _ = _run_steps(dec, seq, P, N)
    err, tol = assert_logits_close(z, z_ref, REL)
    assert np.all(np.abs(lp - lp_ref) <= REL * np.maximum(1.0, np.abs(lp_ref)))
    # at 1e-4 x std nearly every row of an fp32 model is decisive
    assert_argmax_where_gap(am.reshape(-1), z_ref.reshape(-1, s.vocab), tol,
                            min_decisive=int(0.9 * am.size))


def test_rollout_entry_point_equals_step_by_step(tiny, rollout_ref):
    import torch
    s, W, dec = tiny
    seq, P, N, z_ref, lp_ref = rollout_ref
    _, lp_steps, am_steps, _ = _run_steps(dec, seq, P, N)
    B = seq.shape[0]
    kv = dec.new_kv(B, P + N)
    am = torch.empty(B, N + 1, dtype=torch.int32, device="cuda")
    lp = dec.rollout(kv, B, P + N, torch.tensor(seq, device="cuda", dtype=torch.int32), P, argmax=am)
    assert dec.check_status() == 0
    assert np.array_equal(lp.cpu().numpy(), lp_steps)
    assert np.array_equal(am.cpu().numpy(), am_steps)


def test_kv_cache_contents_match_oracle(tiny, rollout_ref):
    s, W, dec = tiny
    seq, P, N, _, _ = rollout_ref
    _, _, _, kv = _run_steps(dec, seq, P, N)
    view = dec.kv_view(kv, seq.shape[0], P + N).cpu().numpy()
    for b in (0, 3):
        ref = oracle.KVDecoder(s, W)
        ref.prefill(seq[b, :P + N])
        for layer in range(s.n_layers):
            k_ref = ref.k[layer].transpose(1, 0, 2)  # [nkv, S, d]
            v_ref = ref.v[layer].transpose(1, 0, 2)
            assert np.max(np.abs(view[layer, 0, b] - k_ref)) <= 1e-4 * max(1.0, np.abs(k_ref).max())
            assert np.max(np.abs(view[layer, 1, b] - v_ref)) <= 1e-4 * max(1.0, np.abs(v_ref).max())


def test_score_logprobs_matches_oracle(tiny):
    import torch
    s, W, dec = tiny
    for B, T in ((4, 81), (3, 2), (1, 130)):
        toks = synth.tokens((B, T), s.vocab, stream=40 + T)
        am = torch.empty(B, T - 1, dtype=torch.int32, device="cuda")
        lp = dec.score(torch.tensor(toks, device="cuda", dtype=torch.int32), argmax=am).cpu().numpy()
        assert dec.check_status() == 0
        for b in range(B):
            lp_ref, am_ref, gap = oracle.score_sequence(s, W, toks[b])
            assert np.all(np.abs(lp[b] - lp_ref) <= REL * np.maximum(1.0, np.abs(lp_ref)))
            z = oracle.forward_logits(s, W, toks[b])[:-1]
            assert_argmax_where_gap(am[b].cpu().numpy(), z, REL * np.std(z),
                                    min_decisive=int(0.9 * (T - 1)))


def test_ragged_positions_in_one_decode_step(tiny):
    """Rows at different positions share one decode step (row b at pos[b])."""
    import torch
    s, W, dec = tiny
    B, S = 3, 40
    lens = [5, 17, 33]
    seqs = synth.tokens((B, S), s.vocab, stream=60)
    kv = dec.new_kv(B, S)
    dt = torch.tensor(seqs, device="cuda", dtype=torch.int32)
    # prefill each row separately to its own length (rows share the cache buffer)
    for b, L in enumerate(lens):
        sub = dec.kv_view(kv, B, S)
        tmp = dec.new_kv(1, S)
        dec.prefill(tmp, 1, S, dt[b:b + 1, :L].contiguous())
        sub[:, :, b] = dec.kv_view(tmp, 1, S)[:, :, 0]
    pos = torch.tensor(lens, dtype=torch.int32, device="cuda")
    toks = torch.tensor([seqs[b, L] for b, L in enumerate(lens)], dtype=torch.int32, device="cuda")
    z = torch.empty(B, s.vocab, device="cuda")
    dec.decode_step(kv, B, S, toks, pos, z)
    assert dec.check_status() == 0
    for b, L in enumerate(lens):
        z_ref = oracle.forward_logits(s, W, seqs[b, :L + 1])[-1]
        assert_logits_close(z[b].cpu().numpy(), z_ref, REL)


def test_bad_token_sets_status_and_is_clamped(tiny):
    import torch
    s, W, dec = tiny
    kv = dec.new_kv(1, 8)
    toks = torch.tensor([[1, 2, s.vocab + 5]], dtype=torch.int32, device="cuda")
    dec.prefill(kv, 1, 8, toks)
    import paper_2609_12471_gb300 as qk
    assert dec.check_status() & qk.QK_STATUS_BAD_TOKEN
    assert dec.check_status() == 0  # cleared by the read


def test_bad_position_sets_status(tiny):
    import torch
    s, W, dec = tiny
    kv = dec.new_kv(2, 8)
    dec.prefill(kv, 2, 8, torch.ones(2, 4, dtype=torch.int32, device="cuda"))
    pos = torch.tensor([4, 9], dtype=torch.int32, device="cuda")
    dec.decode_step(kv, 2, 8, torch.ones(2, dtype=torch.int32, device="cuda"), pos)
    import paper_2609_12471_gb300 as qk
    assert dec.check_status() & qk.QK_STATUS_BAD_POS


def test_rollout_inside_caller_graph_capture(tiny):
    """Inside a caller's own stream capture the rollout launches its steps directly
    (no nested capture); replaying the caller's graph gives the direct call's numbers."""
    import torch
    s, W, dec = tiny
    B, P, N = 2, 16, 6
    seq = torch.tensor(synth.tokens((B, P + N + 1), s.vocab, stream=80), dtype=torch.int32,
                       device="cuda")
    kv = dec.new_kv(B, P + N)
    ref = dec.rollout(kv, B, P + N, seq, P).clone()
    out = torch.empty(B, N + 1, device="cuda")
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        dec.rollout(kv, B, P + N, seq, P, logprobs=out)  # warm the workspace outside capture
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side, capture_error_mode="thread_local"):
            dec.rollout(kv, B, P + N, seq, P, logprobs=out)
    torch.cuda.current_stream().wait_stream(side)
    out.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert dec.check_status() == 0
    assert torch.equal(out, ref)
