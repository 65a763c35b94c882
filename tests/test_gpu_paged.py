"""Paged KV cache.  The rollouts of one batch and their appended turns end at
different lengths (Sec. "Multi-Turn On-Policy Reflection"); a paged cache lets
rows take pages from one pool instead of reserving max_seq positions each.

The multi-turn sequence of the dense-cache test (prompts of different lengths,
decode steps at per-row positions, feedback appended at each row's own position)
runs over a pool whose pages a shuffled table hands out, several pages per row and
spare pages left over.  The same kernels read the same keys from other addresses,
so every logit must equal the dense cache's bit for bit; the last logits are also
checked against the fp64 oracle.  Further cases: a prompt prefix written once into
a page that two rows share, a bad page id (status bit, no fault: the entry reads
page 0), and the host-side argument checks."""
import numpy as np
import pytest

import oracle
import synth
from _bf16_floor import forward_logits_bf16_activations
from _gpu import assert_logits_close, decoder

pytestmark = pytest.mark.gpu

PAGE = 128


def _cu(a):
    import torch
    return torch.tensor(np.ascontiguousarray(a), dtype=torch.int32, device="cuda")


def _turns(s, lens1, lens3, steps, T1, T3, seed_stream, prefill, decode):
    """Turn 1 prefill, `steps` decode steps, turn 3 append; returns the logits of each
    call (turn 1, every decode step, turn 3) and the row sequences."""
    import torch
    B = len(lens1)
    V = s.vocab
    toks1 = synth.tokens((B, T1), V, stream=seed_stream)
    dec_toks = synth.tokens((B, steps), V, stream=seed_stream + 1)
    toks3 = synth.tokens((B, T3), V, stream=seed_stream + 2)
    out = []
    z = torch.empty(B, V, device="cuda")
    prefill(_cu(toks1), _cu(np.zeros(B)), _cu(lens1), z)
    out.append(z.cpu().numpy())
    pos = np.array(lens1)
    for j in range(steps):
        z = torch.empty(B, V, device="cuda")
        decode(_cu(dec_toks[:, j]), _cu(pos), z)
        out.append(z.cpu().numpy())
        pos = pos + 1
    z = torch.empty(B, V, device="cuda")
    prefill(_cu(toks3), _cu(pos), _cu(lens3), z)
    out.append(z.cpu().numpy())
    seqs = [np.concatenate([toks1[b, :lens1[b]], dec_toks[b], toks3[b, :lens3[b]]]) for b in range(B)]
    return out, seqs


def _dense_and_paged(s, dec, lens1, lens3, steps, T1, T3, seed_stream):
    B = len(lens1)
    longest = max(l1 + steps + T3 for l1 in lens1)
    per_row = -(-longest // PAGE)
    max_seq = per_row * PAGE  # the dense cache holds as many positions per row as the paged one
    kv = dec.new_kv(B, max_seq)
    dense, seqs = _turns(
        s, lens1, lens3, steps, T1, T3, seed_stream,
        lambda t, st, ln, z: dec.prefill_rows(kv, B, max_seq, t, st, ln, z),
        lambda t, p, z: dec.decode_step(kv, B, max_seq, t, p, z))
    assert dec.check_status() == 0
    del kv
    # a pool with spare pages; each row's pages scattered over it in shuffled order
    n_pages = B * per_row + 5
    rng = np.random.default_rng(seed_stream)
    table = rng.permutation(n_pages)[:B * per_row].reshape(B, per_row).astype(np.int32)
    pool = dec.new_kv_pages(n_pages, PAGE)
    pool.fill_(0xFF)  # NaN patterns in every unwritten position (bf16 and fp32)
    tab = _cu(table)
    paged, _ = _turns(
        s, lens1, lens3, steps, T1, T3, seed_stream,
        lambda t, st, ln, z: dec.prefill_rows_paged(pool, tab, n_pages, PAGE, t, st, ln, z),
        lambda t, p, z: dec.decode_step_paged(pool, tab, n_pages, PAGE, t, p, z))
    assert dec.check_status() == 0
    return dense, paged, seqs, per_row


def test_paged_equals_dense_fp32():
    s = synth.shape("tiny_fp32")
    dec, W = decoder(s, synth.LazyWeights(s))
    # the first row's prompt crosses into its second page
    dense, paged, seqs, per_row = _dense_and_paged(s, dec, lens1=[140, 17, 5], lens3=[4, 9, 6], steps=3,
                                                   T1=140, T3=9, seed_stream=400)
    assert per_row == 2
    for i, (zd, zp) in enumerate(zip(dense, paged)):
        assert np.array_equal(zd, zp), f"call {i}: paged logits differ from the dense cache's"
    for b, seq in enumerate(seqs):
        assert_logits_close(paged[-1][b], oracle.forward_logits(s, W, seq)[-1], 1e-4)


def test_paged_equals_dense_bf16():
    """The tensor-core prefill attention (128-key tiles, one page each) and the split
    decode attention (64-key tiles) over pages."""
    s = synth.ModelShape("attn_bf16", 2, 512, 4, 2, 128, 256, 1024, "bf16")
    dec, W = decoder(s, synth.LazyWeights(s))
    dense, paged, seqs, per_row = _dense_and_paged(s, dec, lens1=[70, 130, 9], lens3=[66, 3, 20], steps=2,
                                                   T1=130, T3=66, seed_stream=410)
    assert per_row == 2
    for i, (zd, zp) in enumerate(zip(dense, paged)):
        assert np.array_equal(zd, zp), f"call {i}: paged logits differ from the dense cache's"
    for b, seq in enumerate(seqs):
        z = oracle.forward_logits(s, W, seq)
        zf = forward_logits_bf16_activations(s, W, seq)
        rel = max(3e-2, 2 * float(np.abs(zf[-1] - z[-1]).max() / z[-1].std()))
        assert_logits_close(paged[-1][b], z[-1], rel)


def test_shared_prefix_page_bf16():
    """Two rows share the page holding a common 128-token prompt, written once through
    row 0; each row then appends its own continuation into a page of its own."""
    import torch
    s = synth.ModelShape("attn_bf16", 2, 512, 4, 2, 128, 256, 1024, "bf16")
    dec, W = decoder(s, synth.LazyWeights(s))
    V = s.vocab
    prefix = synth.tokens((1, PAGE), V, stream=420)
    cont = synth.tokens((2, 12), V, stream=421)
    lens = [12, 7]
    n_pages = 6
    table = _cu(np.array([[4, 1], [4, 3]]))  # page 4 shared; pages 1 and 3 private
    pool = dec.new_kv_pages(n_pages, PAGE)
    pool.fill_(0xFF)
    dec.prefill_rows_paged(pool, table[:1], n_pages, PAGE, _cu(prefix), _cu([0]), None, None)
    z = torch.empty(2, V, device="cuda")
    dec.prefill_rows_paged(pool, table, n_pages, PAGE, _cu(cont), _cu([PAGE, PAGE]), _cu(lens), z)
    assert dec.check_status() == 0
    z = z.cpu().numpy()
    for b in range(2):
        seq = np.concatenate([prefix[0], cont[b, :lens[b]]])
        ref = oracle.forward_logits(s, W, seq)
        zf = forward_logits_bf16_activations(s, W, seq)
        rel = max(3e-2, 2 * float(np.abs(zf[-1] - ref[-1]).max() / ref[-1].std()))
        assert_logits_close(z[b], ref[-1], rel)


def test_bad_page_id_sets_the_status_bit():
    import torch
    import paper_2609_12471_gb300 as qk
    s = synth.shape("tiny_fp32")
    dec, _ = decoder(s, synth.LazyWeights(s))
    n_pages = 4
    pool = dec.new_kv_pages(n_pages, PAGE)
    pool.zero_()
    toks = _cu(synth.tokens((2, 8), s.vocab, stream=430))
    good = _cu(np.array([[0, 1], [2, 3]]))
    dec.prefill_rows_paged(pool, good, n_pages, PAGE, toks, _cu([0, 0]), None, None)
    assert dec.check_status() == 0
    # row 1's first page id is out of the pool (-1 and n_pages + 5 alike): page 0 is used
    for badid in (-1, n_pages + 5):
        bad = _cu(np.array([[0, 1], [badid, 3]]))
        z = torch.empty(2, s.vocab, device="cuda")
        dec.decode_step_paged(pool, bad, n_pages, PAGE, toks[:, 0].contiguous(), _cu([8, 8]), z)
        assert dec.check_status() & qk.QK_STATUS_BAD_PAGE
        assert np.isfinite(z.cpu().numpy()).all()


def test_paged_arguments_are_checked_on_the_host():
    import paper_2609_12471_gb300 as qk
    s = synth.shape("tiny_fp32")
    dec, _ = decoder(s, synth.LazyWeights(s))
    pool = dec.new_kv_pages(4, PAGE)
    toks = _cu([[1], [2]])
    pos = _cu([0, 0])
    tab = _cu(np.array([[0, 1], [2, 3]]))
    h = dec.handle

    def code(**kw):  # a one-byte workspace: the valid call stops at QK_ENOSPACE
        a = dict(kv=pool, table=tab, per_row=2, n_pages=4, page_size=PAGE)
        a.update(kw)
        with pytest.raises(qk.QKError) as e:
            qk.qk_decode_step_paged(h, a["kv"], a["table"], a["per_row"], a["n_pages"], a["page_size"],
                                    toks, pos, 2, workspace=pool, ws_bytes=1, stream=0)
        return e.value.code

    assert code(table=None) == qk.QK_EINVAL
    assert code(kv=None) == qk.QK_EINVAL
    assert code(page_size=100) == qk.QK_ESHAPE          # not a multiple of 128
    assert code(n_pages=0) == qk.QK_ESHAPE
    assert code(per_row=10 ** 6) == qk.QK_ESHAPE        # more positions than the RoPE table
    assert code() == qk.QK_ENOSPACE                     # valid arguments, workspace too small
    with pytest.raises(qk.QKError) as e:
        qk.qk_kv_pages_bytes(h, 4, 96)
    assert e.value.code == qk.QK_ESHAPE
    assert qk.qk_kv_pages_bytes(h, 4, PAGE) == qk.qk_kv_bytes(h, 4, PAGE)


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_paged_rollouts_equal_dense(dtype):
    """Whole rollouts (the prompt prefill, then decode steps replayed from a captured
    graph) over a paged cache: the teacher-forced log-probs and arg-maxes, and at a
    fixed seed the sampled tokens and their log-probs, bit-identical to the dense
    cache's.  P + N crosses into each row's second page."""
    import torch
    if dtype == "fp32":
        s = synth.shape("tiny_fp32")
    else:
        s = synth.ModelShape("attn_bf16", 2, 512, 4, 2, 128, 256, 1024, "bf16")
    dec, _ = decoder(s, synth.LazyWeights(s))
    B, P, N, per_row = 6, 70, 80, 2
    max_seq = per_row * PAGE
    seq = _cu(synth.tokens((B, P + N + 1), s.vocab, stream=440))
    prompt = seq[:, :P].contiguous()
    kv = dec.new_kv(B, max_seq)
    am_d = torch.empty(B, N + 1, dtype=torch.int32, device="cuda")
    lp_d = dec.rollout(kv, B, max_seq, seq, P, argmax=am_d)
    tok_d, slp_d = dec.rollout_sampled(kv, B, max_seq, prompt, N, tau=1.0, seed=7)
    assert dec.check_status() == 0
    del kv
    n_pages = B * per_row + 3
    rng = np.random.default_rng(441)
    tab = _cu(rng.permutation(n_pages)[:B * per_row].reshape(B, per_row))
    pool = dec.new_kv_pages(n_pages, PAGE)
    pool.fill_(0xFF)
    am_p = torch.empty(B, N + 1, dtype=torch.int32, device="cuda")
    lp_p = dec.rollout_paged(pool, tab, n_pages, PAGE, seq, P, argmax=am_p)
    tok_p, slp_p = dec.rollout_sampled_paged(pool, tab, n_pages, PAGE, prompt, N, tau=1.0, seed=7)
    assert dec.check_status() == 0
    assert torch.equal(lp_d, lp_p) and torch.equal(am_d, am_p)
    assert torch.equal(tok_d, tok_p) and torch.equal(slp_d, slp_p)
    assert bool(torch.isfinite(lp_p).all()) and bool(torch.isfinite(slp_p).all())
