"""Pins for the fp64 oracle: each check ties it to something other than itself.

Properties and closed forms (RoPE preserves norms, softmax rows sum to one,
attention over one key returns that key's value, exp(log-softmax) sums to
one, uniform logits give -log V, RMSNorm gives unit RMS), independent library
routines (torch's rms_norm, scaled_dot_product_attention, log_softmax, silu,
complex-number rotation), a scalar brute force of a one-layer two-token model,
and the equality of two code paths (full causal forward and incremental KV
decode).  A dropped term, a wrong sign or index or a transposed operand in the
oracle fails at least one of them.
"""
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
CF = json.load(open(os.path.join(GOLDEN, "closed_forms.json")))
rng = np.random.default_rng(1234)


# ---------------------------------------------------------------- RoPE

def test_rope_preserves_norm_and_identity_at_zero():
    x = rng.standard_normal((7, 3, 64))
    pos = np.array([0, 1, 2, 100, 1000, 4095, 8191])
    y = oracle.apply_rope(x, pos, 1e6)
    assert np.allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-13)
    y0 = oracle.apply_rope(x[:1], [0], 1e6)
    assert np.array_equal(y0, x[:1])


def test_rope_relative_position():
    q = rng.standard_normal((1, 1, 128))
    k = rng.standard_normal((1, 1, 128))
    def dot(pq, pk):
        return float(np.sum(oracle.apply_rope(q, [pq], 1e6) * oracle.apply_rope(k, [pk], 1e6)))
    assert dot(10, 3) == pytest.approx(dot(1007, 1000), rel=1e-10, abs=1e-10)
    assert dot(5000, 5000) == pytest.approx(dot(0, 0), rel=1e-10, abs=1e-10)


def test_rope_matches_complex_rotation():
    # Pair (x_i, x_{i+d/2}) as the complex number x_i + j x_{i+d/2}, multiply by
    # exp(j p w_i) with w_i = theta^(-2i/d), computed through torch.polar.
    d = 64
    x = rng.standard_normal((5, 2, d))
    pos = np.array([0, 3, 77, 2048, 8000])
    xt = torch.tensor(x)
    z = torch.complex(xt[..., : d // 2], xt[..., d // 2:])
    w = torch.tensor([1e6 ** (-2.0 * i / d) for i in range(d // 2)], dtype=torch.float64)
    ang = torch.tensor(pos, dtype=torch.float64)[:, None, None] * w
    r = z * torch.polar(torch.ones_like(ang), ang)
    ref = torch.cat([r.real, r.imag], dim=-1).numpy()
    assert np.allclose(oracle.apply_rope(x, pos, 1e6), ref, rtol=1e-12, atol=1e-12)


def test_rope_inverse_frequency_closed_form():
    g = CF["rope_theta"]
    a64 = oracle.rope_angles([1], 64, g["theta"])[0]
    a128 = oracle.rope_angles([1], 128, g["theta"])[0]
    assert a64[0] == 1.0 and a128[0] == 1.0
    assert a64[-1] == pytest.approx(g["inv_freq_last_d64"], rel=1e-12)
    assert a128[-1] == pytest.approx(g["inv_freq_last_d128"], rel=1e-12)


# ---------------------------------------------------------------- softmax / log-softmax

def test_softmax_rows_sum_to_one_and_shift_invariance():
    s = rng.standard_normal((9, 33)) * 5
    p = oracle.softmax(s)
    assert np.allclose(p.sum(-1), 1.0, rtol=0, atol=1e-14)
    assert np.allclose(oracle.softmax(s + 123.0), p, atol=1e-14)
    assert np.allclose(p, torch.softmax(torch.tensor(s), -1).numpy(), atol=1e-15)


def test_log_softmax_normalised_and_uniform_closed_form():
    z = rng.standard_normal((4, 1000)) * 3
    lp = oracle.log_softmax(z)
    assert np.allclose(np.exp(lp).sum(-1), 1.0, atol=1e-13)
    assert np.allclose(lp, torch.log_softmax(torch.tensor(z), -1).numpy(), atol=1e-13)
    for V in (4096, 151936):
        u = oracle.log_softmax(np.full((1, V), 0.37))
        assert u[0, 0] == pytest.approx(CF["uniform_log_softmax"][str(V)], abs=1e-12)
        assert np.allclose(u, u[0, 0])


def test_token_logprobs_argmax_and_gap():
    z = np.array([[0.0, 2.0, 2.0, -1.0], [5.0, 1.0, 4.5, 5.0]])
    assert list(oracle.argmax_lowest(z)) == [1, 0]  # ties -> lowest index
    assert np.allclose(oracle.top2_gap(z), [0.0, 0.0])
    lp = oracle.token_logprobs(z, [3, 2])
    ref = [-1 - math.log(1 + 2 * math.e ** 2 + math.e ** -1),
           4.5 - math.log(2 * math.e ** 5 + math.e + math.e ** 4.5)]
    assert np.allclose(lp, ref, atol=1e-13)


# ---------------------------------------------------------------- RMSNorm / SiLU

def test_rms_norm_unit_rms_scale_invariance_and_torch():
    x = rng.standard_normal((6, 256)) * 7
    y = oracle.rms_norm(x, np.ones(256), 0.0)
    assert np.allclose(np.sqrt(np.mean(y * y, -1)), 1.0, atol=1e-14)
    assert np.allclose(oracle.rms_norm(3.5 * x, np.ones(256), 0.0), y, atol=1e-14)
    g = 1 + 0.02 * rng.standard_normal(256)
    ref = F.rms_norm(torch.tensor(x), (256,), torch.tensor(g), eps=1e-6).numpy()
    assert np.allclose(oracle.rms_norm(x, g, 1e-6), ref, atol=1e-13)
    # eps sits inside the square root: a zero row stays zero, a tiny row is damped
    t = np.full((1, 4), 1e-4)
    assert oracle.rms_norm(t, np.ones(4), 1e-6)[0, 0] == pytest.approx(1e-4 / math.sqrt(1e-8 + 1e-6))


def test_silu_special_cases():
    assert oracle.silu(np.array([0.0]))[0] == 0.0
    assert oracle.silu(np.array([40.0]))[0] == pytest.approx(40.0, rel=1e-15)
    assert abs(oracle.silu(np.array([-800.0]))[0]) < 1e-300
    z = rng.standard_normal(100) * 4
    assert np.allclose(oracle.silu(z), F.silu(torch.tensor(z)).numpy(), atol=1e-15)


# ---------------------------------------------------------------- attention

def test_attention_single_key_returns_value():
    q = rng.standard_normal((1, 4, 64))
    k = rng.standard_normal((1, 2, 64))
    v = rng.standard_normal((1, 2, 64))
    o = oracle.attention(q, k, v, [0], [0])
    assert np.array_equal(o[0, 0], v[0, 0]) and np.array_equal(o[0, 1], v[0, 0])
    assert np.array_equal(o[0, 2], v[0, 1]) and np.array_equal(o[0, 3], v[0, 1])


def test_attention_equal_keys_give_mean_value():
    q = rng.standard_normal((1, 2, 16))
    k = np.repeat(rng.standard_normal((1, 1, 16)), 9, axis=0)
    v = rng.standard_normal((9, 1, 16))
    o = oracle.attention(q, k, v, [8], np.arange(9))
    assert np.allclose(o[0, 0], v[:, 0].mean(0), atol=1e-14)


def test_attention_matches_torch_sdpa_gqa_causal():
    T, nq, nkv, d = 13, 8, 2, 32
    q = rng.standard_normal((T, nq, d))
    k = rng.standard_normal((T, nkv, d))
    v = rng.standard_normal((T, nkv, d))
    o = oracle.attention(q, k, v, np.arange(T), np.arange(T))
    qt = torch.tensor(q).permute(1, 0, 2)
    kt = torch.tensor(k).permute(1, 0, 2).repeat_interleave(nq // nkv, dim=0)
    vt = torch.tensor(v).permute(1, 0, 2).repeat_interleave(nq // nkv, dim=0)
    ref = F.scaled_dot_product_attention(qt, kt, vt, is_causal=True).permute(1, 0, 2).numpy()
    assert np.allclose(o, ref, atol=1e-13)


def test_gqa_with_equal_heads_is_mha():
    T, n, d = 6, 4, 16
    q = rng.standard_normal((T, n, d))
    k = rng.standard_normal((T, n, d))
    v = rng.standard_normal((T, n, d))
    o = oracle.attention(q, k, v, np.arange(T), np.arange(T))
    for h in range(n):
        s = q[:, h] @ k[:, h].T / math.sqrt(d)
        s[np.triu_indices(T, 1)] = -np.inf
        p = np.exp(s - s.max(-1, keepdims=True))
        p /= p.sum(-1, keepdims=True)
        assert np.allclose(o[:, h], p @ v[:, h], atol=1e-14)


# ---------------------------------------------------------------- whole forward

def _torch_forward_logits(cfg, W, tokens):
    """The same decoder assembled from torch library routines (float64, CPU)."""
    def t(name):
        return torch.tensor(oracle.widen(W[name]))
    T = len(tokens)
    nq, nkv, d, H = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.hidden
    x = t("embed")[torch.tensor(tokens, dtype=torch.long)]
    w = torch.tensor([cfg.rope_theta ** (-2.0 * i / d) for i in range(d // 2)], dtype=torch.float64)
    ang = torch.arange(T, dtype=torch.float64)[:, None, None] * w
    rot = torch.polar(torch.ones_like(ang), ang)

    def rope(y):
        z = torch.complex(y[..., : d // 2], y[..., d // 2:]) * rot
        return torch.cat([z.real, z.imag], -1)
    for layer in range(cfg.n_layers):
        p = f"layers.{layer}."
        u = F.rms_norm(x, (H,), t(p + "attn_norm"), eps=cfg.rms_eps)
        q = F.linear(u, t(p + "wq")).view(T, nq, d)
        k = F.linear(u, t(p + "wk")).view(T, nkv, d)
        v = F.linear(u, t(p + "wv")).view(T, nkv, d)
        q = rope(F.rms_norm(q, (d,), t(p + "q_norm"), eps=cfg.rms_eps))
        k = rope(F.rms_norm(k, (d,), t(p + "k_norm"), eps=cfg.rms_eps))
        rep = nq // nkv
        o = F.scaled_dot_product_attention(
            q.permute(1, 0, 2), k.permute(1, 0, 2).repeat_interleave(rep, 0),
            v.permute(1, 0, 2).repeat_interleave(rep, 0), is_causal=True)
        x = x + F.linear(o.permute(1, 0, 2).reshape(T, nq * d), t(p + "wo"))
        u = F.rms_norm(x, (H,), t(p + "mlp_norm"), eps=cfg.rms_eps)
        x = x + F.linear(F.silu(F.linear(u, t(p + "wg"))) * F.linear(u, t(p + "wu")), t(p + "wd"))
    hn = F.rms_norm(x, (H,), t("final_norm"), eps=cfg.rms_eps)
    return F.linear(hn, t("lm_head")).numpy()


def test_forward_matches_torch_library_decoder(tiny_shape, tiny_weights):
    toks = synth.tokens((40,), tiny_shape.vocab, stream=11)
    z = oracle.forward_logits(tiny_shape, tiny_weights, toks)
    ref = _torch_forward_logits(tiny_shape, tiny_weights, toks)
    assert np.abs(z - ref).max() < 1e-11 * max(1.0, np.abs(ref).max())


def test_incremental_decode_equals_full_forward(tiny_shape, tiny_weights):
    seq = synth.tokens((4, 81), tiny_shape.vocab)[2]
    z_full = oracle.forward_logits(tiny_shape, tiny_weights, seq[:80])
    z_roll, lp = oracle.rollout_teacher_forced(tiny_shape, tiny_weights, seq, 64)
    assert z_roll.shape == (17, tiny_shape.vocab)
    assert np.abs(z_roll - z_full[63:80]).max() < 1e-12
    lp_s, am, gap = oracle.score_sequence(tiny_shape, tiny_weights, seq)
    assert np.allclose(lp, lp_s[63:80], atol=1e-12)
    assert np.array_equal(am, oracle.argmax_lowest(oracle.forward_logits(tiny_shape, tiny_weights, seq)[:-1]))


def test_causality_prefix_independence(tiny_shape, tiny_weights):
    a = synth.tokens((30,), tiny_shape.vocab, stream=21)
    b = a.copy()
    b[17:] = synth.tokens((13,), tiny_shape.vocab, stream=22)
    za = oracle.forward_logits(tiny_shape, tiny_weights, a)
    zb = oracle.forward_logits(tiny_shape, tiny_weights, b)
    assert np.array_equal(za[:17], zb[:17])
    assert np.abs(za[17:] - zb[17:]).max() > 1e-3


def test_layer_decode_step_matches_incremental_decoder(tiny_shape, tiny_weights):
    # The one-layer workload routine, checked against KVDecoder's cache on a
    # one-layer model: same new residual, same appended key and value.
    one = synth.shape("tiny_fp32", n_layers=1)
    W = synth.LazyWeights(one)
    toks = synth.tokens((12,), one.vocab, stream=31)
    dec = oracle.KVDecoder(one, W)
    dec.prefill(toks[:11])
    k_cache = dec.k[0].transpose(1, 0, 2)[None]
    v_cache = dec.v[0].transpose(1, 0, 2)[None]
    x = oracle.embed(W, toks[11:12])
    out, kn, vn = oracle.layer_decode_step(one, oracle.layer_weights(W, 0), x, k_cache, v_cache, [11])
    xo, kr, vr = oracle.decoder_layer(one, oracle.layer_weights(W, 0), x, [11], dec.k[0], dec.v[0],
                                      np.arange(11))
    assert np.allclose(out, xo, atol=1e-13)
    dec.step(toks[11])
    assert np.allclose(kn[0], dec.k[0][11], atol=1e-13) and np.allclose(vn[0], dec.v[0][11], atol=1e-13)


def test_brute_force_one_layer_two_tokens():
    """A scalar, loop-by-loop evaluation of a micro one-layer model, two tokens."""
    cfg = synth.ModelShape("micro", 1, 8, 2, 1, 4, 6, 10, "f32")
    W = synth.LazyWeights(cfg, seed=77)
    tokens = [3, 7]
    eps, theta = cfg.rms_eps, cfg.rope_theta

    def m(name):
        return oracle.widen(W[name]).tolist()

    def norm(vec, g):
        r = math.sqrt(sum(a * a for a in vec) / len(vec) + eps)
        return [a / r * gi for a, gi in zip(vec, g)]

    def matvec(Wm, vec):
        return [sum(Wm[o][i] * vec[i] for i in range(len(vec))) for o in range(len(Wm))]

    def rot(vec, p):
        half = len(vec) // 2
        out = list(vec)
        for i in range(half):
            a = p * theta ** (-2.0 * i / len(vec))
            out[i] = vec[i] * math.cos(a) - vec[i + half] * math.sin(a)
            out[i + half] = vec[i + half] * math.cos(a) + vec[i] * math.sin(a)
        return out

    E = m("embed")
    xs = [list(E[t]) for t in tokens]
    ks, vs, qs = [], [], []
    for p, x in enumerate(xs):
        u = norm(x, m("layers.0.attn_norm"))
        q = matvec(m("layers.0.wq"), u)
        k = matvec(m("layers.0.wk"), u)
        v = matvec(m("layers.0.wv"), u)
        qh = [rot(norm(q[h * 4:(h + 1) * 4], m("layers.0.q_norm")), p) for h in range(2)]
        ks.append(rot(norm(k, m("layers.0.k_norm")), p))
        vs.append(v)
        qs.append(qh)
    logits = []
    for p, x in enumerate(xs):
        o = []
        for h in range(2):  # both q heads read the single kv head
            sc = [sum(a * b for a, b in zip(qs[p][h], ks[j])) / 2.0 for j in range(p + 1)]
            mx = max(sc)
            e = [math.exp(s - mx) for s in sc]
            o += [sum(e[j] * vs[j][c] for j in range(p + 1)) / sum(e) for c in range(4)]
        x = [a + b for a, b in zip(x, matvec(m("layers.0.wo"), o))]
        u = norm(x, m("layers.0.mlp_norm"))
        gt = matvec(m("layers.0.wg"), u)
        up = matvec(m("layers.0.wu"), u)
        hh = [g / (1 + math.exp(-g)) * w for g, w in zip(gt, up)]
        x = [a + b for a, b in zip(x, matvec(m("layers.0.wd"), hh))]
        logits.append(matvec(m("lm_head"), norm(x, m("final_norm"))))
    z = oracle.forward_logits(cfg, W, tokens)
    assert np.allclose(z, np.array(logits), atol=1e-13)


def test_layer_decode_step_batched_rows_match_per_row_layers(tiny_shape, tiny_weights):
    # Rows with different cache lengths; each must equal decoder_layer on that row alone.
    Lw = oracle.layer_weights(tiny_weights, 1)
    r = np.random.default_rng(5)
    B, S = 3, 20
    kc = r.standard_normal((B, tiny_shape.n_kv_heads, S, tiny_shape.head_dim))
    vc = r.standard_normal((B, tiny_shape.n_kv_heads, S, tiny_shape.head_dim))
    x = r.standard_normal((B, tiny_shape.hidden))
    pos = [19, 0, 7]
    out, kn, vn = oracle.layer_decode_step(tiny_shape, Lw, x, kc, vc, pos)
    for b in range(B):
        p = pos[b]
        xo, k1, v1 = oracle.decoder_layer(tiny_shape, Lw, x[b:b + 1], [p],
                                          kc[b, :, :p].transpose(1, 0, 2),
                                          vc[b, :, :p].transpose(1, 0, 2), np.arange(p))
        assert np.allclose(out[b], xo[0], atol=1e-12)
        assert np.allclose(kn[b], k1[0], atol=1e-13) and np.allclose(vn[b], v1[0], atol=1e-13)
