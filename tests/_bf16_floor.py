"""bf16 noise floor: the decoder evaluated with exact bf16 rounding (round to
nearest even) at the points where the bf16 GPU path stores an activation, and
float64 everywhere else.

Test infrastructure only.  It is built from the oracle's own functions; the
only difference from oracle.forward_logits is where values are rounded.  The
two GPU paths round at different points, and each is modelled:

* prefill / scoring (tokens at positions < decode_from): the RMSNorm'd input
  u = bf16(RMSNorm(x) g) of every linear layer, the q/k/v projections, q and k
  after QK-norm + RoPE (the bf16 KV cache), the attention output and the
  SwiGLU output;
* decode steps (positions >= decode_from): the norm is split around the
  linear, so the stored input is bf16(x g) and the RMSNorm scale s =
  rsqrt(mean(x^2) + eps) multiplies the fp32 product afterwards (W (x g s) =
  s W (x g)); q, k and v are not stored before QK-norm + RoPE (the fused
  epilogue works on the fp32 accumulator), so only the rotated q and k and the
  scaled v are rounded; then the attention output, bf16(x g_mlp) before
  gate/up, the SwiGLU output, and bf16(x g_final) before the lm_head.

The distance between this and the float64 oracle is the error any
implementation that stores those activations in bf16 carries; the GPU path is
judged against a multiple of it on the 36-layer model, where the fixed 3e-2 x
std bound is below that floor.
"""
import numpy as np

import oracle


def bf16_round(x) -> np.ndarray:
    f = np.asarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    r = (((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16).astype(np.uint32)
    return r.view(np.float32).astype(np.float64)


def _rms_scale(x, eps):
    return 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)


def forward_logits_bf16_activations(cfg, W, tokens, decode_from=None) -> np.ndarray:
    """Logits [T, V] with bf16 rounding at the prefill path's storage points for
    positions < decode_from and at the decode path's for the rest (decode_from
    None: every position as prefill / scoring)."""
    tokens = np.asarray(tokens)
    T = len(tokens)
    pos = np.arange(T)
    dec = (pos >= (T if decode_from is None else decode_from))[:, None]  # decode-path rows
    eps, nq, nkv, d = cfg.rms_eps, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim
    r = bf16_round

    def pick(a_prefill, a_decode):
        if not dec.any():
            return a_prefill
        m = dec.reshape((T,) + (1,) * (a_prefill.ndim - 1))
        return np.where(m, a_decode, a_prefill)

    def linear_in(x, g, Wt):
        """Normed input times W^T as each path forms it."""
        pre = r(oracle.rms_norm(x, g, eps)) @ Wt
        if not dec.any():
            return pre
        return pick(pre, (r(x * g) @ Wt) * _rms_scale(x, eps))

    x = oracle.embed(W, tokens)
    for layer in range(cfg.n_layers):
        Lw = oracle.layer_weights(W, layer)
        q_raw = linear_in(x, Lw["attn_norm"], Lw["wq"].T)
        k_raw = linear_in(x, Lw["attn_norm"], Lw["wk"].T)
        v_raw = linear_in(x, Lw["attn_norm"], Lw["wv"].T)
        q_in = pick(r(q_raw), q_raw).reshape(T, nq, d)   # the prefill path stores raw q, k, v
        k_in = pick(r(k_raw), k_raw).reshape(T, nkv, d)
        v = r(v_raw).reshape(T, nkv, d)
        q = r(oracle.apply_rope(oracle.rms_norm(q_in, Lw["q_norm"], eps), pos, cfg.rope_theta))
        k = r(oracle.apply_rope(oracle.rms_norm(k_in, Lw["k_norm"], eps), pos, cfg.rope_theta))
        o = r(oracle.attention(q, k, v, pos, pos).reshape(T, nq * d))
        x = x + o @ Lw["wo"].T
        g = linear_in(x, Lw["mlp_norm"], Lw["wg"].T)
        u = linear_in(x, Lw["mlp_norm"], Lw["wu"].T)
        x = x + r(oracle.silu(g) * u) @ Lw["wd"].T
    h = oracle.final_hidden(cfg, W, x)
    z = oracle.lm_logits(W, r(h))
    if dec.any():
        gf = oracle.widen(W["final_norm"])
        z = pick(z, oracle.lm_logits(W, r(x * gf)) * _rms_scale(x, eps))
    return z
