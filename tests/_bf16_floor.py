"""bf16 noise floor: the decoder evaluated with exact bf16 rounding (round to
nearest even) at the points where the bf16 GPU path stores an activation, and
float64 everywhere else.

Test infrastructure only.  It is built from the oracle's own functions; the
only difference from oracle.forward_logits is the rounding applied to: the
RMSNorm'd input of every linear layer, the q/k/v projections, q and k after
QK-norm + RoPE (the bf16 KV cache), the attention output and the SwiGLU output.
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


def forward_logits_bf16_activations(cfg, W, tokens) -> np.ndarray:
    tokens = np.asarray(tokens)
    T = len(tokens)
    pos = np.arange(T)
    eps, nq, nkv, d = cfg.rms_eps, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim
    r = bf16_round
    x = oracle.embed(W, tokens)
    for layer in range(cfg.n_layers):
        Lw = oracle.layer_weights(W, layer)
        u = r(oracle.rms_norm(x, Lw["attn_norm"], eps))
        q = r(u @ Lw["wq"].T).reshape(T, nq, d)
        k = r(u @ Lw["wk"].T).reshape(T, nkv, d)
        v = r(u @ Lw["wv"].T).reshape(T, nkv, d)
        q = r(oracle.apply_rope(oracle.rms_norm(q, Lw["q_norm"], eps), pos, cfg.rope_theta))
        k = r(oracle.apply_rope(oracle.rms_norm(k, Lw["k_norm"], eps), pos, cfg.rope_theta))
        o = r(oracle.attention(q, k, v, pos, pos).reshape(T, nq * d))
        x = x + o @ Lw["wo"].T
        u = r(oracle.rms_norm(x, Lw["mlp_norm"], eps))
        x = x + r(oracle.silu(u @ Lw["wg"].T) * (u @ Lw["wu"].T)) @ Lw["wd"].T
    return oracle.lm_logits(W, r(oracle.final_hidden(cfg, W, x)))
