"""fp64 CPU oracle: the Qwen3-architecture decoder forward pass, written from its definition.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference arm may use it.  It shares no code with
the CUDA path; both sides read the same seeded inputs from ``synth``.

What it computes.  The paper trains a Qwen3-8B policy with the SFT objective
(Sec. "Task Serialization and SFT Objective", Eq. sft: the log-likelihood
log pi_theta(y* | x) of each target token) and with GRPO under a PPO-clipped
objective (Sec. "GRPO Optimization", Eq. ppo: the ratio rho_t of the current to
the old policy's token probability, plus a KL term to a reference policy).
Both consume the per-token log-probability log pi_theta(y_t | x, y_<t) produced
by the policy's causal forward pass; rollouts (Sec. "Implementation
Components": the SLIME-style rollout loop) produce those tokens by
autoregressive decode.  The paper cites the Qwen3 architecture without stating
it, so every layer below follows the public Qwen3 decoder design:

  x_0 = E[token]
  per layer:   u = RMSNorm(x) * g_attn
               q, k, v = W_q u, W_k u, W_v u           (no biases)
               q_h = RMSNorm_d(q_h) * g_q ; k_h = RMSNorm_d(k_h) * g_k   (per head)
               q, k = RoPE_rotate_half(q, k; position, theta = 1e6)
               o_h = sum_j softmax_j(q_h . k_j / sqrt(d)) v_j   over j <= position,
                     kv head of q head h = floor(h / (n_q / n_kv))
               x = x + W_o o
               u = RMSNorm(x) * g_mlp
               x = x + W_down (silu(W_gate u) * (W_up u))
  z = W_lm (RMSNorm(x) * g_final)                     (lm_head separate from E)
  log p(t) = z_t - logsumexp(z) ;  argmax = lowest index attaining max z

Everything is float64.  Weights arrive as bf16 bit patterns (uint16) or
float32 and are widened exactly.  Matrix products use numpy's matmul as a
library step.  The only restructuring is of independent work: the lm_head is
evaluated in vocabulary chunks and token chunks so that no [T, V] float64 array
larger than a chunk is held; every logit is still one full dot product.

Readings where the paper is silent (each also listed in the design notes):
RMSNorm epsilon 1e-6 inside the square root; QK-norm before RoPE with one gain
vector of length head_dim shared by all heads; rotate-half RoPE pairing
(i, i + d/2) with inverse frequency theta^(-2i/d); contiguous GQA groups;
attention scale 1/sqrt(head_dim); positions start at 0.

Every function here is pinned by ``tests/test_oracle_pins.py`` against
properties, closed forms, independent library routines (torch's
scaled_dot_product_attention, rms_norm, log_softmax, complex rotation) and a
scalar brute force; none is "parity unpinned".
"""
from __future__ import annotations

import numpy as np

__all__ = [
    "widen", "rms_norm", "rope_angles", "apply_rope", "softmax", "log_softmax", "silu",
    "attention", "layer_weights", "decoder_layer", "embed", "final_hidden", "lm_logits",
    "forward_hidden",
    "forward_logits", "token_logprobs", "argmax_lowest", "top2_gap", "score_sequence",
    "KVDecoder", "rollout_teacher_forced", "layer_decode_step",
]


def widen(a) -> np.ndarray:
    """bf16 bit patterns (uint16) or fp32/fp64 values -> float64, exactly."""
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


def rms_norm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * g."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * g


def rope_angles(pos, head_dim: int, theta: float) -> np.ndarray:
    """Rotation angles [T, d/2]: position p times inverse frequency theta^(-2i/d), i < d/2."""
    i = np.arange(head_dim // 2, dtype=np.float64)
    inv_freq = theta ** (-2.0 * i / head_dim)
    return np.asarray(pos, dtype=np.float64)[:, None] * inv_freq[None, :]


def apply_rope(x: np.ndarray, pos, theta: float) -> np.ndarray:
    """Rotate-half RoPE of x [T, heads, d] at positions pos [T].

    Element i < d/2 is paired with element i + d/2 and the pair (a, b) is rotated
    by angle p * theta^(-2i/d): (a cos - b sin, b cos + a sin).
    """
    d = x.shape[-1]
    half = d // 2
    ang = rope_angles(pos, d, theta)[:, None, :]
    c, s = np.cos(ang), np.sin(ang)
    a, b = x[..., :half], x[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def softmax(s: np.ndarray, axis: int = -1) -> np.ndarray:
    """Max-subtracted softmax; -inf entries get probability 0."""
    m = np.max(s, axis=axis, keepdims=True)
    e = np.exp(s - m)
    return e / np.sum(e, axis=axis, keepdims=True)


def log_softmax(z: np.ndarray, axis: int = -1) -> np.ndarray:
    """z - logsumexp(z), with the maximum subtracted before exponentiating."""
    m = np.max(z, axis=axis, keepdims=True)
    return z - (m + np.log(np.sum(np.exp(z - m), axis=axis, keepdims=True)))


def silu(z: np.ndarray) -> np.ndarray:
    """silu(z) = z * sigmoid(z) = z / (1 + exp(-z))."""
    with np.errstate(over="ignore"):
        return z / (1.0 + np.exp(-z))


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, q_pos, k_pos) -> np.ndarray:
    """Masked grouped-query attention.

    q [T, n_q, d]; k, v [S, n_kv, d]; query t attends key j iff k_pos[j] <= q_pos[t].
    Query head h reads kv head h // (n_q // n_kv).  Scale 1/sqrt(d).
    """
    T, n_q, d = q.shape
    n_kv = k.shape[1]
    group = n_q // n_kv
    q_pos = np.asarray(q_pos)
    k_pos = np.asarray(k_pos)
    visible = k_pos[None, :] <= q_pos[:, None]
    out = np.empty((T, n_q, d), dtype=np.float64)
    for h in range(n_q):
        g = h // group
        s = (q[:, h, :] @ k[:, g, :].T) / np.sqrt(d)
        s = np.where(visible, s, -np.inf)
        out[:, h, :] = softmax(s, axis=-1) @ v[:, g, :]
    return out


def layer_weights(W, layer: int) -> dict:
    """Widen one layer's tensors from the weight mapping to float64."""
    return {nm: widen(W[f"layers.{layer}.{nm}"]) for nm in
            ("attn_norm", "wq", "wk", "wv", "q_norm", "k_norm", "wo", "mlp_norm", "wg", "wu", "wd")}


def decoder_layer(cfg, Lw: dict, x: np.ndarray, pos, k_past=None, v_past=None, past_pos=None):
    """One decoder layer over T new tokens.

    x [T, H] float64 residual stream at positions pos [T].  k_past / v_past
    [S0, n_kv, d] are earlier keys / values (already normed and rotated) at
    positions past_pos [S0].  Returns (x_out [T, H], k_new, v_new [T, n_kv, d]).
    """
    T = x.shape[0]
    nq, nkv, d, eps = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.rms_eps
    pos = np.asarray(pos)
    u = rms_norm(x, Lw["attn_norm"], eps)
    q = (u @ Lw["wq"].T).reshape(T, nq, d)
    k = (u @ Lw["wk"].T).reshape(T, nkv, d)
    v = (u @ Lw["wv"].T).reshape(T, nkv, d)
    q = rms_norm(q, Lw["q_norm"], eps)
    k = rms_norm(k, Lw["k_norm"], eps)
    q = apply_rope(q, pos, cfg.rope_theta)
    k = apply_rope(k, pos, cfg.rope_theta)
    if k_past is not None and len(k_past):
        K = np.concatenate([k_past, k], axis=0)
        V = np.concatenate([v_past, v], axis=0)
        kpos = np.concatenate([np.asarray(past_pos), pos])
    else:
        K, V, kpos = k, v, pos
    o = attention(q, K, V, pos, kpos).reshape(T, nq * d)
    x = x + o @ Lw["wo"].T
    u = rms_norm(x, Lw["mlp_norm"], eps)
    h = silu(u @ Lw["wg"].T) * (u @ Lw["wu"].T)
    x = x + h @ Lw["wd"].T
    return x, k, v


def embed(W, tokens) -> np.ndarray:
    """x_0 = E[token] for each token (rows of the embedding table)."""
    E = W["embed"]
    return widen(E[np.asarray(tokens)])


def final_hidden(cfg, W, x: np.ndarray) -> np.ndarray:
    return rms_norm(x, widen(W["final_norm"]), cfg.rms_eps)


def lm_logits(W, hn: np.ndarray, vocab_chunk: int = 16384) -> np.ndarray:
    """z = W_lm hn for hn [T, H]; the vocabulary is widened chunk by chunk."""
    Wl = W["lm_head"]
    V = Wl.shape[0]
    z = np.empty((hn.shape[0], V), dtype=np.float64)
    for v0 in range(0, V, vocab_chunk):
        z[:, v0:v0 + vocab_chunk] = hn @ widen(Wl[v0:v0 + vocab_chunk]).T
    return z


def forward_hidden(cfg, W, tokens) -> np.ndarray:
    """Full causal forward over one sequence; returns the final-normed hidden states [T, H]."""
    tokens = np.asarray(tokens)
    pos = np.arange(len(tokens))
    x = embed(W, tokens)
    for layer in range(cfg.n_layers):
        x, _, _ = decoder_layer(cfg, layer_weights(W, layer), x, pos)
    return final_hidden(cfg, W, x)


def forward_logits(cfg, W, tokens) -> np.ndarray:
    """Logits [T, V] of the full causal forward over one sequence."""
    return lm_logits(W, forward_hidden(cfg, W, tokens))


def token_logprobs(z: np.ndarray, targets) -> np.ndarray:
    """log p(target) = z[target] - logsumexp(z), per row of z [T, V]."""
    lsm = log_softmax(z, axis=-1)
    return lsm[np.arange(z.shape[0]), np.asarray(targets)]


def argmax_lowest(z: np.ndarray) -> np.ndarray:
    """Index of the largest logit per row; ties go to the lowest index."""
    return np.argmax(z, axis=-1)


def top2_gap(z: np.ndarray) -> np.ndarray:
    """Largest minus second-largest logit per row."""
    part = np.partition(z, -2, axis=-1)
    return part[..., -1] - part[..., -2]


def score_sequence(cfg, W, tokens, token_chunk: int = 256):
    """Teacher-forced scoring of one sequence (Eq. sft / Eq. ppo inputs).

    Returns lp [T-1] with lp[t] = log p(tokens[t+1] | tokens[<=t]), argmax [T-1]
    and top-2 gap [T-1] of the logits at positions t < T-1.  Positions are
    independent after the decoder stack, so the lm_head runs token_chunk rows
    at a time.
    """
    tokens = np.asarray(tokens)
    hn = forward_hidden(cfg, W, tokens)[:-1]
    T1 = hn.shape[0]
    lp = np.empty(T1)
    am = np.empty(T1, dtype=np.int64)
    gap = np.empty(T1)
    for t0 in range(0, T1, token_chunk):
        z = lm_logits(W, hn[t0:t0 + token_chunk])
        lp[t0:t0 + token_chunk] = token_logprobs(z, tokens[t0 + 1:t0 + 1 + z.shape[0]])
        am[t0:t0 + token_chunk] = argmax_lowest(z)
        gap[t0:t0 + token_chunk] = top2_gap(z)
    return lp, am, gap


class KVDecoder:
    """Incremental decoding of one sequence with a per-layer key/value cache.

    A second code path for the same function as forward_logits: prefill runs the
    prompt, every step appends one token at the next position and attends to the
    whole cache.
    """

    def __init__(self, cfg, W):
        self.cfg, self.W = cfg, W
        self.Lw = [layer_weights(W, layer) for layer in range(cfg.n_layers)]
        self.k = [np.zeros((0, cfg.n_kv_heads, cfg.head_dim)) for _ in range(cfg.n_layers)]
        self.v = [np.zeros((0, cfg.n_kv_heads, cfg.head_dim)) for _ in range(cfg.n_layers)]
        self.n = 0

    def _run(self, tokens) -> np.ndarray:
        tokens = np.asarray(tokens)
        pos = np.arange(self.n, self.n + len(tokens))
        x = embed(self.W, tokens)
        for layer in range(self.cfg.n_layers):
            x, kn, vn = decoder_layer(self.cfg, self.Lw[layer], x, pos, self.k[layer],
                                      self.v[layer], np.arange(self.n))
            self.k[layer] = np.concatenate([self.k[layer], kn])
            self.v[layer] = np.concatenate([self.v[layer], vn])
        self.n += len(tokens)
        return lm_logits(self.W, final_hidden(self.cfg, self.W, x))

    def prefill(self, tokens) -> np.ndarray:
        """Logits of the last prompt position [V]."""
        return self._run(tokens)[-1]

    def step(self, token) -> np.ndarray:
        """Logits [V] after appending one token."""
        return self._run([token])[-1]


def rollout_teacher_forced(cfg, W, seq, P: int):
    """Teacher-forced rollout of one sequence seq = prompt[0:P] ++ c[0..N].

    Prefill over the prompt scores c[0]; decode step j (j = 0..N-1) consumes
    c[j] at position P + j and scores c[j+1].  Returns (logits [N+1, V],
    lp [N+1]) where row j holds the logits that score c[j].
    """
    seq = np.asarray(seq)
    N = len(seq) - P - 1
    dec = KVDecoder(cfg, W)
    rows = [dec.prefill(seq[:P])]
    for j in range(N):
        rows.append(dec.step(seq[P + j]))
    z = np.stack(rows)
    return z, token_logprobs(z, seq[P:P + N + 1])


def layer_decode_step(cfg, Lw: dict, x: np.ndarray, k_cache: np.ndarray, v_cache: np.ndarray, pos):
    """One decoder layer, one decode step per batch row (the one-layer workload).

    x [B, H] residual stream; k_cache / v_cache [B, n_kv, S, d] hold keys and
    values already normed and rotated at positions 0..pos[b]-1.  The new token
    sits at pos[b], its key and value are appended and attended.  Returns
    (x_out [B, H], k_new [B, n_kv, d], v_new [B, n_kv, d]).

    Same steps as decoder_layer; the B rows share the linear layers (each row is
    an independent matrix-vector product) and differ only in their caches.
    """
    B = x.shape[0]
    nq, nkv, d, eps = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.rms_eps
    pos = np.asarray(pos)
    x = widen(x)
    u = rms_norm(x, Lw["attn_norm"], eps)
    q = rms_norm((u @ Lw["wq"].T).reshape(B, nq, d), Lw["q_norm"], eps)
    k = rms_norm((u @ Lw["wk"].T).reshape(B, nkv, d), Lw["k_norm"], eps)
    v = (u @ Lw["wv"].T).reshape(B, nkv, d)
    q = apply_rope(q, pos, cfg.rope_theta)
    k = apply_rope(k, pos, cfg.rope_theta)
    o = np.empty((B, nq, d))
    for b in range(B):
        p = int(pos[b])
        K = np.concatenate([widen(k_cache[b, :, :p, :]).transpose(1, 0, 2), k[b:b + 1]])
        V = np.concatenate([widen(v_cache[b, :, :p, :]).transpose(1, 0, 2), v[b:b + 1]])
        o[b] = attention(q[b:b + 1], K, V, [p], np.arange(p + 1))[0]
    x = x + o.reshape(B, nq * d) @ Lw["wo"].T
    u = rms_norm(x, Lw["mlp_norm"], eps)
    x = x + (silu(u @ Lw["wg"].T) * (u @ Lw["wu"].T)) @ Lw["wd"].T
    return x, k, v
