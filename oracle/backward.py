"""fp64 CPU oracle: the gradient of the SFT objective of the Qwen3-architecture decoder.

TEST INFRASTRUCTURE ONLY (see the package docstring).

What it computes.  The SFT objective (Sec. "Task Serialization and SFT
Objective", Eq. sft) maximises the log-likelihood of the target tokens; as a
loss to minimise over a batch of teacher-forced sequences it is

    loss = scale * sum_{b, t < T-1, mask[b, t]} -log p(tokens[b, t+1] | tokens[b, <= t])

(scale = 1 / number of target tokens gives the token mean).  The general form
computed here weights each token by a coefficient c[b, t],
loss = sum c[b, t] (-log p(...)); SFT takes c = scale * mask, and the GRPO
objective of Eq. ppo takes c = -d L / d lp (grpo.grpo_coef), whose gradient
is then the gradient of the GRPO loss.  The gradient of
this loss with respect to every weight tensor of the decoder is obtained here by
writing out the backward pass of each forward step of the oracle (qwen3.py), in
reverse order, from the chain rule:

  log-softmax:   d loss / dz_t = scale * mask_t * (softmax(z_t) - onehot(target_t))
  linear y = x W^T:          dx = dy W,  dW = dy^T x
  RMSNorm y = x r g, r = (mean(x^2) + eps)^(-1/2) over the last axis (n entries):
                 dg = sum over rows of dy x r,
                 dx = r (dy g) - (r^3 / n) x sum_i (dy_i g_i x_i)
  RoPE (rotate-half, a rotation R(p)):  dx = R(p)^T dy  (the rotation by -theta)
  causal attention, per query head h with its kv head:
                 S = q k^T / sqrt(d) (keys after the query masked), P = softmax(S),
                 o = P v:   dP = do v^T,  dv += P^T do,
                 dS = P (dP - rowsum(dP P)),  dq = dS k / sqrt(d),  dk += dS^T q / sqrt(d)
  SwiGLU h = silu(g) u, silu(g) = g s(g), s the logistic function:
                 dg = dh u s(g) (1 + g (1 - s(g))),  du = dh silu(g)
  residual x + f(x):  the incoming gradient passes through unchanged and adds to f's
  embedding x_0 = E[token]:  dE[token] += dx_0 (every occurrence).

Pinned by ``tests/test_oracle_backward.py`` against central finite differences of
the loss (an independent evaluation of the same function) and against
torch.autograd through a decoder assembled from torch library routines, and by
planted mistakes that those pins must catch.
"""
from __future__ import annotations

import numpy as np

from .qwen3 import apply_rope, forward_logits, layer_weights, silu, softmax, token_logprobs, widen

__all__ = ["policy_loss", "policy_loss_and_grads", "sft_loss", "sft_loss_and_grads"]

_LAYER = ("attn_norm", "wq", "wk", "wv", "q_norm", "k_norm", "wo", "mlp_norm", "wg", "wu", "wd")


def _rms_scale(x, eps):
    return 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)


def _rms_backward(x, r, g, dy):
    """Backward of y = x r g (r per row of the last axis): returns dx, dg (summed over rows)."""
    n = x.shape[-1]
    a = dy * g
    dx = r * a - (r ** 3 / n) * x * np.sum(a * x, axis=-1, keepdims=True)
    dg = np.sum((dy * x * r).reshape(-1, n), axis=0)
    return dx, dg


def _rope_backward(dy, pos, theta):
    """R(p)^T dy for the rotate-half RoPE of apply_rope (rotation by -theta)."""
    d = dy.shape[-1]
    half = d // 2
    inv = theta ** (-2.0 * np.arange(half) / d)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]
    c, s = np.cos(ang), np.sin(ang)
    shape = (dy.shape[0],) + (1,) * (dy.ndim - 2) + (half,)
    c, s = c.reshape(shape), s.reshape(shape)
    d1, d2 = dy[..., :half], dy[..., half:]
    return np.concatenate([d1 * c + d2 * s, -d1 * s + d2 * c], axis=-1)


def _forward_cache(cfg, W, tokens):
    """Forward over one sequence keeping what the backward needs."""
    T = len(tokens)
    nq, nkv, d, eps = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.rms_eps
    group = nq // nkv
    pos = np.arange(T)
    visible = pos[None, :] <= pos[:, None]
    x = widen(W["embed"][np.asarray(tokens)])
    cache = []
    for layer in range(cfg.n_layers):
        Lw = layer_weights(W, layer)
        c = {"x_in": x}
        c["r1"] = _rms_scale(x, eps)
        u1 = x * c["r1"] * Lw["attn_norm"]
        c["u1"] = u1
        q = (u1 @ Lw["wq"].T).reshape(T, nq, d)
        k = (u1 @ Lw["wk"].T).reshape(T, nkv, d)
        v = (u1 @ Lw["wv"].T).reshape(T, nkv, d)
        c["q_raw"], c["k_raw"], c["v"] = q, k, v
        c["rq"], c["rk"] = _rms_scale(q, eps), _rms_scale(k, eps)
        qn = q * c["rq"] * Lw["q_norm"]
        kn = k * c["rk"] * Lw["k_norm"]
        qr, kr = apply_rope(qn, pos, cfg.rope_theta), apply_rope(kn, pos, cfg.rope_theta)
        c["qr"], c["kr"] = qr, kr
        P = np.empty((nq, T, T))
        o = np.empty((T, nq, d))
        for h in range(nq):
            g = h // group
            s = np.where(visible, (qr[:, h] @ kr[:, g].T) / np.sqrt(d), -np.inf)
            P[h] = softmax(s, axis=-1)
            o[:, h] = P[h] @ v[:, g]
        c["P"], c["o"] = P, o.reshape(T, nq * d)
        x = x + c["o"] @ Lw["wo"].T
        c["x_mid"] = x
        c["r2"] = _rms_scale(x, eps)
        u2 = x * c["r2"] * Lw["mlp_norm"]
        c["u2"] = u2
        gl, up = u2 @ Lw["wg"].T, u2 @ Lw["wu"].T
        c["g"], c["up"] = gl, up
        c["h"] = silu(gl) * up
        x = x + c["h"] @ Lw["wd"].T
        cache.append(c)
    rf = _rms_scale(x, eps)
    hn = x * rf * widen(W["final_norm"])
    z = hn @ widen(W["lm_head"]).T
    return cache, x, rf, hn, z


def _coef(tokens, coef):
    """Per-token weights [B, T-1] as float64 (all ones when None)."""
    B, T = tokens.shape
    if coef is None:
        return np.ones((B, T - 1))
    c = np.asarray(coef, dtype=np.float64).reshape(B, T - 1)
    return c


def policy_loss(cfg, W, tokens, coef=None) -> float:
    """sum_{b, t < T-1} coef[b, t] * (-log p(tokens[b, t+1] | tokens[b, <= t])), tokens [B, T].

    Evaluated through the forward oracle (forward_logits, token_logprobs), not through
    the forward pass kept by the backward below.
    """
    tokens = np.atleast_2d(np.asarray(tokens))
    c = _coef(tokens, coef)
    total = 0.0
    for b in range(tokens.shape[0]):
        z = forward_logits(cfg, W, tokens[b])
        lp = token_logprobs(z[:-1], tokens[b, 1:])
        total += float(np.sum(c[b] * -lp))
    return total


def sft_loss(cfg, W, tokens, mask=None, scale=1.0) -> float:
    """Eq. sft as a loss: scale * sum of -log p(target) over the target tokens (mask [B, T-1])."""
    tokens = np.atleast_2d(np.asarray(tokens))
    m = _coef(tokens, mask)
    return policy_loss(cfg, W, tokens, scale * m)


def sft_loss_and_grads(cfg, W, tokens, mask=None, scale=1.0):
    """(loss, grads) of sft_loss (see policy_loss_and_grads)."""
    tokens = np.atleast_2d(np.asarray(tokens))
    return policy_loss_and_grads(cfg, W, tokens, scale * _coef(tokens, mask))


def policy_loss_and_grads(cfg, W, tokens, coef=None):
    """(loss, grads) of policy_loss: grads[name] has the shape of weight tensor `name` (float64).

    With coef = -d L / d lp_t of any token-level objective L of the log-probs (Eq. ppo
    through grpo_coef), grads is d L / d theta.
    """
    tokens = np.atleast_2d(np.asarray(tokens))
    cf = _coef(tokens, coef)
    nq, nkv, d = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim
    group = nq // nkv
    grads = {"embed": np.zeros(W["embed"].shape), "final_norm": np.zeros(W["final_norm"].shape),
             "lm_head": np.zeros(W["lm_head"].shape)}
    for layer in range(cfg.n_layers):
        for nm in _LAYER:
            grads[f"layers.{layer}.{nm}"] = np.zeros(W[f"layers.{layer}.{nm}"].shape)
    Wlm, gf = widen(W["lm_head"]), widen(W["final_norm"])
    layers = [layer_weights(W, layer) for layer in range(cfg.n_layers)]
    total = 0.0
    for b in range(tokens.shape[0]):
        tok = tokens[b]
        T = len(tok)
        pos = np.arange(T)
        cache, xL, rf, hn, z = _forward_cache(cfg, W, tok)
        # rows t < T-1 score tokens[t+1]; the last row has no target (weight 0)
        w = np.zeros(T)
        w[:T - 1] = cf[b]
        tgt = np.zeros(T, dtype=np.int64)
        tgt[:T - 1] = np.asarray(tok)[1:]
        m = np.max(z, axis=-1, keepdims=True)
        lse = (m + np.log(np.sum(np.exp(z - m), axis=-1, keepdims=True)))[:, 0]
        total += float(np.sum(w * (lse - z[np.arange(T), tgt])))
        # log-softmax: d(-log p(tgt)) / dz = softmax(z) - onehot(tgt)
        dz = softmax(z, axis=-1)
        dz[np.arange(T), tgt] -= 1.0
        dz *= w[:, None]
        grads["lm_head"] += dz.T @ hn
        dx, dgf = _rms_backward(xL, rf, gf, dz @ Wlm)
        grads["final_norm"] += dgf
        for layer in reversed(range(cfg.n_layers)):
            c, Lw = cache[layer], layers[layer]
            G = lambda nm: grads[f"layers.{layer}.{nm}"]
            # MLP: x_out = x_mid + W_d (silu(W_g u2) * (W_u u2)), u2 = RMSNorm(x_mid) g_mlp
            G("wd")[...] += dx.T @ c["h"]
            dh = dx @ Lw["wd"]
            sg = 1.0 / (1.0 + np.exp(-c["g"]))
            dg = dh * c["up"] * sg * (1.0 + c["g"] * (1.0 - sg))
            dup = dh * c["g"] * sg
            G("wg")[...] += dg.T @ c["u2"]
            G("wu")[...] += dup.T @ c["u2"]
            du2 = dg @ Lw["wg"] + dup @ Lw["wu"]
            dxm, dg2 = _rms_backward(c["x_mid"], c["r2"], Lw["mlp_norm"], du2)
            G("mlp_norm")[...] += dg2
            dx = dx + dxm
            # attention: x_mid = x_in + W_o o
            G("wo")[...] += dx.T @ c["o"]
            do = (dx @ Lw["wo"]).reshape(T, nq, d)
            dqr = np.zeros((T, nq, d))
            dkr = np.zeros((T, nkv, d))
            dv = np.zeros((T, nkv, d))
            for h in range(nq):
                g = h // group
                P = c["P"][h]
                dP = do[:, h] @ c["v"][:, g].T
                dv[:, g] += P.T @ do[:, h]
                dS = P * (dP - np.sum(dP * P, axis=-1, keepdims=True))
                dqr[:, h] = dS @ c["kr"][:, g] / np.sqrt(d)
                dkr[:, g] += dS.T @ c["qr"][:, h] / np.sqrt(d)
            dqn = _rope_backward(dqr, pos, cfg.rope_theta)
            dkn = _rope_backward(dkr, pos, cfg.rope_theta)
            dq, dgq = _rms_backward(c["q_raw"], c["rq"], Lw["q_norm"], dqn)
            dk, dgk = _rms_backward(c["k_raw"], c["rk"], Lw["k_norm"], dkn)
            G("q_norm")[...] += dgq
            G("k_norm")[...] += dgk
            dq, dk, dv = dq.reshape(T, nq * d), dk.reshape(T, nkv * d), dv.reshape(T, nkv * d)
            G("wq")[...] += dq.T @ c["u1"]
            G("wk")[...] += dk.T @ c["u1"]
            G("wv")[...] += dv.T @ c["u1"]
            du1 = dq @ Lw["wq"] + dk @ Lw["wk"] + dv @ Lw["wv"]
            dxi, dg1 = _rms_backward(c["x_in"], c["r1"], Lw["attn_norm"], du1)
            G("attn_norm")[...] += dg1
            dx = dx + dxi
        np.add.at(grads["embed"], np.asarray(tok), dx)
    return total, grads
