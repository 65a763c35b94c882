"""fp64 CPU oracle: the GRPO token loss of the paper's RL stage, written from its definition.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference arm may use it.  It shares no code with
the CUDA path.

What it computes (Sec. "GRPO Optimization"):
  * Eq. advantage: the group-relative advantage without variance
    normalisation, A_i = r_i - mean_{j in group(i)} r_j, where a group is the
    G rollouts of one prompt (G consecutive rows here);
  * Eq. ppo: the PPO-clipped surrogate with a KL penalty,
        L_t = -min(rho_t A, clip(rho_t, 1 - eps_low, 1 + eps_high) A) + beta KL_t,
    rho_t = pi_theta(y_t) / pi_old(y_t) = exp(lp_t - lp_old_t), for every
    response token t of a rollout, A being its rollout's advantage;
  * the loss is the mean of L_t over the response tokens of the batch.

Readings where the paper is silent (also listed in the design notes):
  * the KL estimator: k3, KL_t = exp(lp_ref_t - lp_t) - (lp_ref_t - lp_t) - 1
    (non-negative, zero where the two policies agree);
  * "clip(rho, 1 +- eps)" with the hyperparameter table's two values 0.2 / 0.28
    is read as eps_low = 0.2, eps_high = 0.28 (0.2 / 0.2 for the single-turn run);
  * the expectation is a token mean over all response tokens of the batch
    (mask = 1), not a mean of per-sequence means.
"""
from __future__ import annotations

import numpy as np


def group_advantages(rewards, group: int) -> np.ndarray:
    """Eq. advantage: A_i = r_i - (mean reward of row i's group of `group` rows)."""
    r = np.asarray(rewards, dtype=np.float64)
    if group < 1 or r.shape[0] % group:
        raise ValueError("the batch is not a whole number of groups")
    g = r.reshape(-1, group)
    return (g - g.mean(axis=1, keepdims=True)).reshape(-1)


def kl_k3(lp, lp_ref) -> np.ndarray:
    """k3 estimate of KL(pi_theta || pi_ref) at a sampled token: e^x - x - 1, x = lp_ref - lp."""
    x = np.asarray(lp_ref, dtype=np.float64) - np.asarray(lp, dtype=np.float64)
    return np.exp(x) - x - 1.0


def grpo_token_loss(lp, lp_old, lp_ref, adv_rows, eps_low: float, eps_high: float,
                    beta: float) -> np.ndarray:
    """Eq. ppo per token: lp, lp_old, lp_ref [B, T] (lp_ref may be None when beta = 0),
    adv_rows [B]; returns L [B, T]."""
    lp = np.asarray(lp, dtype=np.float64)
    rho = np.exp(lp - np.asarray(lp_old, dtype=np.float64))
    a = np.asarray(adv_rows, dtype=np.float64)[:, None]
    surrogate = np.minimum(rho * a, np.clip(rho, 1.0 - eps_low, 1.0 + eps_high) * a)
    loss = -surrogate
    if beta != 0.0:
        loss = loss + beta * kl_k3(lp, lp_ref)
    return loss


def grpo_token_grad(lp, lp_old, lp_ref, adv_rows, eps_low: float, eps_high: float,
                    beta: float) -> np.ndarray:
    """d L_t / d lp_t of Eq. ppo per token (same arguments as grpo_token_loss).

    d rho / d lp = rho.  The min picks the unclipped term rho A where rho A <=
    clip(rho) A; there its derivative is rho A.  Elsewhere the clipped term is
    smaller, which happens only with rho outside [1 - eps_low, 1 + eps_high],
    where clip(rho) is constant: derivative 0.  d k3 / d lp = 1 - e^x,
    x = lp_ref - lp.
    """
    lp = np.asarray(lp, dtype=np.float64)
    rho = np.exp(lp - np.asarray(lp_old, dtype=np.float64))
    a = np.asarray(adv_rows, dtype=np.float64)[:, None]
    unclipped = rho * a <= np.clip(rho, 1.0 - eps_low, 1.0 + eps_high) * a
    g = -np.where(unclipped, rho * a, 0.0)
    if beta != 0.0:
        g = g + beta * (1.0 - np.exp(np.asarray(lp_ref, dtype=np.float64) - lp))
    return g


def grpo_coef(lp, lp_old, lp_ref, adv_rows, eps_low: float, eps_high: float, beta: float,
              mask=None) -> np.ndarray:
    """Per-token weights c with d(grpo_loss_mean)/d theta = d/d theta sum c (-lp).

    The batch loss is sum(mask L) / sum(mask), so c_t = -mask_t (dL_t/dlp_t) / sum(mask)
    (all zero for an empty mask).
    """
    g = grpo_token_grad(lp, lp_old, lp_ref, adv_rows, eps_low, eps_high, beta)
    m = np.ones_like(g) if mask is None else np.asarray(mask, dtype=np.float64)
    n = m.sum()
    return -m * g / n if n > 0 else np.zeros_like(g)


def grpo_loss_mean(loss_tok, mask=None) -> float:
    """Token mean over the response tokens (mask 1) of the whole batch."""
    loss_tok = np.asarray(loss_tok, dtype=np.float64)
    m = np.ones_like(loss_tok) if mask is None else np.asarray(mask, dtype=np.float64)
    n = m.sum()
    return float((loss_tok * m).sum() / n) if n > 0 else 0.0
