"""fp64 CPU oracle: temperature sampling of rollout tokens by the Gumbel-max rule.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference arm may use it.  It shares no code with
the CUDA path.

What it computes.  The paper's rollouts and its pass@k evaluation sample the
policy at temperature 1.0 (Table "Pass@K results on ROCmBench"; Sec.
"Implementation Components" for the rollout loop).  A token is drawn from
softmax(z / tau) over the vocabulary.  The Gumbel-max rule gives the same
distribution as a deterministic function of independent uniforms:
    c = argmax_v ( z_v / tau + G_v ),   G_v = -log(-log(u_v)),  u_v ~ U(0, 1)
(ties go to the lowest index).  The uniforms come from one counter-based
generator so that the GPU and this oracle draw the same numbers:
  * SplitMix64 (Steele, Lea, Flood, OOPSLA 2014): the i-th output of the stream
    seeded with `seed` is mix64(seed + (i + 1) * 0x9E3779B97F4A7C15) (mod 2^64),
    mix64 the published finaliser;
  * the uniform for (row b, sampling step j, token v) is output
    i = b * 2^40 + j * 2^18 + v (v < 2^18, j < 2^22), mapped to the 24-bit grid
    u = (floor(x / 2^40) + 1/2) / 2^24, which lies strictly inside (0, 1).
The log-probability reported for a sampled token is log softmax(z / tau)[c].

Rollout: prompt p[0:P]; the prefill's last logits sample c[0] (step 0); decode
step j consumes c[j] at position P + j and its logits sample c[j + 1].
"""
from __future__ import annotations

import numpy as np

from .qwen3 import KVDecoder, log_softmax

GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def mix64(z: np.ndarray) -> np.ndarray:
    """SplitMix64's output finaliser on uint64 arrays (wrapping arithmetic)."""
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def splitmix64_at(seed: int, idx) -> np.ndarray:
    """Outputs idx (array) of the SplitMix64 stream seeded with `seed`."""
    i = np.asarray(idx, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return mix64(np.uint64(seed) + (i + np.uint64(1)) * GAMMA)


def sample_uniforms(seed: int, b: int, j: int, V: int) -> np.ndarray:
    """u[v] for v < V at (row b, step j): float64 on the 24-bit grid, in (0, 1)."""
    idx = (np.uint64(b) << np.uint64(40)) + (np.uint64(j) << np.uint64(18)) + np.arange(V, dtype=np.uint64)
    x = splitmix64_at(seed, idx)
    return ((x >> np.uint64(40)).astype(np.float64) + 0.5) * 2.0 ** -24


def gumbel(u: np.ndarray) -> np.ndarray:
    return -np.log(-np.log(u))


def sample_token(z: np.ndarray, tau: float, seed: int, b: int, j: int):
    """Gumbel-max draw from softmax(z / tau): (token, log p(token), sorted top-2 gap of the
    perturbed scores)."""
    z = np.asarray(z, dtype=np.float64)
    y = z / tau + gumbel(sample_uniforms(seed, b, j, z.shape[-1]))
    c = int(np.argmax(y))  # numpy returns the first (lowest) index of the maximum
    top2 = np.partition(y, -2)[-2:]
    return c, float(log_softmax(z / tau)[c]), float(top2[1] - top2[0])


def rollout_sampled(cfg, W, prompt, N: int, tau: float, seed: int, b: int = 0, forced=None):
    """Sampled rollout of one row b.  Returns (tokens [N+1], lp [N+1], gaps [N+1], z [N+1, V]).
    With `forced` (tokens [N+1]) the sequence follows the given tokens instead of the
    oracle's own draws (so a GPU rollout can be checked step by step), while the
    oracle's draw, log-prob of the forced token and gap are still reported."""
    dec = KVDecoder(cfg, W)
    z = dec.prefill(np.asarray(prompt))
    toks, lps, gaps, zs = [], [], [], []
    for j in range(N + 1):
        c, _, gap = sample_token(z, tau, seed, b, j)
        t = c if forced is None else int(forced[j])
        toks.append(c)
        lps.append(float(log_softmax(np.asarray(z, dtype=np.float64) / tau)[t]))
        gaps.append(gap)
        zs.append(z)
        if j < N:
            z = dec.step(t)
    return np.array(toks), np.array(lps), np.array(gaps), np.stack(zs)
