"""Seeded synthetic inputs for the Qwen3-architecture decoder workloads.

This module is shared by the fp64 oracle (``oracle/``) and the GPU path
(``paper_2609_12471_gb300``).  It holds none of the decoder's arithmetic:
it names the model shapes, assigns every tensor a generator stream, and turns
(seed, stream, index) into bf16 / fp32 / int32 values through ``gen.c``.

Workload recipe (random-init stand-ins for the trained Qwen3-8B policy, whose
weights are not available):
  * linear and embedding weights ~ N(0, 0.02), stored in the model dtype;
  * RMSNorm gains ~ 1 + N(0, 0.02) (perturbed so that a missing or
    mis-indexed gain multiply is visible);
  * token ids uniform over [0, vocab), seed 1;
  * one-layer decode workload: KV cache N(0, 1) bf16 (seed 2, K stream 0,
    V stream 1) and input hidden state N(0, 1) fp32 (seed 3).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass, replace

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gen.c")
_LIB_PATH = os.path.join(_HERE, "libsynth.so")
_lock = threading.Lock()
_lib = None

WEIGHT_SEED = 0
TOKEN_SEED = 1
KV_FILL_SEED = 2
HIDDEN_SEED = 3


def build(force: bool = False) -> str:
    """Compile gen.c into libsynth.so next to it (gcc, no vendor code)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call([
            "gcc", "-O2", "-fPIC", "-shared", "-pthread", "-ffp-contract=off",
            "-o", tmp, _SRC, "-lm",
        ])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            u64, i32, dbl = ctypes.c_uint64, ctypes.c_int32, ctypes.c_double
            for name in ("synth_normal_bf16", "synth_normal_f32"):
                f = getattr(lib, name)
                f.argtypes = [u64, u64, u64, u64, dbl, dbl, ctypes.c_void_p, ctypes.c_int]
                f.restype = ctypes.c_int
            lib.synth_uniform_i32.argtypes = [u64, u64, u64, u64, i32, i32, ctypes.c_void_p, ctypes.c_int]
            lib.synth_uniform_i32.restype = ctypes.c_int
            lib.synth_raw_draw.argtypes = [u64, u64, u64]
            lib.synth_raw_draw.restype = u64
            _lib = lib
    return _lib


def raw_draw(seed: int, stream: int, ctr: int) -> int:
    return int(_load().synth_raw_draw(seed, stream, ctr))


def normal(seed: int, stream: int, shape, dtype: str, mean: float = 0.0, sigma: float = 1.0,
           offset: int = 0, nthreads: int = 0) -> np.ndarray:
    """Normal values; dtype 'bf16' returns the raw bf16 bit patterns as uint16."""
    n = int(np.prod(shape, dtype=np.int64)) if len(tuple(shape)) else 1
    if dtype == "bf16":
        out = np.empty(n, dtype=np.uint16)
        _load().synth_normal_bf16(seed, stream, offset, n, mean, sigma, out.ctypes.data, nthreads)
    elif dtype == "f32":
        out = np.empty(n, dtype=np.float32)
        _load().synth_normal_f32(seed, stream, offset, n, mean, sigma, out.ctypes.data, nthreads)
    else:
        raise ValueError(dtype)
    return out.reshape(shape)


def uniform_int(seed: int, stream: int, shape, lo: int, hi: int, offset: int = 0,
                nthreads: int = 0) -> np.ndarray:
    n = int(np.prod(shape, dtype=np.int64))
    out = np.empty(n, dtype=np.int32)
    rc = _load().synth_uniform_i32(seed, stream, offset, n, lo, hi, out.ctypes.data, nthreads)
    if rc != 0:
        raise ValueError("empty integer range")
    return out.reshape(shape)


# --------------------------------------------------------------------------------------
# Model shapes


@dataclass(frozen=True)
class ModelShape:
    name: str
    n_layers: int
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    intermediate: int
    vocab: int
    dtype: str  # "bf16" | "f32"
    rms_eps: float = 1e-6
    rope_theta: float = 1e6


SHAPES = {
    "tiny_fp32": ModelShape("tiny_fp32", 2, 256, 4, 2, 64, 768, 4096, "f32"),
    "q8b": ModelShape("q8b", 36, 4096, 32, 8, 128, 12288, 151936, "bf16"),
    "q8b_layer": ModelShape("q8b_layer", 1, 4096, 32, 8, 128, 12288, 151936, "bf16"),
}


def shape(name: str, **over) -> ModelShape:
    s = SHAPES[name]
    return replace(s, **over) if over else s


LAYER_TENSORS = ("attn_norm", "wq", "wk", "wv", "q_norm", "k_norm", "wo",
                 "mlp_norm", "wg", "wu", "wd")


def tensor_list(s: ModelShape):
    """Ordered (name, shape, kind, stream) for every weight tensor, HF [out, in] layout.

    kind 'w' is drawn N(0, 0.02); kind 'g' (an RMSNorm gain) is drawn 1 + N(0, 0.02).
    """
    H, d, nq, nkv, I, V = s.hidden, s.head_dim, s.n_q_heads, s.n_kv_heads, s.intermediate, s.vocab
    per_layer = {
        "attn_norm": ((H,), "g"), "wq": ((nq * d, H), "w"), "wk": ((nkv * d, H), "w"),
        "wv": ((nkv * d, H), "w"), "q_norm": ((d,), "g"), "k_norm": ((d,), "g"),
        "wo": ((H, nq * d), "w"), "mlp_norm": ((H,), "g"), "wg": ((I, H), "w"),
        "wu": ((I, H), "w"), "wd": ((H, I), "w"),
    }
    out = [("embed", (V, H), "w", 0)]
    for layer in range(s.n_layers):
        for t, nm in enumerate(LAYER_TENSORS):
            shp, kind = per_layer[nm]
            out.append((f"layers.{layer}.{nm}", shp, kind, 1 + len(LAYER_TENSORS) * layer + t))
    out.append(("final_norm", (H,), "g", 1 + len(LAYER_TENSORS) * s.n_layers))
    out.append(("lm_head", (V, H), "w", 2 + len(LAYER_TENSORS) * s.n_layers))
    return out


def gen_tensor(s: ModelShape, name: str, seed: int = WEIGHT_SEED, rows=None) -> np.ndarray:
    """One weight tensor (or a row range [r0, r1) of it) in the model dtype.

    bf16 tensors come back as uint16 bit patterns, fp32 as float32.
    """
    for nm, shp, kind, stream in tensor_list(s):
        if nm == name:
            mean = 1.0 if kind == "g" else 0.0
            if rows is None:
                return normal(seed, stream, shp, s.dtype, mean=mean, sigma=0.02)
            r0, r1 = rows
            cols = int(np.prod(shp[1:], dtype=np.int64))
            return normal(seed, stream, (r1 - r0,) + tuple(shp[1:]), s.dtype, mean=mean,
                          sigma=0.02, offset=r0 * cols)
    raise KeyError(name)


class LazyWeights:
    """Mapping name -> array that generates each tensor on access (optionally cached)."""

    def __init__(self, s: ModelShape, seed: int = WEIGHT_SEED, cache: bool = True):
        self.shape = s
        self.seed = seed
        self._cache = {} if cache else None
        self._names = [t[0] for t in tensor_list(s)]

    def __getitem__(self, name):
        if self._cache is not None and name in self._cache:
            return self._cache[name]
        a = gen_tensor(self.shape, name, self.seed)
        if self._cache is not None:
            self._cache[name] = a
        return a

    def __contains__(self, name):
        return name in self._names

    def keys(self):
        return list(self._names)

    def drop(self, name):
        if self._cache is not None:
            self._cache.pop(name, None)


def tokens(shape_, vocab: int, seed: int = TOKEN_SEED, stream: int = 0) -> np.ndarray:
    return uniform_int(seed, stream, shape_, 0, vocab)


def kv_fill(B: int, n_kv: int, S: int, d: int):
    """One-layer decode workload: K and V caches [B, n_kv, S, d] ~ N(0, 1) as bf16 bits."""
    k = normal(KV_FILL_SEED, 0, (B, n_kv, S, d), "bf16")
    v = normal(KV_FILL_SEED, 1, (B, n_kv, S, d), "bf16")
    return k, v


def hidden_input(B: int, H: int) -> np.ndarray:
    """One-layer decode workload: input residual stream [B, H] ~ N(0, 1) fp32."""
    return normal(HIDDEN_SEED, 0, (B, H), "f32")
