"""Helpers for the GPU parity tests: build + load the library, tolerance checks."""
import numpy as np
import pytest


def require_gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_12471_gb300 import build
    build.build()
    import paper_2609_12471_gb300 as qk
    return qk


def decoder(shape, weights=None, **cfg_over):
    """Build a libqk model for a synth.ModelShape (weights default to the seeded ones)."""
    import synth
    qk = require_gpu()
    from paper_2609_12471_gb300.runtime import Decoder
    base = {"tiny_fp32": "tiny_fp32", "q8b": "q8b", "q8b_layer": "q8b_layer"}.get(shape.name, "q8b")
    cfg = qk.qk_config_preset(base)
    for f in ("n_layers", "hidden", "n_q_heads", "n_kv_heads", "head_dim", "intermediate", "vocab"):
        setattr(cfg, f, getattr(shape, f))
    cfg.dtype = qk.QK_DTYPE_BF16 if shape.dtype == "bf16" else qk.QK_DTYPE_F32
    for k, v in cfg_over.items():
        setattr(cfg, k, v)
    W = weights if weights is not None else synth.LazyWeights(shape, cache=False)
    return Decoder(cfg, (W[n] for n in [t[0] for t in synth.tensor_list(shape)])), W


def bf16_bits_to_f64(a):
    return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def assert_logits_close(got, ref, rel):
    """max |got - ref| <= rel * std(ref) over the whole compared tensor."""
    got = np.asarray(got, dtype=np.float64)
    tol = rel * float(np.std(ref))
    err = float(np.max(np.abs(got - ref)))
    assert err <= tol, f"max |dlogit| {err:.3e} > {tol:.3e} ({rel} x std {np.std(ref):.4f})"
    return err, tol


def assert_argmax_where_gap(got, ref_logits, logit_tol, min_decisive=1, distinct=None):
    """Arg-max must match where the oracle's top-2 gap exceeds 10x the logit tolerance,
    and at least `min_decisive` rows must be decisive (so the check cannot pass
    vacuously).  distinct: columns holding the distinct logit values when the vocabulary
    repeats values on purpose (the gap is then taken over those columns only)."""
    import oracle
    ref_logits = np.asarray(ref_logits)
    gap = oracle.top2_gap(ref_logits if distinct is None else ref_logits[:, distinct])
    am = oracle.argmax_lowest(ref_logits)
    mask = gap > 10 * logit_tol
    n = int(mask.sum())
    bad = np.nonzero(mask & (np.asarray(got) != am))[0]
    assert bad.size == 0, f"argmax differs at {bad[:10]} (of {n} decisive rows)"
    assert n >= min_decisive, f"only {n} of {len(mask)} rows decisive (need {min_decisive})"
    return n
