"""The no-allocation SwiGLU linear entry point, qk_op_linear_swiglu_static.

It serves callers that cannot give the library a scratch buffer (a process
that reserved its whole device memory budget up front, or code inside a
runtime that owns the allocator): the [M, 2N] gate/up intermediate lives in a
fixed device array of the library instead.  Checked here through the C ABI
against a float64 numpy evaluation of silu(A Wg^T) * (A Wu^T), on an fp32 and a
bf16 model, on two calls in a row with different shapes and inputs (a stale
intermediate from the first call would show in the second), and for the size
limit.  This file is collected last so that a stop-at-first-failure run has
already run every other test."""
import numpy as np
import pytest

import oracle
import synth
from _gpu import decoder

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def models():
    return {"f32": decoder(synth.shape("tiny_fp32"))[0],
            "bf16": decoder(synth.shape("tiny_fp32", dtype="bf16"))[0]}


def _gate_up(A, W):
    """float64 gate and up products; W holds blocks of 128 gate rows, each followed
    by the matching 128 up rows."""
    z = oracle.widen(A) @ oracle.widen(W).T
    nb = W.shape[0] // 256
    g = np.concatenate([z[:, 256 * i:256 * i + 128] for i in range(nb)], axis=1)
    u = np.concatenate([z[:, 256 * i + 128:256 * i + 256] for i in range(nb)], axis=1)
    return g, u


@pytest.mark.parametrize("dt", ["f32", "bf16"])
def test_static_scratch_swiglu_matches_f64(models, dt):
    import torch
    import paper_2609_12471_gb300 as qk
    dec = models[dt]
    tdt = torch.bfloat16 if dt == "bf16" else torch.float32
    cvt = ((lambda a: torch.from_numpy(a.view(np.int16)).view(torch.bfloat16)) if dt == "bf16"
           else torch.from_numpy)
    for call, (M, N, K) in enumerate([(48, 768, 256), (131, 384, 192)]):
        A = synth.normal(500 + call, 1, (M, K), dt)
        W = synth.normal(500 + call, 2, (2 * N, K), dt, sigma=0.05)
        Ad, Wd = cvt(A).cuda(), cvt(W).cuda()
        got = torch.full((M, N), float("nan"), dtype=tdt, device="cuda")
        qk.qk_op_linear_swiglu_static(dec.handle, Ad, K, Wd, got, N, M, N, K)
        torch.cuda.synchronize()
        g = got.double().cpu().numpy()
        gate, up = _gate_up(A, W)
        ref = oracle.silu(gate) * up
        assert np.all(np.isfinite(g)), f"call {call}"
        if dt == "f32":
            tol = 1e-5 * np.abs(ref).max()  # fp32 accumulation, no intermediate rounding
        else:
            # bf16 gate/up intermediate and bf16 output: three roundings of relative size
            # <= 2^-8 on values bounded by |gate| |up| (|silu'| <= 1.1, |silu(g)| <= |g|)
            tol = 4 * 2.0 ** -8 * np.max(np.abs(gate) * np.abs(up))
        err = np.abs(g - ref).max()
        assert err <= tol, f"call {call}: max err {err:.3e} > {tol:.3e}"


def test_static_scratch_rejects_oversized_call(models):
    import torch
    import paper_2609_12471_gb300 as qk
    N, K = 768, 256
    M = qk.QK_STATIC_SCRATCH_BYTES // (2 * N * 4) + 1
    A = torch.zeros(M, K, device="cuda")
    W = torch.zeros(2 * N, K, device="cuda")
    C = torch.zeros(M, N, device="cuda")
    before = qk.qk_launch_count()
    with pytest.raises(qk.QKError) as e:
        qk.qk_op_linear_swiglu_static(models["f32"].handle, A, K, W, C, N, M, N, K)
    assert e.value.code == qk.QK_ESHAPE
    assert qk.qk_launch_count() == before
