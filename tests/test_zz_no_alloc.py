"""The no-allocation SwiGLU linear entry point, qk_op_linear_swiglu_static.

It serves callers that cannot give the library a scratch buffer (a process
that reserved its whole device memory budget up front, or code inside a
runtime that owns the allocator): the [M, 2N] gate/up intermediate lives in a
fixed device array of the library instead.  Checked here through the C ABI
against qk_op_linear with QK_EPI_SWIGLU and a caller-supplied scratch buffer,
on two calls in a row with different shapes and inputs (a stale intermediate
from the first call would show in the second), and for the size limit.
This file is collected last so that a stop-at-first-failure run has already
run every other test."""
import numpy as np
import pytest

import synth
from _gpu import decoder

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tiny_model():
    return decoder(synth.shape("tiny_fp32"))[0]


def test_static_scratch_swiglu_matches_scratch_buffer_version(tiny_model):
    import torch
    import paper_2609_12471_gb300 as qk
    dec = tiny_model
    for call, (M, N, K) in enumerate([(48, 768, 256), (131, 384, 192)]):
        A = synth.normal(500 + call, 1, (M, K), "f32")
        W = synth.normal(500 + call, 2, (2 * N, K), "f32", sigma=0.05)
        Ad, Wd = torch.from_numpy(A).cuda(), torch.from_numpy(W).cuda()
        ref = torch.zeros(M, N, dtype=torch.float32, device="cuda")
        scratch = torch.empty(M * 2 * N * 4, dtype=torch.uint8, device="cuda")
        qk.qk_op_linear(dec.handle, Ad, K, Wd, ref, N, M, N, K, qk.QK_EPI_SWIGLU, scratch)
        got = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
        qk.qk_op_linear_swiglu_static(dec.handle, Ad, K, Wd, got, N, M, N, K)
        torch.cuda.synchronize()
        r, g = ref.cpu().numpy(), got.cpu().numpy()
        assert np.all(np.isfinite(g))
        assert np.abs(g - r).max() <= 1e-5 * np.abs(r).max(), f"call {call}"


def test_static_scratch_rejects_oversized_call(tiny_model):
    import torch
    import paper_2609_12471_gb300 as qk
    N, K = 768, 256
    M = qk.QK_STATIC_SCRATCH_BYTES // (2 * N * 4) + 1
    A = torch.zeros(M, K, device="cuda")
    W = torch.zeros(2 * N, K, device="cuda")
    C = torch.zeros(M, N, device="cuda")
    with pytest.raises(qk.QKError) as e:
        qk.qk_op_linear_swiglu_static(tiny_model.handle, A, K, W, C, N, M, N, K)
    assert e.value.code == qk.QK_ESHAPE
