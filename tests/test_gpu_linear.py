"""Per-kernel parity of the linear layers (qk_op_linear) against float64 matmul.

Covers the three paths the model uses: the bf16 weight-streaming GEMV (<= 16
token rows), the tcgen05 GEMM (> 16 rows; token tiles 32/64/128/256 with ragged
tails, several feature tiles, K of one and many k-blocks) and the fp32 CUDA-core
GEMM, with every epilogue (store, fp32 store, residual add, SwiGLU).  Inputs are
bf16 (or fp32) values from the seeded generator; the reference widens them to
float64 exactly and multiplies (numpy matmul)."""
import numpy as np
import pytest

import oracle
import synth
from _gpu import decoder

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def models():
    bf = synth.shape("tiny_fp32", dtype="bf16")
    f32 = synth.shape("tiny_fp32")
    return {"bf16": decoder(bf)[0], "f32": decoder(f32)[0]}


def _ref(A, W, epi, C0):
    z = oracle.widen(A) @ oracle.widen(W).T
    if epi == 3:  # SwiGLU over 128-row gate / up blocks
        N = W.shape[0] // 2
        g = np.concatenate([z[:, 256 * i:256 * i + 128] for i in range(N // 128)], axis=1)
        u = np.concatenate([z[:, 256 * i + 128:256 * i + 256] for i in range(N // 128)], axis=1)
        return oracle.silu(g) * u
    if epi == 2:
        return C0 + z
    return z


CASES = [  # (M, N, K)
    (1, 384, 256), (4, 256, 512), (5, 128, 4096), (16, 640, 192), (17, 384, 256), (31, 128, 64),
    (33, 256, 4096), (64, 128, 512), (100, 384, 256), (129, 256, 320), (300, 128, 4096),
    (1000, 640, 256),
]


@pytest.mark.parametrize("dt", ["bf16", "f32"])
@pytest.mark.parametrize("epi", [0, 1, 2, 3])
@pytest.mark.parametrize("M,N,K", CASES)
def test_linear_matches_f64(models, dt, epi, M, N, K):
    import torch
    import paper_2609_12471_gb300 as qk
    if dt == "f32" and M * N * K > 40_000_000:
        pytest.skip("fp32 CUDA-core path: large shapes covered by bf16")
    dec = models[dt]
    seed = M * 7919 + N * 31 + K + epi
    Wrows = 2 * N if epi == 3 else N
    A = synth.normal(seed, 1, (M, K), dt)
    W = synth.normal(seed, 2, (Wrows, K), dt, sigma=0.05)
    tdt = torch.bfloat16 if dt == "bf16" else torch.float32
    cvt = (lambda a: torch.from_numpy(a.view(np.int16)).view(torch.bfloat16)) if dt == "bf16" else torch.from_numpy
    Ad, Wd = cvt(A).cuda(), cvt(W).cuda()
    out_f32 = epi in (1, 2)
    C0 = synth.normal(seed, 3, (M, N), "f32")
    Cd = torch.from_numpy(C0).cuda() if out_f32 else torch.zeros(M, N, dtype=tdt, device="cuda")
    scratch = torch.empty(M * 2 * N * 4, dtype=torch.uint8, device="cuda") if epi == 3 else None
    qk.qk_op_linear(dec.handle, Ad, K, Wd, Cd, N, M, N, K, epi, scratch)
    torch.cuda.synchronize()
    got = Cd.double().cpu().numpy()
    ref = _ref(A, W, epi, C0.astype(np.float64))
    scale = np.abs(ref).max() + 1e-30
    if dt == "f32":
        tol = 1e-5 * scale
    elif out_f32:
        tol = 2e-5 * scale                     # fp32 accumulation of exact bf16 products
    else:
        tol = 2 ** -8 * scale                  # one bf16 rounding of the output
    err = np.abs(got - ref).max()
    assert err <= tol, f"max err {err:.3e} > {tol:.3e} (scale {scale:.3e})"


@pytest.mark.parametrize("dt", ["bf16", "f32"])
def test_misaligned_operands_are_refused_before_any_launch(models, dt):
    """A, W off a 16-byte boundary, a row stride that breaks the rows' 16-byte
    alignment, or C off its element size: refused on the host, nothing launched."""
    import torch
    import paper_2609_12471_gb300 as qk
    dec = models[dt]
    es = 2 if dt == "bf16" else 4
    M, N, K = 20, 128, 64
    buf = torch.zeros(8 << 20, dtype=torch.uint8, device="cuda")  # every case stays in bounds
    A, W, C = buf.data_ptr(), buf.data_ptr() + (1 << 20), buf.data_ptr() + (2 << 20)
    bad_lda = K + (4 if dt == "bf16" else 2)
    cases = [dict(A=A + es), dict(W=W + 8), dict(lda=bad_lda), dict(C=C + 2, epi=qk.QK_EPI_STORE_F32)]
    for over in cases:
        a = dict(A=A, W=W, C=C, lda=K, epi=qk.QK_EPI_STORE)
        a.update(over)
        before = qk.qk_launch_count()
        with pytest.raises(qk.QKError) as e:
            qk.qk_op_linear(dec.handle, a["A"], a["lda"], a["W"], a["C"], N, M, N, K, a["epi"])
        assert e.value.code in (qk.QK_EINVAL, qk.QK_ESHAPE), over
        assert qk.qk_launch_count() == before, over
        if "epi" in over:
            continue  # the static variant always stores in the model dtype
        with pytest.raises(qk.QKError) as e:
            qk.qk_op_linear_swiglu_static(dec.handle, a["A"], a["lda"], a["W"], a["C"], N, M, N, K)
        assert e.value.code in (qk.QK_EINVAL, qk.QK_ESHAPE), over
        assert qk.qk_launch_count() == before, over
