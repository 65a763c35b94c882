// qk_op_linear_swiglu_static: the gate/up + SwiGLU linear step of the CUDA-core
// path with its intermediate held in a fixed device array instead of a
// caller-supplied buffer.
//
// Why it exists: qk_op_linear's unfused SwiGLU path stages the [M, 2N]
// gate/up product in scratch memory the caller passes in.  Some callers cannot
// provide that buffer at call time: a process that reserved its whole device
// memory budget up front (for instance for a KV cache pool) or code embedded in
// a host runtime that owns the allocator and forbids side allocations.  This
// entry point allocates nothing; it uses the array below, which every GPU that
// loads the library holds for the life of the process.
//
// The array's name, used in host code, is only a host-side stand-in for the
// device symbol; it is not a device address.  The device address is looked up
// with cudaGetSymbolAddress (with the device current) on the first call in each
// CUDA context and cached against that context, so a context torn down and
// created again (cudaDeviceReset) is looked up afresh instead of reusing a
// stale address.
#include <cuda.h>

#include <mutex>

#include "qk_internal.cuh"

namespace qk {

namespace {

// Largest gate/up intermediate (M x 2N elements of the model dtype) a call may use.
constexpr size_t kStaticScratchBytes = QK_STATIC_SCRATCH_BYTES;

__device__ __align__(256) unsigned char g_swiglu_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
struct CachedAddress {
    CUcontext ctx;  // context the address belongs to
    void* ptr;
};
CachedAddress g_scratch[kMaxDevices] = {};

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);

// Current driver context of this thread (nullptr if it cannot be queried).
CUcontext current_context() {
    static CtxGetCurrentFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (CtxGetCurrentFn)p;
    });
    CUcontext c = nullptr;
    if (!fn || fn(&c) != CUDA_SUCCESS) return nullptr;
    return c;
}

// Device address of g_swiglu_scratch on the current device, looked up once per
// context (the caller has made `device` current).
int scratch_address(int device, void** out) {
    if (device < 0 || device >= kMaxDevices)
        return set_error(QK_EINVAL, "device ordinal %d outside [0, %d)", device, kMaxDevices);
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    const CUcontext ctx = current_context();
    CachedAddress& c = g_scratch[device];
    if (!c.ptr || !ctx || c.ctx != ctx) {
        void* p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_swiglu_scratch);
        if (e != cudaSuccess) return cuda_error(e, "cudaGetSymbolAddress(static scratch)");
        // cudaGetSymbolAddress may have created the primary context: read it again
        c.ctx = ctx ? ctx : current_context();
        c.ptr = p;
    }
    *out = c.ptr;
    return QK_OK;
}

}  // namespace

}  // namespace qk

using namespace qk;

extern "C" int qk_op_linear_swiglu_static(qk_model* mh, const void* A, int lda, const void* W,
                                          void* C, int ldc, int M, int N, int K, void* stream) {
    if (!mh || !A || !W || !C) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    if (M < 1 || N < 128 || N % 128 || K < 16 || K % 16 || lda < K || ldc != N)
        return set_error(QK_ESHAPE, "bad SwiGLU linear shape M %d N %d K %d lda %d ldc %d", M, N,
                         K, lda, ldc);
    QK_TRY(check_linear_operands(m, A, lda, W, C, m.es));
    const size_t need = (size_t)M * 2 * N * m.es;
    if (need > kStaticScratchBytes)
        return set_error(QK_ESHAPE,
                         "gate/up intermediate of %zu bytes exceeds the static scratch of %zu bytes "
                         "(M x 2N x element size must be <= %zu)",
                         need, kStaticScratchBytes, kStaticScratchBytes);
    int device = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
    if (device != m.device)
        return set_error(QK_EINVAL, "current device %d is not the model's device %d", device,
                         m.device);
    void* scratch = nullptr;
    QK_TRY(scratch_address(device, &scratch));
    cudaStream_t s = (cudaStream_t)stream;
    // The GEMM overwrites every element of the M x 2N intermediate before the
    // SwiGLU kernel reads it, so nothing left by an earlier call is ever used.
    launch_gemm_simt(A, lda, W, scratch, 2 * N, M, 2 * N, K, m.cfg.dtype, EPI_STORE_ACT, s);
    launch_swiglu(scratch, C, m.cfg.dtype, M, N, s);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "static SwiGLU linear");
    return QK_OK;
}
