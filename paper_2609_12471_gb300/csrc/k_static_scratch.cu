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
// once per device with cudaGetSymbolAddress (with that device current) and
// cached; the first call on each device performs that lookup.
#include <mutex>

#include "qk_internal.cuh"

namespace qk {

namespace {

// Largest gate/up intermediate (M x 2N elements of the model dtype) a call may use.
constexpr size_t kStaticScratchBytes = QK_STATIC_SCRATCH_BYTES;

__device__ __align__(256) unsigned char g_swiglu_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_swiglu_scratch on the current device (looked up once per device).
int scratch_address(int device, void** out) {
    if (device < 0 || device >= kMaxDevices)
        return set_error(QK_EINVAL, "device ordinal %d outside [0, %d)", device, kMaxDevices);
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_ptr[device]) {
        void* p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_swiglu_scratch);
        if (e != cudaSuccess) return cuda_error(e, "cudaGetSymbolAddress(static scratch)");
        g_scratch_ptr[device] = p;
    }
    *out = g_scratch_ptr[device];
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
    const size_t need = (size_t)M * 2 * N * m.es;
    if (need > kStaticScratchBytes)
        return set_error(QK_ESHAPE,
                         "gate/up intermediate of %zu bytes exceeds the static scratch of %zu bytes "
                         "(M x 2N x element size must be <= %zu)",
                         need, kStaticScratchBytes, kStaticScratchBytes);
    int device = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
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
