/*
 * qk_ops.h -- single steps of the libqk forward pass on caller buffers.
 *
 * These run exactly the kernels the model entry points of qk.h launch for the
 * same step, so each step can be checked against the oracle on its own (odd
 * shapes, several tiles, ragged tails).  Conventions as in qk.h: device
 * pointers, caller-owned memory, asynchronous on `stream`, QK_E* codes.
 */
#ifndef QK_OPS_H
#define QK_OPS_H

#include "qk.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Epilogues of qk_op_linear (values match the library's internal codes). */
#define QK_EPI_STORE 0     /* C (model dtype) = A W^T                                  */
#define QK_EPI_STORE_F32 1 /* C (fp32) = A W^T                                         */
#define QK_EPI_RESID_F32 2 /* C (fp32) += A W^T                                        */
#define QK_EPI_SWIGLU 3    /* C (model dtype) [M, N] = silu(A Wg^T) * (A Wu^T), where W  */
                           /* holds 2N rows: blocks of 128 gate rows, each followed by   */
                           /* the matching 128 up rows                                   */

/* One linear layer of the model's dtype (m supplies dtype, SM count and the
 * status word): A [M, K] (row stride lda elements), W [N, K] row-major ([2N, K]
 * for QK_EPI_SWIGLU), C [M, ldc].  This is the step the Qwen3 layer uses for its
 * QKV, output, gate/up and down projections and for the lm_head (logits =
 * W_lm h).  scratch: device buffer of M * 2N elements of the model dtype, needed
 * only for QK_EPI_SWIGLU on the fp32 model (else may be NULL and is ignored).  K must be a
 * multiple of 16, N of 128 for QK_EPI_SWIGLU.
 * Alignment (every path reads A and W with 8- or 16-byte vector loads): A and W
 * start on a 16-byte boundary and lda is a multiple of 16 bytes (8 bf16 or 4 fp32
 * elements), else QK_EINVAL / QK_ESHAPE; C is aligned to its element size (4 bytes
 * for the fp32 epilogues), else QK_EINVAL.  Nothing is launched on an error. */
int qk_op_linear(qk_model* m, const void* A, int lda, const void* W, void* C, int ldc, int M,
                 int N, int K, int epilogue, void* scratch, size_t scratch_bytes, void* stream);

/* The QK_EPI_SWIGLU linear step on the CUDA-core path (the one that stages the
 * [M, 2N] gate/up product in scratch before applying SwiGLU), for callers that
 * cannot hand the library a scratch buffer: e.g. a process that reserved its
 * whole device memory budget up front, or code embedded in a runtime that owns
 * the allocator and forbids side allocations.  The paper has no counterpart;
 * this is a service entry point of the library.
 *
 * It allocates nothing: the gate/up product lives in a file-scope device array
 * of QK_STATIC_SCRATCH_BYTES (8 MiB) that every GPU loading libqk holds until
 * the process exits.  Inputs and outputs are the caller's, as in qk_op_linear
 * with QK_EPI_SWIGLU: A [M, K] (row stride lda), W [2N, K] (128-row gate/up
 * blocks), C [M, N] with ldc == N, all in the model's dtype, with the alignment
 * rules of qk_op_linear.  The model's device must be the current device
 * (else QK_EINVAL).
 *  - Limit: M * 2N * element size must not exceed QK_STATIC_SCRATCH_BYTES;
 *    larger calls return QK_ESHAPE and launch nothing.
 *  - Set-up: the first call in each CUDA context looks up the array's device
 *    address (cudaGetSymbolAddress, with that device current) and caches it
 *    against the context (a context created again after cudaDeviceReset is
 *    looked up again); make that first call before any stream capture.
 *  - Sharing: every call on a device uses the same array and it keeps the last
 *    call's contents (each call overwrites all of the part it reads, so nothing
 *    needs clearing).  Calls that overlap on the GPU (other streams, other host
 *    threads) race on the array; serialise them. */
/* Test hook of the bounded-wait status path (a service call; the paper has no
 * counterpart).  Every wait of the library's kernels on a copy, an MMA or
 * another CTA is bounded: when one expires the kernel sets QK_STATUS_TIMEOUT,
 * waits (bounded) for its own copies in flight, frees its tensor memory and
 * returns, so the context stays usable.  After this call, the next plain
 * tensor-core GEMM launched for the model (qk_op_linear on a bf16 model with
 * M > 4 rows, a prefill / scoring linear, which then runs on the swap-AB kernel,
 * or a GEMM of qk_backward_logprob) lets its first CTA wait at most wait_cycles
 * SM cycles and issues no copy for that CTA's first k-block, so that CTA's wait
 * for it expires: its output (and what the call computes from it) is undefined,
 * QK_STATUS_TIMEOUT is set and qk_check_status returns QK_ETIMEOUT.  The hook
 * disarms at that launch.
 * wait_cycles in [1, 2^31]; QK_EINVAL otherwise. */
int qk_debug_expire_next_wait(qk_model* m, long long wait_cycles);

#define QK_STATIC_SCRATCH_BYTES (8u << 20)
int qk_op_linear_swiglu_static(qk_model* m, const void* A, int lda, const void* W, void* C,
                               int ldc, int M, int N, int K, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* QK_OPS_H */
