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
 * only for QK_EPI_SWIGLU on the fp32 model (else may be NULL).  K must be a
 * multiple of 16, N of 128 for QK_EPI_SWIGLU. */
int qk_op_linear(qk_model* m, const void* A, int lda, const void* W, void* C, int ldc, int M,
                 int N, int K, int epilogue, void* scratch, size_t scratch_bytes, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* QK_OPS_H */
