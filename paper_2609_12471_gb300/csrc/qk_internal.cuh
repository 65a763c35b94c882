// Internal declarations shared by the libqk translation units: the model
// object, error helpers, epilogue kinds and the kernel launchers.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include "qk.h"
#include "qk_ops.h"

namespace qk {

using bf16 = __nv_bfloat16;

// ---------------------------------------------------------------- errors
int set_error(int code, const char* fmt, ...);
int cuda_error(cudaError_t e, const char* what);
#define QK_TRY_CUDA(expr)                                   \
    do {                                                    \
        cudaError_t _e = (expr);                            \
        if (_e != cudaSuccess) return ::qk::cuda_error(_e, #expr); \
    } while (0)
#define QK_TRY(expr)              \
    do {                          \
        int _r = (expr);          \
        if (_r != QK_OK) return _r; \
    } while (0)

// ---------------------------------------------------------------- model
struct LayerW {
    float* attn_norm;
    float* q_norm;
    float* k_norm;
    float* mlp_norm;
    void* w_qkv;  // [(nq + 2 nkv) d, H]: rows of wq, then wk, then wv
    void* w_o;    // [H, nq d]
    void* w_gu;   // [2 I, H]: blocks of 128 gate rows followed by the matching 128 up rows
    void* w_d;    // [H, I]
};

struct Model {
    qk_config cfg;
    int es;  // bytes per element of the model dtype
    char* packed;
    size_t packed_bytes;
    uint32_t* status;  // device status word (QK_STATUS_* bits)
    float* rope_cos;   // [max_positions, d/2]
    float* rope_sin;
    void* embed;       // [V, H]
    std::vector<LayerW> layers;
    float* final_norm;
    void* lm_head;     // [V, H]
    int device;
    int num_sms;
    // Event bracketing of one kernel class during decode steps (qk_profile_begin).
    int prof_kind = -1;
    bool in_decode = false;
    std::vector<cudaEvent_t> prof_ev;
    int prof_used = 0;
    // First host-side failure of a launch inside an orchestration (0 = none);
    // reported and cleared by the entry point that made the launches.
    int deferred_error = 0;
};

// Records the opening event of a bracketed launch; returns whether it did.
bool prof_open(Model& m, int kind, cudaStream_t s);
void prof_close(Model& m, bool opened, cudaStream_t s);
// Counts kernel launches (qk_launch_count).
void note_launch(int n = 1);

// Byte offsets of every packed region (shared by the size query and the loader).
struct PackedLayout {
    size_t status, rope_cos, rope_sin, embed, final_norm, lm_head, total;
    struct L {
        size_t attn_norm, q_norm, k_norm, mlp_norm, w_qkv, w_o, w_gu, w_d;
    };
    std::vector<L> layers;
};
int packed_layout(const qk_config& c, PackedLayout* out);
int validate_config(const qk_config& c);

// ---------------------------------------------------------------- kernels
enum Epi : int {
    EPI_STORE_ACT = 0,   // C (model activation dtype, ldc) = acc
    EPI_STORE_F32 = 1,   // C (fp32, ldc) = acc
    EPI_RESID_F32 = 2,   // C (fp32, ldc) += acc
    EPI_SWIGLU = 3,      // W holds gate/up blocks of 128 rows; C[m, j] = silu(gate) * up, N = I
};

// Token id of flattened row r: tokens[(r / T) * ld + off + r % T].
struct TokIndex {
    const int32_t* ptr;
    int T, ld, off;
};

// Position of flattened row r: pos_dev ? pos_dev[r / T] + r % T : start + r % T.
struct PosIndex {
    const int32_t* pos_dev;
    int start, T;
};

// Where the log-prob / argmax of flattened logits row r goes.  b = r / T, t = r % T;
// the row is skipped when t >= out_lim; target = tgt[b * tgt_ld + tgt_off + t];
// outputs at index b * out_ld + out_off + t.
// Rows are numbered from row0 (a chunk of a larger set of rows).
struct OutIndex {
    int T, out_lim, out_ld, out_off;
    const int32_t* tgt;
    int tgt_ld, tgt_off, row0;
};

void launch_embed(const void* E, int dtype, int V, int H, TokIndex tok, int M, float* x,
                  uint32_t* status, cudaStream_t s);
// out[r] = x[r * in_step + in_off] * rsqrt(mean(x^2) + eps) * g, stored in out_dtype.
void launch_rmsnorm(const float* x, int in_step, int in_off, const float* g, int H, float eps,
                    void* out, int out_dtype, int M, cudaStream_t s);
// Per-head RMSNorm of q and k, RoPE of q and k, q written in place, k and v to the cache.
void launch_qk_norm_rope(void* qkv, int dtype, int M, int nq, int nkv, int d, const float* gq,
                         const float* gk, float eps, const float* rope_cos, const float* rope_sin,
                         int max_positions, PosIndex pos, void* k_cache, void* v_cache,
                         int max_seq, uint32_t* status, cudaStream_t s);
void launch_swiglu(const void* gu, void* h, int dtype, int M, int I, cudaStream_t s);
void launch_logits_reduce(const float* logits, int M, int V, OutIndex oi, float* lp,
                          int32_t* argmax, uint32_t* status, cudaStream_t s);
void launch_rope_table(float* cos_t, float* sin_t, int max_positions, int d, double theta,
                       cudaStream_t s);
void launch_widen_gain(const void* src, int dtype, float* dst, int n, cudaStream_t s);

// Attention.  q rows of q_ld elements holding nq heads of d (row r = b * T + t),
// caches [B_max, nkv, max_seq, d] of one layer; row r attends cache positions
// 0 .. pos(r) inclusive; o [M, nq * d].
void launch_attention_simt(const void* q, int q_ld, const void* k_cache, const void* v_cache,
                           int dtype, int M, int nq, int nkv, int d, int max_seq, PosIndex pos,
                           void* o, uint32_t* status, cudaStream_t s);

// GEMMs: C[M, N] = A[M, K] * W[N, K]^T with an epilogue (see Epi).
void launch_gemm_simt(const void* A, int lda, const void* W, void* C, int ldc, int M, int N,
                      int K, int dtype, int epi, cudaStream_t s);
void launch_gemv_bf16(const bf16* A, int lda, const bf16* W, void* C, int ldc, int M, int N,
                      int K, int epi, cudaStream_t s);
// tcgen05 path (k_gemm_tc.cu): N % 128 == 0, K % 64 == 0, A 16-byte aligned, lda % 8 == 0.
bool gemm_tc_supported(const void* A, int lda, int N, int K);
int launch_gemm_tc(const bf16* A, int lda, const bf16* W, void* C, int ldc, int M, int N, int K,
                   int epi, int num_sms, uint32_t* status, cudaStream_t s);

// Kernel selection (k_dispatch.cu).  linear: C = A W^T with epilogue `epi`; for
// EPI_SWIGLU, N is the SwiGLU width I and W holds 2 I interleaved rows; `gu` is
// scratch [M, 2 I] for paths that cannot fuse the SwiGLU epilogue.
void linear(Model& m, const void* A, int lda, const void* W, void* C, int ldc, int M, int N,
            int K, int epi, void* gu, cudaStream_t s);
void launch_attention(const Model& m, const void* q, int q_ld, const void* k_cache,
                      const void* v_cache, int M, int max_batch, int max_seq, PosIndex pos,
                      void* o, cudaStream_t s);

}  // namespace qk
