// Internal declarations shared by the libqk translation units: the model
// object, error helpers, epilogue kinds and the kernel launchers.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>
#include <vector>

#include "qk.h"
#include "qk_ops.h"

namespace qk {

using bf16 = __nv_bfloat16;

// Programmatic dependent launch: a kernel launched with launch_k may start while
// the previous kernel on the stream is still running; it must execute
// pdl_wait() before its first global-memory access (read or write) that can
// depend on or conflict with earlier kernels.  Launched normally, pdl_wait() is
// a no-op.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Lets the next kernel on the stream be scheduled (its pdl_wait still waits for this one to finish).
__device__ __forceinline__ void pdl_trigger() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
inline void launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                     Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// bf16 linear layers over at most this many token rows stream the weights through
// the CUDA-core GEMV (fused epilogues); larger ones run on the tensor cores.
constexpr int kGemvMaxRows = 4;

// ---------------------------------------------------------------- errors
int set_error(int code, const char* fmt, ...);
int cuda_error(cudaError_t e, const char* what);
struct Model;
// Host check of the operands of a caller-facing linear step (qk_op_linear and its
// static-scratch variant): A and W must start on a 16-byte boundary, lda must keep
// every row of A on one (a multiple of 8 bf16 / 4 fp32 elements), and C must be
// aligned to its element size (out_es bytes).  The CUDA-core, GEMV and tcgen05
// kernels all read A and W with 8- or 16-byte vector loads.
int check_linear_operands(const Model& m, const void* A, int lda, const void* W, const void* C,
                          int out_es);
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

// Temperature sampling of rollout tokens by the Gumbel-max rule: a kernel that forms
// a row's logits z draws c = argmax_v (z_v / tau + G(seed, row, step, v)) and reports
// log softmax(z / tau)[c]; out_tokens == nullptr disables it.
struct SampleArgs {
    unsigned long long seed;
    float inv_tau;
    int32_t* out_tokens;  // written at the same index as the log-prob
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
    // Instantiated decode-step graphs of qk_rollout_teacher_forced, keyed by the call's
    // pointers and sizes (every kernel parameter of a step is fixed by them).
    struct StepGraph {
        uint64_t key[17];
        cudaGraphExec_t exec;
        int kernels;  // kernel nodes of one step (for the launch counter)
    };
    std::vector<StepGraph> graphs;
    // Library-owned stream on which step graphs are captured (capture records only;
    // the graphs are launched on the caller's stream).  Created on first use.
    cudaStream_t capture_stream = nullptr;
    // First host-side failure of a launch inside an orchestration (0 = none);
    // reported and cleared by the entry point that made the launches.
    int deferred_error = 0;
    SampleArgs sampling{};  // set only while a sampled rollout runs
    // qk_debug_expire_next_wait: wait limit (SM cycles) of the next plain tcgen05 GEMM
    // launch, which then skips one copy so that the wait expires; 0 = off.
    long long test_wait_cycles = 0;
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
    EPI_PARTIAL_F32 = 4, // split-K unit s writes its fp32 partial to C[s][m][n] (ldc = N)
    EPI_LSE = 5,         // lm_head: per (token row, 128-entry vocabulary tile) the max, sum of
                         // exponentials and lowest arg-max of the logits, and the target's logit
                         // (Fuse::lse_*); no logits are stored
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

// Where a layer's cache keeps the keys and values of row b's positions.  Each of a
// layer's K and V is a pool of n_pages pages, [n_pages, nkv, page, d]; position p of
// row b sits at offset p % page of page table[b * per_row + p / page].  A dense cache
// [max_batch, nkv, max_seq, d] is the same with one page per row: table null, page b,
// page = max_seq, per_row = 1.  A row holds per_row * page positions (cap()).
struct KvPages {
    const int32_t* table;  // device [rows, per_row] page ids, or null (dense)
    int per_row;
    int n_pages;
    int page;
    __host__ __device__ int cap() const { return per_row * page; }
    static KvPages dense(int max_batch, int max_seq) { return KvPages{nullptr, 1, max_batch, max_seq}; }
};

// Row index, in the 2-D view [n_pages nkv page, d] of a layer's K (or V), of position
// p of (row b, kv head g).  A page id outside [0, n_pages) sets QK_STATUS_BAD_PAGE (when
// status is given) and reads page 0.
__device__ __forceinline__ int kv_row(const KvPages& kp, int nkv, int b, int g, int p,
                                      uint32_t* status) {
    int pg = b, off = p;
    if (kp.table) {
        pg = kp.table[(size_t)b * kp.per_row + p / kp.page];
        off = p % kp.page;
        if ((unsigned)pg >= (unsigned)kp.n_pages) {
            if (status) atomicOr(status, QK_STATUS_BAD_PAGE);
            pg = 0;
        }
    }
    return (pg * nkv + g) * kp.page + off;
}

// Where the log-prob / argmax of flattened logits row r goes.  b = r / T, t = r % T;
// the row is skipped when t >= out_lim; target = tgt[b * tgt_ld + tgt_off + t];
// outputs at index b * out_ld + out_off + t.
// Rows are numbered from row0 (a chunk of a larger set of rows).  With dyn_off set,
// *dyn_off (read on the device) is added to the output index.
struct OutIndex {
    int T, out_lim, out_ld, out_off;
    const int32_t* tgt;
    int tgt_ld, tgt_off, row0;
    const int32_t* dyn_off = nullptr;
};

void launch_embed(const void* E, int dtype, int V, int H, TokIndex tok, int M, float* x,
                  uint32_t* status, cudaStream_t s);
// out[r] = x[r * in_step + in_off] * rsqrt(mean(x^2) + eps) * g, stored in out_dtype.
// With row_len, row r reads x[r * in_step + row_len[r] - 1] instead (per-row last token).
void launch_rmsnorm(const float* x, int in_step, int in_off, const float* g, int H, float eps,
                    void* out, int out_dtype, int M, cudaStream_t s,
                    const int32_t* row_len = nullptr);
// Per-head RMSNorm of q and k, RoPE of q and k, q written in place, k and v to the cache.
void launch_qk_norm_rope(void* qkv, int dtype, int M, int nq, int nkv, int d, const float* gq,
                         const float* gk, float eps, const float* rope_cos, const float* rope_sin,
                         int max_positions, PosIndex pos, void* k_cache, void* v_cache,
                         const KvPages& kp, uint32_t* status, cudaStream_t s);
void launch_swiglu(const void* gu, void* h, int dtype, int M, int I, cudaStream_t s);
// GRPO token loss (Sec. "GRPO Optimization"): inputs and output of Eq. ppo for the
// tokens whose log-prob a kernel forms; loss_tok == nullptr disables it.
struct GrpoArgs {
    const float* lp_old;
    const float* lp_ref;   // may be null when beta == 0
    const float* rewards;  // [B]
    const uint8_t* mask;   // [B, ld] or null (all ones)
    float* loss_tok;       // [B, ld]
    int group, ld;
    float eps_low, eps_high, beta;
};

// Eq. advantage: A_b = r_b - mean of r over b's group (summed in row order).
__device__ __forceinline__ float grpo_advantage(const float* rewards, int b, int group) {
    const int g0 = b - b % group;
    float s = 0.f;
    for (int i = 0; i < group; ++i) s += rewards[g0 + i];
    return rewards[b] - s / (float)group;
}

// Eq. ppo for one token: -min(rho A, clip(rho, 1 - eps_low, 1 + eps_high) A) + beta k3,
// rho = exp(lp - lp_old), k3 = e^x - x - 1 with x = lp_ref - lp (as expm1(x) - x).
__device__ __forceinline__ float grpo_token(float lp, float lp_old, float lp_ref, float A,
                                            const GrpoArgs& g) {
    const float rho = expf(lp - lp_old);
    const float clipped = fminf(fmaxf(rho, 1.f - g.eps_low), 1.f + g.eps_high);
    float L = -fminf(rho * A, clipped * A);
    if (g.beta != 0.f) {
        const float x = lp_ref - lp;
        L += g.beta * (expm1f(x) - x);
    }
    return L;
}

void launch_logits_reduce(const float* logits, int M, int V, OutIndex oi, float* lp,
                          int32_t* argmax, uint32_t* status, cudaStream_t s,
                          const GrpoArgs* grpo = nullptr, const SampleArgs* samp = nullptr);
// GRPO reductions (k_grpo.cu).  With `compute`, loss_tok is formed from lp (else it
// was formed by the scoring epilogue); then per-row sums of mask * loss and of the
// mask go to `rows` ([B] float2) and loss_mean (if not null) = their ratio.
size_t grpo_scratch_bytes(int B);
void launch_grpo_loss(const float* lp, int B, int T, const GrpoArgs& g, bool compute,
                      void* scratch, float* loss_mean, cudaStream_t s);
// Per-token coefficients of the GRPO gradient (after launch_grpo_loss filled `scratch`):
// coef = -mask * (d loss_tok / d lp) / sum(mask), same indexing as lp.
void launch_grpo_coef(const float* lp, int B, int T, const GrpoArgs& g, const void* scratch, float* coef,
                      cudaStream_t s);
// Workspace of qk_backward_logprob (qk_backward.cu).
int backward_workspace_bytes(const Model& m, int B, int T, size_t* bytes);
// Rollout cursor: s = *step; pos[b] = P + s; tok[b] = seq[b, P + s]; tgt[b] = seq[b, P + s + 1];
// *out_off = s + 1; *step = s + 1.
void launch_rollout_prepare(const int32_t* seq, int L, int P, int B, int32_t* step, int32_t* pos,
                            int32_t* tok, int32_t* tgt, int32_t* out_off, cudaStream_t s);
// Sampled rollout cursor: s = *step; pos[b] = P + s; tok[b] = sampled[b * ld + s];
// *out_off = s + 1; *step = s + 1.
void launch_rollout_prepare_sampled(const int32_t* sampled, int ld, int P, int B, int32_t* step,
                                    int32_t* pos, int32_t* tok, int32_t* out_off, cudaStream_t s);
void launch_rope_table(float* cos_t, float* sin_t, int max_positions, int d, double theta,
                       cudaStream_t s);
void launch_widen_gain(const void* src, int dtype, float* dst, int n, cudaStream_t s);

// Attention.  q rows of q_ld elements holding nq heads of d (row r = b * T + t),
// one layer's caches laid out as kp says; row r attends cache positions 0 .. pos(r)
// inclusive; o [M, nq * d].
void launch_attention_simt(const void* q, int q_ld, const void* k_cache, const void* v_cache,
                           int dtype, int M, int nq, int nkv, int d, const KvPages& kp, PosIndex pos,
                           void* o, uint32_t* status, cudaStream_t s);

// GEMMs: C[M, N] = A[M, K] * W[N, K]^T with an epilogue (see Epi).
void launch_gemm_simt(const void* A, int lda, const void* W, void* C, int ldc, int M, int N,
                      int K, int dtype, int epi, cudaStream_t s);
void launch_gemv_bf16(const bf16* A, int lda, const bf16* W, void* C, int ldc, int M, int N,
                      int K, int epi, cudaStream_t s);
// tcgen05 path (k_gemm_tc.cu): N % 128 == 0, K % 64 == 0, A 16-byte aligned, lda % 8 == 0.
bool gemm_tc_supported(const void* A, int lda, int N, int K);
struct Fuse;
// test_wait > 0: bounded-wait test launch (CTA 0 skips its first copy and gives up
// after test_wait SM cycles; the output is undefined and QK_STATUS_TIMEOUT is set).
int launch_gemm_tc(const bf16* A, int lda, const bf16* W, void* C, int ldc, int M, int N, int K,
                   int epi, int num_sms, uint32_t* status, cudaStream_t s, long long test_wait = 0,
                   const Fuse* lse = nullptr);
// Combines the EPI_LSE partials of M logits rows over n_vt vocabulary tiles into the
// log-prob of each row's target, its arg-max and (grpo) its GRPO token loss, with the
// output indexing of launch_logits_reduce (k_misc.cu).
void launch_lse_combine(const float2* ms, const int* idx, const float* zt, int n_vt, int V, int M,
                        OutIndex oi, float* lp, int32_t* argmax, uint32_t* status, cudaStream_t s,
                        const GrpoArgs* grpo = nullptr);

// Fused epilogue of a decode-sized linear (one token tile, M <= 64 rows).  The
// N/128 x K/64 k-block iterations are split evenly over the CTAs; a CTA that holds
// only part of a tile's k range writes its fp32 partial [M][128] to slot (CTA +
// tile) of `part` and takes the tile's ticket, and the last of them (the last of a
// gate/up tile pair for FUSE_SWIGLU, whose halves always go through `part`) sums
// the slots in k order and applies `op`.  `part` holds gemm_fused_part_floats()
// floats, `tickets` N/128 ints (zero on entry, zero again on exit).  The linear's input is x * g (bf16, not yet
// normalised); the RMSNorm scale s_m = rsqrt(sum_t ssq_in[t][m] / H + eps) of
// token row m is applied after the product (W (x g s) = s W (x g)).
enum FuseOp : int {
    FUSE_NONE = 0,
    FUSE_QKV = 1,       // tile = one head: s, per-head RMSNorm + RoPE for q/k, q -> q_out, k/v -> cache
    FUSE_RESID = 2,     // x += sum; xg_out = bf16(x * g_next); ssq_out[tile][m] = sum of x^2 over the tile
    FUSE_SWIGLU = 3,    // tiles 2j (gate) and 2j+1 (up): h[m, 128 j + r] = silu(s g) * (s u)
    FUSE_COLSCALE = 4,  // fp32 store of s_m * (x g W^T)[m, n] (lm_head logits)
};

struct Fuse {
    int op;
    int* tickets;
    float* part;
    const float* ssq_in;  // [n_ssq][M]
    int n_ssq, H;
    float eps;
    // FUSE_QKV
    int nq, nkv;
    const float* gq;
    const float* gk;
    const float* rope_cos;
    const float* rope_sin;
    int max_positions;
    PosIndex pos;
    bf16* q_out;
    int q_ld;
    bf16* k_cache;
    bf16* v_cache;
    KvPages kv;
    uint32_t* status;
    // FUSE_RESID
    float* x;
    const float* g_next;
    bf16* xg_out;
    float* ssq_out;
    // FUSE_SWIGLU
    bf16* h_out;
    // EPI_LSE (plain tcgen05 GEMM over the lm_head): token row m of the launch is
    // global row g = lse_row0 + m of tokens [., lse_T]; its target is tokens[g + 1]
    // when g % lse_T < lse_T - 1 (an id outside [0, V) counts as 0).  Outputs per
    // (row, vocabulary tile v): lse_ms[m * n_vt + v] = (max, sum exp(z - max)),
    // lse_idx[...] = lowest index of the max; lse_zt[m] = the target's logit.
    float2* lse_ms;
    int* lse_idx;
    float* lse_zt;
    const int32_t* lse_tok;
    int lse_T, lse_row0;
};

// Decode linear with a fused epilogue (k_gemm_tc.cu): A = bf16 [M, K] (M <= 64),
// W [N, K]; out is the op's fp32 logits for FUSE_COLSCALE, unused otherwise.
int launch_gemm_tc_fused(const bf16* A, int lda, const bf16* W, float* out, int M, int N, int K,
                         const Fuse& f, int num_sms, uint32_t* status, cudaStream_t s);
inline size_t gemm_fused_part_floats(int M, int N, int num_sms) {
    return ((size_t)num_sms + (size_t)(N / 128)) * (size_t)M * 128;
}
// x = E[token] (embed) or the given x; xg = bf16(x * g); ssq[t][m] = sum over features
// 128 t .. 128 t + 127 of x^2 (k_misc.cu).
void launch_embed_gain(const void* E, int V, TokIndex tok, bool do_embed, float* x, const float* g,
                       bf16* xg, float* ssq, int M, int H, uint32_t* status, cudaStream_t s);

// Kernel selection (k_dispatch.cu).  linear: C = A W^T with epilogue `epi`; for
// EPI_SWIGLU, N is the SwiGLU width I and W holds 2 I interleaved rows; `gu` is
// scratch [M, 2 I] for paths that cannot fuse the SwiGLU epilogue.
void linear(Model& m, const void* A, int lda, const void* W, void* C, int ldc, int M, int N,
            int K, int epi, void* gu, cudaStream_t s);
// Decode rows (pos.T == 1) of a bf16 model go to the split tensor-core kernel,
// whose partials use `scratch` (attn_decode_scratch_bytes); other cases run the
// SIMT kernel.
void launch_attention(Model& m, const void* q, int q_ld, const void* k_cache, const void* v_cache,
                      int M, const KvPages& kp, PosIndex pos, void* o, void* scratch,
                      cudaStream_t s);
// Causal tensor-core attention for prefill / scoring (k_attn_prefill.cu): M = B x T
// query rows at positions start_b .. start_b+T-1, start_b = start_dev[b] when given,
// else start; head_dim 128.
bool attn_prefill_supported(int d, int nq, int nkv);
// lse (may be null): [B, nq, T] natural-log log-sum-exp of each row's scaled scores.
int launch_attn_prefill(const bf16* q, int q_ld, const void* k_layer, int nq, int nkv,
                        const KvPages& kp, int B, int T, int start,
                        const int32_t* start_dev, bf16* o, int num_sms, uint32_t* status,
                        cudaStream_t s, float* lse = nullptr);
// Fused causal attention backward on tcgen05 (k_attn_bwd.cu): head_dim 128, T % 128 == 0.
// q, dO [B T, nq d] bf16; kvh [2][B][nkv][T][d] bf16 (K then V); lse, D [B nq T] fp32;
// dq [B T, nq d] fp32 (zero on entry: added into); dk [B T, nkv d] fp32; dv at columns
// dv_col0 .. of dv_base [B T, dv_ld] bf16.
bool attn_bwd_supported(int d, int nq, int nkv, int T);
int launch_attn_bwd(const bf16* q, const bf16* dO, const bf16* kvh, const float* lse, const float* D,
                    float* dq, float* dk, bf16* dv_base, int dv_ld, int dv_col0, int B, int T, int nq, int nkv,
                    int num_sms, uint32_t* status, cudaStream_t s);
// Split tensor-core decode attention (k_attn_decode.cu); head_dim 128, G <= 8.
void attn_decode_split(int B, int nkv, int max_seq, int num_sms, int* chunk, int* n_split);
size_t attn_decode_scratch_bytes(int B, int nq, int nkv, int max_seq, int num_sms);
// Merge tickets inside that scratch; zero them (B * nkv ints) before a decode step.
int* attn_decode_tickets(void* scratch, int B, int nq, int nkv, int max_seq, int num_sms);
// The partial, (m, l) and ticket regions of that scratch.
void attn_scratch_parts(void* scratch, int B, int nq, int nkv, int max_seq, int num_sms, int n_split,
                        float** part_o, float2** part_ml, int** tickets);
// 3-D TMA map over `layers` layers' K / V caches (k_layer0 = layer 0's K, layer stride
// layer_bytes; ignored for one layer), each layer's K then V pools laid out as kp says.
bool make_kv_map(CUtensorMap* map, const void* k_layer0, const KvPages& kp, int nkv, int layers,
                 size_t layer_bytes);
bool attn_decode_supported(int d, int nq, int nkv);
int launch_attn_decode(const bf16* q, int q_ld, const void* k_layer, int nq, int nkv,
                       const KvPages& kp, int B, PosIndex pos, void* scratch, bf16* o,
                       int num_sms, uint32_t* status, cudaStream_t s);

}  // namespace qk
