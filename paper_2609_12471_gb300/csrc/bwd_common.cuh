// Backward pass of the decoder (gradient of the token-weighted log-likelihood of
// Eq. sft; with GRPO coefficients, of Eq. ppo): the batched GEMM descriptors and
// the epilogue arithmetic shared by the tcgen05 GEMM (bf16 models) and its
// CUDA-core twin (fp32 models), so that both paths run the same epilogue code.
//
// Every product of the backward pass is one batched GEMM
//     D_z[m, n] = sum_k A_z[m, k] B_z[n, k],   z < Z, m < M, n < N, k in the tile's range,
// whose operands are addressed by Op (below) inside row-major 2-D buffers, so that
// attention heads, GQA groups and the transposed operands of dX = dY W and
// dW = dY^T X need no copies: a batch index picks a (row, column) offset, an
// operand is K-major (k along the row) or MN-major (m or n along the row), and a
// reduction may run over several heads of a group (kwrap).
#pragma once

#include "qk_internal.cuh"

namespace qk {
namespace bwd {

// Element (z, i, k) of an operand (i = m for A, n for B):
//   z1 = z / zdiv;  x0 = xb + (z1 % zq) * zx;  y0 = yb + (z1 / zq) * zy
//   kwrap > 0: s = k / kwrap, kk = k % kwrap;  else s = 0, kk = k
//   ic = (i / 128) * pitch + i % 128
//   mn:      column x0 + ic + s * kwx, row y0 + kk + s * kwy
//   k-major: column x0 + kk + s * kwx, row y0 + ic + s * kwy
// of the buffer ptr [rows, cols] with row stride ld elements.
struct Op {
    const void* ptr;
    long long ld;
    int rows, cols;
    int mn;
    int xb, yb;
    int zdiv, zq, zx, zy;
    int kwrap, kwx, kwy;
    int pitch;
};

// Output element (z, m, n) is C[(z / zq) * zrow + m, (z % zq) * zcol + n] of the buffer
// C [rows, cols] (row stride ldc).
struct Out {
    void* C;
    long long ldc;
    int rows, cols;
    int zq, zrow, zcol;
    const float* addend;  // E_F32: C = addend + acc, addend indexed like C (may be C itself)
};

enum Mode : int {
    E_F32 = 0,      // fp32 store of acc (plus addend)
    E_ACT = 1,      // store in the activation type
    E_STATS = 2,    // per (row, column tile): max and sum of exp over the unmasked t = scale * acc,
                    // and the target column's t (no matrix is stored)
    E_SOFTMAX = 3,  // (exp(scale * acc - lse_row) - [n == tgt_row]) * w_row; masked entries 0
    E_DS = 4,       // P * (acc - D_row) * scale, P read from a buffer laid out like C
    E_SWIGLU_BWD = 5,  // acc = dh[m, n] of h = silu(g) u: with (g, u) read from gu (the packed
                       // [M, 2 I] gate / up layout, row stride ldc), writes dg and du into C
                       // (laid out like gu) at the gate and up columns of n
    E_SWIGLU_FWD = 6,  // acc = [gate | up] of a 256-column tile of the packed gate / up product:
                       // C[m, 128 t + c] = bf16(silu(gate c) up c)  (tensor-core path, 256-row tiles)
};

// Row vectors (lse, w, tgt, zt, D, stats) are indexed r = z * rows_per_z + m.
struct Epi {
    int mode;
    float scale;
    int causal;        // column n > row m is masked (E_STATS, E_SOFTMAX)
    int rows_per_z;
    const float* lse;  // E_SOFTMAX
    const float* w;    // E_SOFTMAX row weight (null: 1)
    const int* tgt;    // E_STATS capture / E_SOFTMAX one-hot: target column, < 0 none (null: none)
    float* zt;         // E_STATS: t at the target column
    float2* stats;     // E_STATS: [r][n_ct]
    int n_ct;
    const void* P;     // E_DS; E_SWIGLU_BWD: gu
    const float* D;    // E_DS
};

// Tile schedule of one launch (per batch entry z: M x N outputs in BM x BN tiles).
enum Red : int {
    RED_FULL = 0,    // k < K
    RED_PREFIX = 1,  // k < min(K, m0 + BM): causal keys of a query tile
    RED_SUFFIX = 2,  // in each of K / seg segments, offsets m0 .. seg - 1: causal queries of a key tile
};
struct Sched {
    int Z, M, N, K;
    int red, seg;
    int tri;     // only tiles with n0 < m0 + BM (the others are fully masked); needs BM == BN
    int desc_m;  // m tiles in descending order (heaviest first under RED_PREFIX)
};

__host__ __device__ __forceinline__ int cdiv(int a, int b) { return (a + b - 1) / b; }

// Tiles of one batch entry.
__host__ __device__ __forceinline__ long long tiles_per_z(const Sched& s, int BM, int BN) {
    const int nm = cdiv(s.M, BM), nn = cdiv(s.N, BN);
    if (!s.tri) return (long long)nm * nn;
    long long t = 0;
    for (int i = 0; i < nm; ++i) t += (i + 1 < nn ? i + 1 : nn);
    return t;
}

constexpr int kGroupM = 16;

// Tile t of the launch -> (z, m tile, n tile).
__device__ __forceinline__ void tile_at(const Sched& s, int BM, int BN, long long per, long long t,
                                        int& z, int& mt, int& nt) {
    z = (int)(t / per);
    long long r = t - (long long)z * per;
    const int nm = cdiv(s.M, BM), nn = cdiv(s.N, BN);
    if (s.tri) {  // row i holds i + 1 tiles (nn == nm)
        int i = (int)((sqrtf(8.f * (float)r + 1.f) - 1.f) * 0.5f);
        while ((long long)(i + 1) * (i + 2) / 2 <= r) ++i;
        while ((long long)i * (i + 1) / 2 > r) --i;
        mt = i;
        nt = (int)(r - (long long)i * (i + 1) / 2);
    } else {
        // groups of kGroupM m tiles: within a group the m tile runs fastest, so a wave of
        // concurrent tiles touches a few n tiles of B and at most kGroupM m tiles of A
        // (both L2-resident) instead of streaming one operand from DRAM each wave
        const long long gsz = (long long)kGroupM * nn;
        const int g = (int)(r / gsz);
        const long long loc = r - (long long)g * gsz;
        const int gm = nm - g * kGroupM < kGroupM ? nm - g * kGroupM : kGroupM;
        mt = g * kGroupM + (int)(loc % gm);
        nt = (int)(loc / gm);
        if (s.desc_m) mt = nm - 1 - mt;
    }
}

// Reduction blocks of BK of a tile whose first row is m0; block j covers [k0, k0 + BK)
// clipped to its valid range [k0, kend).
__device__ __forceinline__ int kblocks(const Sched& s, int BM, int BK, int m0) {
    if (s.red == RED_FULL) return cdiv(s.K, BK);
    if (s.red == RED_PREFIX) {
        const int lim = s.K < m0 + BM ? s.K : m0 + BM;
        return cdiv(lim, BK);
    }
    const int per = s.seg > m0 ? cdiv(s.seg - m0, BK) : 0;
    return (s.K / s.seg) * per;
}
__device__ __forceinline__ void kblock_at(const Sched& s, int BM, int BK, int m0, int j, int& k0,
                                          int& kend) {
    if (s.red == RED_FULL) {
        k0 = j * BK;
        kend = s.K;
    } else if (s.red == RED_PREFIX) {
        k0 = j * BK;
        kend = s.K < m0 + BM ? s.K : m0 + BM;
    } else {
        const int per = cdiv(s.seg - m0, BK);
        const int sg = j / per;
        k0 = sg * s.seg + m0 + (j - sg * per) * BK;
        kend = (sg + 1) * s.seg;
    }
}

__device__ __forceinline__ void op_xy(const Op& o, int z, int i, int k, int& x, int& y) {
    const int z1 = z / o.zdiv;
    const int x0 = o.xb + (z1 % o.zq) * o.zx, y0 = o.yb + (z1 / o.zq) * o.zy;
    int s = 0, kk = k;
    if (o.kwrap) {
        s = k / o.kwrap;
        kk = k - s * o.kwrap;
    }
    const int ic = (i >> 7) * o.pitch + (i & 127);
    if (o.mn) {
        x = x0 + ic + s * o.kwx;
        y = y0 + kk + s * o.kwy;
    } else {
        x = x0 + kk + s * o.kwx;
        y = y0 + ic + s * o.kwy;
    }
}

__device__ __forceinline__ float ld_act(const float* p) { return *p; }
__device__ __forceinline__ float ld_act(const bf16* p) { return __bfloat162float(*p); }
__device__ __forceinline__ void st_act(float* p, float v) { *p = v; }
__device__ __forceinline__ void st_act(bf16* p, float v) { *p = __float2bfloat16_rn(v); }

// Element offset of output (z, m, n) in C.
__device__ __forceinline__ size_t out_offset(const Out& o, int z, int m, int n) {
    const size_t row = (size_t)(z / o.zq) * o.zrow + m;
    return row * (size_t)o.ldc + (size_t)(z % o.zq) * o.zcol + n;
}

constexpr float kLog2e = 1.4426950408889634f;
// 2^x on the special-function unit (relative error about 2^-22; 2^-inf = 0).
__device__ __forceinline__ float exp2f_fast(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

struct RowStat {
    float mx, sm;
};

__device__ __forceinline__ void stat_merge(RowStat& a, float m2, float s2) {
    if (s2 == 0.f) return;
    if (a.sm == 0.f) {
        a.mx = m2;
        a.sm = s2;
        return;
    }
    const float mx = fmaxf(a.mx, m2);
    a.sm = a.sm * expf(a.mx - mx) + s2 * expf(m2 - mx);
    a.mx = mx;
}

// Epilogue values of nv <= 16 consecutive outputs (z, m, n .. n + nv - 1) from the
// accumulators v: E_STATS updates st and returns false (nothing to store); the other
// modes fill y (E_SWIGLU_BWD: y and y2, for the gate and up columns) and return true.
// VEC: nv == 16 and every address 16-byte aligned.
template <typename act_t, bool VEC, int MODE>
__device__ __forceinline__ bool epi_values(const Epi& e, const Out& o, int z, int m, int n, int nv,
                                           const float (&v)[16], RowStat& st, float (&y)[16],
                                           float (&y2)[16]) {
    const int r = z * e.rows_per_z + m;
    if constexpr (MODE == E_STATS) {
        float t[16];
        float cmax = -INFINITY;
        const int tg = e.tgt ? e.tgt[r] : -1;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const bool ok = j < nv && !(e.causal && n + j > m);
            t[j] = ok ? v[j] * e.scale : -INFINITY;
            cmax = fmaxf(cmax, t[j]);
            if (ok && n + j == tg) e.zt[r] = t[j];
        }
        if (cmax == -INFINITY) return false;
        // e^(t - cmax) = 2^((t - cmax) log2 e); masked entries give 2^-inf = 0
        const float c2 = cmax * kLog2e;
        float cs = 0.f;
#pragma unroll
        for (int j = 0; j < 16; ++j) cs += exp2f_fast(fmaf(t[j], kLog2e, -c2));
        stat_merge(st, cmax, cs);
        return false;
    }
    const size_t off = out_offset(o, z, m, n);
    if constexpr (MODE == E_F32 || MODE == E_ACT) {
#pragma unroll
        for (int j = 0; j < 16; ++j) y[j] = v[j];
        if (MODE == E_F32 && o.addend) {
            const float* a = o.addend + off;
            if constexpr (VEC) {
#pragma unroll
                for (int j = 0; j < 16; j += 4) {
                    const float4 q = *(const float4*)(a + j);
                    y[j] += q.x, y[j + 1] += q.y, y[j + 2] += q.z, y[j + 3] += q.w;
                }
            } else {
                for (int j = 0; j < nv; ++j) y[j] += a[j];
            }
        }
    } else if constexpr (MODE == E_SOFTMAX) {
        // e^(scale acc - lse) = 2^(acc scale log2 e - lse log2 e)
        const float l2 = e.lse[r] * kLog2e, c = e.scale * kLog2e;
        const float w = e.w ? e.w[r] : 1.f;
        const int tg = e.tgt ? e.tgt[r] : -1;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const bool masked = e.causal && n + j > m;
            const float p = masked ? 0.f : exp2f_fast(fmaf(v[j], c, -l2));
            y[j] = (p - (n + j == tg ? 1.f : 0.f)) * w;
        }
    } else if constexpr (MODE == E_SWIGLU_BWD) {
        // gate of column n at packed column (n / 128) 256 + n % 128, up 128 further;
        // y = dg, y2 = du
        const size_t go = (size_t)m * o.ldc + (size_t)(n >> 7) * 256 + (n & 127);  // one batch entry
        const act_t* G = (const act_t*)e.P + go;
        float gv[16], uv[16];
        if constexpr (VEC && sizeof(act_t) == 2) {
            const uint4 q0 = *(const uint4*)G, q1 = *(const uint4*)(G + 8);
            const uint4 u0 = *(const uint4*)(G + 128), u1 = *(const uint4*)(G + 136);
            const bf16* a0 = (const bf16*)&q0;
            const bf16* a1 = (const bf16*)&q1;
            const bf16* b0 = (const bf16*)&u0;
            const bf16* b1 = (const bf16*)&u1;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                gv[j] = __bfloat162float(a0[j]), gv[j + 8] = __bfloat162float(a1[j]);
                uv[j] = __bfloat162float(b0[j]), uv[j + 8] = __bfloat162float(b1[j]);
            }
        } else {
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                gv[j] = j < nv ? ld_act(G + j) : 0.f;
                uv[j] = j < nv ? ld_act(G + 128 + j) : 0.f;
            }
        }
#pragma unroll
        // SwiGLU backward (h = silu(g) u, s = sigmoid(g)): dg = dh u s (1 + g (1 - s)), du = dh g s
        for (int j = 0; j < 16; ++j) {
            const float sg = 1.f / (1.f + __expf(-gv[j]));
            y[j] = v[j] * uv[j] * sg * (1.f + gv[j] * (1.f - sg));
            y2[j] = v[j] * gv[j] * sg;
        }
    } else {  // E_DS
        const float d = e.D[r];
        const act_t* P = (const act_t*)e.P + off;
        float p[16];
        if constexpr (VEC && sizeof(act_t) == 2) {
            const uint4 q0 = *(const uint4*)P, q1 = *(const uint4*)(P + 8);
            const bf16* b0 = (const bf16*)&q0;
            const bf16* b1 = (const bf16*)&q1;
#pragma unroll
            for (int j = 0; j < 8; ++j) p[j] = __bfloat162float(b0[j]), p[j + 8] = __bfloat162float(b1[j]);
        } else {
#pragma unroll
            for (int j = 0; j < 16; ++j) p[j] = j < nv ? ld_act(P + j) : 0.f;
        }
#pragma unroll
        for (int j = 0; j < 16; ++j) y[j] = p[j] * (v[j] - d) * e.scale;
    }
    return true;
}

// The epilogue of nv <= 16 consecutive outputs with plain stores (CUDA-core path).
template <typename act_t, int MODE>
__device__ __forceinline__ void epi16_mode(const Epi& e, const Out& o, int z, int m, int n, int nv,
                                           const float (&v)[16], RowStat& st) {
    float y[16], y2[16];
    if (!epi_values<act_t, false, MODE>(e, o, z, m, n, nv, v, st, y, y2)) return;
    if constexpr (MODE == E_SWIGLU_BWD) {
        act_t* c = (act_t*)o.C + (size_t)m * o.ldc + (size_t)(n >> 7) * 256 + (n & 127);
        for (int j = 0; j < nv; ++j) st_act(c + j, y[j]), st_act(c + 128 + j, y2[j]);
        return;
    }
    const size_t off = out_offset(o, z, m, n);
    if constexpr (MODE == E_F32) {
        float* c = (float*)o.C + off;
        for (int j = 0; j < nv; ++j) c[j] = y[j];
    } else {
        act_t* c = (act_t*)o.C + off;
        for (int j = 0; j < nv; ++j) st_act(c + j, y[j]);
    }
}

template <typename act_t>
__device__ __forceinline__ void epi16(const Epi& e, const Out& o, int z, int m, int n, int nv,
                                      const float (&v)[16], RowStat& st) {
    switch (e.mode) {
        case E_F32: epi16_mode<act_t, E_F32>(e, o, z, m, n, nv, v, st); break;
        case E_ACT: epi16_mode<act_t, E_ACT>(e, o, z, m, n, nv, v, st); break;
        case E_STATS: epi16_mode<act_t, E_STATS>(e, o, z, m, n, nv, v, st); break;
        case E_SOFTMAX: epi16_mode<act_t, E_SOFTMAX>(e, o, z, m, n, nv, v, st); break;
        case E_DS: epi16_mode<act_t, E_DS>(e, o, z, m, n, nv, v, st); break;
        default: epi16_mode<act_t, E_SWIGLU_BWD>(e, o, z, m, n, nv, v, st); break;
    }
}

// One GEMM of the backward pass.
struct Gemm {
    Op A, B;
    Out out;
    Epi epi;
    Sched sc;
};

// Runs g on the model's path: tcgen05 for bf16 models, CUDA cores for fp32 models.
int run_gemm(Model& m, const Gemm& g, cudaStream_t s);
// bf16 linear C = A W^T for M >= 256 rows through this GEMM's 256 x 256 tiles (the forward
// pass's prefill / scoring linears): epi EPI_STORE_ACT, EPI_STORE_F32, EPI_RESID_F32 or
// EPI_SWIGLU (N = I, W the packed gate / up rows).  Returns false (nothing launched) when
// the shape or alignment does not fit those tiles; the caller then uses its other kernels.
bool linear_large(Model& m, const void* A, int lda, const void* W, void* C, int ldc, int M, int N,
                  int K, int epi, cudaStream_t s);

// Column width of the E_STATS partials of the kernel run_gemm picks for N columns
// (half its N tile on the tensor-core path, its tile on the CUDA-core path).
int gemm_tile_n(const Model& m, int N, int tri);

// ---------------------------------------------------------------- row / elementwise kernels
// tgt[r] = tokens[b, t + 1] and w[r] = coef[b, t] for r = b T + t, t < T - 1; -1 and 0 for t = T - 1.
void launch_rows_prep(const int32_t* tokens, int B, int T, const float* coef, int V, int* tgt, float* w,
                      uint32_t* status, cudaStream_t s);
// From the raw projections qkv [M, (nq + 2 nkv) d] (row stride ld) of M = B Tlen rows at
// positions r % Tlen: qr [M, nq d] = RoPE(RMSNorm(q head) g_q) (token major); kvh =
// [2][B][nkv][Tlen][d], K = RoPE(RMSNorm(k head) g_k) then V = the raw v heads (head major).
void launch_qk_fwd(const void* qkv, int ld, int M, int Tlen, int nq, int nkv, int d, const float* gq,
                   const float* gk, float eps, const float* rc, const float* rs, void* qr, void* kvh,
                   int dtype, cudaStream_t s);
// lse[r] from the E_STATS partials st [R][n_ct] (column tiles of ct_w; causal: only the
// tiles at or left of the diagonal of row r % rows_per_z); loss_rows (may be null).
void launch_stats_combine(const float2* st, int n_ct, int ct_w, int causal, int R, int rows_per_z,
                          float* lse, const float* w, const float* zt, float* loss_rows, cudaStream_t s);
// RMSNorm backward (fp32 x, g, dy [M, H], H % 4 == 0): dres (+)= dx, dres_act = act(dres); gain partials
// part [rms_part_rows(M)][H].
int rms_part_rows(int M);
void launch_rms_bwd(const float* x, const float* g, const float* dy, int M, int H, float eps, int init,
                    float* dres, void* dres_act, float* part, int dtype, cudaStream_t s);
void launch_gain_reduce(const float* part, int nb, int n, int stride, float* out, int accumulate,
                        cudaStream_t s);
// QK-norm + RoPE backward into the q / k columns of dqkv (row stride ld); gain partials
// part [rms_part_rows(M)][2 d] (q gain, then k gain).
void launch_qk_bwd(const float* dqr, const float* dkr, const void* qkv, int ld, int M, int Tlen, int nq,
                   int nkv, int d, const float* gq, const float* gk, float eps, const float* rc,
                   const float* rs, void* dqkv, float* part, int dtype, cudaStream_t s);
void launch_attn_d(const void* dO, const void* O, int M, int Tlen, int nq, int d, float* Dv, int dtype,
                   cudaStream_t s);
void launch_embed_bwd(const int32_t* tokens, const float* dx, int M, int H, int V, float* dE, cudaStream_t s);
// h [M, I] = silu(gate) * up from the packed gate / up product gu [M, 2 I] (I % 128 == 0).
void launch_swiglu_fwd(const void* gu, int M, int I, void* h, int dtype, cudaStream_t s);
void launch_sum(const float* v, int n, float* out, cudaStream_t s);
// tok_p [B, Tp] / coef_p [B, Tp - 1]: the rows of tok [B, T] / coef [B, T - 1] followed by
// token 0 and coefficient 0 up to Tp positions.
void launch_pad_rows(const int32_t* tok, const float* coef, int B, int T, int Tp, int32_t* tok_p, float* coef_p,
                     cudaStream_t s);

}  // namespace bwd
}  // namespace qk
