// Row-wise and elementwise kernels of the backward pass (gradient of the
// token-weighted log-likelihood, Eq. sft / Eq. ppo): per-row targets and weights,
// the per-head QK-RMSNorm + RoPE forward that keeps the raw projections, the
// softmax-statistics combine, RMSNorm / QK-norm / RoPE / embedding backward,
// D = rowsum(dO * O) of the attention backward, and the deterministic
// reductions of gain gradients and of the loss.  fp32 arithmetic throughout;
// activations are read and written in the model dtype (act_t).
//
// Backward of the pieces (chain rule on their definitions):
//   RMSNorm y = x r g, r = (mean(x^2) + eps)^-1/2 over n entries:
//     dx = r (dy g) - (r^3 / n) x sum(dy g x),   dg = sum over rows of dy x r
//   RoPE (rotation of the pair (a, b) = (x_j, x_{j + d/2}) by angle p w_j):
//     (da, db) = (dy_a cos + dy_b sin, -dy_a sin + dy_b cos)
//   embedding x_0 = E[token]:  dE[token] += dx_0
#include <math.h>

#include <type_traits>

#include "bwd_common.cuh"

namespace qk {
namespace bwd {

namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// (sum a, sum b) over a block of 256 threads; every thread gets the totals.
__device__ __forceinline__ float2 block_sum2(float a, float b, float2* red) {
    a = warp_sum(a);
    b = warp_sum(b);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    __syncthreads();
    if (l == 0) red[w] = make_float2(a, b);
    __syncthreads();
    float2 t = make_float2(0.f, 0.f);
#pragma unroll
    for (int i = 0; i < 8; ++i) t.x += red[i].x, t.y += red[i].y;
    return t;
}

__global__ void rows_prep_kernel(const int32_t* __restrict__ tokens, int B, int T,
                                 const float* __restrict__ coef, int V, int* __restrict__ tgt,
                                 float* __restrict__ w, uint32_t* status) {
    pdl_wait();
    const int r = blockIdx.x * blockDim.x + threadIdx.x;
    if (r >= B * T) return;
    const int b = r / T, t = r % T;
    if (t < T - 1) {
        int id = tokens[(size_t)b * T + t + 1];
        if (id < 0 || id >= V) {
            atomicOr(status, QK_STATUS_BAD_TOKEN);
            id = 0;
        }
        tgt[r] = id;
        w[r] = coef[(size_t)b * (T - 1) + t];
    } else {
        tgt[r] = -1;
        w[r] = 0.f;
    }
}

// One warp per (token row r = b T + t, head of qkv): q heads -> qr [M, nq D] (token
// major) = RoPE(RMSNorm(raw) g_q); k heads -> kvh rows (b nkv + g) T + t = RoPE(RMSNorm(raw) g_k);
// v heads copied to kvh rows M nkv + (b nkv + g) T + t (K then V, head major, the layout
// of a KV cache holding B rows of T positions).
template <typename T, int D>
__global__ void qk_fwd_kernel(const T* __restrict__ qkv, int ld, int M, int Tlen, int nq, int nkv,
                              const float* __restrict__ gq, const float* __restrict__ gk, float eps,
                              const float* __restrict__ rc, const float* __restrict__ rs,
                              T* __restrict__ qr, T* __restrict__ kvh) {
    constexpr int E = D / 32, HALF = D / 2;
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const long long item = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int nh = nq + 2 * nkv;
    if (item >= (long long)M * nh) return;
    const int r = (int)(item / nh), hh = (int)(item % nh);
    const int b = r / Tlen, p = r % Tlen;
    const T* src = qkv + (size_t)r * ld + (size_t)hh * D;
    if (hh >= nq + nkv) {
        const int g = hh - nq - nkv;
        T* dst = kvh + ((size_t)M * nkv + ((size_t)b * nkv + g) * Tlen + p) * D;
#pragma unroll
        for (int i = 0; i < E; ++i) dst[lane + 32 * i] = src[lane + 32 * i];
        return;
    }
    float e[E];
#pragma unroll
    for (int i = 0; i < E; ++i) e[i] = ld_act(src + lane + 32 * i);
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < E; ++i) ss += e[i] * e[i];
    const float sc = rsqrtf(warp_sum(ss) / (float)D + eps);
    const float* g = hh < nq ? gq : gk;
#pragma unroll
    for (int i = 0; i < E; ++i) e[i] = e[i] * sc * g[lane + 32 * i];
#pragma unroll
    for (int i = 0; i < E / 2; ++i) {
        const int j = lane + 32 * i;
        const float c = rc[(size_t)p * HALF + j], sn = rs[(size_t)p * HALF + j];
        const float a = e[i], bb = e[i + E / 2];
        e[i] = a * c - bb * sn;
        e[i + E / 2] = bb * c + a * sn;
    }
    T* dst = hh < nq ? qr + (size_t)r * nq * D + (size_t)hh * D
                     : kvh + (((size_t)b * nkv + (hh - nq)) * Tlen + p) * D;
#pragma unroll
    for (int i = 0; i < E; ++i) st_act(dst + lane + 32 * i, e[i]);
}

// One warp per row: merge the (max, sum) partials of the row's unmasked column tiles
// into lse = max + log(sum); with loss_rows, loss_rows[r] = w_r (lse - zt_r) (0 where w_r == 0).
__global__ void stats_combine_kernel(const float2* __restrict__ st, int n_ct, int ct_w, int causal,
                                     int R, int rows_per_z, float* __restrict__ lse,
                                     const float* __restrict__ w, const float* __restrict__ zt,
                                     float* __restrict__ loss_rows) {
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const long long r = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (r >= R) return;
    const int m = (int)(r % rows_per_z);
    int nct = n_ct;
    if (causal) {
        const int lim = m / ct_w + 1;
        nct = lim < n_ct ? lim : n_ct;
    }
    RowStat a{-INFINITY, 0.f};
    for (int c = lane; c < nct; c += 32) {
        const float2 v = st[(size_t)r * n_ct + c];
        stat_merge(a, v.x, v.y);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, a.mx, o);
        const float s2 = __shfl_xor_sync(0xffffffffu, a.sm, o);
        stat_merge(a, m2, s2);
    }
    if (lane == 0) {
        const float l = a.mx + logf(a.sm);
        lse[r] = l;
        if (loss_rows) {
            const float wr = w[r];
            loss_rows[r] = wr != 0.f ? wr * (l - zt[r]) : 0.f;
        }
    }
}

// RMSNorm backward over rows [8 b, 8 b + 8) of CTA b (256 threads; H % 4 == 0: thread i
// owns the float4 column groups i, i + 256, ...): dres = (init ? 0 : dres) + dx,
// dres_act = act(dres), part[b][c] = sum over the CTA's rows of dy x r (column c).
constexpr int kRmsRows = 8;

template <typename T>
__global__ void __launch_bounds__(256)
    rms_bwd_kernel(const float* __restrict__ x, const float* __restrict__ g, const float* __restrict__ dy,
                   int M, int H, float eps, int init, float* __restrict__ dres, T* __restrict__ dres_act,
                   float* __restrict__ part) {
    extern __shared__ float dgs[];
    __shared__ float2 red[8];
    pdl_wait();
    const int H4 = H >> 2;
    for (int c = threadIdx.x; c < H; c += 256) dgs[c] = 0.f;
    const float4* g4 = (const float4*)g;
    const int r0 = blockIdx.x * kRmsRows;
    for (int r = r0; r < r0 + kRmsRows && r < M; ++r) {
        const float4* xr = (const float4*)(x + (size_t)r * H);
        const float4* dr = (const float4*)(dy + (size_t)r * H);
        float ss = 0.f, sa = 0.f;
        for (int c = threadIdx.x; c < H4; c += 256) {
            const float4 xv = xr[c], dv = dr[c], gv = g4[c];
            ss += xv.x * xv.x + xv.y * xv.y + xv.z * xv.z + xv.w * xv.w;
            sa += dv.x * gv.x * xv.x + dv.y * gv.y * xv.y + dv.z * gv.z * xv.z + dv.w * gv.w * xv.w;
        }
        const float2 t = block_sum2(ss, sa, red);
        const float rr = rsqrtf(t.x / (float)H + eps);
        const float k3 = rr * rr * rr / (float)H * t.y;
        float4* d4 = (float4*)(dres + (size_t)r * H);
        T* da = dres_act + (size_t)r * H;
        for (int c = threadIdx.x; c < H4; c += 256) {
            const float4 xv = xr[c], dv = dr[c], gv = g4[c];
            float4 o = init ? make_float4(0.f, 0.f, 0.f, 0.f) : d4[c];
            o.x += rr * dv.x * gv.x - k3 * xv.x;
            o.y += rr * dv.y * gv.y - k3 * xv.y;
            o.z += rr * dv.z * gv.z - k3 * xv.z;
            o.w += rr * dv.w * gv.w - k3 * xv.w;
            d4[c] = o;
            st_act(da + 4 * c, o.x);
            st_act(da + 4 * c + 1, o.y);
            st_act(da + 4 * c + 2, o.z);
            st_act(da + 4 * c + 3, o.w);
            dgs[4 * c] += dv.x * xv.x * rr;
            dgs[4 * c + 1] += dv.y * xv.y * rr;
            dgs[4 * c + 2] += dv.z * xv.z * rr;
            dgs[4 * c + 3] += dv.w * xv.w * rr;
        }
    }
    __syncthreads();
    for (int c = threadIdx.x; c < H; c += 256) part[(size_t)blockIdx.x * H + c] = dgs[c];
}

// out[c] (+)= sum over the nb partial rows of part[.][c] (row stride `stride`): CTA
// b takes columns 32 b .. 32 b + 31, warp w the rows w, w + 8, ... (lane = column),
// then the eight warp sums are added in warp order (a fixed order).
__global__ void __launch_bounds__(256)
    gain_reduce_kernel(const float* __restrict__ part, int nb, int n, int stride, float* __restrict__ out,
                       int accumulate) {
    __shared__ float red[8][32];
    pdl_wait();
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int c = blockIdx.x * 32 + lane;
    float s = 0.f;
    if (c < n)
        for (int b = w; b < nb; b += 8) s += part[(size_t)b * stride + c];
    red[w][lane] = s;
    __syncthreads();
    if (w == 0 && c < n) {
        float t = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) t += red[i][lane];
        out[c] = accumulate ? out[c] + t : t;
    }
}

// QK-norm + RoPE backward.  CTA b (8 warps) takes token rows [16 b, 16 b + 16); a warp
// handles one (row, q or k head) at a time: the gradient of the rotated output (dqr /
// dkr, fp32) goes back through the rotation and the head RMSNorm to the raw
// projection (written in the activation type into dqkv), and the gain gradients
// accumulate per lane; part[b][0 .. D) gets the q gain's, part[b][D .. 2 D) the k gain's.
template <typename T, int D>
__global__ void __launch_bounds__(256)
    qk_bwd_kernel(const float* __restrict__ dqr, const float* __restrict__ dkr,
                  const T* __restrict__ qkv, int ld, int M, int Tlen, int nq, int nkv,
                  const float* __restrict__ gq, const float* __restrict__ gk, float eps,
                  const float* __restrict__ rc, const float* __restrict__ rs, T* __restrict__ dqkv,
                  float* __restrict__ part) {
    constexpr int E = D / 32, HALF = D / 2;
    __shared__ float red[8][2 * D];
    pdl_wait();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nh = nq + nkv;
    const int r0 = blockIdx.x * kRmsRows;
    const int rows = M - r0 < kRmsRows ? M - r0 : kRmsRows;
    float accq[E], acck[E];
#pragma unroll
    for (int i = 0; i < E; ++i) accq[i] = acck[i] = 0.f;
    for (int it = warp; it < rows * nh; it += 8) {
        const int r = r0 + it / nh, hh = it % nh;
        const int p = r % Tlen;
        const bool isq = hh < nq;
        const float* gsrc = isq ? dqr + (size_t)r * nq * D + (size_t)hh * D
                                : dkr + (size_t)r * nkv * D + (size_t)(hh - nq) * D;
        float e[E], xv[E];
#pragma unroll
        for (int i = 0; i < E; ++i) e[i] = gsrc[lane + 32 * i];
#pragma unroll
        for (int i = 0; i < E / 2; ++i) {  // transpose of the rotation
            const int j = lane + 32 * i;
            const float c = rc[(size_t)p * HALF + j], sn = rs[(size_t)p * HALF + j];
            const float a = e[i], b = e[i + E / 2];
            e[i] = a * c + b * sn;
            e[i + E / 2] = -a * sn + b * c;
        }
        const T* raw = qkv + (size_t)r * ld + (size_t)hh * D;
        const float* g = isq ? gq : gk;
        float ss = 0.f, sa = 0.f;
#pragma unroll
        for (int i = 0; i < E; ++i) {
            xv[i] = ld_act(raw + lane + 32 * i);
            ss += xv[i] * xv[i];
            sa += e[i] * g[lane + 32 * i] * xv[i];
        }
        ss = warp_sum(ss);
        sa = warp_sum(sa);
        const float rr = rsqrtf(ss / (float)D + eps);
        const float k3 = rr * rr * rr / (float)D * sa;
        T* dst = dqkv + (size_t)r * ld + (size_t)hh * D;
#pragma unroll
        for (int i = 0; i < E; ++i) {
            st_act(dst + lane + 32 * i, rr * e[i] * g[lane + 32 * i] - k3 * xv[i]);
            const float dg = e[i] * xv[i] * rr;
            if (isq) accq[i] += dg; else acck[i] += dg;
        }
    }
#pragma unroll
    for (int i = 0; i < E; ++i) {
        red[warp][lane + 32 * i] = accq[i];
        red[warp][D + lane + 32 * i] = acck[i];
    }
    __syncthreads();
    for (int c = threadIdx.x; c < 2 * D; c += 256) {
        float s = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) s += red[w][c];
        part[(size_t)blockIdx.x * 2 * D + c] = s;
    }
}

// One warp per (token row r = b T + t, head h): D[(b nq + h) T + t] = sum_j dO * O.
template <typename T>
__global__ void attn_d_kernel(const T* __restrict__ dO, const T* __restrict__ O, int M, int Tlen,
                              int nq, int d, float* __restrict__ Dv) {
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const long long item = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (item >= (long long)M * nq) return;
    const int r = (int)(item / nq), h = (int)(item % nq);
    const size_t o = (size_t)r * nq * d + (size_t)h * d;
    float s = 0.f;
    for (int j = lane; j < d; j += 32) s += ld_act(dO + o + j) * ld_act(O + o + j);
    s = warp_sum(s);
    if (lane == 0) Dv[((size_t)(r / Tlen) * nq + h) * Tlen + r % Tlen] = s;
}

// h = silu(g) u from gu [M, 2 I] in the packed order (blocks of 128 gate columns, then
// the matching 128 up columns); thread e takes 8 consecutive columns (one 16-byte load of
// gate, one of up, one 16-byte store of h).  I % 128 == 0.
template <typename T>
__global__ void swiglu_fwd_kernel(const T* __restrict__ gu, int M, int I, T* __restrict__ h) {
    constexpr int V = 16 / sizeof(T);
    pdl_wait();
    const size_t n = (size_t)M * I / V;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const size_t j0 = e * V;
        const size_t m = j0 / I;
        const int j = (int)(j0 - m * I);
        const T* gp = gu + m * 2 * I + (size_t)(j >> 7) * 256 + (j & 127);
        uint4 gq = *(const uint4*)gp, uq = *(const uint4*)(gp + 128), hq;
        const T* ga = (const T*)&gq;
        const T* ua = (const T*)&uq;
        T* ha = (T*)&hq;
#pragma unroll
        for (int k = 0; k < V; ++k) {
            const float gv = ld_act(ga + k);
            st_act(ha + k, gv / (1.f + __expf(-gv)) * ld_act(ua + k));
        }
        *(uint4*)(h + j0) = hq;
    }
}

// dE[token[r]] += dx[r] (fp32 atomics: rows that share a token add in any order).
__global__ void embed_bwd_kernel(const int32_t* __restrict__ tokens, const float* __restrict__ dx, int H,
                                 int V, float* __restrict__ dE) {
    pdl_wait();
    const int r = blockIdx.x;
    int id = tokens[r];
    if (id < 0 || id >= V) id = 0;  // flagged by the forward embedding
    for (int c = threadIdx.x; c < H; c += blockDim.x) atomicAdd(dE + (size_t)id * H + c, dx[(size_t)r * H + c]);
}

// Rows padded from T to Tp positions: tokens id 0 and coefficients 0 past the row's end.
__global__ void pad_rows_kernel(const int32_t* __restrict__ tok, const float* __restrict__ coef, int B, int T,
                                int Tp, int32_t* __restrict__ tok_p, float* __restrict__ coef_p) {
    pdl_wait();
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (long long)B * Tp) return;
    const int b = (int)(i / Tp), t = (int)(i % Tp);
    tok_p[i] = t < T ? tok[(size_t)b * T + t] : 0;
    if (t < Tp - 1) coef_p[(size_t)b * (Tp - 1) + t] = t < T - 1 ? coef[(size_t)b * (T - 1) + t] : 0.f;
}

// *out = sum of v[0 .. n) in a fixed order (one CTA of 256 threads).
__global__ void sum_kernel(const float* __restrict__ v, int n, float* __restrict__ out) {
    __shared__ float2 red[8];
    pdl_wait();
    float s = 0.f;
    for (int i = threadIdx.x; i < n; i += 256) s += v[i];
    const float2 t = block_sum2(s, 0.f, red);
    if (threadIdx.x == 0) *out = t.x;
}

template <typename F>
void launch_act(int dtype, F f) {
    if (dtype == QK_DTYPE_BF16) f((bf16*)nullptr); else f((float*)nullptr);
}

}  // namespace

void launch_rows_prep(const int32_t* tokens, int B, int T, const float* coef, int V, int* tgt, float* w,
                      uint32_t* status, cudaStream_t s) {
    const int n = B * T;
    launch_k(rows_prep_kernel, dim3(cdiv(n, 256)), dim3(256), 0, s, tokens, B, T, coef, V, tgt, w, status);
    note_launch();
}

void launch_qk_fwd(const void* qkv, int ld, int M, int Tlen, int nq, int nkv, int d, const float* gq,
                   const float* gk, float eps, const float* rc, const float* rs, void* qr, void* kvh,
                   int dtype, cudaStream_t s) {
    const long long items = (long long)M * (nq + 2 * nkv);
    const dim3 grid((unsigned)((items + 7) / 8));
    launch_act(dtype, [&](auto* tp) {
        using A = std::remove_pointer_t<decltype(tp)>;
        if (d == 128)
            launch_k(qk_fwd_kernel<A, 128>, grid, dim3(256), 0, s, (const A*)qkv, ld, M, Tlen, nq, nkv, gq,
                     gk, eps, rc, rs, (A*)qr, (A*)kvh);
        else
            launch_k(qk_fwd_kernel<A, 64>, grid, dim3(256), 0, s, (const A*)qkv, ld, M, Tlen, nq, nkv, gq,
                     gk, eps, rc, rs, (A*)qr, (A*)kvh);
    });
    note_launch();
}

void launch_stats_combine(const float2* st, int n_ct, int ct_w, int causal, int R, int rows_per_z,
                          float* lse, const float* w, const float* zt, float* loss_rows, cudaStream_t s) {
    launch_k(stats_combine_kernel, dim3(cdiv(R, 8)), dim3(256), 0, s, st, n_ct, ct_w, causal, R, rows_per_z,
             lse, w, zt, loss_rows);
    note_launch();
}

int rms_part_rows(int M) { return cdiv(M, kRmsRows); }

void launch_rms_bwd(const float* x, const float* g, const float* dy, int M, int H, float eps, int init,
                    float* dres, void* dres_act, float* part, int dtype, cudaStream_t s) {
    const size_t smem = (size_t)H * 4;
    launch_act(dtype, [&](auto* tp) {
        using A = std::remove_pointer_t<decltype(tp)>;
        launch_k(rms_bwd_kernel<A>, dim3(cdiv(M, kRmsRows)), dim3(256), smem, s, x, g, dy, M, H, eps, init,
                 dres, (A*)dres_act, part);
    });
    note_launch();
}

void launch_gain_reduce(const float* part, int nb, int n, int stride, float* out, int accumulate,
                        cudaStream_t s) {
    launch_k(gain_reduce_kernel, dim3(cdiv(n, 32)), dim3(256), 0, s, part, nb, n, stride, out, accumulate);
    note_launch();
}

void launch_qk_bwd(const float* dqr, const float* dkr, const void* qkv, int ld, int M, int Tlen, int nq,
                   int nkv, int d, const float* gq, const float* gk, float eps, const float* rc,
                   const float* rs, void* dqkv, float* part, int dtype, cudaStream_t s) {
    const dim3 grid(cdiv(M, kRmsRows));
    launch_act(dtype, [&](auto* tp) {
        using A = std::remove_pointer_t<decltype(tp)>;
        if (d == 128)
            launch_k(qk_bwd_kernel<A, 128>, grid, dim3(256), 0, s, dqr, dkr, (const A*)qkv, ld, M, Tlen, nq,
                     nkv, gq, gk, eps, rc, rs, (A*)dqkv, part);
        else
            launch_k(qk_bwd_kernel<A, 64>, grid, dim3(256), 0, s, dqr, dkr, (const A*)qkv, ld, M, Tlen, nq,
                     nkv, gq, gk, eps, rc, rs, (A*)dqkv, part);
    });
    note_launch();
}

void launch_attn_d(const void* dO, const void* O, int M, int Tlen, int nq, int d, float* Dv, int dtype,
                   cudaStream_t s) {
    const long long items = (long long)M * nq;
    const dim3 grid((unsigned)((items + 7) / 8));
    launch_act(dtype, [&](auto* tp) {
        using A = std::remove_pointer_t<decltype(tp)>;
        launch_k(attn_d_kernel<A>, grid, dim3(256), 0, s, (const A*)dO, (const A*)O, M, Tlen, nq, d, Dv);
    });
    note_launch();
}

void launch_swiglu_fwd(const void* gu, int M, int I, void* h, int dtype, cudaStream_t s) {
    const size_t n = (size_t)M * I / (dtype == QK_DTYPE_BF16 ? 8 : 4);
    const int blocks = (int)(n / 256 + 1 < 152 * 16 ? n / 256 + 1 : 152 * 16);
    launch_act(dtype, [&](auto* tp) {
        using A = std::remove_pointer_t<decltype(tp)>;
        launch_k(swiglu_fwd_kernel<A>, dim3(blocks), dim3(256), 0, s, (const A*)gu, M, I, (A*)h);
    });
    note_launch();
}

void launch_embed_bwd(const int32_t* tokens, const float* dx, int M, int H, int V, float* dE, cudaStream_t s) {
    launch_k(embed_bwd_kernel, dim3(M), dim3(256), 0, s, tokens, dx, H, V, dE);
    note_launch();
}

void launch_pad_rows(const int32_t* tok, const float* coef, int B, int T, int Tp, int32_t* tok_p, float* coef_p,
                     cudaStream_t s) {
    const long long n = (long long)B * Tp;
    launch_k(pad_rows_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, tok, coef, B, T, Tp, tok_p, coef_p);
    note_launch();
}

void launch_sum(const float* v, int n, float* out, cudaStream_t s) {
    launch_k(sum_kernel, dim3(1), dim3(256), 0, s, v, n, out);
    note_launch();
}

}  // namespace bwd
}  // namespace qk
