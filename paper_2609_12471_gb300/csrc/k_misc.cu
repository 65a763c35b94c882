// Elementwise and row-wise kernels of the decoder forward pass: embedding
// gather, RMSNorm, per-head QK-RMSNorm + RoPE + KV-cache write, SwiGLU, the
// vocabulary reduce (log-softmax / gather / arg-max, the Gumbel-max draw of a
// sampled rollout and the GRPO token loss where a log-prob is formed), the
// rollout cursors, and the load-time RoPE table.
#include <math.h>

#include "qk_internal.cuh"

namespace qk {

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(bf16 v) { return __bfloat162float(v); }
template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Sum over a block whose size is a multiple of 32 (at most 1024); every thread gets the total.
__device__ float block_sum(float v, float* red) {
    v = warp_sum(v);
    int w = threadIdx.x >> 5, l = threadIdx.x & 31, nw = blockDim.x >> 5;
    __syncthreads();
    if (l == 0) red[w] = v;
    __syncthreads();
    float t = l < nw ? red[l] : 0.f;
    return warp_sum(t);
}

// ---------------------------------------------------------------- embedding (x_0 = E[token])
template <typename T>
__global__ void embed_kernel(const T* __restrict__ E, int V, int H, TokIndex tok,
                             float* __restrict__ x, uint32_t* status) {
    pdl_wait();
    pdl_trigger();  // short kernel: let the next one launch and prefetch now
    int r = blockIdx.x;
    int id = tok.ptr[(size_t)(r / tok.T) * tok.ld + tok.off + r % tok.T];
    if (id < 0 || id >= V) {
        if (threadIdx.x == 0) atomicOr(status, QK_STATUS_BAD_TOKEN);
        id = 0;
    }
    const T* src = E + (size_t)id * H;
    float* dst = x + (size_t)r * H;
    for (int i = threadIdx.x; i < H; i += blockDim.x) dst[i] = to_f(src[i]);
}

void launch_embed(const void* E, int dtype, int V, int H, TokIndex tok, int M, float* x,
                  uint32_t* status, cudaStream_t s) {
    note_launch();
    if (M <= 0) return;
    if (dtype == QK_DTYPE_BF16)
        launch_k(embed_kernel<bf16>, dim3(M), dim3(256), 0, s, (const bf16*)E, V, H, tok, x, status);
    else
        launch_k(embed_kernel<float>, dim3(M), dim3(256), 0, s, (const float*)E, V, H, tok, x, status);
}

// ---------------------------------------------------------------- embedding + gain (fused decode)
// One CTA per (128-feature tile, row): x = E[token] (or the given x), xg = bf16(x * g) and
// the tile's sum of squares ssq[tile][row] (the input-norm statistics of the next linear).
__global__ void __launch_bounds__(128)
    embed_gain_kernel(const bf16* __restrict__ E, int V, TokIndex tok, int do_embed,
                      float* __restrict__ x, const float* __restrict__ g, bf16* __restrict__ xg,
                      float* __restrict__ ssq, int M, int H, uint32_t* status) {
    __shared__ float red[4];
    pdl_wait();
    const int m = blockIdx.y, f = blockIdx.x * 128 + threadIdx.x;
    float xv;
    if (do_embed) {
        int id = tok.ptr[(size_t)(m / tok.T) * tok.ld + tok.off + m % tok.T];
        if (id < 0 || id >= V) {
            if (threadIdx.x == 0 && blockIdx.x == 0) atomicOr(status, QK_STATUS_BAD_TOKEN);
            id = 0;
        }
        xv = __bfloat162float(E[(size_t)id * H + f]);
        x[(size_t)m * H + f] = xv;
    } else {
        xv = x[(size_t)m * H + f];
    }
    xg[(size_t)m * H + f] = __float2bfloat16_rn(xv * g[f]);
    const float sq = warp_sum(xv * xv);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = sq;
    __syncthreads();
    if (threadIdx.x == 0) ssq[(size_t)blockIdx.x * M + m] = red[0] + red[1] + red[2] + red[3];
}

void launch_embed_gain(const void* E, int V, TokIndex tok, bool do_embed, float* x, const float* g,
                       bf16* xg, float* ssq, int M, int H, uint32_t* status, cudaStream_t s) {
    note_launch();
    if (M <= 0) return;
    launch_k(embed_gain_kernel, dim3(H / 128, M), dim3(128), 0, s, (const bf16*)E, V, tok,
             do_embed ? 1 : 0, x, g, xg, ssq, M, H, status);
}

// ---------------------------------------------------------------- RMSNorm
template <typename OutT>
__global__ void rmsnorm_kernel(const float* __restrict__ x, int in_step, int in_off,
                               const int32_t* __restrict__ row_len, const float* __restrict__ g,
                               int H, float eps, OutT* __restrict__ out) {
    __shared__ float red[32];
    pdl_wait();
    pdl_trigger();  // short kernel: let the next one launch and prefetch now
    int r = blockIdx.x;
    int off = in_off;
    if (row_len) {  // row r's last valid token: row_len[r] - 1, clamped into the row
        off = row_len[r] - 1;
        off = off < 0 ? 0 : (off >= in_step ? in_step - 1 : off);
    }
    const float* xr = x + ((size_t)r * in_step + off) * H;
    float ss = 0.f;
    for (int i = threadIdx.x * 4; i < H; i += blockDim.x * 4) {
        float4 v = *reinterpret_cast<const float4*>(xr + i);
        ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
    }
    ss = block_sum(ss, red);
    float scale = rsqrtf(ss / (float)H + eps);
    OutT* o = out + (size_t)r * H;
    for (int i = threadIdx.x * 4; i < H; i += blockDim.x * 4) {
        float4 v = *reinterpret_cast<const float4*>(xr + i);
        float4 gg = *reinterpret_cast<const float4*>(g + i);
        o[i + 0] = from_f<OutT>(v.x * scale * gg.x);
        o[i + 1] = from_f<OutT>(v.y * scale * gg.y);
        o[i + 2] = from_f<OutT>(v.z * scale * gg.z);
        o[i + 3] = from_f<OutT>(v.w * scale * gg.w);
    }
}

void launch_rmsnorm(const float* x, int in_step, int in_off, const float* g, int H, float eps,
                    void* out, int out_dtype, int M, cudaStream_t s, const int32_t* row_len) {
    note_launch();
    if (M <= 0) return;
    int threads = H >= 1024 ? 256 : 64;
    if (out_dtype == QK_DTYPE_BF16)
        launch_k(rmsnorm_kernel<bf16>, dim3(M), dim3(threads), 0, s, x, in_step, in_off, row_len, g,
                 H, eps, (bf16*)out);
    else
        launch_k(rmsnorm_kernel<float>, dim3(M), dim3(threads), 0, s, x, in_step, in_off, row_len, g,
                 H, eps, (float*)out);
}

// ---------------------------------------------------------------- QK-norm + RoPE + cache write
// One warp per (token, head) of the fused qkv row; lane owns elements lane + 32 i.
template <typename T, int D>
__global__ void qk_norm_rope_kernel(T* __restrict__ qkv, int nq, int nkv, const float* __restrict__ gq,
                                    const float* __restrict__ gk, float eps,
                                    const float* __restrict__ rc, const float* __restrict__ rs,
                                    int max_positions, PosIndex pos, T* __restrict__ kc,
                                    T* __restrict__ vc, KvPages kp, uint32_t* status) {
    constexpr int E = D / 32, HALF = D / 2;
    pdl_wait();
    pdl_trigger();  // short kernel: let the next one launch and prefetch now
    int lane = threadIdx.x & 31;
    int hh = blockIdx.y * (blockDim.x >> 5) + (threadIdx.x >> 5);
    int nh = nq + 2 * nkv;
    if (hh >= nh) return;
    int r = blockIdx.x;
    int b = r / pos.T, t = r % pos.T;
    int p = pos.pos_dev ? pos.pos_dev[b] + t : pos.start + t;
    int lim = kp.cap() < max_positions ? kp.cap() : max_positions;
    if (p < 0 || p >= lim) {
        if (lane == 0) atomicOr(status, QK_STATUS_BAD_POS);
        p = p < 0 ? 0 : lim - 1;
    }
    T* src = qkv + (size_t)r * nh * D + (size_t)hh * D;
    float e[E];
#pragma unroll
    for (int i = 0; i < E; ++i) e[i] = to_f(src[lane + 32 * i]);
    if (hh >= nq + nkv) {  // value head: straight to the cache
        int kvh = hh - nq - nkv;
        T* dst = vc + (size_t)kv_row(kp, nkv, b, kvh, p, lane == 0 ? status : nullptr) * D;
#pragma unroll
        for (int i = 0; i < E; ++i) dst[lane + 32 * i] = src[lane + 32 * i];
        return;
    }
    const float* g = hh < nq ? gq : gk;
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < E; ++i) ss += e[i] * e[i];
    ss = warp_sum(ss);
    float scale = rsqrtf(ss / (float)D + eps);
#pragma unroll
    for (int i = 0; i < E; ++i) e[i] = e[i] * scale * g[lane + 32 * i];
    const float* cr = rc + (size_t)p * HALF;
    const float* sr = rs + (size_t)p * HALF;
#pragma unroll
    for (int i = 0; i < E / 2; ++i) {
        int j = lane + 32 * i;  // j < d/2, partner j + d/2 is element i + E/2 of this lane
        float c = cr[j], sn = sr[j];
        float a = e[i], bb = e[i + E / 2];
        e[i] = a * c - bb * sn;
        e[i + E / 2] = bb * c + a * sn;
    }
    T* dst;
    if (hh < nq) {
        dst = src;
    } else {
        int kvh = hh - nq;
        dst = kc + (size_t)kv_row(kp, nkv, b, kvh, p, lane == 0 ? status : nullptr) * D;
    }
#pragma unroll
    for (int i = 0; i < E; ++i) dst[lane + 32 * i] = from_f<T>(e[i]);
}

void launch_qk_norm_rope(void* qkv, int dtype, int M, int nq, int nkv, int d, const float* gq,
                         const float* gk, float eps, const float* rope_cos, const float* rope_sin,
                         int max_positions, PosIndex pos, void* k_cache, void* v_cache,
                         const KvPages& kp, uint32_t* status, cudaStream_t s) {
    note_launch();
    if (M <= 0) return;
    dim3 grid(M, (nq + 2 * nkv + 7) / 8);
#define QK_NR(T, D)                                                                          \
    launch_k(qk_norm_rope_kernel<T, D>, grid, dim3(256), 0, s, (T*)qkv, nq, nkv, gq, gk, eps,  \
             rope_cos, rope_sin, max_positions, pos, (T*)k_cache, (T*)v_cache, kp, status)
    if (dtype == QK_DTYPE_BF16) {
        if (d == 128) QK_NR(bf16, 128); else QK_NR(bf16, 64);
    } else {
        if (d == 128) QK_NR(float, 128); else QK_NR(float, 64);
    }
#undef QK_NR
}

// ---------------------------------------------------------------- SwiGLU (unfused path)
template <typename T>
__global__ void swiglu_kernel(const T* __restrict__ gu, T* __restrict__ h, int M, int I) {
    pdl_wait();
    pdl_trigger();  // short kernel: let the next one launch and prefetch now
    size_t n = (size_t)M * I;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n;
         e += (size_t)gridDim.x * blockDim.x) {
        size_t m = e / I;
        int j = (int)(e % I);
        const T* row = gu + m * 2 * I + (size_t)(j >> 7) * 256 + (j & 127);
        float g = to_f(row[0]), u = to_f(row[128]);
        h[e] = from_f<T>(g / (1.f + expf(-g)) * u);
    }
}

void launch_swiglu(const void* gu, void* h, int dtype, int M, int I, cudaStream_t s) {
    note_launch();
    if (M <= 0) return;
    size_t n = (size_t)M * I;
    int blocks = (int)((n + 255) / 256);
    if (blocks > 65535) blocks = 65535;
    if (dtype == QK_DTYPE_BF16)
        launch_k(swiglu_kernel<bf16>, dim3(blocks), dim3(256), 0, s, (const bf16*)gu, (bf16*)h, M, I);
    else
        launch_k(swiglu_kernel<float>, dim3(blocks), dim3(256), 0, s, (const float*)gu, (float*)h, M,
                 I);
}

// ---------------------------------------------------------------- log-softmax / gather / argmax
// One block per logits row: max and lowest arg-max, then logsumexp, then the target's log-prob.
// Online (max, arg-max, sum of exp) over a stream of logits: the running sum is kept
// relative to the running max (rescaled when the max grows); ties keep the lowest index.
struct MaxSum {
    float m, s;
    int i;
    float ym;  // sampling: the largest perturbed score z / tau + G and its token
    int yi;
};

__device__ __forceinline__ void ms_push(MaxSum& a, float v, int i) {
    if (v > a.m) {
        a.s = (a.m == -INFINITY ? 0.f : a.s * expf(a.m - v)) + 1.f;
        a.m = v;
        a.i = i;
    } else {
        a.s += expf(v - a.m);
    }
}

// a followed by b (b covers later indices, or is an unordered peer: ties take the lower index)
__device__ __forceinline__ MaxSum ms_merge(MaxSum a, MaxSum b) {
    MaxSum r;
    r.ym = fmaxf(a.ym, b.ym);
    r.yi = a.ym > b.ym ? a.yi : (b.ym > a.ym ? b.yi : min(a.yi, b.yi));
    r.m = fmaxf(a.m, b.m);
    if (r.m == -INFINITY) {
        a.ym = r.ym, a.yi = r.yi;
        return a;
    }
    r.s = (a.m == -INFINITY ? 0.f : a.s * expf(a.m - r.m)) + (b.m == -INFINITY ? 0.f : b.s * expf(b.m - r.m));
    r.i = a.m > b.m ? a.i : (b.m > a.m ? b.i : min(a.i, b.i));
    return r;
}

// Gumbel noise for (row b, sampling step j, token v): the uniform is output
// i = b 2^40 + j 2^18 + v of the SplitMix64 stream seeded with `seed` (Steele, Lea,
// Flood, OOPSLA 2014: state seed + (i + 1) gamma through the published finaliser),
// on the 24-bit grid u = (x / 2^40 + 1/2) / 2^24 (exact in fp32, strictly inside
// (0, 1)); G = -log(-log u).
__device__ __forceinline__ float gumbel_noise(unsigned long long seed, int b, int j, int v) {
    const unsigned long long i =
        ((unsigned long long)b << 40) + ((unsigned long long)j << 18) + (unsigned long long)v;
    unsigned long long z = seed + (i + 1ull) * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    z ^= z >> 31;
    const float u = ((float)(z >> 40) + 0.5f) * 5.9604644775390625e-8f;  // 2^-24
    return -logf(-logf(u));
}

// One logits row per cluster of kLogitCtas CTAs: CTA k of the cluster reduces the
// k-th slice of the row in one pass, then CTA 0 combines the slices' (max, arg-max,
// sum of exp) in slice order through distributed shared memory and writes
//   argmax, and log p(target) = z[target] - (max + log sum exp(z - max)).
constexpr int kLogitCtas = 8;

__global__ void __cluster_dims__(kLogitCtas, 1, 1) __launch_bounds__(256)
    logits_reduce_kernel(const float* __restrict__ logits, int V, OutIndex oi,
                         float* __restrict__ lp, int32_t* __restrict__ am, uint32_t* status,
                         GrpoArgs grpo, SampleArgs samp) {
    __shared__ MaxSum red[8];
    __shared__ MaxSum part;
    pdl_wait();
    pdl_trigger();  // short kernel: let the next one launch and prefetch now
    const int r = blockIdx.y, k = blockIdx.x;
    const int g = oi.row0 + r;
    const int b = g / oi.T, t = g % oi.T;
    const bool active = t < oi.out_lim;  // uniform over the cluster (one row per cluster)
    const float* z = logits + (size_t)r * V;
    const bool sampling = samp.out_tokens != nullptr;
    // the output column is the sampling step (prefill: 0; rollout decode step s: s + 1)
    const int step = t + oi.out_off + (oi.dyn_off ? *oi.dyn_off : 0);
    const float inv_tau = sampling ? samp.inv_tau : 1.f;
    int tg = 0;
    float z_tg = 0.f;
    if (active && !sampling && k == 0 && threadIdx.x == 0 && lp && oi.tgt) {  // fetched early, used last
        tg = oi.tgt[(size_t)b * oi.tgt_ld + oi.tgt_off + t];
        if (tg < 0 || tg >= V) {
            atomicOr(status, QK_STATUS_BAD_TOKEN);
            tg = 0;
        }
        z_tg = z[tg];
    }
    MaxSum a{-INFINITY, 0.f, 0x7fffffff, -INFINITY, 0x7fffffff};
    // z / tau into the max / sum of exponentials; with sampling also z / tau + G into (ym, yi)
    auto push = [&](float zv, int i) {
        const float zz = zv * inv_tau;
        ms_push(a, zz, i);
        if (sampling) {
            const float y = zz + gumbel_noise(samp.seed, b, step, i);
            if (y > a.ym) a.ym = y, a.yi = i;
        }
    };
    if (active) {
        // slice k: [lo, hi), a multiple of 4 wide except at the row's end
        const int per = ((V + kLogitCtas - 1) / kLogitCtas + 3) & ~3;
        const int lo = min(V, k * per), hi = min(V, lo + per);
        if ((V & 3) == 0) {
            for (int i = lo + threadIdx.x * 4; i < hi; i += blockDim.x * 4) {
                const float4 v = *reinterpret_cast<const float4*>(z + i);
                push(v.x, i);
                push(v.y, i + 1);
                push(v.z, i + 2);
                push(v.w, i + 3);
            }
        } else {
            for (int i = lo + threadIdx.x; i < hi; i += blockDim.x) push(z[i], i);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        MaxSum p;
        p.m = __shfl_xor_sync(0xffffffffu, a.m, o);
        p.s = __shfl_xor_sync(0xffffffffu, a.s, o);
        p.i = __shfl_xor_sync(0xffffffffu, a.i, o);
        p.ym = __shfl_xor_sync(0xffffffffu, a.ym, o);
        p.yi = __shfl_xor_sync(0xffffffffu, a.yi, o);
        a = ms_merge(a, p);
    }
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    if (l == 0) red[w] = a;
    __syncthreads();
    if (threadIdx.x == 0) {
        MaxSum c = red[0];
        for (int i = 1; i < (int)(blockDim.x >> 5); ++i) c = ms_merge(c, red[i]);
        part = c;
    }
    // every slice's partial is in its CTA's shared memory before CTA 0 reads them
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
    if (active && k == 0 && threadIdx.x == 0) {
        MaxSum c{-INFINITY, 0.f, 0x7fffffff, -INFINITY, 0x7fffffff};
        const uint32_t local = (uint32_t)__cvta_generic_to_shared(&part);
        for (int q = 0; q < kLogitCtas; ++q) {
            uint32_t remote;
            asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(q));
            MaxSum p;
            asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(p.m) : "r"(remote));
            asm volatile("ld.shared::cluster.f32 %0, [%1+4];" : "=f"(p.s) : "r"(remote));
            asm volatile("ld.shared::cluster.s32 %0, [%1+8];" : "=r"(p.i) : "r"(remote));
            asm volatile("ld.shared::cluster.f32 %0, [%1+12];" : "=f"(p.ym) : "r"(remote));
            asm volatile("ld.shared::cluster.s32 %0, [%1+16];" : "=r"(p.yi) : "r"(remote));
            c = ms_merge(c, p);
        }
        const size_t o = (size_t)b * oi.out_ld + oi.out_off + t + (oi.dyn_off ? *oi.dyn_off : 0);
        if (am) am[o] = c.i;
        if (sampling) {  // the drawn token and log softmax(z / tau) at it
            int tok = c.yi;
            if (tok < 0 || tok >= V) {  // only non-finite logits leave no maximum
                atomicOr(status, QK_STATUS_BAD_TOKEN);
                tok = 0;
            }
            samp.out_tokens[o] = tok;
            if (lp) lp[o] = z[tok] * inv_tau - (c.m + logf(c.s));
        } else if (lp && oi.tgt) {
            const float l = z_tg - (c.m + logf(c.s));
            lp[o] = l;
            if (grpo.loss_tok) {  // Eq. ppo for this token, where its log-prob is formed
                const size_t go = (size_t)b * grpo.ld + t;
                const float ref = grpo.lp_ref ? grpo.lp_ref[go] : l;
                grpo.loss_tok[go] = grpo_token(l, grpo.lp_old[go], ref,
                                               grpo_advantage(grpo.rewards, b, grpo.group), grpo);
            }
        }
    }
    // no CTA leaves while CTA 0 may still read its shared memory
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

void launch_logits_reduce(const float* logits, int M, int V, OutIndex oi, float* lp,
                          int32_t* argmax, uint32_t* status, cudaStream_t s, const GrpoArgs* grpo,
                          const SampleArgs* samp) {
    note_launch();
    if (M <= 0) return;
    GrpoArgs g{};
    if (grpo) g = *grpo;
    SampleArgs sa{};
    if (samp) sa = *samp;
    launch_k(logits_reduce_kernel, dim3(kLogitCtas, M), dim3(256), 0, s, logits, V, oi, lp, argmax,
             status, g, sa);
}

// ---------------------------------------------------------------- vocabulary-tile combine
// One block of 128 threads per logits row: merges the row's per-tile (max, sum of
// exponentials, lowest arg-max) in a fixed order (thread i takes tiles i, i + 128, ...
// ascending, then a fixed tree; equal maxima keep the lower index), then
//   log p(target) = z[target] - (max + log sum exp(z - max)),
// the arg-max and, with grpo, the GRPO token loss, with the output indexing of
// logits_reduce_kernel.
__device__ __forceinline__ void tile_merge(float& m, float& s, int& i, float m2, float s2, int i2) {
    const float mx = fmaxf(m, m2);
    if (mx == -INFINITY) return;
    s = (m == -INFINITY ? 0.f : s * expf(m - mx)) + (m2 == -INFINITY ? 0.f : s2 * expf(m2 - mx));
    i = m > m2 ? i : (m2 > m ? i2 : min(i, i2));
    m = mx;
}

__global__ void __launch_bounds__(128)
    lse_combine_kernel(const float2* __restrict__ ms, const int* __restrict__ idx,
                       const float* __restrict__ zt, int n_vt, int V, OutIndex oi,
                       float* __restrict__ lp, int32_t* __restrict__ am, uint32_t* status,
                       GrpoArgs grpo) {
    __shared__ float sm[4], ss[4];
    __shared__ int si[4];
    pdl_wait();
    pdl_trigger();
    const int r = blockIdx.x;
    const int g = oi.row0 + r;
    const int b = g / oi.T, t = g % oi.T;
    if (t >= oi.out_lim) return;  // uniform over the block
    float m = -INFINITY, sum = 0.f;
    int i = 0x7fffffff;
    const float2* row = ms + (size_t)r * n_vt;
    const int* rowi = idx + (size_t)r * n_vt;
    for (int v = threadIdx.x; v < n_vt; v += 128) {
        const float2 p = row[v];
        tile_merge(m, sum, i, p.x, p.y, rowi[v]);
    }
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
        const float s2 = __shfl_xor_sync(0xffffffffu, sum, o);
        const int i2 = __shfl_xor_sync(0xffffffffu, i, o);
        tile_merge(m, sum, i, m2, s2, i2);
    }
    const int w = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) sm[w] = m, ss[w] = sum, si[w] = i;
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int k = 1; k < 4; ++k) tile_merge(m, sum, i, sm[k], ss[k], si[k]);
        const size_t o = (size_t)b * oi.out_ld + oi.out_off + t + (oi.dyn_off ? *oi.dyn_off : 0);
        if (am) am[o] = i;
        if (lp && oi.tgt) {
            const int tg = oi.tgt[(size_t)b * oi.tgt_ld + oi.tgt_off + t];
            if (tg < 0 || tg >= V) atomicOr(status, QK_STATUS_BAD_TOKEN);  // token 0 was used
            const float l = zt[r] - (m + logf(sum));
            lp[o] = l;
            if (grpo.loss_tok) {  // Eq. ppo for this token, where its log-prob is formed
                const size_t go = (size_t)b * grpo.ld + t;
                const float ref = grpo.lp_ref ? grpo.lp_ref[go] : l;
                grpo.loss_tok[go] = grpo_token(l, grpo.lp_old[go], ref,
                                               grpo_advantage(grpo.rewards, b, grpo.group), grpo);
            }
        }
    }
}

void launch_lse_combine(const float2* ms, const int* idx, const float* zt, int n_vt, int V, int M,
                        OutIndex oi, float* lp, int32_t* argmax, uint32_t* status, cudaStream_t s,
                        const GrpoArgs* grpo) {
    note_launch();
    if (M <= 0) return;
    GrpoArgs g{};
    if (grpo) g = *grpo;
    launch_k(lse_combine_kernel, dim3(M), dim3(128), 0, s, ms, idx, zt, n_vt, V, oi, lp, argmax,
             status, g);
}

// ---------------------------------------------------------------- rollout cursor
__global__ void rollout_prepare_kernel(const int32_t* __restrict__ seq, int L, int P, int B,
                                       int32_t* step, int32_t* pos, int32_t* tok, int32_t* tgt,
                                       int32_t* out_off) {
    pdl_wait();
    pdl_trigger();  // short kernel: let the next one launch and prefetch now
    const int s = *step;
    __syncthreads();  // every thread has read the step before it advances
    for (int b = threadIdx.x; b < B; b += blockDim.x) {
        pos[b] = P + s;
        tok[b] = seq[(size_t)b * L + P + s];
        tgt[b] = seq[(size_t)b * L + P + s + 1];
    }
    if (threadIdx.x == 0) {
        *out_off = s + 1;
        *step = s + 1;
    }
}

void launch_rollout_prepare(const int32_t* seq, int L, int P, int B, int32_t* step, int32_t* pos,
                            int32_t* tok, int32_t* tgt, int32_t* out_off, cudaStream_t s) {
    note_launch();
    launch_k(rollout_prepare_kernel, dim3(1), dim3(256), 0, s, seq, L, P, B, step, pos, tok, tgt,
             out_off);
}

__global__ void rollout_prepare_sampled_kernel(const int32_t* __restrict__ sampled, int ld, int P,
                                               int B, int32_t* step, int32_t* pos, int32_t* tok,
                                               int32_t* out_off) {
    pdl_wait();
    pdl_trigger();
    const int s = *step;
    __syncthreads();  // every thread has read the step before it advances
    for (int b = threadIdx.x; b < B; b += blockDim.x) {
        pos[b] = P + s;
        tok[b] = sampled[(size_t)b * ld + s];
    }
    if (threadIdx.x == 0) {
        *out_off = s + 1;
        *step = s + 1;
    }
}

void launch_rollout_prepare_sampled(const int32_t* sampled, int ld, int P, int B, int32_t* step,
                                    int32_t* pos, int32_t* tok, int32_t* out_off, cudaStream_t s) {
    note_launch();
    launch_k(rollout_prepare_sampled_kernel, dim3(1), dim3(256), 0, s, sampled, ld, P, B, step, pos,
             tok, out_off);
}

// ---------------------------------------------------------------- load-time tables
// cos / sin of p * theta^(-2i/d) in double precision, stored as fp32 [max_positions, d/2].
__global__ void rope_table_kernel(float* cos_t, float* sin_t, int max_positions, int d,
                                  double theta) {
    int half = d / 2;
    size_t n = (size_t)max_positions * half;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n;
         e += (size_t)gridDim.x * blockDim.x) {
        int p = (int)(e / half), i = (int)(e % half);
        double inv_freq = pow(theta, -2.0 * i / d);
        double ang = (double)p * inv_freq;
        double sn, c;
        sincos(ang, &sn, &c);
        cos_t[e] = (float)c;
        sin_t[e] = (float)sn;
    }
}

void launch_rope_table(float* cos_t, float* sin_t, int max_positions, int d, double theta,
                       cudaStream_t s) {
    note_launch();
    size_t n = (size_t)max_positions * (d / 2);
    int blocks = (int)((n + 255) / 256);
    if (blocks > 4096) blocks = 4096;
    rope_table_kernel<<<blocks, 256, 0, s>>>(cos_t, sin_t, max_positions, d, theta);
}

template <typename T>
__global__ void widen_kernel(const T* src, float* dst, int n) {
    int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) dst[i] = to_f(src[i]);
}

void launch_widen_gain(const void* src, int dtype, float* dst, int n, cudaStream_t s) {
    note_launch();
    int blocks = (n + 255) / 256;
    if (dtype == QK_DTYPE_BF16)
        widen_kernel<bf16><<<blocks, 256, 0, s>>>((const bf16*)src, dst, n);
    else
        widen_kernel<float><<<blocks, 256, 0, s>>>((const float*)src, dst, n);
}

}  // namespace qk
