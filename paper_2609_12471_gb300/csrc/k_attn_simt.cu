// Causal grouped-query attention over a per-layer KV cache, SIMT version.
//
// Used for the fp32 model (no tensor cores may touch it: TF32 would break the
// 1e-4 tolerance) and for any head_dim / grouping the tensor-core kernels do
// not cover.  One warp per (token row, query head); the warps of a block are the
// query heads sharing one kv head, so K/V rows are read once from DRAM and then
// hit in L1/L2.  Online softmax (running max m, running sum l) over blocks of 32
// keys: lane j scores key kb + j, then every lane accumulates its d/32 output
// dimensions over the block.
#include <math.h>

#include "qk_internal.cuh"

namespace qk {

namespace {

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(bf16 v) { return __bfloat162float(v); }
template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

// Dot product of a cache row with q (fp32, in shared memory), 16-byte loads.
template <typename T, int D>
__device__ __forceinline__ float row_dot(const T* __restrict__ row, const float* q) {
    constexpr int PER = 16 / sizeof(T);
    float s = 0.f;
#pragma unroll
    for (int c = 0; c < D / PER; ++c) {
        uint4 raw = *reinterpret_cast<const uint4*>(row + c * PER);
        const T* v = reinterpret_cast<const T*>(&raw);
#pragma unroll
        for (int e = 0; e < PER; ++e) s += to_f(v[e]) * q[c * PER + e];
    }
    return s;
}

template <typename T, int D>
__global__ void attention_simt_kernel(const T* __restrict__ q, int q_ld, const T* __restrict__ kc,
                                      const T* __restrict__ vc, int nq, int nkv, KvPages kp,
                                      PosIndex pos, T* __restrict__ o, uint32_t* status) {
    constexpr int E = D / 32;
    extern __shared__ float qs[];  // [warps][D]
    pdl_wait();
    int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int group = nq / nkv;
    int r = blockIdx.x, kvh = blockIdx.y, h = kvh * group + warp;
    int b = r / pos.T, t = r % pos.T;
    int p = pos.pos_dev ? pos.pos_dev[b] + t : pos.start + t;
    const int cap = kp.cap();
    if (p < 0 || p >= cap) {
        if (lane == 0) atomicOr(status, QK_STATUS_BAD_POS);
        p = p < 0 ? 0 : cap - 1;
    }
    float* qw = qs + warp * D;
    const T* qrow = q + (size_t)r * q_ld + (size_t)h * D;
    float scale = rsqrtf((float)D);
#pragma unroll
    for (int i = 0; i < E; ++i) qw[lane + 32 * i] = to_f(qrow[lane + 32 * i]) * scale;
    __syncwarp();
    // row of key position j in the K and V views
    auto krow = [&](int j) { return (size_t)kv_row(kp, nkv, b, kvh, j, status) * D; };
    float m = -INFINITY, l = 0.f, acc[E];
#pragma unroll
    for (int i = 0; i < E; ++i) acc[i] = 0.f;
    for (int kb = 0; kb <= p; kb += 32) {
        int j = kb + lane;
        const size_t jr = j <= p ? krow(j) : 0;  // this lane's key's row in K and in V
        float s = j <= p ? row_dot<T, D>(kc + jr, qw) : -INFINITY;
        float mb = s;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) mb = fmaxf(mb, __shfl_xor_sync(0xffffffffu, mb, off));
        float m_new = fmaxf(m, mb);
        float corr = expf(m - m_new);
        float pj = j <= p ? expf(s - m_new) : 0.f;
        float ps = pj;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, off);
        l = l * corr + ps;
#pragma unroll
        for (int i = 0; i < E; ++i) acc[i] *= corr;
        int nk = p - kb + 1 < 32 ? p - kb + 1 : 32;
        for (int jj = 0; jj < nk; ++jj) {
            float w = __shfl_sync(0xffffffffu, pj, jj);
            const T* vr = vc + __shfl_sync(0xffffffffu, jr, jj);
#pragma unroll
            for (int i = 0; i < E; ++i) acc[i] += w * to_f(vr[lane + 32 * i]);
        }
        m = m_new;
    }
    float inv = 1.f / l;
    T* orow = o + ((size_t)r * nq + h) * D;
#pragma unroll
    for (int i = 0; i < E; ++i) orow[lane + 32 * i] = from_f<T>(acc[i] * inv);
}

}  // namespace

void launch_attention_simt(const void* q, int q_ld, const void* k_cache, const void* v_cache,
                           int dtype, int M, int nq, int nkv, int d, const KvPages& kp, PosIndex pos,
                           void* o, uint32_t* status, cudaStream_t s) {
    note_launch();
    if (M <= 0) return;
    int group = nq / nkv;
    dim3 grid(M, nkv);
    int threads = 32 * group;
    size_t smem = (size_t)group * d * sizeof(float);
#define QK_ATT(T, D)                                                                           \
    launch_k(attention_simt_kernel<T, D>, grid, dim3(threads), smem, s, (const T*)q, q_ld,    \
             (const T*)k_cache, (const T*)v_cache, nq, nkv, kp, pos, (T*)o, status)
    if (dtype == QK_DTYPE_BF16) {
        if (d == 128) QK_ATT(bf16, 128); else QK_ATT(bf16, 64);
    } else {
        if (d == 128) QK_ATT(float, 128); else QK_ATT(float, 64);
    }
#undef QK_ATT
}

}  // namespace qk
