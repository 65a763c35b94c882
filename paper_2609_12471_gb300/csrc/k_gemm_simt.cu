// CUDA-core linear layers: C[M, N] = A[M, K] * W[N, K]^T (+ epilogue).
//
//  * gemm_simt: a 64x64x16 shared-memory tiled GEMM in fp32 arithmetic, used for
//    the fp32 model (the 1e-4 tolerance of that model rules out TF32 tensor cores).
//  * gemv_bf16: the weight-streaming path for a handful of token rows (decode at
//    batch <= 16): each warp streams R weight rows with 16-byte loads, U chunks in
//    flight per lane, and multiplies them against every token row.  At this size
//    the layer is bound by reading W once from HBM; the SwiGLU and residual
//    epilogues are fused so no intermediate leaves the SM.
#include <math.h>

#include "qk_internal.cuh"

namespace qk {

namespace {

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(bf16 v) { return __bfloat162float(v); }

template <typename T>
__device__ __forceinline__ void load4(const T* p, float* out) {
    if constexpr (sizeof(T) == 4) {
        float4 v = *reinterpret_cast<const float4*>(p);
        out[0] = v.x; out[1] = v.y; out[2] = v.z; out[3] = v.w;
    } else {
        uint2 v = *reinterpret_cast<const uint2*>(p);
        const bf16* h = reinterpret_cast<const bf16*>(&v);
        out[0] = to_f(h[0]); out[1] = to_f(h[1]); out[2] = to_f(h[2]); out[3] = to_f(h[3]);
    }
}

template <typename T>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const T* __restrict__ A, int lda,
                                                        const T* __restrict__ W,
                                                        void* __restrict__ C, int ldc, int M,
                                                        int N, int K, int epi) {
    constexpr int BM = 64, BN = 64, BK = 16;
    __shared__ float As[BK][BM + 4];
    __shared__ float Ws[BK][BN + 4];
    pdl_wait();
    int tid = threadIdx.x;
    int tx = tid % 16, ty = tid / 16;
    int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
    int lr = tid / 4, lk = (tid % 4) * 4;
    float acc[4][4] = {};
    for (int k0 = 0; k0 < K; k0 += BK) {
        float a[4] = {0.f, 0.f, 0.f, 0.f}, w[4] = {0.f, 0.f, 0.f, 0.f};
        if (m0 + lr < M) load4(A + (size_t)(m0 + lr) * lda + k0 + lk, a);
        if (n0 + lr < N) load4(W + (size_t)(n0 + lr) * K + k0 + lk, w);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            As[lk + e][lr] = a[e];
            Ws[lk + e][lr] = w[e];
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < BK; ++kk) {
            float av[4], wv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) av[i] = As[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) wv[j] = Ws[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], wv[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        int m = m0 + ty * 4 + i;
        if (m >= M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            int n = n0 + tx * 4 + j;
            if (n >= N) continue;
            size_t o = (size_t)m * ldc + n;
            if (epi == EPI_STORE_ACT) {
                if constexpr (sizeof(T) == 2) ((bf16*)C)[o] = __float2bfloat16_rn(acc[i][j]);
                else ((float*)C)[o] = acc[i][j];
            } else if (epi == EPI_STORE_F32)
                ((float*)C)[o] = acc[i][j];
            else
                ((float*)C)[o] += acc[i][j];
        }
    }
}

// Dot of 8 bf16 weights with 8 bf16 activations, accumulated in fp32.
__device__ __forceinline__ float dot8(const uint4& w, const uint4& x) {
    const __nv_bfloat162* wp = reinterpret_cast<const __nv_bfloat162*>(&w);
    const __nv_bfloat162* xp = reinterpret_cast<const __nv_bfloat162*>(&x);
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float2 a = __bfloat1622float2(wp[i]);
        float2 b = __bfloat1622float2(xp[i]);
        s = fmaf(a.x, b.x, s);
        s = fmaf(a.y, b.y, s);
    }
    return s;
}

// Each warp owns R output features (2R weight rows for SwiGLU: gate rows then up rows).
template <int MT, int R, bool SW>
__global__ void __launch_bounds__(256) gemv_bf16_kernel(const bf16* __restrict__ A, int lda,
                                                        const bf16* __restrict__ W,
                                                        void* __restrict__ C, int ldc, int N,
                                                        int K, int epi) {
    constexpr int NR = SW ? 2 * R : R;
    constexpr int U = 2;
    pdl_wait();
    int lane = threadIdx.x & 31;
    int f0 = (blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5)) * R;
    if (f0 >= N) return;
    const bf16* rows[NR];
#pragma unroll
    for (int i = 0; i < R; ++i) {
        int f = min(f0 + i, N - 1);
        if (SW) {
            size_t g = (size_t)(f >> 7) * 256 + (f & 127);
            rows[i] = W + g * K;
            rows[R + i] = W + (g + 128) * K;
        } else {
            rows[i] = W + (size_t)f * K;
        }
    }
    float acc[NR][MT];
#pragma unroll
    for (int i = 0; i < NR; ++i)
#pragma unroll
        for (int t = 0; t < MT; ++t) acc[i][t] = 0.f;
    int k = lane * 8;
    for (; k + (U - 1) * 256 < K; k += U * 256) {
        uint4 w[U][NR];
#pragma unroll
        for (int u = 0; u < U; ++u)
#pragma unroll
            for (int i = 0; i < NR; ++i)
                w[u][i] = __ldcs(reinterpret_cast<const uint4*>(rows[i] + k + u * 256));
#pragma unroll
        for (int u = 0; u < U; ++u)
#pragma unroll
            for (int t = 0; t < MT; ++t) {
                uint4 x = __ldg(reinterpret_cast<const uint4*>(A + (size_t)t * lda + k + u * 256));
#pragma unroll
                for (int i = 0; i < NR; ++i) acc[i][t] += dot8(w[u][i], x);
            }
    }
    for (; k < K; k += 256) {
#pragma unroll
        for (int t = 0; t < MT; ++t) {
            uint4 x = __ldg(reinterpret_cast<const uint4*>(A + (size_t)t * lda + k));
#pragma unroll
            for (int i = 0; i < NR; ++i)
                acc[i][t] += dot8(__ldcs(reinterpret_cast<const uint4*>(rows[i] + k)), x);
        }
    }
#pragma unroll
    for (int i = 0; i < NR; ++i)
#pragma unroll
        for (int t = 0; t < MT; ++t)
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) acc[i][t] += __shfl_xor_sync(0xffffffffu, acc[i][t], o);
#pragma unroll
    for (int i = 0; i < R; ++i) {
        int f = f0 + i;
#pragma unroll
        for (int t = 0; t < MT; ++t) {
            if (lane != ((i * MT + t) & 31) || f >= N) continue;
            size_t o = (size_t)t * ldc + f;
            if (SW) {
                float g = acc[i][t], u = acc[R + i][t];
                ((bf16*)C)[o] = __float2bfloat16_rn(g / (1.f + expf(-g)) * u);
            } else if (epi == EPI_STORE_ACT) {
                ((bf16*)C)[o] = __float2bfloat16_rn(acc[i][t]);
            } else if (epi == EPI_STORE_F32) {
                ((float*)C)[o] = acc[i][t];
            } else {
                ((float*)C)[o] += acc[i][t];
            }
        }
    }
}

template <int MT>
void gemv_dispatch(const bf16* A, int lda, const bf16* W, void* C, int ldc, int N, int K, int epi,
                   cudaStream_t s) {
    constexpr int R = 2;
    int warps = (N + R - 1) / R;
    int blocks = (warps + 7) / 8;
    if (epi == EPI_SWIGLU)
        launch_k(gemv_bf16_kernel<MT, R, true>, dim3(blocks), dim3(256), 0, s, A, lda, W, C, ldc, N,
                 K, epi);
    else
        launch_k(gemv_bf16_kernel<MT, R, false>, dim3(blocks), dim3(256), 0, s, A, lda, W, C, ldc, N,
                 K, epi);
}

}  // namespace

void launch_gemm_simt(const void* A, int lda, const void* W, void* C, int ldc, int M, int N,
                      int K, int dtype, int epi, cudaStream_t s) {
    note_launch();
    if (M <= 0 || N <= 0) return;
    dim3 grid((N + 63) / 64, (M + 63) / 64);
    if (dtype == QK_DTYPE_BF16)
        launch_k(gemm_simt_kernel<bf16>, grid, dim3(256), 0, s, (const bf16*)A, lda,
                 (const bf16*)W, C, ldc, M, N, K, epi);
    else
        launch_k(gemm_simt_kernel<float>, grid, dim3(256), 0, s, (const float*)A, lda,
                 (const float*)W, C, ldc, M, N, K, epi);
}

// M <= 16 token rows (the model uses it up to kGemvMaxRows); N output features (I for SwiGLU).
void launch_gemv_bf16(const bf16* A, int lda, const bf16* W, void* C, int ldc, int M, int N,
                      int K, int epi, cudaStream_t s) {
    note_launch();
    switch (M) {
        case 1: gemv_dispatch<1>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 2: gemv_dispatch<2>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 3: gemv_dispatch<3>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 4: gemv_dispatch<4>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 5: gemv_dispatch<5>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 6: gemv_dispatch<6>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 7: gemv_dispatch<7>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 8: gemv_dispatch<8>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 9: gemv_dispatch<9>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 10: gemv_dispatch<10>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 11: gemv_dispatch<11>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 12: gemv_dispatch<12>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 13: gemv_dispatch<13>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 14: gemv_dispatch<14>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 15: gemv_dispatch<15>(A, lda, W, C, ldc, N, K, epi, s); break;
        case 16: gemv_dispatch<16>(A, lda, W, C, ldc, N, K, epi, s); break;
        default: break;
    }
}

}  // namespace qk
