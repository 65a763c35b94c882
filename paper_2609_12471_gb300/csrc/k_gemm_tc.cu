// Tensor-core linear layers on tcgen05 / TMEM / TMA:
//     C[M, N] = X[M, K] * W[N, K]^T   (bf16 in, fp32 accumulate) + fused epilogue.
//
// Operand roles ("swap AB"): the weight tile is the 128-row MMA operand (A) and
// the token tile the N-side operand (B), so one MMA shape serves decode (a few
// tokens, N = 16..64) and prefill/scoring (N = 128 or 256 tokens per tile).
// D[feature, token] sits in TMEM with one feature per lane; an epilogue thread
// owns one output feature and walks the tile's tokens, so stores of a warp hit
// 32 consecutive features of one token row (coalesced), and the residual add,
// SwiGLU and fp32 logits store happen on the accumulator without another pass.
//
// Per CTA (persistent, one per SM, 192 threads):
//   warp 0, one lane : TMA producer over a STAGES-deep ring of (W, X) k-blocks;
//   warp 1           : TMEM allocation; one lane issues tcgen05.mma + commits;
//   warps 2..5       : epilogue, warp w reads TMEM lanes 32*(w%4) .. +31.
// Two TMEM accumulators alternate so the epilogue of tile t overlaps the
// mainloop of tile t+1.  SwiGLU tiles carry 256 weight rows (128 gate rows and
// the matching 128 up rows, packed that way at load) and two accumulators.
//
// Every mbarrier wait is bounded (tc::mbar_wait).  On a timeout the CTA sets its
// abort flag and QK_STATUS_TIMEOUT in the model status word; every role leaves
// its loop, the producer waits (bounded) for the copies it issued, the MMA
// thread waits (bounded) for its MMAs, then TMEM is freed and the CTA exits.
#include <cuda.h>
#include <mutex>

#include "qk_internal.cuh"
#include "tc_ptx.cuh"

namespace qk {

namespace {

constexpr int kThreads = 192;
constexpr int kBK = 64;  // bf16 elements per k-block: one 128-byte swizzle row

__host__ __device__ constexpr int pow2_at_least(int v) {
    int p = 32;
    while (p < v) p <<= 1;
    return p;
}

template <int BN, bool SWIGLU, int STAGES>
struct Cfg {
    static constexpr int A_ROWS = SWIGLU ? 256 : 128;
    static constexpr int A_BYTES = A_ROWS * 128;
    static constexpr int B_BYTES = BN * 128;
    static constexpr int ACC_COLS = SWIGLU ? 2 * BN : BN;
    static constexpr int TMEM_COLS = pow2_at_least(2 * ACC_COLS);
    static constexpr int SMEM = STAGES * (A_BYTES + B_BYTES) + 1024 /*align*/ + 256 /*barriers*/;
    static_assert(TMEM_COLS <= 512, "accumulators exceed TMEM");
    static_assert(BN % 16 == 0 && BN >= 16 && BN <= 256, "invalid MMA N");
};

__device__ __forceinline__ float silu(float g) { return g / (1.f + __expf(-g)); }

template <int BN, bool SWIGLU, int STAGES>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                   void* __restrict__ C, int ldc, int M, int N, int K, int epi, int n_split,
                   uint32_t* __restrict__ status) {
    using G = Cfg<BN, SWIGLU, STAGES>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* sA = smem;
    uint8_t* sB = smem + STAGES * G::A_BYTES;
    uint64_t* full = (uint64_t*)(sB + STAGES * G::B_BYTES);
    uint64_t* empty = full + STAGES;
    uint64_t* tfull = empty + STAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint32_t* tmem_slot = (uint32_t*)(drain + 1);
    volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_feat = N / 128;
    const int n_tok = (M + BN - 1) / BN;
    // Work unit t = ((feat * n_tok) + tok) * n_split + split; a split covers k-blocks
    // [split * kblocks / n_split, (split + 1) * kblocks / n_split).
    const int num_tiles = n_feat * n_tok * n_split;
    const int kblocks = K / kBK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            tc::mbar_init(&full[s], 1);
            tc::mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            tc::mbar_init(&tfull[a], 1);
            tc::mbar_init(&tempty[a], 4);
        }
        tc::mbar_init(drain, 1);
        *abort_flag = 0;
        tc::fence_mbar_init();
        tc::tma_prefetch_desc(&tmW);
        tc::tma_prefetch_desc(&tmX);
    }
    if (warp == 1) tc::tmem_alloc(tmem_slot, G::TMEM_COLS);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;
    // Everything above touched only shared memory and TMEM.  The producer thread
    // waits for the previous kernel after it has issued the first ring of weight
    // tiles (weights are never written by a kernel); every other thread waits now.
    if (!(warp == 0 && lane == 0)) pdl_wait();

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------ TMA producer
            int stage = 0;
            uint32_t phase = 0;
            int armed[STAGES];
            for (int s = 0; s < STAGES; ++s) armed[s] = -1;
            bool ok = true;
            // activation loads held back until the dependency wait: (stage, x, y)
            int pend_stage[STAGES], pend_x[STAGES], pend_y[STAGES];
            int npend = 0;
            bool waited = false;
            auto release_pending = [&]() {
                pdl_wait();
                waited = true;
                for (int i = 0; i < npend; ++i)
                    tc::tma_load_2d(sB + pend_stage[i] * G::B_BYTES, &tmX, pend_x[i], pend_y[i],
                                    &full[pend_stage[i]]);
                npend = 0;
            };
            for (int t = blockIdx.x; ok && t < num_tiles; t += gridDim.x) {
                const int split = t % n_split, rest = t / n_split;
                const int feat = rest / n_tok, tok = rest % n_tok;
                const int kb0 = split * kblocks / n_split, kb1 = (split + 1) * kblocks / n_split;
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!tc::mbar_wait(&empty[stage], phase ^ 1, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc::mbar_expect_tx(&full[stage], G::A_BYTES + G::B_BYTES);
                    tc::tma_load_2d(sA + stage * G::A_BYTES, &tmW, kb * kBK, feat * G::A_ROWS,
                                    &full[stage]);
                    if (waited) {
                        tc::tma_load_2d(sB + stage * G::B_BYTES, &tmX, kb * kBK, tok * BN,
                                        &full[stage]);
                    } else {
                        pend_stage[npend] = stage;
                        pend_x[npend] = kb * kBK;
                        pend_y[npend] = tok * BN;
                        if (++npend == STAGES) release_pending();
                    }
                    armed[stage] = (int)phase;
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
            }
            if (!waited) release_pending();
            pdl_trigger();  // every load of this CTA is issued: the next kernel may be scheduled
            if (!ok) {  // abort path: let every copy this thread issued land before exit
                for (int s = 0; s < STAGES; ++s)
                    if (armed[s] >= 0) tc::mbar_wait_drain(&full[s], (uint32_t)armed[s]);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ------------------------------------------------ MMA issuer
            constexpr uint32_t idesc = tc::idesc_bf16(128, BN);
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true, issued = false;
            for (int t = blockIdx.x; ok && t < num_tiles; t += gridDim.x) {
                const int split = t % n_split;
                const int kb0 = split * kblocks / n_split, kb1 = (split + 1) * kblocks / n_split;
                if (!tc::mbar_wait(&tempty[acc], acc_phase ^ 1, abort_flag)) {
                    ok = false;
                    break;
                }
                tc::fence_after_sync();
                const uint32_t d = tmem_base + (uint32_t)(acc * G::ACC_COLS);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!tc::mbar_wait(&full[stage], phase, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc::fence_after_sync();
                    const uint32_t a0 = tc::smem_u32(sA + stage * G::A_BYTES);
                    const uint32_t b0 = tc::smem_u32(sB + stage * G::B_BYTES);
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k) {
                        const uint64_t bd = tc::sw128_desc(b0 + k * 32);
                        const uint32_t accum = (kb != kb0 || k) ? 1u : 0u;
                        tc::mma_bf16(d, tc::sw128_desc(a0 + k * 32), bd, idesc, accum);
                        if (SWIGLU)
                            tc::mma_bf16(d + BN, tc::sw128_desc(a0 + 128 * 128 + k * 32), bd, idesc,
                                         accum);
                    }
                    issued = true;
                    tc::mma_commit(&empty[stage]);
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
                if (!ok) break;
                tc::mma_commit(&tfull[acc]);
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1;
            }
            if (!ok && issued) {  // abort path: wait for the MMAs in flight
                tc::mma_commit(drain);
                tc::mbar_wait_drain(drain, 0);
            }
        }
    } else {
        // ---------------------------------------------------- epilogue (warps 2..5)
        const int q = warp & 3;
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
            const int split = t % n_split, rest = t / n_split;
            const int feat = rest / n_tok, tok = rest % n_tok;
            bool ok = tc::mbar_wait(&tfull[acc], acc_phase, abort_flag);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            tc::fence_after_sync();
            const int f = feat * 128 + q * 32 + lane;
            const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * G::ACC_COLS);
            for (int c0 = 0; c0 < BN; c0 += 16) {
                const int tok0 = tok * BN + c0;
                if (tok0 >= M) break;
                uint32_t r[16];
                tc::tmem_ld16(tbase + c0, r);
                uint32_t u[16];
                if (SWIGLU) tc::tmem_ld16(tbase + BN + c0, u);
                tc::tmem_wait_ld();
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const int m = tok0 + j;
                    if (m >= M) break;
                    const size_t o = (size_t)m * ldc + f;
                    const float v = __uint_as_float(r[j]);
                    if (SWIGLU) {
                        ((bf16*)C)[o] = __float2bfloat16_rn(silu(v) * __uint_as_float(u[j]));
                    } else if (epi == EPI_PARTIAL_F32) {
                        ((float*)C)[(size_t)split * M * ldc + o] = v;
                    } else if (epi == EPI_STORE_ACT) {
                        ((bf16*)C)[o] = __float2bfloat16_rn(v);
                    } else if (epi == EPI_STORE_F32) {
                        ((float*)C)[o] = v;
                    } else {
                        ((float*)C)[o] += v;
                    }
                }
            }
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&tempty[acc]);
            acc ^= 1;
            if (acc == 0) acc_phase ^= 1;
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    if (threadIdx.x == 0 && *abort_flag) atomicOr(status, QK_STATUS_TIMEOUT);
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem_base, G::TMEM_COLS);
    }
}

// ---------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)p;
    });
    return fn;
}

// 2-D bf16 tensor map over rows of `inner` elements (row stride `ld` elements),
// box of 64 elements x box_rows rows, 128-byte swizzle, zero fill out of range.
bool make_map(CUtensorMap* map, const void* base, int inner, int rows, int ld, int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                    box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

template <int BN, bool SWIGLU, int STAGES>
int launch_cfg(const bf16* A, int lda, const bf16* W, void* C, int ldc, int M, int N, int K,
               int epi, int n_split, int num_sms, uint32_t* status, cudaStream_t s) {
    using G = Cfg<BN, SWIGLU, STAGES>;
    static bool attr_set = false;
    if (!attr_set) {
        if (cudaFuncSetAttribute(gemm_tc_kernel<BN, SWIGLU, STAGES>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, G::SMEM) != cudaSuccess)
            return QK_ECUDA;
        attr_set = true;
    }
    CUtensorMap tmW, tmX;
    const int w_rows = SWIGLU ? 2 * N : N;
    if (!make_map(&tmW, W, K, w_rows, K, G::A_ROWS) || !make_map(&tmX, A, K, M, lda, BN))
        return QK_ECUDA;
    const int tiles = (N / 128) * ((M + BN - 1) / BN) * n_split;
    const int grid = tiles < num_sms ? tiles : num_sms;
    launch_k(gemm_tc_kernel<BN, SWIGLU, STAGES>, dim3(grid), dim3(kThreads), G::SMEM, s, tmW, tmX, C,
             ldc, M, N, K, epi, n_split, status);
    note_launch();
    return QK_OK;
}

}  // namespace

bool gemm_tc_supported(const void* A, int lda, int N, int K) {
    return N % 128 == 0 && K % kBK == 0 && lda % 8 == 0 && ((uintptr_t)A & 15) == 0 &&
           encode_fn() != nullptr;
}

// bf16 linear layer on the tensor cores; token-tile width chosen from M.
int launch_gemm_tc(const bf16* A, int lda, const bf16* W, void* C, int ldc, int M, int N, int K,
                   int epi, int num_sms, uint32_t* status, cudaStream_t s) {
    if (M <= 0) return QK_OK;
    if (epi == EPI_SWIGLU) {
        if (M <= 16) return launch_cfg<16, true, 6>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s);
        if (M <= 32) return launch_cfg<32, true, 6>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s);
        if (M <= 64) return launch_cfg<64, true, 5>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s);
        return launch_cfg<128, true, 4>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s);
    }
    if (M <= 16) return launch_cfg<16, false, 8>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s);
    if (M <= 32) return launch_cfg<32, false, 8>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s);
    if (M <= 64) return launch_cfg<64, false, 8>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s);
    if (M <= 128) return launch_cfg<128, false, 6>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s);
    return launch_cfg<256, false, 4>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s);
}

// Split count for a decode-sized GEMM (one token tile): the smallest S whose
// N/128 * S work units fill the persistent grid to >= 90 % of its last round,
// with at least 4 k-blocks per unit; the best S found otherwise.
int gemm_tc_split(int N, int K, int num_sms) {
    const int n_feat = N / 128, kblocks = K / kBK;
    int best = 1;
    double best_eff = 0.0;
    for (int S = 1; S <= 32 && kblocks / S >= 4; ++S) {
        const int units = n_feat * S;
        const int rounds = (units + num_sms - 1) / num_sms;
        const double eff = (double)units / ((double)rounds * num_sms);
        if (eff >= 0.9) return S;
        if (eff > best_eff + 1e-9) {
            best_eff = eff;
            best = S;
        }
    }
    return best;
}

// Decode-sized linear (M <= 64 rows) split over K: unit `split` writes its fp32 partial
// product to part[split][M][N]; consumers add the n_split partials in order.
int launch_gemm_tc_splitk(const bf16* A, int lda, const bf16* W, float* part, int M, int N, int K,
                          int n_split, int num_sms, uint32_t* status, cudaStream_t s) {
    if (M <= 0) return QK_OK;
    if (M <= 16)
        return launch_cfg<16, false, 8>(A, lda, W, part, N, M, N, K, EPI_PARTIAL_F32, n_split,
                                        num_sms, status, s);
    if (M <= 32)
        return launch_cfg<32, false, 8>(A, lda, W, part, N, M, N, K, EPI_PARTIAL_F32, n_split,
                                        num_sms, status, s);
    return launch_cfg<64, false, 8>(A, lda, W, part, N, M, N, K, EPI_PARTIAL_F32, n_split,
                                    num_sms, status, s);
}

}  // namespace qk
