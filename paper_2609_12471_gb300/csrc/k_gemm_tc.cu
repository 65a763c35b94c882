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

template <int BN, bool SWIGLU, int STAGES, bool FUSED = false>
struct Cfg {
    static constexpr int A_ROWS = SWIGLU ? 256 : 128;
    static constexpr int A_BYTES = A_ROWS * 128;
    static constexpr int B_BYTES = BN * 128;
    static constexpr int ACC_COLS = SWIGLU ? 2 * BN : BN;
    static constexpr int TMEM_COLS = pow2_at_least(2 * ACC_COLS);
    // fused epilogue scratch (floats): s_row[64], p_row[64] (int), red[4][64], xch[128][BN], flag
    static constexpr int FUSE_FLOATS = FUSED ? 64 + 64 + 4 * 64 + 128 * BN + 4 : 0;
    static constexpr int SMEM =
        STAGES * (A_BYTES + B_BYTES) + 1024 /*align*/ + 256 /*barriers*/ + FUSE_FLOATS * 4;
    static_assert(TMEM_COLS <= 512, "accumulators exceed TMEM");
    static_assert(BN % 16 == 0 && BN >= 16 && BN <= 256, "invalid MMA N");
};

__device__ __forceinline__ float silu(float g) { return g / (1.f + __expf(-g)); }

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

template <int BN, bool SWIGLU, int STAGES, bool FUSED>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                   void* __restrict__ C, int ldc, int M, int N, int K, int epi, int n_split,
                   uint32_t* __restrict__ status, const __grid_constant__ Fuse fz) {
    using G = Cfg<BN, SWIGLU, STAGES, FUSED>;
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
    float* fscr = (float*)(smem + STAGES * (G::A_BYTES + G::B_BYTES) + 256);  // fused scratch

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
    } else if constexpr (FUSED) {
        // ---------------------------------------------------- fused epilogue (warps 2..5)
        // One token tile (M <= BN).  Each unit: TMEM -> registers, release the
        // accumulator, write the fp32 partial, take the tile's ticket; the last unit
        // of a tile sums the partials in split order and applies fz.op.
        const int q = warp & 3;
        const int e = threadIdx.x - 64;  // 0..127 across the epilogue warps
        const int row = q * 32 + lane;   // accumulator row (TMEM lane) = feature within the tile
        // Per-token values used by every unit are computed once: the input-norm scale
        // s_row and (QKV) the clamped cache position p_row.  Loops over the tile's
        // tokens are predicated (no early exit) so their independent loads overlap.
        float* s_row = fscr;                      // [64]
        int* p_row = (int*)(fscr + 64);           // [64]
        float* red = fscr + 128;                  // [4][64]
        float* xch = fscr + 128 + 256;            // [128][BN]
        volatile int* flag = (volatile int*)(fscr + 128 + 256 + 128 * BN);
        if (fz.op == FUSE_QKV || fz.op == FUSE_SWIGLU || fz.op == FUSE_COLSCALE) {
            for (int j = e; j < BN; j += 128) {
                float t = 0.f;
                if (j < M)
                    for (int i = 0; i < fz.n_ssq; ++i) t += fz.ssq_in[(size_t)i * M + j];
                s_row[j] = j < M ? rsqrtf(t / (float)fz.H + fz.eps) : 0.f;
            }
        }
        if (fz.op == FUSE_QKV) {
            const int lim = fz.max_seq < fz.max_positions ? fz.max_seq : fz.max_positions;
            for (int j = e; j < BN; j += 128) {
                int p = 0;
                if (j < M) {
                    p = fz.pos.pos_dev ? fz.pos.pos_dev[j] : fz.pos.start;
                    if (p < 0 || p >= lim) {
                        atomicOr(fz.status, QK_STATUS_BAD_POS);
                        p = p < 0 ? 0 : lim - 1;
                    }
                }
                p_row[j] = p;
            }
        }
        epi_bar();
        int acc = 0;
        uint32_t acc_phase = 0;
        const size_t sstride = (size_t)M * N;
        for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
            const int split = t % n_split, feat = t / n_split;
            bool ok = tc::mbar_wait(&tfull[acc], acc_phase, abort_flag);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            tc::fence_after_sync();
            const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * G::ACC_COLS);
            float v[BN];
#pragma unroll
            for (int j = 0; j < BN; ++j) v[j] = 0.f;
#pragma unroll
            for (int c0 = 0; c0 < BN; c0 += 16) {
                if (c0 < M) {
                    uint32_t r[16];
                    tc::tmem_ld16(tbase + c0, r);
                    tc::tmem_wait_ld();
#pragma unroll
                    for (int j = 0; j < 16; ++j) v[c0 + j] = __uint_as_float(r[j]);
                }
            }
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&tempty[acc]);
            acc ^= 1;
            if (acc == 0) acc_phase ^= 1;

            const int f = feat * 128 + row;
            const bool swiglu = fz.op == FUSE_SWIGLU;
            const bool ticketed = swiglu || n_split > 1;
            const int key = swiglu ? feat >> 1 : feat;
            if (ticketed) {
#pragma unroll
                for (int j = 0; j < BN; ++j)
                    if (j < M) fz.part[split * sstride + (size_t)j * N + f] = v[j];
                // The barrier orders every epilogue thread's stores before the ticket
                // thread's fence, which publishes them at GPU scope before the atomic; the
                // last unit's ticket thread fences again before its peers read (L2 loads).
                epi_bar();
                if (e == 0) {
                    const int need = swiglu ? 2 * n_split : n_split;
                    __threadfence();
                    const bool last = atomicAdd(&fz.tickets[key], 1) == need - 1;
                    if (last) __threadfence();
                    *flag = last;
                }
                epi_bar();
                const bool last = *flag != 0;
                if (!last) continue;  // uniform over the four warps
                if (!swiglu) {
                    // sum in split order; the loads of one split are independent, so each
                    // split costs one L2 round trip (this unit's own split is in registers)
                    float a[BN];
#pragma unroll
                    for (int j = 0; j < BN; ++j) a[j] = 0.f;
                    for (int sp = 0; sp < n_split; ++sp) {
                        if (sp == split) {
#pragma unroll
                            for (int j = 0; j < BN; ++j) a[j] += v[j];
                        } else {
                            float ld[BN];
#pragma unroll
                            for (int j = 0; j < BN; ++j)
                                ld[j] = j < M ? __ldcg(&fz.part[sp * sstride + (size_t)j * N + f]) : 0.f;
#pragma unroll
                            for (int j = 0; j < BN; ++j) a[j] += ld[j];
                        }
                    }
#pragma unroll
                    for (int j = 0; j < BN; ++j) v[j] = a[j];
                }
            }
            if (fz.op == FUSE_QKV) {
                const int hh = feat, nq = fz.nq, nkv = fz.nkv;
#pragma unroll
                for (int j = 0; j < BN; ++j) v[j] *= s_row[j];
                if (hh < nq + nkv) {
                    // per-head RMSNorm over the 128 rows of the tile, per token
#pragma unroll
                    for (int j = 0; j < BN; ++j) {
                        float sq = v[j] * v[j];
#pragma unroll
                        for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
                        if (lane == 0) red[q * 64 + j] = sq;
                    }
                    epi_bar();
                    const float gain = hh < nq ? fz.gq[row] : fz.gk[row];
#pragma unroll
                    for (int j = 0; j < BN; ++j) {
                        const float tot = red[j] + red[64 + j] + red[128 + j] + red[192 + j];
                        v[j] = v[j] * rsqrtf(tot / 128.f + fz.eps) * gain;
                        xch[row * BN + j] = v[j];
                    }
                    epi_bar();
                    // rotate-half RoPE: row i < 64 pairs with row i + 64
                    const int i = row & 63;
                    float c[BN], sn[BN];
#pragma unroll
                    for (int j = 0; j < BN; ++j) {
                        c[j] = fz.rope_cos[(size_t)p_row[j] * 64 + i];
                        sn[j] = fz.rope_sin[(size_t)p_row[j] * 64 + i];
                    }
#pragma unroll
                    for (int j = 0; j < BN; ++j) {
                        const float partner = xch[(row ^ 64) * BN + j];
                        const float o = row < 64 ? v[j] * c[j] - partner * sn[j] : v[j] * c[j] + partner * sn[j];
                        if (j < M) {
                            if (hh < nq)
                                fz.q_out[(size_t)j * fz.q_ld + (size_t)hh * 128 + row] = __float2bfloat16_rn(o);
                            else
                                fz.k_cache[(((size_t)j * nkv + (hh - nq)) * fz.max_seq + p_row[j]) * 128 + row] =
                                    __float2bfloat16_rn(o);
                        }
                    }
                } else {
#pragma unroll
                    for (int j = 0; j < BN; ++j)
                        if (j < M)
                            fz.v_cache[(((size_t)j * nkv + (hh - nq - nkv)) * fz.max_seq + p_row[j]) * 128 + row] =
                                __float2bfloat16_rn(v[j]);
                }
            } else if (fz.op == FUSE_RESID) {
                const float gn = fz.g_next[f];
                float xo[BN];
#pragma unroll
                for (int j = 0; j < BN; ++j) xo[j] = j < M ? fz.x[(size_t)j * N + f] : 0.f;
#pragma unroll
                for (int j = 0; j < BN; ++j) {
                    const float xn = xo[j] + v[j];
                    if (j < M) {
                        fz.x[(size_t)j * N + f] = xn;
                        fz.xg_out[(size_t)j * N + f] = __float2bfloat16_rn(xn * gn);
                    }
                    float sq = j < M ? xn * xn : 0.f;
#pragma unroll
                    for (int k = 16; k > 0; k >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, k);
                    if (lane == 0) red[q * 64 + j] = sq;
                }
                epi_bar();
                if (e < M) fz.ssq_out[(size_t)feat * M + e] = red[e] + red[64 + e] + red[128 + e] + red[192 + e];
            } else if (fz.op == FUSE_SWIGLU) {
                // this unit completed the pair: gate tile 2 jb, up tile 2 jb + 1
                const int jb = feat >> 1, I = N / 2;
                const int fg = (2 * jb) * 128 + row, fu = fg + 128;
                float gs[BN], us[BN];
#pragma unroll
                for (int j = 0; j < BN; ++j) gs[j] = us[j] = 0.f;
                for (int sp = 0; sp < n_split; ++sp) {
                    float lg[BN], lu[BN];
#pragma unroll
                    for (int j = 0; j < BN; ++j) {
                        lg[j] = j < M ? __ldcg(&fz.part[sp * sstride + (size_t)j * N + fg]) : 0.f;
                        lu[j] = j < M ? __ldcg(&fz.part[sp * sstride + (size_t)j * N + fu]) : 0.f;
                    }
#pragma unroll
                    for (int j = 0; j < BN; ++j) {
                        gs[j] += lg[j];
                        us[j] += lu[j];
                    }
                }
#pragma unroll
                for (int j = 0; j < BN; ++j) {
                    const float g = gs[j] * s_row[j], u = us[j] * s_row[j];
                    if (j < M)
                        fz.h_out[(size_t)j * I + (size_t)jb * 128 + row] =
                            __float2bfloat16_rn(g / (1.f + __expf(-g)) * u);
                }
            } else if (fz.op == FUSE_COLSCALE) {
#pragma unroll
                for (int j = 0; j < BN; ++j)
                    if (j < M) ((float*)C)[(size_t)j * ldc + f] = v[j] * s_row[j];
            }
            if (ticketed && e == 0) fz.tickets[key] = 0;
            epi_bar();  // scratch (red, xch, flag) is reused by the next unit
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

template <int BN, bool SWIGLU, int STAGES, bool FUSED = false>
int launch_cfg(const bf16* A, int lda, const bf16* W, void* C, int ldc, int M, int N, int K,
               int epi, int n_split, int num_sms, uint32_t* status, cudaStream_t s,
               const Fuse* fz = nullptr) {
    using G = Cfg<BN, SWIGLU, STAGES, FUSED>;
    static bool attr_set = false;
    if (!attr_set) {
        if (cudaFuncSetAttribute(gemm_tc_kernel<BN, SWIGLU, STAGES, FUSED>,
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
    Fuse none{};
    launch_k(gemm_tc_kernel<BN, SWIGLU, STAGES, FUSED>, dim3(grid), dim3(kThreads), G::SMEM, s, tmW,
             tmX, C, ldc, M, N, K, epi, n_split, status, fz ? *fz : none);
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
// N/128 * S work units fill the persistent grid to >= 80 % of its last round,
// with at least 12 k-blocks per unit (each unit ends in a fused epilogue); the
// best S found otherwise.
int gemm_tc_split(int N, int K, int num_sms) {
    const int n_feat = N / 128, kblocks = K / kBK;
    int best = 1;
    double best_eff = 0.0;
    for (int S = 1; S <= 32 && kblocks / S >= 12; ++S) {
        const int units = n_feat * S;
        const int rounds = (units + num_sms - 1) / num_sms;
        const double eff = (double)units / ((double)rounds * num_sms);
        if (eff >= 0.8) return S;
        if (eff > best_eff + 1e-9) {
            best_eff = eff;
            best = S;
        }
    }
    return best;
}

// Decode linear with a fused epilogue (see Fuse); one token tile of M <= 64 rows.
int launch_gemm_tc_fused(const bf16* A, int lda, const bf16* W, float* out, int M, int N, int K,
                         int n_split, const Fuse& f, int num_sms, uint32_t* status, cudaStream_t s) {
    if (M <= 0) return QK_OK;
    if (M > 64) return QK_ESHAPE;
    if (M <= 16)
        return launch_cfg<16, false, 8, true>(A, lda, W, out, N, M, N, K, EPI_PARTIAL_F32, n_split,
                                              num_sms, status, s, &f);
    if (M <= 32)
        return launch_cfg<32, false, 8, true>(A, lda, W, out, N, M, N, K, EPI_PARTIAL_F32, n_split,
                                              num_sms, status, s, &f);
    return launch_cfg<64, false, 7, true>(A, lda, W, out, N, M, N, K, EPI_PARTIAL_F32, n_split,
                                          num_sms, status, s, &f);
}

}  // namespace qk
