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
// Per CTA (persistent, one per SM, 192 threads; the 16-row decode configuration
// is small enough for a CTA of the next kernel to become resident beside it):
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
// A launch with test_wait > 0 (the qk_debug_expire_next_wait hook of the plain
// GEMM) exercises that path: CTA 0 issues no copy for its first k-block and
// waits at most test_wait cycles, so its MMA thread's wait for that copy expires.
#include <cuda.h>
#include <mutex>

#include "qk_internal.cuh"
#include "tc_ptx.cuh"

namespace qk {

namespace {

constexpr int kThreads = 192;
constexpr int kBK = 64;  // bf16 elements per k-block: one 128-byte swizzle row
// Decode (fused, 16-row) configuration.  Five ring stages (109 KB of shared
// memory) and at most 168 registers a thread let a CTA of the next kernel become
// resident beside one of this kernel, so its weight prefetch starts while this
// kernel's last tiles finish (measured faster than an 8-stage ring that needs the
// whole SM); partial slots are loaded two at a time to stay inside the registers
// (four at a time, measured, gained nothing).
constexpr int kFused16Stages = 5;
constexpr int kFusedCtasPerSm = 2;
constexpr int kFused16PartialBatch = 2;

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
    // fused epilogue scratch (floats): s_row[64], p_row[64] (int), red[4][64], xch[BN][128],
    // cos / sin [2][BN][64], flag, c_row[64] (int)
    // plain GEMM: the EPI_LSE transpose buffer [16 tokens][128 features] and the tile's targets
    static constexpr int FUSE_FLOATS = FUSED ? 64 + 64 + 4 * 64 + 128 * BN + 128 * BN + 4 + 64
                                             : 16 * 128 + (BN > 16 ? BN : 16);
    static constexpr int SMEM =
        STAGES * (A_BYTES + B_BYTES) + 1024 /*align*/ + 256 /*barriers*/ + FUSE_FLOATS * 4;
    static_assert(TMEM_COLS <= 512, "accumulators exceed TMEM");
    static_assert(BN % 16 == 0 && BN >= 16 && BN <= 256, "invalid MMA N");
};

__device__ __forceinline__ float silu(float g) { return g / (1.f + __expf(-g)); }

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// One level of a reduce-scatter butterfly over the warp: C values per lane become
// C / 2, each the sum of two lanes' values; lanes with `mask` set keep the upper half.
template <int C>
__device__ __forceinline__ void rs_level(float* v, int lane, int mask) {
    const bool up = (lane & mask) != 0;
#pragma unroll
    for (int i = 0; i < C / 2; ++i) {
        const float send = up ? v[i] : v[i + C / 2];
        const float keep = up ? v[i + C / 2] : v[i];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, mask);
    }
}

// out[i] = sum over the warp's 32 lanes of v[i], i < N (N = 16 or 32): log2 N
// butterfly levels (N - 1 shuffles, then 5 - log2 N plain ones) instead of N
// separate five-level reductions.  v is clobbered.
template <int N>
__device__ __forceinline__ void warp_col_sums(float (&v)[N], float* out, int lane) {
    static_assert(N == 16 || N == 32, "16 or 32 values per lane");
    rs_level<N>(v, lane, 16);
    rs_level<N / 2>(v, lane, 8);
    rs_level<N / 4>(v, lane, 4);
    rs_level<N / 8>(v, lane, 2);
    if constexpr (N == 32) rs_level<2>(v, lane, 1);
    else v[0] += __shfl_xor_sync(0xffffffffu, v[0], 1);
    // the value a lane holds: bits 4..1 (and 0 for N = 32) of the lane pick halves
    int idx = ((lane >> 4) & 1) * (N / 2) + ((lane >> 3) & 1) * (N / 4) + ((lane >> 2) & 1) * (N / 8) +
              ((lane >> 1) & 1) * (N / 16);
    if constexpr (N == 32) idx += lane & 1;
    if (N == 32 || (lane & 1) == 0) out[idx] = v[0];
}

// A CTA's work as a sequence of segments: tile (feat, tok) over k-blocks [kb0, kb1).
//  * plain: unit t = blockIdx.x + i * gridDim.x of n_feat x n_tok x n_split, one
//    segment per unit (split s covers k-blocks [s K / S, (s + 1) K / S));
//  * FUSED (one token tile): the n_feat x kblocks k-block iterations are cut into
//    gridDim.x equal ranges; CTA c takes [c I / C, (c + 1) I / C) and a segment is
//    the part of its range inside one tile.  Every CTA streams the same weight
//    bytes; a tile shared by several CTAs is finished by the last of them.
struct Seg {
    int feat, tok, split, kb0, kb1;
    long long next;  // where the following segment starts
};

template <bool FUSED>
__device__ __forceinline__ bool seg_at(Seg& sg, long long at, long long hi, int n_tok, int n_split,
                                       int kblocks) {
    if (at >= hi) return false;
    if constexpr (FUSED) {
        sg.feat = (int)(at / kblocks);
        sg.tok = 0;
        sg.split = 0;
        sg.kb0 = (int)(at - (long long)sg.feat * kblocks);
        const long long tile_end = (long long)(sg.feat + 1) * kblocks;
        const long long end = hi < tile_end ? hi : tile_end;
        sg.kb1 = sg.kb0 + (int)(end - at);
        sg.next = end;
    } else {
        const int t = (int)at;
        sg.split = t % n_split;
        const int rest = t / n_split;
        sg.feat = rest / n_tok;
        sg.tok = rest % n_tok;
        sg.kb0 = sg.split * kblocks / n_split;
        sg.kb1 = (sg.split + 1) * kblocks / n_split;
        sg.next = at + gridDim.x;
    }
    return true;
}

// CTA owning k-block iteration `it` of a FUSED launch (I iterations, C CTAs).
__device__ __forceinline__ int it_owner(long long it, long long I, int C) {
    return (int)(((it + 1) * C - 1) / I);
}

// Fused epilogue of one decode-sized linear (warps 2..5 of the block; see Fuse): the
// segments [seg_lo, seg_hi) of k-block iterations of this CTA (`cta`, of n_cta), in
// order.  acc / acc_phase: the TMEM accumulator ring position, carried across calls
// by a persistent caller.  C / ldc: the FUSE_COLSCALE output.  Returns false if a
// wait gave up (the abort flag is raised).
template <int BN, int STAGES>
__device__ __forceinline__ bool fused_epilogue(const Fuse& fz, float* C, int ldc, int M, int N,
                                               int kblocks, long long n_iter, long long seg_lo,
                                               long long seg_hi, int n_cta, uint32_t tmem_base,
                                               uint64_t* tfull, uint64_t* tempty, int& acc,
                                               uint32_t& acc_phase, float* fscr,
                                               volatile int* abort_flag, int cta = -1) {
    using G = Cfg<BN, false, STAGES, true>;
    if (cta < 0) cta = (int)blockIdx.x;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // One token tile (M <= BN).  Per segment: prefetch the op's inputs, TMEM ->
    // registers, release the accumulator; a segment holding part of its tile's k
    // range writes its fp32 partial and takes the tile's ticket, and the last one
    // sums the tile's slots in k order; then the op.  Global loads on this path are
    // issued in batches ahead of their use: under the weight stream of the next
    // kernel's prefetch, one L2 round trip costs about a microsecond.
    const int q = warp & 3;
    const int e = threadIdx.x - 64;  // 0..127 across the epilogue warps
    const int row = q * 32 + lane;   // accumulator row (TMEM lane) = feature within the tile
    float* s_row = fscr;                  // [64] input-norm scale per token
    int* p_row = (int*)(fscr + 64);       // [64] clamped cache position per token (QKV)
    float* red = fscr + 128;              // [4][64] per-warp sums
    float* xch = fscr + 384;              // [BN][128]: QKV partner exchange, RESID x prefetch
    float* rope_c = xch + 128 * BN;       // [BN][64] cos / sin at each token's position (QKV)
    float* rope_s = rope_c + 64 * BN;
    volatile int* flag = (volatile int*)(rope_s + 64 * BN);
    int* c_row = (int*)(rope_s + 64 * BN + 4);  // [64] cache row of kv head 0 per token (QKV)
    constexpr int kParts = 128 / BN;
    {
        // s_row[j] = rsqrt(sum_i ssq_in[i][j] / H + eps): 128 / BN threads per token
        // each sum every (128 / BN)-th tile sum, then token j's thread adds them in order
        const bool need_s = fz.op == FUSE_QKV || fz.op == FUSE_SWIGLU || fz.op == FUSE_COLSCALE;
        const int j = e % BN, part = e / BN;
        float t = 0.f;
        if (need_s && j < M)
#pragma unroll 8
            for (int i = part; i < fz.n_ssq; i += kParts) t += fz.ssq_in[(size_t)i * M + j];
        xch[part * BN + j] = t;
        if (fz.op == FUSE_QKV && e < BN) {
            const int lim = fz.kv.cap() < fz.max_positions ? fz.kv.cap() : fz.max_positions;
            int p = 0;
            if (e < M) {
                p = fz.pos.pos_dev ? fz.pos.pos_dev[e] : fz.pos.start;
                if (p < 0 || p >= lim) {
                    atomicOr(fz.status, QK_STATUS_BAD_POS);
                    p = p < 0 ? 0 : lim - 1;
                }
            }
            p_row[e] = p;
            // kv head g of the token sits g x page rows further: (page id x nkv + g) x page + offset
            c_row[e] = e < M ? kv_row(fz.kv, fz.nkv, e, 0, p, fz.status) : 0;
        }
        epi_bar();
        if (e < BN) {
            float tt = 0.f;
            for (int pp = 0; pp < kParts; ++pp) tt += xch[pp * BN + e];
            s_row[e] = e < M ? rsqrtf(tt / (float)fz.H + fz.eps) : 0.f;
        }
        if (fz.op == FUSE_QKV) {
            for (int idx = e; idx < M * 64; idx += 128) {
                const int jj = idx >> 6, i = idx & 63;
                tc::cp_async4(&rope_c[idx], &fz.rope_cos[(size_t)p_row[jj] * 64 + i]);
                tc::cp_async4(&rope_s[idx], &fz.rope_sin[(size_t)p_row[jj] * 64 + i]);
            }
            tc::cp_async_commit();
        }
        epi_bar();  // s_row, p_row and xch settled
    }
    constexpr int PB = BN <= 16 ? kFused16PartialBatch : (BN <= 32 ? 3 : 1);  // partial slots per load batch
    // Partials: slot (CTA + tile) holds one segment's [M][128] fp32 sums; the slots of
    // tile f are owner(first k-block) + f .. owner(last k-block) + f, in k order.
    auto slot0 = [&](int ft) { return it_owner((long long)ft * kblocks, n_iter, n_cta) + ft; };
    auto slot1 = [&](int ft) { return it_owner((long long)ft * kblocks + kblocks - 1, n_iter, n_cta) + ft; };
    Seg sg;
    for (bool have = seg_at<true>(sg, seg_lo, seg_hi, 1, 1, kblocks); have;
         have = seg_at<true>(sg, sg.next, seg_hi, 1, 1, kblocks)) {
        const int feat = sg.feat;
        const int f = feat * 128 + row;
        // ---- op inputs, loaded while the accumulator is still being produced
        float gain = 0.f;
        if (fz.op == FUSE_QKV) {
            if (feat < fz.nq) gain = fz.gq[row];
            else if (feat < fz.nq + fz.nkv) gain = fz.gk[row];
        } else if (fz.op == FUSE_RESID) {
            gain = fz.g_next[f];
#pragma unroll
            for (int j = 0; j < BN; ++j)
                if (j < M) tc::cp_async4(&xch[j * 128 + row], &fz.x[(size_t)j * N + f]);
            tc::cp_async_commit();
        }
        // the outcome of the wait is made uniform over the four warps, which meet at
        // named barriers below
        const bool ok = tc::bar128_and(tc::mbar_wait(&tfull[acc], acc_phase, abort_flag));
        if (!ok) {
            tc::cp_async_wait_all();
            return false;
        }
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

        const bool swiglu = fz.op == FUSE_SWIGLU;
        // a tile done whole by this CTA needs no partials (SwiGLU pairs two tiles: always)
        const bool ticketed = swiglu || sg.kb0 != 0 || sg.kb1 != kblocks;
        const int key = swiglu ? feat >> 1 : feat;
        const int my_slot = cta + feat;
        if (ticketed) {
#pragma unroll
            for (int j = 0; j < BN; ++j)
                if (j < M) fz.part[((size_t)my_slot * M + j) * 128 + row] = v[j];
            // The barrier orders every epilogue thread's stores before the ticket
            // thread's release (cumulative over the barrier); its acquire orders the
            // last segment's reads after every other segment's stores.
            epi_bar();
            if (e == 0) {
                const int need = swiglu ? slot1(2 * key) - slot0(2 * key) + slot1(2 * key + 1) -
                                              slot0(2 * key + 1) + 2
                                        : slot1(feat) - slot0(feat) + 1;
                *flag = tc::atom_add_acq_rel_gpu(&fz.tickets[key], 1) == need - 1;
            }
            epi_bar();
            const bool last = *flag != 0;
            if (!last) continue;  // uniform over the four warps
            if (!swiglu) {
                // sum the tile's slots in k order (this CTA's own slot from registers)
                float a[BN];
#pragma unroll
                for (int j = 0; j < BN; ++j) a[j] = 0.f;
                const int s0 = slot0(feat), s1 = slot1(feat);
                for (int base = s0; base <= s1; base += PB) {
                    float ld[PB][BN];
#pragma unroll
                    for (int k = 0; k < PB; ++k) {
                        const int sl = base + k;
                        const bool rd = sl <= s1 && sl != my_slot;
#pragma unroll
                        for (int j = 0; j < BN; ++j)
                            ld[k][j] = rd && j < M ? __ldcg(&fz.part[((size_t)sl * M + j) * 128 + row]) : 0.f;
                    }
#pragma unroll
                    for (int k = 0; k < PB; ++k) {
                        const bool mine = base + k == my_slot;
#pragma unroll
                        for (int j = 0; j < BN; ++j) a[j] += mine ? v[j] : ld[k][j];
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
                constexpr int RW = BN < 32 ? BN : 32;
#pragma unroll
                for (int h = 0; h < BN; h += RW) {
                    float sq[RW];
#pragma unroll
                    for (int i = 0; i < RW; ++i) sq[i] = v[h + i] * v[h + i];
                    warp_col_sums<RW>(sq, red + q * 64 + h, lane);
                }
                tc::cp_async_wait_all();  // this thread's share of the cos / sin table
                epi_bar();
#pragma unroll
                for (int j = 0; j < BN; ++j) {
                    const float tot = red[j] + red[64 + j] + red[128 + j] + red[192 + j];
                    v[j] = v[j] * rsqrtf(tot / 128.f + fz.eps) * gain;
                    xch[j * 128 + row] = v[j];
                }
                epi_bar();
                // rotate-half RoPE: row i < 64 pairs with row i + 64
                const int i = row & 63;
#pragma unroll
                for (int j = 0; j < BN; ++j) {
                    const float c = rope_c[j * 64 + i], sn = rope_s[j * 64 + i];
                    const float partner = xch[j * 128 + (row ^ 64)];
                    const float o = row < 64 ? v[j] * c - partner * sn : v[j] * c + partner * sn;
                    if (j < M) {
                        if (hh < nq)
                            fz.q_out[(size_t)j * fz.q_ld + (size_t)hh * 128 + row] = __float2bfloat16_rn(o);
                        else
                            fz.k_cache[(size_t)(c_row[j] + (hh - nq) * fz.kv.page) * 128 + row] =
                                __float2bfloat16_rn(o);
                    }
                }
            } else {
#pragma unroll
                for (int j = 0; j < BN; ++j)
                    if (j < M)
                        fz.v_cache[(size_t)(c_row[j] + (hh - nq - nkv) * fz.kv.page) * 128 + row] =
                            __float2bfloat16_rn(v[j]);
            }
        } else if (fz.op == FUSE_RESID) {
            tc::cp_async_wait_all();  // this thread's x values (prefetched at segment start)
#pragma unroll
            for (int j = 0; j < BN; ++j) {
                const float xn = (j < M ? xch[j * 128 + row] : 0.f) + v[j];
                if (j < M) {
                    fz.x[(size_t)j * N + f] = xn;
                    fz.xg_out[(size_t)j * N + f] = __float2bfloat16_rn(xn * gain);
                }
                v[j] = j < M ? xn : 0.f;
            }
            constexpr int RW = BN < 32 ? BN : 32;
#pragma unroll
            for (int h = 0; h < BN; h += RW) {
                float sq[RW];
#pragma unroll
                for (int i = 0; i < RW; ++i) sq[i] = v[h + i] * v[h + i];
                warp_col_sums<RW>(sq, red + q * 64 + h, lane);
            }
            epi_bar();
            if (e < M) fz.ssq_out[(size_t)feat * M + e] = red[e] + red[64 + e] + red[128 + e] + red[192 + e];
        } else if (fz.op == FUSE_SWIGLU) {
            // this segment completed the pair: gate tile 2 jb, up tile 2 jb + 1, each
            // summed over its slots in k order; both tiles' loads go out in one batch
            const int jb = feat >> 1, I = N / 2;
            constexpr int PS = PB > 1 ? PB / 2 : 1;
            float gs[BN], us[BN];
#pragma unroll
            for (int j = 0; j < BN; ++j) gs[j] = us[j] = 0.f;
            const int g0 = slot0(2 * jb), g1 = slot1(2 * jb), u0 = slot0(2 * jb + 1), u1 = slot1(2 * jb + 1);
            const int nb = max(g1 - g0, u1 - u0) + 1;
            for (int base = 0; base < nb; base += PS) {
                float lg[PS][BN], lu[PS][BN];
#pragma unroll
                for (int k = 0; k < PS; ++k) {
                    const int sg_ = g0 + base + k, su = u0 + base + k;
#pragma unroll
                    for (int j = 0; j < BN; ++j) {
                        lg[k][j] = sg_ <= g1 && j < M ? __ldcg(&fz.part[((size_t)sg_ * M + j) * 128 + row]) : 0.f;
                        lu[k][j] = su <= u1 && j < M ? __ldcg(&fz.part[((size_t)su * M + j) * 128 + row]) : 0.f;
                    }
                }
#pragma unroll
                for (int k = 0; k < PS; ++k)
#pragma unroll
                    for (int j = 0; j < BN; ++j) {
                        gs[j] += lg[k][j];
                        us[j] += lu[k][j];
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
                if (j < M) C[(size_t)j * ldc + f] = v[j] * s_row[j];
        }
        if (ticketed && e == 0) fz.tickets[key] = 0;
        epi_bar();  // scratch (red, xch, flag) is reused by the next segment
    }
    tc::cp_async_wait_all();  // no copy into shared memory outlives the segment's op
    return true;
}

template <int BN, bool SWIGLU, int STAGES, bool FUSED>
__global__ void __launch_bounds__(kThreads, FUSED && BN == 16 ? kFusedCtasPerSm : 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                   void* __restrict__ C, int ldc, int M, int N, int K, int epi, int n_split,
                   uint32_t* __restrict__ status, const __grid_constant__ Fuse fz,
                   long long test_wait) {
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
    // Plain work unit t = ((feat * n_tok) + tok) * n_split + split; a split covers k-blocks
    // [split * kblocks / n_split, (split + 1) * kblocks / n_split).  FUSED: see seg_at.
    const int num_tiles = n_feat * n_tok * n_split;
    const int kblocks = K / kBK;
    // segment iteration range: k-block iterations (FUSED) or unit indices (plain)
    const long long n_iter = (long long)n_feat * kblocks;
    const long long seg_lo = FUSED ? (long long)blockIdx.x * n_iter / gridDim.x : (long long)blockIdx.x;
    const long long seg_hi = FUSED ? (long long)(blockIdx.x + 1) * n_iter / gridDim.x : (long long)num_tiles;
    // bounded-wait test: CTA 0 skips its first copy and waits test_wait cycles at most
    const bool test_skip = !FUSED && test_wait > 0 && blockIdx.x == 0;
    const long long wlim = test_skip ? test_wait : tc::kWaitCycles;

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
            bool skip_next = test_skip;
            Seg sg;
            for (bool have = seg_at<FUSED>(sg, seg_lo, seg_hi, n_tok, n_split, kblocks); ok && have;
                 have = seg_at<FUSED>(sg, sg.next, seg_hi, n_tok, n_split, kblocks)) {
                const int feat = sg.feat, tok = sg.tok;
                for (int kb = sg.kb0; kb < sg.kb1; ++kb) {
                    if (!tc::mbar_wait(&empty[stage], phase ^ 1, abort_flag, wlim)) {
                        ok = false;
                        break;
                    }
                    if (skip_next) {  // bounded-wait test: this stage's copy is never issued
                        skip_next = false;
                        if (++stage == STAGES) {
                            stage = 0;
                            phase ^= 1;
                        }
                        continue;
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
            Seg sg;
            for (bool have = seg_at<FUSED>(sg, seg_lo, seg_hi, n_tok, n_split, kblocks); ok && have;
                 have = seg_at<FUSED>(sg, sg.next, seg_hi, n_tok, n_split, kblocks)) {
                const int kb0 = sg.kb0, kb1 = sg.kb1;
                if (!tc::mbar_wait(&tempty[acc], acc_phase ^ 1, abort_flag, wlim)) {
                    ok = false;
                    break;
                }
                tc::fence_after_sync();
                const uint32_t d = tmem_base + (uint32_t)(acc * G::ACC_COLS);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!tc::mbar_wait(&full[stage], phase, abort_flag, wlim)) {
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
        int acc = 0;
        uint32_t acc_phase = 0;
        fused_epilogue<BN, STAGES>(fz, (float*)C, ldc, M, N, kblocks, n_iter, seg_lo, seg_hi,
                                   (int)gridDim.x, tmem_base, tfull, tempty, acc, acc_phase, fscr,
                                   abort_flag);
        tc::cp_async_wait_all();  // no copy into shared memory outlives the CTA
    } else {
        // ---------------------------------------------------- epilogue (warps 2..5)
        const int q = warp & 3;
        int acc = 0;
        uint32_t acc_phase = 0;
        const int e = threadIdx.x - 64;
        float* tr = fscr;                        // EPI_LSE: [16][128] logits of a token chunk
        int* tgt_s = (int*)(fscr + 16 * 128);    // EPI_LSE: the tile's targets
        const bool lse = !SWIGLU && epi == EPI_LSE;
        const int n_vt = N / 128;
        for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
            const int split = t % n_split, rest = t / n_split;
            const int feat = rest / n_tok, tok = rest % n_tok;
            if (lse) {
                // targets of the tile's tokens (rows past M and last positions: none)
                for (int j = e; j < BN; j += 128) {
                    const int m = tok * BN + j;
                    int tg = -1;
                    if (m < M) {
                        const int g = fz.lse_row0 + m;
                        if (g % fz.lse_T < fz.lse_T - 1) {
                            tg = fz.lse_tok[g + 1];
                            if (tg < 0 || tg >= N) tg = 0;  // flagged by the combine
                        }
                    }
                    tgt_s[j] = tg;
                }
            }
            bool ok = tc::mbar_wait(&tfull[acc], acc_phase, abort_flag, wlim);
            ok = lse ? tc::bar128_and(ok) : __all_sync(0xffffffffu, ok);
            if (!ok) break;
            tc::fence_after_sync();
            const int f = feat * 128 + q * 32 + lane;
            const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * G::ACC_COLS);
            // Residual add: the residual values of each 16-token chunk are loaded one
            // chunk ahead, before the current chunk's stores, so the loads of a tile are
            // pipelined instead of one read-modify-write round trip per token.
            const bool resid = !SWIGLU && epi == EPI_RESID_F32;
            float xo[16], xn[16];
            auto load_x = [&](int tok0, float (&dst)[16]) {
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const int m = tok0 + j;
                    dst[j] = m < M ? ((const float*)C)[(size_t)m * ldc + f] : 0.f;
                }
            };
            if (resid) load_x(tok * BN, xo);
            for (int c0 = 0; c0 < BN; c0 += 16) {
                const int tok0 = tok * BN + c0;
                if (tok0 >= M) break;
                if (resid && c0 + 16 < BN && tok0 + 16 < M) load_x(tok0 + 16, xn);
                uint32_t r[16];
                tc::tmem_ld16(tbase + c0, r);
                uint32_t u[16];
                if (SWIGLU) tc::tmem_ld16(tbase + BN + c0, u);
                tc::tmem_wait_ld();
                if (lse) {
                    // 16 tokens x 128 features through shared memory, then 8 threads per
                    // token: max / lowest arg-max / sum exp over 16 features each, merged
                    // over the 8 lanes in a fixed order
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const float v = __uint_as_float(r[j]);
                        tr[j * 128 + q * 32 + lane] = v;
                        if (tgt_s[c0 + j] == f && tok0 + j < M) fz.lse_zt[tok0 + j] = v;
                    }
                    tc::bar128();
                    const int col = e >> 3, part = e & 7;
                    const float* zc = tr + col * 128 + part * 16;
                    float mv = zc[0];
                    int mi = part * 16;
#pragma unroll
                    for (int k = 1; k < 16; ++k)
                        if (zc[k] > mv) mv = zc[k], mi = part * 16 + k;
                    float sv = 0.f;
#pragma unroll
                    for (int k = 0; k < 16; ++k) sv += expf(zc[k] - mv);
#pragma unroll
                    for (int o = 1; o < 8; o <<= 1) {
                        const float m2 = __shfl_xor_sync(0xffffffffu, mv, o);
                        const float s2 = __shfl_xor_sync(0xffffffffu, sv, o);
                        const int i2 = __shfl_xor_sync(0xffffffffu, mi, o);
                        const float mx = fmaxf(mv, m2);
                        sv = sv * expf(mv - mx) + s2 * expf(m2 - mx);
                        mi = mv > m2 ? mi : (m2 > mv ? i2 : min(mi, i2));
                        mv = mx;
                    }
                    const int m = tok0 + col;
                    if (part == 0 && m < M) {
                        fz.lse_ms[(size_t)m * n_vt + feat] = make_float2(mv, sv);
                        fz.lse_idx[(size_t)m * n_vt + feat] = feat * 128 + mi;
                    }
                    tc::bar128();  // the buffer is rewritten by the next chunk
                    continue;
                }
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
                        ((float*)C)[o] = xo[j] + v;
                    }
                }
                if (resid) {
#pragma unroll
                    for (int j = 0; j < 16; ++j) xo[j] = xn[j];
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
               const Fuse* fz = nullptr, long long test_wait = 0) {
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
    const long long units = FUSED ? (long long)(N / 128) * (K / kBK)
                                  : (long long)(N / 128) * ((M + BN - 1) / BN) * n_split;
    const int grid = units < num_sms ? (int)units : num_sms;
    Fuse none{};
    launch_k(gemm_tc_kernel<BN, SWIGLU, STAGES, FUSED>, dim3(grid), dim3(kThreads), G::SMEM, s, tmW,
             tmX, C, ldc, M, N, K, epi, n_split, status, fz ? *fz : none, test_wait);
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
                   int epi, int num_sms, uint32_t* status, cudaStream_t s, long long test_wait,
                   const Fuse* lse) {
    if (M <= 0) return QK_OK;
    if (epi == EPI_LSE) {
        if (!lse || N % 128) return QK_EINVAL;
        if (M <= 16) return launch_cfg<16, false, 8>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, lse, test_wait);
        if (M <= 32) return launch_cfg<32, false, 8>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, lse, test_wait);
        if (M <= 64) return launch_cfg<64, false, 8>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, lse, test_wait);
        if (M <= 128) return launch_cfg<128, false, 6>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, lse, test_wait);
        return launch_cfg<256, false, 4>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, lse, test_wait);
    }
    const long long tw = test_wait;
    if (epi == EPI_SWIGLU) {
        if (M <= 16) return launch_cfg<16, true, 6>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, nullptr, tw);
        if (M <= 32) return launch_cfg<32, true, 6>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, nullptr, tw);
        if (M <= 64) return launch_cfg<64, true, 5>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, nullptr, tw);
        return launch_cfg<128, true, 4>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, nullptr, tw);
    }
    if (M <= 16) return launch_cfg<16, false, 8>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, nullptr, tw);
    if (M <= 32) return launch_cfg<32, false, 8>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, nullptr, tw);
    if (M <= 64) return launch_cfg<64, false, 8>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, nullptr, tw);
    if (M <= 128) return launch_cfg<128, false, 6>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, nullptr, tw);
    return launch_cfg<256, false, 4>(A, lda, W, C, ldc, M, N, K, epi, 1, num_sms, status, s, nullptr, tw);
}

// Decode linear with a fused epilogue (see Fuse); one token tile of M <= 64 rows.
int launch_gemm_tc_fused(const bf16* A, int lda, const bf16* W, float* out, int M, int N, int K,
                         const Fuse& f, int num_sms, uint32_t* status, cudaStream_t s) {
    if (M <= 0) return QK_OK;
    if (M > 64) return QK_ESHAPE;
    // every launch may split a tile over CTAs: partial slots and tickets are required
    if (!f.part || !f.tickets || !f.status) return QK_EINVAL;
    if (M <= 16)
        return launch_cfg<16, false, kFused16Stages, true>(A, lda, W, out, N, M, N, K, EPI_PARTIAL_F32, 1,
                                              num_sms, status, s, &f);
    if (M <= 32)
        return launch_cfg<32, false, 8, true>(A, lda, W, out, N, M, N, K, EPI_PARTIAL_F32, 1,
                                              num_sms, status, s, &f);
    return launch_cfg<64, false, 6, true>(A, lda, W, out, N, M, N, K, EPI_PARTIAL_F32, 1,
                                          num_sms, status, s, &f);
}


}  // namespace qk
