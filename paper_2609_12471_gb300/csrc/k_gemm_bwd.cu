// The batched GEMM of the backward pass (bwd_common.cuh): a tcgen05 / TMEM / TMA
// kernel for bf16 models and a CUDA-core kernel for fp32 models, both over the
// same operand descriptors, tile schedule and epilogue.
//
// tcgen05 kernel, one persistent CTA per SM, 320 threads:
//   warp 0, one lane : TMA producer over a STAGES-deep ring of (A, B) k-blocks of 64;
//   warp 1           : TMEM allocation; one lane issues tcgen05.mma (M 128, N BN, K 16)
//                      and the commits;
//   warps 2..9       : epilogue; warp w reads TMEM lanes 32 (w % 4) .. + 31 (one output
//                      row per thread) and half (w - 2) / 4 of the tile's columns, 16
//                      columns per tcgen05.ld, four loads per wait.
// A K-major operand tile is one 128-byte-swizzled box (64 k x 128 or BN rows); an
// MN-major one is boxes of 64 m/n x 64 k (8 KB each), whose descriptor steps 64
// m/n elements by the leading byte offset (8 KB) and 8 k rows by the stride byte
// offset (1 KB).  Two TMEM accumulators alternate so the epilogue of one tile
// overlaps the main loop of the next.  Every mbarrier wait is bounded; on a timeout
// the CTA raises QK_STATUS_TIMEOUT, drains its copies and MMAs and exits.  A launch
// armed by qk_debug_expire_next_wait exercises that path: CTA 0 issues no copy for
// its first k-block and its waits give up after the armed limit.
#include <cuda.h>
#include <math.h>
#include <string.h>

#include "bwd_common.cuh"
#include "tc_ptx.cuh"

namespace qk {
namespace bwd {

namespace {

// ------------------------------------------------------------------ CUDA-core kernel
constexpr int kSimtTile = 64, kSimtBK = 16, kSimtThreads = 256;

template <typename T>
__device__ __forceinline__ float op_load(const Op& o, int z, int i, int k) {
    int x, y;
    op_xy(o, z, i, k, x, y);
    return ld_act((const T*)o.ptr + (size_t)y * o.ld + x);
}

// One 64 x 64 output tile per CTA; thread t owns row t / 4, columns 16 (t % 4) .. + 15.
template <typename T>
__global__ void __launch_bounds__(kSimtThreads) gemm_bwd_simt_kernel(Gemm g, long long per) {
    __shared__ float As[kSimtBK][kSimtTile + 1], Bs[kSimtBK][kSimtTile + 1];
    pdl_wait();
    const Sched& sc = g.sc;
    int z, mt, nt;
    tile_at(sc, kSimtTile, kSimtTile, per, (long long)blockIdx.x, z, mt, nt);
    const int m0 = mt * kSimtTile, n0 = nt * kSimtTile;
    const int tid = threadIdx.x, r = tid >> 2, cg = tid & 3;
    float acc[16];
#pragma unroll
    for (int c = 0; c < 16; ++c) acc[c] = 0.f;
    const int nkb = kblocks(sc, kSimtTile, kSimtBK, m0);
    for (int j = 0; j < nkb; ++j) {
        int k0, kend;
        kblock_at(sc, kSimtTile, kSimtBK, m0, j, k0, kend);
        for (int e = tid; e < kSimtTile * kSimtBK; e += kSimtThreads) {
            const int i = e % kSimtTile, kq = e / kSimtTile, k = k0 + kq;
            const bool kv = k < kend;
            As[kq][i] = (kv && m0 + i < sc.M) ? op_load<T>(g.A, z, m0 + i, k) : 0.f;
            Bs[kq][i] = (kv && n0 + i < sc.N) ? op_load<T>(g.B, z, n0 + i, k) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kq = 0; kq < kSimtBK; ++kq) {
            const float a = As[kq][r];
#pragma unroll
            for (int c = 0; c < 16; ++c) acc[c] = fmaf(a, Bs[kq][cg * 16 + c], acc[c]);
        }
        __syncthreads();
    }
    const int m = m0 + r, n = n0 + cg * 16;
    int nv = sc.N - n;
    nv = nv < 0 ? 0 : (nv > 16 ? 16 : nv);
    RowStat st{-INFINITY, 0.f};
    if (m < sc.M && nv > 0) epi16<T>(g.epi, g.out, z, m, n, nv, acc, st);
    if (g.epi.mode == E_STATS) {  // merge the row's four 16-column parts
#pragma unroll
        for (int o = 1; o < 4; o <<= 1) {
            const float m2 = __shfl_xor_sync(0xffffffffu, st.mx, o);
            const float s2 = __shfl_xor_sync(0xffffffffu, st.sm, o);
            stat_merge(st, m2, s2);
        }
        if (cg == 0 && m < sc.M)
            g.epi.stats[(size_t)(z * g.epi.rows_per_z + m) * g.epi.n_ct + nt] = make_float2(st.mx, st.sm);
    }
}

// ------------------------------------------------------------------ tcgen05 kernel
constexpr int kEpiWarps = 8;  // two per TMEM lane quadrant, each owning half of the tile's columns
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr int kBK = 64;
constexpr int kBox = 64 * 128;  // one 64 x 64 bf16 box (8 KB)

// BM x BN output tiles.  BM = 256 (two 128-row MMAs per k-step, one accumulator set
// filling TMEM, three 64 KB stages) for the large full-reduction GEMMs: it halves the
// shared-memory bytes per flop of A and lets the ring cover more load latency; BM = 128
// keeps two accumulator sets so the epilogue of a tile overlaps the next main loop.
template <int BN, int BM>
struct TcCfg {
    static constexpr int STAGES = BM == 256 ? 3 : (BN == 256 ? 4 : 6);
    static constexpr int A_BYTES = BM * 128;
    static constexpr int B_BYTES = BN * 128;
    static constexpr int ACC = BM == 256 ? 1 : 2;       // accumulator sets
    static constexpr int ACC_COLS = (BM / 128) * BN;    // TMEM columns of one set
    static constexpr int TMEM_COLS = ACC * ACC_COLS;
    static constexpr int STAGE_OUT = kEpiWarps * 4096;  // per epilogue warp: one 32 x 128-byte block
    static constexpr int SMEM = STAGES * (A_BYTES + B_BYTES) + STAGE_OUT + 1024 + 256;
    static_assert(TMEM_COLS <= 512, "accumulators exceed TMEM");
    static_assert(SMEM <= 232448, "shared memory per CTA");
};

template <int BN, int BM, bool AMN, bool BMN, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_bwd_tc_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
                       const __grid_constant__ CUtensorMap mapC, const __grid_constant__ Gemm g,
                       long long per, long long total, int a3, int b3, uint32_t* __restrict__ status,
                       long long test_wait) {
    using G = TcCfg<BN, BM>;
    constexpr int STAGES = G::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* sA = smem;
    uint8_t* sB = smem + STAGES * G::A_BYTES;
    uint8_t* sOut = sB + STAGES * G::B_BYTES;
    uint64_t* full = (uint64_t*)(sOut + G::STAGE_OUT);
    uint64_t* empty = full + STAGES;
    uint64_t* tfull = empty + STAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint32_t* tmem_slot = (uint32_t*)(drain + 1);
    volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const Sched& sc = g.sc;
    // bounded-wait test (qk_debug_expire_next_wait): CTA 0 issues no copy for its first
    // k-block and its waits give up after test_wait cycles
    const bool test_skip = test_wait > 0 && blockIdx.x == 0;
    const long long wlim = test_skip ? test_wait : tc::kWaitCycles;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            tc::mbar_init(&full[s], 1);
            tc::mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < G::ACC; ++a) {
            tc::mbar_init(&tfull[a], 1);
            tc::mbar_init(&tempty[a], kEpiWarps);
        }
        tc::mbar_init(drain, 1);
        *abort_flag = 0;
        tc::fence_mbar_init();
        tc::tma_prefetch_desc(&mapA);
        tc::tma_prefetch_desc(&mapB);
    }
    if (warp == 1) tc::tmem_alloc(tmem_slot, G::TMEM_COLS);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;
    pdl_wait();

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------ TMA producer
            int stage = 0;
            uint32_t phase = 0;
            int armed[STAGES];
            for (int s = 0; s < STAGES; ++s) armed[s] = -1;
            bool ok = true, skip_next = test_skip;
            for (long long t = blockIdx.x; ok && t < total; t += gridDim.x) {
                int z, mt, nt;
                tile_at(sc, BM, BN, per, t, z, mt, nt);
                const int m0 = mt * BM, n0 = nt * BN;
                const int nkb = kblocks(sc, BM, kBK, m0);
                for (int j = 0; j < nkb; ++j) {
                    int k0, kend;
                    kblock_at(sc, BM, kBK, m0, j, k0, kend);
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
                    uint8_t* a_s = sA + stage * G::A_BYTES;
                    uint8_t* b_s = sB + stage * G::B_BYTES;
                    int x, y;
#pragma unroll
                    for (int h = 0; h < BM / 128; ++h) {  // 128-row blocks of A (16 KB each)
                        uint8_t* ah = a_s + h * 16384;
                        const int mh = m0 + 128 * h;
                        if (AMN) {  // MN chunks of 64: one 3-D box (chunk index as the third axis) or one box each
                            if (a3) {
                                op_xy(g.A, z, mh, k0, x, y);
                                tc::tma_load_3d(ah, &mapA, 0, y, x >> 6, &full[stage]);
                            } else {
#pragma unroll
                                for (int c = 0; c < 2; ++c) {
                                    op_xy(g.A, z, mh + 64 * c, k0, x, y);
                                    tc::tma_load_2d(ah + c * kBox, &mapA, x, y, &full[stage]);
                                }
                            }
                        } else {
                            op_xy(g.A, z, mh, k0, x, y);
                            tc::tma_load_2d(ah, &mapA, x, y, &full[stage]);
                        }
                    }
                    if (BMN) {
                        if (b3) {
                            op_xy(g.B, z, n0, k0, x, y);
                            tc::tma_load_3d(b_s, &mapB, 0, y, x >> 6, &full[stage]);
                        } else {
#pragma unroll
                            for (int c = 0; c < BN / 64; ++c) {
                                op_xy(g.B, z, n0 + 64 * c, k0, x, y);
                                tc::tma_load_2d(b_s + c * kBox, &mapB, x, y, &full[stage]);
                            }
                        }
                    } else {
                        op_xy(g.B, z, n0, k0, x, y);
                        tc::tma_load_2d(b_s, &mapB, x, y, &full[stage]);
                    }
                    armed[stage] = (int)phase;
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
            }
            pdl_trigger();
            if (!ok) {
                for (int s = 0; s < STAGES; ++s)
                    if (armed[s] >= 0) tc::mbar_wait_drain(&full[s], (uint32_t)armed[s]);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ------------------------------------------------ MMA issuer
            constexpr uint32_t idesc =
                tc::idesc_bf16(128, BN) | (AMN ? (1u << 15) : 0u) | (BMN ? (1u << 16) : 0u);
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true, issued = false;
            for (long long t = blockIdx.x; ok && t < total; t += gridDim.x) {
                int z, mt, nt;
                tile_at(sc, BM, BN, per, t, z, mt, nt);
                const int nkb = kblocks(sc, BM, kBK, mt * BM);
                if (!tc::mbar_wait(&tempty[acc], acc_phase ^ 1, abort_flag, wlim)) {
                    ok = false;
                    break;
                }
                tc::fence_after_sync();
                const uint32_t d = tmem_base + (uint32_t)(acc * G::ACC_COLS);
                for (int j = 0; j < nkb; ++j) {
                    if (!tc::mbar_wait(&full[stage], phase, abort_flag, wlim)) {
                        ok = false;
                        break;
                    }
                    tc::fence_after_sync();
                    const uint32_t a0 = tc::smem_u32(sA + stage * G::A_BYTES);
                    const uint32_t b0 = tc::smem_u32(sB + stage * G::B_BYTES);
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k) {
                        const uint64_t bd = BMN ? tc::sw128_desc_mn(b0 + k * 2048, kBox)
                                                : tc::sw128_desc(b0 + k * 32);
#pragma unroll
                        for (int h = 0; h < BM / 128; ++h) {  // rows 128 h .. of the tile
                            const uint32_t ah = a0 + h * 16384;
                            const uint64_t ad = AMN ? tc::sw128_desc_mn(ah + k * 2048, kBox)
                                                    : tc::sw128_desc(ah + k * 32);
                            tc::mma_bf16(d + h * BN, ad, bd, idesc, (j || k) ? 1u : 0u);
                        }
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
                if (++acc == G::ACC) {
                    acc = 0;
                    acc_phase ^= 1;
                }
            }
            if (!ok && issued) {
                tc::mma_commit(drain);
                tc::mbar_wait_drain(drain, 0);
            }
        }
    } else {
        // ---------------------------------------------------- epilogue (warps 2..9)
        // Warp w reads TMEM lanes 32 (w % 4) .. + 31 (its rows) and the columns of half
        // (w - 2) / 4 of the tile (BM = 256: half selects the 128-row block and the warp
        // takes every column), four 16-column blocks per TMEM wait.  Outputs leave through
        // the warp's 4 KB staging buffer, one TMA store per 32 rows x 128 bytes (64 bf16 or
        // 32 fp32 columns), rows stored with the 128-byte swizzle so the writes of a warp hit
        // distinct banks; the two-output SwiGLU backward stores 32 x 16 blocks instead.
        const int q = warp & 3, half = (warp - 2) >> 2;
        constexpr int HC = BM == 256 ? BN : BN / 2;  // columns per warp
        const int c_lo = BM == 256 ? 0 : half * HC, r_lo = BM == 256 ? half * 128 : 0;
        constexpr bool f32 = MODE == E_F32;
        constexpr bool staged = MODE != E_STATS && MODE != E_SWIGLU_BWD && MODE != E_SWIGLU_FWD;
        uint8_t* stg = sOut + (warp - 2) * 4096;
        const int sw = lane & 7;
        int acc = 0;
        uint32_t acc_phase = 0;
        for (long long t = blockIdx.x; t < total; t += gridDim.x) {
            int z, mt, nt;
            tile_at(sc, BM, BN, per, t, z, mt, nt);
            const int m0 = mt * BM + r_lo, n0 = nt * BN;
            bool ok = tc::mbar_wait(&tfull[acc], acc_phase, abort_flag, wlim);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            tc::fence_after_sync();
            const int m = m0 + q * 32 + lane;
            const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) +
                                   (uint32_t)(acc * G::ACC_COLS + (BM == 256 ? half * BN : 0));
            const int orow = (z / g.out.zq) * g.out.zrow + m0 + q * 32;
            const int ocol = (z % g.out.zq) * g.out.zcol;
            RowStat st{-INFINITY, 0.f};
            if constexpr (MODE == E_SWIGLU_FWD) {
                // BM = 256: the warp holds all 256 columns of its rows, gate c at TMEM column
                // c and up c at c + 128 (the packed gate / up rows); 64 outputs per store
                for (int c = 0; c < 128; c += 64) {
                    if (lane == 0) tc::bulk_wait_read<0>();
                    __syncwarp();
                    uint4* row = (uint4*)(stg + lane * 128);
#pragma unroll
                    for (int hh = 0; hh < 2; ++hh) {
                        const int cc = c + 32 * hh;
                        uint32_t gr[2][16], ur[2][16];
                        tc::tmem_ld16(tbase + cc, gr[0]);
                        tc::tmem_ld16(tbase + cc + 16, gr[1]);
                        tc::tmem_ld16(tbase + 128 + cc, ur[0]);
                        tc::tmem_ld16(tbase + 128 + cc + 16, ur[1]);
                        tc::tmem_wait_ld();
#pragma unroll
                        for (int w2 = 0; w2 < 2; ++w2) {
                            uint4 wv[2];
                            bf16* b = (bf16*)wv;
#pragma unroll
                            for (int j = 0; j < 16; ++j) {
                                const float gv = __uint_as_float(gr[w2][j]), uv = __uint_as_float(ur[w2][j]);
                                b[j] = __float2bfloat16_rn(m < sc.M ? gv / (1.f + __expf(-gv)) * uv : 0.f);
                            }
                            row[(hh * 4 + w2 * 2) ^ sw] = wv[0];
                            row[(hh * 4 + w2 * 2 + 1) ^ sw] = wv[1];
                        }
                    }
                    tc::fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        tc::tma_store_2d(&mapC, ocol + nt * 128 + c, orow, stg);
                        tc::bulk_commit();
                    }
                }
            }
            for (int c4 = c_lo; c4 < c_lo + HC && MODE != E_SWIGLU_FWD; c4 += 64) {
                if (n0 + c4 >= sc.N) break;  // uniform over the warp
                uint32_t r[4][16];
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (n0 + c4 + 16 * u < sc.N) tc::tmem_ld16(tbase + c4 + 16 * u, r[u]);
                tc::tmem_wait_ld();
                if constexpr (staged) {  // the previous block's store has read the buffer
                    if (lane == 0) tc::bulk_wait_read<0>();
                    __syncwarp();
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int n = n0 + c4 + 16 * u;
                    const bool in = n < sc.N;
                    float v[16], y[16], y2[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j) v[j] = __uint_as_float(r[u][j]);
                    const bool store =
                        in && m < sc.M && epi_values<bf16, true, MODE>(g.epi, g.out, z, m, n, 16, v, st, y, y2);
                    if constexpr (MODE == E_STATS) continue;
                    if constexpr (MODE == E_SWIGLU_BWD) {
                        if (!in) break;  // uniform
                        // dg and du blocks (bf16, 32 x 16 each) in the staging buffer, two stores
                        if (lane == 0) tc::bulk_wait_read<0>();
                        __syncwarp();
                        uint4 w[4];
                        bf16* b = (bf16*)w;
#pragma unroll
                        for (int j = 0; j < 16; ++j)
                            b[j] = __float2bfloat16_rn(store ? y[j] : 0.f), b[16 + j] = __float2bfloat16_rn(store ? y2[j] : 0.f);
                        uint4* d = (uint4*)(stg + lane * 32);
                        d[0] = w[0];
                        d[1] = w[1];
                        uint4* d2 = (uint4*)(stg + 1024 + lane * 32);
                        d2[0] = w[2];
                        d2[1] = w[3];
                        tc::fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            const int gc = (n >> 7) * 256 + (n & 127);
                            tc::tma_store_2d(&mapC, gc, orow, stg);
                            tc::tma_store_2d(&mapC, gc + 128, orow, stg + 1024);
                            tc::bulk_commit();
                        }
                        continue;
                    }
                    uint4* row = (uint4*)(stg + lane * 128);  // this lane's output row, 8 granules of 16 B
                    if constexpr (f32) {
                        const int ub = u & 1;  // chunk within the 32-column block
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const float4 f = store ? make_float4(y[4 * j], y[4 * j + 1], y[4 * j + 2], y[4 * j + 3])
                                                   : make_float4(0.f, 0.f, 0.f, 0.f);
                            row[(ub * 4 + j) ^ sw] = *reinterpret_cast<const uint4*>(&f);
                        }
                        if (ub == 1) {  // 32 columns staged: store them
                            tc::fence_proxy_async_smem();
                            __syncwarp();
                            if (lane == 0) {
                                tc::tma_store_2d(&mapC, ocol + n0 + c4 + 32 * (u >> 1), orow, stg);
                                tc::bulk_commit();
                            }
                            if (u == 1) {
                                if (lane == 0) tc::bulk_wait_read<0>();
                                __syncwarp();
                            }
                        }
                    } else {
                        uint4 w[2];
                        bf16* b = (bf16*)w;
#pragma unroll
                        for (int j = 0; j < 16; ++j) b[j] = __float2bfloat16_rn(store ? y[j] : 0.f);
                        row[(2 * u) ^ sw] = w[0];
                        row[(2 * u + 1) ^ sw] = w[1];
                    }
                }
                if constexpr (staged && !f32) {  // 64 columns staged: store them
                    tc::fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        tc::tma_store_2d(&mapC, ocol + n0 + c4, orow, stg);
                        tc::bulk_commit();
                    }
                }
            }
            const int ct = nt * 2 + half;  // statistics column tile of HC columns (BM = 128)
            if (MODE == E_STATS && m < sc.M && ct < g.epi.n_ct)
                g.epi.stats[(size_t)(z * g.epi.rows_per_z + m) * g.epi.n_ct + ct] = make_float2(st.mx, st.sm);
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&tempty[acc]);
            if (++acc == G::ACC) {
                acc = 0;
                acc_phase ^= 1;
            }
        }
        if (lane == 0) tc::bulk_wait<0>();  // every store of this warp has completed
    }

    tc::fence_before_sync();
    __syncthreads();
    if (threadIdx.x == 0 && *abort_flag) atomicOr(status, QK_STATUS_TIMEOUT);
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem_base, G::TMEM_COLS);
    }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)p;
    }
    return fn;
}

// bf16 map over the whole operand buffer, box 64 columns x box_rows rows, 128-byte swizzle.
bool make_op_map(CUtensorMap* map, const Op& o, int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)o.cols, (cuuint64_t)o.rows};
    cuuint64_t strides[1] = {(cuuint64_t)o.ld * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(o.ptr), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// MN-major operand as a 3-D map: (element within a 64-column chunk, row, chunk), box
// 64 x 64 rows x nch chunks, so that one copy lands the nch chunks of a k-block one
// after another (8 KB apart), the layout the MMA descriptors expect.
bool make_op_map3(CUtensorMap* map, const Op& o, int nch) {
    EncodeTiledFn fn = encode_fn();
    if (!fn || o.cols % 64) return false;
    cuuint64_t dims[3] = {64, (cuuint64_t)o.rows, (cuuint64_t)(o.cols / 64)};
    cuuint64_t strides[2] = {(cuuint64_t)o.ld * 2, 128};
    cuuint32_t box[3] = {64, 64, (cuuint32_t)nch};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(o.ptr), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Output map over C [rows, cols]: box 32 rows x 128 bytes (64 bf16 / 32 fp32 columns) with
// the 128-byte swizzle, or (narrow) 32 rows x 16 columns unswizzled.
bool make_out_map(CUtensorMap* map, const Out& o, bool f32, bool narrow) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const size_t es = f32 ? 4 : 2;
    cuuint64_t dims[2] = {(cuuint64_t)o.cols, (cuuint64_t)o.rows};
    cuuint64_t strides[1] = {(cuuint64_t)o.ldc * es};
    cuuint32_t box[2] = {narrow ? 16u : (cuuint32_t)(128 / es), 32};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, o.C, dims,
              strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              narrow ? CU_TENSOR_MAP_SWIZZLE_NONE : CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, int BM, bool AMN, bool BMN, int MODE>
int launch_tc_cfg(Model& m, const Gemm& g, cudaStream_t s) {
    using G = TcCfg<BN, BM>;
    auto kern = gemm_bwd_tc_kernel<BN, BM, AMN, BMN, MODE>;
    static bool attr_set = false;
    if (!attr_set) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, G::SMEM) != cudaSuccess)
            return set_error(QK_ECUDA, "backward GEMM: shared-memory attribute");
        attr_set = true;
    }
    CUtensorMap ma, mb, mc;
    int a3 = 0, b3 = 0;
    if (AMN) a3 = make_op_map3(&ma, g.A, 2) ? 1 : 0;
    if (BMN) b3 = make_op_map3(&mb, g.B, BN / 64) ? 1 : 0;
    if ((!a3 && !make_op_map(&ma, g.A, AMN ? 64 : 128)) || (!b3 && !make_op_map(&mb, g.B, BMN ? 64 : BN)))
        return set_error(QK_ECUDA, "backward GEMM: tensor map encoding failed");
    memset(&mc, 0, sizeof(mc));
    if (MODE != E_STATS && !make_out_map(&mc, g.out, MODE == E_F32, MODE == E_SWIGLU_BWD))
        return set_error(QK_ECUDA, "backward GEMM: output tensor map encoding failed");
    const long long per = tiles_per_z(g.sc, BM, BN);
    const long long total = per * g.sc.Z;
    const int grid = total < m.num_sms ? (int)total : m.num_sms;
    const long long test_wait = m.test_wait_cycles;  // one launch only
    m.test_wait_cycles = 0;
    launch_k(kern, dim3(grid), dim3(kThreads), G::SMEM, s, ma, mb, mc, g, per, total, a3, b3, m.status,
             test_wait);
    note_launch();
    return QK_OK;
}

bool big_tiles(const Model& m, const Gemm& g) {
    const long long tiles = (long long)g.sc.Z * (g.sc.M / 256) * cdiv(g.sc.N, 256);
    return g.sc.red == RED_FULL && !g.sc.tri && g.sc.M % 256 == 0 && tiles >= m.num_sms;
}

// 256-row tiles for the large full-reduction GEMMs: whole 256-row blocks, at least one
// tile per SM, and an epilogue light enough to run unoverlapped (not the row statistics
// or the two-output SwiGLU backward, measured slower without a second accumulator set).
template <int BN, bool AMN, bool BMN, int MODE>
int launch_tc_mode(Model& m, const Gemm& g, cudaStream_t s) {
    if constexpr (BN == 256 && MODE != E_STATS && MODE != E_SWIGLU_BWD) {
        if (big_tiles(m, g)) return launch_tc_cfg<BN, 256, AMN, BMN, MODE>(m, g, s);
    }
    if constexpr (MODE == E_SWIGLU_FWD) {
        return set_error(QK_ESHAPE, "SwiGLU forward epilogue needs 256 x 256 tiles");
    } else {
        return launch_tc_cfg<BN, 128, AMN, BMN, MODE>(m, g, s);
    }
}

// The epilogue modes each operand layout is instantiated for (the ones the backward uses).
template <int BN, bool AMN, bool BMN>
int launch_tc(Model& m, const Gemm& g, cudaStream_t s) {
    const int mode = g.epi.mode;
    if (!AMN && !BMN) {
        if (mode == E_SWIGLU_FWD) return launch_tc_mode<BN, AMN, BMN, E_SWIGLU_FWD>(m, g, s);
        if (mode == E_F32) return launch_tc_mode<BN, AMN, BMN, E_F32>(m, g, s);
        if (mode == E_ACT) return launch_tc_mode<BN, AMN, BMN, E_ACT>(m, g, s);
        if (mode == E_STATS) return launch_tc_mode<BN, AMN, BMN, E_STATS>(m, g, s);
        if (mode == E_SOFTMAX) return launch_tc_mode<BN, AMN, BMN, E_SOFTMAX>(m, g, s);
        if (mode == E_DS) return launch_tc_mode<BN, AMN, BMN, E_DS>(m, g, s);
    } else if (!AMN && BMN) {
        if (mode == E_F32) return launch_tc_mode<BN, AMN, BMN, E_F32>(m, g, s);
        if (mode == E_ACT) return launch_tc_mode<BN, AMN, BMN, E_ACT>(m, g, s);
        if (mode == E_SWIGLU_BWD) return launch_tc_mode<BN, AMN, BMN, E_SWIGLU_BWD>(m, g, s);
    } else {
        if (mode == E_F32) return launch_tc_mode<BN, AMN, BMN, E_F32>(m, g, s);
        if (mode == E_ACT) return launch_tc_mode<BN, AMN, BMN, E_ACT>(m, g, s);
    }
    return set_error(QK_EINVAL, "backward GEMM: epilogue %d is not instantiated for this operand layout", mode);
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15) == 0; }

}  // namespace

// Width of the column tiles of the N tile chosen for N columns (tri: causal, square tiles).
static int tile_bn(const Model& m, int N, int tri) {
    if (m.cfg.dtype != QK_DTYPE_BF16) return kSimtTile;
    return (tri || N <= 128) ? 128 : 256;
}

int gemm_tile_n(const Model& m, int N, int tri) {
    return m.cfg.dtype != QK_DTYPE_BF16 ? kSimtTile : tile_bn(m, N, tri) / 2;
}

bool linear_large(Model& m, const void* A, int lda, const void* W, void* C, int ldc, int M, int N,
                  int K, int epi, cudaStream_t s) {
    if (m.cfg.dtype != QK_DTYPE_BF16 || M < 256) return false;
    const bool swiglu = epi == EPI_SWIGLU;
    const int n_gemm = swiglu ? 2 * N : N;
    Gemm g{};
    g.A = Op{A, lda, M, K, 0, 0, 0, 1, 1, 0, 0, 0, 0, 0, 128};
    g.B = Op{W, K, n_gemm, K, 0, 0, 0, 1, 1, 0, 0, 0, 0, 0, 128};
    g.out = Out{C, ldc, M, N, 1, 0, 0, nullptr};
    g.epi = Epi{};
    g.epi.scale = 1.f;
    g.sc = Sched{1, M, n_gemm, K, RED_FULL, 0, 0, 0};
    if (epi == EPI_STORE_ACT) g.epi.mode = E_ACT;
    else if (epi == EPI_STORE_F32) g.epi.mode = E_F32;
    else if (epi == EPI_RESID_F32) g.epi.mode = E_F32, g.out.addend = (const float*)C;
    else if (swiglu) g.epi.mode = E_SWIGLU_FWD;
    else return false;
    if (!big_tiles(m, g) || n_gemm % 256 || K % 64 || lda % 8 || ((uintptr_t)A & 15) || ((uintptr_t)W & 15) ||
        ((uintptr_t)C & 15) || (g.epi.mode == E_F32 ? ldc % 4 : ldc % 8) || ldc < N)
        return false;
    const int rc = run_gemm(m, g, s);
    if (rc != QK_OK && !m.deferred_error) m.deferred_error = rc;
    return true;
}

int run_gemm(Model& m, const Gemm& g, cudaStream_t s) {
    const Sched& sc = g.sc;
    if (sc.Z <= 0 || sc.M <= 0 || sc.N <= 0) return QK_OK;
    if (m.cfg.dtype != QK_DTYPE_BF16) {
        const long long per = tiles_per_z(sc, kSimtTile, kSimtTile);
        const long long total = per * sc.Z;
        if (total >= (1ll << 31)) return set_error(QK_ESHAPE, "backward GEMM: too many tiles");
        launch_k(gemm_bwd_simt_kernel<float>, dim3((unsigned)total), dim3(kSimtThreads), 0, s, g, per);
        note_launch();
        return QK_OK;
    }
    const int BN = tile_bn(m, sc.N, sc.tri);
    // Every k-block is whole, every TMA box starts on a 16-byte boundary and every
    // epilogue access of 16 outputs is 16-byte aligned.
    bool ok = sc.K % kBK == 0 && aligned16(g.A.ptr) && aligned16(g.B.ptr) && g.A.ld % 8 == 0 &&
              g.B.ld % 8 == 0 && sc.N % 16 == 0 && aligned16(g.out.C) && g.out.zcol % 16 == 0;
    ok = ok && (g.epi.mode == E_F32 ? g.out.ldc % 4 == 0 : g.out.ldc % 8 == 0);
    ok = ok && (!g.out.addend || aligned16(g.out.addend)) && (!g.epi.P || aligned16(g.epi.P));
    ok = ok && (sc.red != RED_SUFFIX || (sc.seg % kBK == 0 && sc.seg > 0 && sc.K % sc.seg == 0));
    ok = ok && (!g.A.kwrap || g.A.kwrap % kBK == 0) && (!g.B.kwrap || g.B.kwrap % kBK == 0);
    ok = ok && g.B.pitch == 128 && g.A.pitch % 64 == 0 && (!sc.tri || (BN == 128 && sc.M == sc.N));
    // output tiles are whole 128-row blocks of a batch entry, or clipped at the buffer's last row;
    // stores of 64 (bf16) or 32 (fp32) columns stay inside N, or are clipped at the last column
    ok = ok && (sc.M % 128 == 0 || (sc.Z == 1 && g.out.rows == sc.M)) && g.out.rows > 0 && g.out.cols > 0;
    ok = ok && (sc.N % 64 == 0 || (sc.Z == 1 && g.out.cols == sc.N));
    if (!ok) return set_error(QK_ESHAPE, "backward GEMM: shape or alignment outside the tcgen05 path");
    const bool amn = g.A.mn != 0, bmn = g.B.mn != 0;
    if (BN == 256) {
        if (!amn && !bmn) return launch_tc<256, false, false>(m, g, s);
        if (!amn && bmn) return launch_tc<256, false, true>(m, g, s);
        if (amn && bmn) return launch_tc<256, true, true>(m, g, s);
    } else {
        if (!amn && !bmn) return launch_tc<128, false, false>(m, g, s);
        if (!amn && bmn) return launch_tc<128, false, true>(m, g, s);
        if (amn && bmn) return launch_tc<128, true, true>(m, g, s);
    }
    return set_error(QK_EINVAL, "backward GEMM: MN-major A with K-major B is not instantiated");
}

}  // namespace bwd
}  // namespace qk
