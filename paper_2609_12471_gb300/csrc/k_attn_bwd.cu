// Causal attention backward on tcgen05 / TMEM (bf16, head_dim 128), fused: the
// probabilities P and their gradient dS never leave the SM.
//
// For the causal softmax attention o = P v, P = softmax(q k^T / sqrt(d)) (masked),
// with the forward's per-row log-sum-exp lse and D = rowsum(dO * o):
//     dP = dO v^T,  dS = P (dP - D) / sqrt(d),
//     dV = P^T dO,  dK = dS^T q,  dQ = dS k,
// dV and dK summed over the query heads of each GQA group.
//
// Work item = (row b, kv head g, 128-key tile j), heaviest (smallest j) first, dealt
// to the CTAs in rounds whose CTA order reverses every round.  One persistent CTA per
// SM, 320 threads: warp 0 lane 0 the TMA producer, warp 1 the TMEM owner whose lane 0
// issues the MMAs, warps 2..9 the epilogue, two warps per TMEM lane quadrant (one key
// row, or for dQ one query row, per thread; each warp of a pair takes half of the
// columns).  Per item K_j and V_j are loaded once; per
// step (query head h of the group, 128-query tile i >= j) Q and dO are loaded and
//   1. S^T = K Q^T and dP^T = V dO^T (M 128 keys, N 128 queries, K = d) into TMEM
//      columns [0, 128) and [128, 256);
//   2. the epilogue forms P^T = exp(S^T / sqrt(d) - lse) (keys after the query
//      masked) and dS^T = P^T (dP^T - D) / sqrt(d) in bf16 into shared memory (rows =
//      keys, 128-byte swizzle);
//   3. dV += P^T dO, dK += dS^T Q (TMEM columns [256, 384), [384, 512)) and
//      dQ = dS K (columns [0, 128)); the epilogue adds dQ into the fp32 global dQ by
//      TMA reduce-add (other key tiles add theirs: the sum's order varies).
// Each shared-memory tile serves both majorness orders: a K-major [rows x 128] tile
// of X is the MN-major tile of X^T.  At the item's end dK (fp32) and dV (bf16) are
// stored by TMA.  Every mbarrier wait is bounded; on a timeout the CTA records
// QK_STATUS_TIMEOUT, waits (bounded) for its copies and MMAs and exits.
#include <cuda.h>
#include <math.h>
#include <string.h>

#include "qk_internal.cuh"
#include "tc_ptx.cuh"

namespace qk {

namespace {

constexpr int kD = 128, kT = 128;
constexpr int kThreads = 320;
constexpr int kEpiWarps = 8;
constexpr int kTile = 2 * 16384;  // 128 rows x 128 bf16 as two 64-column boxes
constexpr int kOffK = 0, kOffV = kTile, kOffQ = 2 * kTile, kOffDO = 3 * kTile, kOffP = 4 * kTile,
              kOffDS = 5 * kTile, kOffStage = 6 * kTile, kOffLse = kOffStage + kEpiWarps * 4096,
              kOffBar = kOffLse + 2 * 128 * 4;
constexpr int kSmem = kOffBar + 256 + 1024;
static_assert(kSmem <= 232448, "shared memory per CTA");
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ void tma_reduce_add_2d(const CUtensorMap* map, int x, int y, const void* src) {
    asm volatile("cp.reduce.async.bulk.tensor.2d.global.shared::cta.add.tile.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                     map),
                 "r"(x), "r"(y), "r"(tc::smem_u32(src))
                 : "memory");
}

// Named barrier 1 over the epilogue warps; returns whether `pred` held in all of them.
__device__ __forceinline__ bool epi_bar_and(bool pred) {
    uint32_t r;
    asm volatile(
        "{\n"
        ".reg .pred p, q;\n"
        "setp.ne.u32 p, %1, 0;\n"
        "bar.red.and.pred q, 1, %2, p;\n"
        "selp.u32 %0, 1, 0, q;\n"
        "}\n"
        : "=r"(r)
        : "r"((uint32_t)pred), "n"(kEpiWarps * 32)
        : "memory");
    return r != 0;
}

struct Args {
    int B, T, nq, nkv, n_items, nt;
    const float* lse;  // [B nq T]
    const float* D;    // [B nq T]
    float scale;
    uint32_t* status;
};

// The CTA's item in round r, or -1 after the last: round r deals items r G .. r G + G - 1
// (G CTAs) to CTAs 0 .. G - 1 on even rounds and G - 1 .. 0 on odd ones.  An item's work
// falls with its index, so alternating the order evens the CTAs' sums (with 2 x 8 x 32
// items on 152 CTAs the busiest CTA has 1.05 x the mean work, 1.3 x with plain rounds).
__device__ __forceinline__ int item_of(int r, int n_items) {
    const int c = (r & 1) ? (int)gridDim.x - 1 - (int)blockIdx.x : (int)blockIdx.x;
    const int it = r * (int)gridDim.x + c;
    return it < n_items ? it : -1;
}

// Item `it`: key tile j = it / (B nkv) (ascending j: descending work), (b, g) = it % (B nkv).
__device__ __forceinline__ void item_at(const Args& a, int it, int& b, int& g, int& j) {
    const int bg = it % (a.B * a.nkv);
    j = it / (a.B * a.nkv);
    b = bg / a.nkv;
    g = bg % a.nkv;
}

__global__ void __launch_bounds__(kThreads, 1)
    attn_bwd_kernel(const __grid_constant__ CUtensorMap mQ, const __grid_constant__ CUtensorMap mDO,
                    const __grid_constant__ CUtensorMap mKV, const __grid_constant__ CUtensorMap mDQ,
                    const __grid_constant__ CUtensorMap mDK, const __grid_constant__ CUtensorMap mDV,
                    const __grid_constant__ Args a, int dv_col0) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* sK = smem + kOffK;
    uint8_t* sV = smem + kOffV;
    uint8_t* sQ = smem + kOffQ;
    uint8_t* sDO = smem + kOffDO;
    uint8_t* sP = smem + kOffP;
    uint8_t* sDS = smem + kOffDS;
    float* sLse = (float*)(smem + kOffLse);
    float* sD = sLse + 128;
    uint64_t* bar = (uint64_t*)(smem + kOffBar);
    uint64_t* kv_full = bar + 0;
    uint64_t* kv_empty = bar + 1;
    uint64_t* qd_full = bar + 2;
    uint64_t* qd_empty = bar + 3;
    uint64_t* sp_full = bar + 4;
    uint64_t* pds_ready = bar + 5;
    uint64_t* mm2_done = bar + 6;
    uint64_t* s_free = bar + 7;
    uint64_t* acc_full = bar + 8;
    uint64_t* acc_free = bar + 9;
    uint64_t* drain = bar + 10;
    uint32_t* tmem_slot = (uint32_t*)(bar + 11);
    volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int G = a.nq / a.nkv;
    if (threadIdx.x == 0) {
        tc::mbar_init(kv_full, 1);
        tc::mbar_init(kv_empty, 1);
        tc::mbar_init(qd_full, 1);
        tc::mbar_init(qd_empty, 1);
        tc::mbar_init(sp_full, 1);
        tc::mbar_init(pds_ready, kEpiWarps);
        tc::mbar_init(mm2_done, 1);
        tc::mbar_init(s_free, kEpiWarps);
        tc::mbar_init(acc_full, 1);
        tc::mbar_init(acc_free, kEpiWarps);
        tc::mbar_init(drain, 1);
        *abort_flag = 0;
        tc::fence_mbar_init();
        tc::tma_prefetch_desc(&mQ);
        tc::tma_prefetch_desc(&mDO);
        tc::tma_prefetch_desc(&mKV);
    }
    if (warp == 1) tc::tmem_alloc(tmem_slot, 512);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = *tmem_slot;
    pdl_wait();
    const int kv_rows = a.B * a.T * a.nkv;  // V starts this many rows into the K/V map

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------ TMA producer
            bool ok = true;
            int st = 0;  // steps of this CTA
            int kv_armed = -1, qd_armed = -1;
            for (int n = 0, it; ok && (it = item_of(n, a.n_items)) >= 0; ++n) {
                int b, g, j;
                item_at(a, it, b, g, j);
                if (n > 0 && !tc::mbar_wait(kv_empty, (uint32_t)((n - 1) & 1), abort_flag)) {
                    ok = false;
                    break;
                }
                const int krow = (b * a.nkv + g) * a.T + j * kT;
                tc::mbar_expect_tx(kv_full, 2 * kTile);
                tc::tma_load_2d(sK, &mKV, 0, krow, kv_full);
                tc::tma_load_2d(sK + 16384, &mKV, 64, krow, kv_full);
                tc::tma_load_2d(sV, &mKV, 0, kv_rows + krow, kv_full);
                tc::tma_load_2d(sV + 16384, &mKV, 64, kv_rows + krow, kv_full);
                kv_armed = n & 1;
                for (int h = 0; ok && h < G; ++h) {
                    for (int i = j; i < a.nt; ++i, ++st) {
                        if (st > 0 && !tc::mbar_wait(qd_empty, (uint32_t)((st - 1) & 1), abort_flag)) {
                            ok = false;
                            break;
                        }
                        const int qrow = b * a.T + i * kT, qcol = (g * G + h) * kD;
                        const size_t r0 = ((size_t)b * a.nq + g * G + h) * a.T + (size_t)i * kT;
                        tc::mbar_expect_tx(qd_full, 2 * kTile + 2 * 128 * 4);
                        tc::tma_load_2d(sQ, &mQ, qcol, qrow, qd_full);
                        tc::tma_load_2d(sQ + 16384, &mQ, qcol + 64, qrow, qd_full);
                        tc::tma_load_2d(sDO, &mDO, qcol, qrow, qd_full);
                        tc::tma_load_2d(sDO + 16384, &mDO, qcol + 64, qrow, qd_full);
                        // the step's log-sum-exp and D rows (read by the epilogue before
                        // the stage is released again)
                        tc::bulk_load(sLse, a.lse + r0, 128 * 4, qd_full);
                        tc::bulk_load(sD, a.D + r0, 128 * 4, qd_full);
                        qd_armed = st & 1;
                    }
                }
            }
            pdl_trigger();
            if (!ok) {  // let every issued copy land before the CTA exits
                if (kv_armed >= 0) tc::mbar_wait_drain(kv_full, (uint32_t)kv_armed);
                if (qd_armed >= 0) tc::mbar_wait_drain(qd_full, (uint32_t)qd_armed);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ------------------------------------------------ MMA issuer
            constexpr uint32_t id_kk = tc::idesc_bf16(128, 128);                 // A, B K-major
            constexpr uint32_t id_km = tc::idesc_bf16(128, 128) | (1u << 16);    // B MN-major
            constexpr uint32_t id_mm = tc::idesc_bf16(128, 128) | (3u << 15);    // A, B MN-major
            const uint32_t aK = tc::smem_u32(sK), aV = tc::smem_u32(sV), aQ = tc::smem_u32(sQ),
                           aDO = tc::smem_u32(sDO), aP = tc::smem_u32(sP), aDS = tc::smem_u32(sDS);
            // K-major descriptor at k-step kk (16 elements) of a [128 x 128] tile; MN-major
            // descriptor at k-step kk (16 rows) with the second 64-column box 16 KB further
            auto km = [](uint32_t base, int kk) { return tc::sw128_desc(base + (kk >> 2) * 16384 + (kk & 3) * 32); };
            auto mn = [](uint32_t base, int kk) { return tc::sw128_desc_mn(base + kk * 2048, 16384); };
            bool ok = true, issued = false;
            int st = 0;
            for (int n = 0, it; ok && (it = item_of(n, a.n_items)) >= 0; ++n) {
                int b, g, j;
                item_at(a, it, b, g, j);
                if (!tc::mbar_wait(kv_full, (uint32_t)(n & 1), abort_flag)) {
                    ok = false;
                    break;
                }
                int e = 0;  // step within the item
                for (int h = 0; ok && h < G; ++h) {
                    for (int i = j; i < a.nt; ++i, ++st, ++e) {
                        if (!tc::mbar_wait(qd_full, (uint32_t)(st & 1), abort_flag) ||
                            (st > 0 && !tc::mbar_wait(s_free, (uint32_t)((st - 1) & 1), abort_flag))) {
                            ok = false;
                            break;
                        }
                        tc::fence_after_sync();
                        // 1. S^T = K Q^T, dP^T = V dO^T
#pragma unroll
                        for (int kk = 0; kk < kD / 16; ++kk) {
                            tc::mma_bf16(tmem + 0, km(aK, kk), km(aQ, kk), id_kk, kk ? 1u : 0u);
                            tc::mma_bf16(tmem + 128, km(aV, kk), km(aDO, kk), id_kk, kk ? 1u : 0u);
                        }
                        issued = true;
                        tc::mma_commit(sp_full);
                        // 3. after the epilogue wrote P^T and dS^T
                        if (!tc::mbar_wait(pds_ready, (uint32_t)(st & 1), abort_flag) ||
                            (e == 0 && n > 0 && !tc::mbar_wait(acc_free, (uint32_t)((n - 1) & 1), abort_flag))) {
                            ok = false;
                            break;
                        }
                        tc::fence_after_sync();
#pragma unroll
                        for (int kk = 0; kk < kT / 16; ++kk) {
                            const uint32_t acc = (e > 0 || kk > 0) ? 1u : 0u;
                            tc::mma_bf16(tmem + 256, km(aP, kk), mn(aDO, kk), id_km, acc);   // dV += P^T dO
                            tc::mma_bf16(tmem + 384, km(aDS, kk), mn(aQ, kk), id_km, acc);   // dK += dS^T Q
                        }
                        tc::mma_commit(qd_empty);  // Q and dO read: the next step's copies may start
#pragma unroll
                        for (int kk = 0; kk < kT / 16; ++kk)
                            tc::mma_bf16(tmem + 0, mn(aDS, kk), mn(aK, kk), id_mm, kk ? 1u : 0u);  // dQ = dS K
                        tc::mma_commit(mm2_done);
                    }
                }
                if (!ok) break;
                tc::mma_commit(kv_empty);
                tc::mma_commit(acc_full);
            }
            if (!ok && issued) {
                tc::mma_commit(drain);
                tc::mbar_wait_drain(drain, 0);
            }
        }
    } else {
        // ---------------------------------------------------- epilogue (warps 2..9)
        const int q = warp & 3;           // TMEM lane quadrant
        const int half = (warp - 2) >> 2;  // columns [64 half, 64 half + 64) of each tile
        const int row = q * 32 + lane;    // key row (steps 1-2, dV / dK) or query row (dQ)
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        uint8_t* stg = smem + kOffStage + (warp - 2) * 4096;
        const int sw = lane & 7;
        const float c2 = a.scale * kLog2e;
        bool ok = true;
        int st = 0;
        for (int n = 0, it; ok && (it = item_of(n, a.n_items)) >= 0; ++n) {
            int b, g, j;
            item_at(a, it, b, g, j);
            for (int h = 0; ok && h < G; ++h) {
                const int hq = g * G + h;
                for (int i = j; i < a.nt; ++i, ++st) {
                    // S^T and dP^T in TMEM; the step's log-sum-exp and D rows in shared
                    // memory (copied with Q and dO)
                    ok = tc::mbar_wait(sp_full, (uint32_t)(st & 1), abort_flag) &&
                         tc::mbar_wait(qd_full, (uint32_t)(st & 1), abort_flag);
                    ok = epi_bar_and(ok);
                    if (!ok) break;
                    tc::fence_after_sync();
                    // 2. P^T and dS^T of this key row and the warp's 64 queries (the box
                    // `half` of the tile), 32 queries per TMEM wait
                    const bool diag = i == j;
                    uint8_t* prow = sP + half * 16384 + (row >> 3) * 1024 + (row & 7) * 128;
                    uint8_t* drow = sDS + half * 16384 + (row >> 3) * 1024 + (row & 7) * 128;
#pragma unroll 1
                    for (int c0 = half * 64; c0 < half * 64 + 64; c0 += 32) {
                        uint32_t sr[2][16], dr[2][16];
#pragma unroll
                        for (int u = 0; u < 2; ++u) {
                            tc::tmem_ld16(tmem + lane_off + c0 + 16 * u, sr[u]);
                            tc::tmem_ld16(tmem + lane_off + 128 + c0 + 16 * u, dr[u]);
                        }
                        tc::tmem_wait_ld();
                        uint32_t pw[16], dw[16];
#pragma unroll
                        for (int u = 0; u < 2; ++u) {
#pragma unroll
                            for (int k2 = 0; k2 < 16; k2 += 2) {
                                const int qc = c0 + 16 * u + k2;  // query column within the tile
                                float p0 = ex2(fmaf(__uint_as_float(sr[u][k2]), c2, -sLse[qc] * kLog2e));
                                float p1 = ex2(fmaf(__uint_as_float(sr[u][k2 + 1]), c2, -sLse[qc + 1] * kLog2e));
                                if (diag) {  // key after the query: masked
                                    if (qc < row) p0 = 0.f;
                                    if (qc + 1 < row) p1 = 0.f;
                                }
                                const float d0 = p0 * (__uint_as_float(dr[u][k2]) - sD[qc]) * a.scale;
                                const float d1 = p1 * (__uint_as_float(dr[u][k2 + 1]) - sD[qc + 1]) * a.scale;
                                pw[u * 8 + k2 / 2] = pack2(p0, p1);
                                dw[u * 8 + k2 / 2] = pack2(d0, d1);
                            }
                        }
                        // 32 queries = granules (c0 % 64) / 8 .. + 3 of the row in box `half`
#pragma unroll
                        for (int gi = 0; gi < 4; ++gi) {
                            const int pos = ((((c0 & 63) >> 3) + gi) ^ (row & 7)) << 4;
                            *reinterpret_cast<uint4*>(prow + pos) =
                                make_uint4(pw[4 * gi], pw[4 * gi + 1], pw[4 * gi + 2], pw[4 * gi + 3]);
                            *reinterpret_cast<uint4*>(drow + pos) =
                                make_uint4(dw[4 * gi], dw[4 * gi + 1], dw[4 * gi + 2], dw[4 * gi + 3]);
                        }
                    }
                    tc::fence_proxy_async_smem();
                    tc::fence_before_sync();
                    __syncwarp();  // this warp's rows written and its sLse / sD reads done
                    if (lane == 0) tc::mbar_arrive(pds_ready);
                    // dQ of the step: TMEM columns [0, 128), one query row per thread, the
                    // warp's 64 columns
                    ok = tc::mbar_wait(mm2_done, (uint32_t)(st & 1), abort_flag);
                    ok = __all_sync(0xffffffffu, ok);
                    if (!ok) break;
                    tc::fence_after_sync();
                    const int qrow = b * a.T + i * kT + q * 32;
                    {
                        uint32_t r[4][16];  // the row's 64 dQ columns, one TMEM wait
#pragma unroll
                        for (int u = 0; u < 4; ++u) tc::tmem_ld16(tmem + lane_off + half * 64 + 16 * u, r[u]);
                        tc::tmem_wait_ld();
                        tc::fence_before_sync();
                        __syncwarp();
                        if (lane == 0) tc::mbar_arrive(s_free);  // TMEM columns [0, 128) free
#pragma unroll
                        for (int c = 0; c < 2; ++c) {  // 32 fp32 columns per reduction
                            if (lane == 0) tc::bulk_wait_read<0>();
                            __syncwarp();
                            uint4* srow = (uint4*)(stg + lane * 128);
#pragma unroll
                            for (int gi = 0; gi < 8; ++gi) {
                                const uint32_t* w = &r[2 * c + (gi >> 2)][(gi & 3) * 4];
                                srow[gi ^ sw] = make_uint4(w[0], w[1], w[2], w[3]);
                            }
                            tc::fence_proxy_async_smem();
                            __syncwarp();
                            if (lane == 0) {
                                tma_reduce_add_2d(&mDQ, hq * kD + half * 64 + 32 * c, qrow, stg);
                                tc::bulk_commit();
                            }
                        }
                    }
                }
            }
            if (!ok) break;
            // the item's dV (bf16) and dK (fp32): TMEM columns [256, 384) and [384, 512)
            ok = tc::mbar_wait(acc_full, (uint32_t)(n & 1), abort_flag);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            tc::fence_after_sync();
            const int krow = b * a.T + j * kT + q * 32;
            {  // dV: the warp's 64 bf16 columns, one store
                const int c0 = half * 64;
                uint32_t r[4][16];
#pragma unroll
                for (int u = 0; u < 4; ++u) tc::tmem_ld16(tmem + lane_off + 256 + c0 + 16 * u, r[u]);
                tc::tmem_wait_ld();
                if (lane == 0) tc::bulk_wait_read<0>();
                __syncwarp();
                uint4* srow = (uint4*)(stg + lane * 128);
#pragma unroll
                for (int gi = 0; gi < 8; ++gi) {
                    const uint32_t* w = &r[gi >> 1][(gi & 1) * 8];
                    srow[gi ^ sw] = make_uint4(pack2(__uint_as_float(w[0]), __uint_as_float(w[1])),
                                               pack2(__uint_as_float(w[2]), __uint_as_float(w[3])),
                                               pack2(__uint_as_float(w[4]), __uint_as_float(w[5])),
                                               pack2(__uint_as_float(w[6]), __uint_as_float(w[7])));
                }
                tc::fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tc::tma_store_2d(&mDV, dv_col0 + g * kD + c0, krow, stg);
                    tc::bulk_commit();
                }
            }
#pragma unroll
            for (int c0 = half * 64; c0 < half * 64 + 64; c0 += 32) {  // dK: 32 fp32 columns per store
                uint32_t r[2][16];
                tc::tmem_ld16(tmem + lane_off + 384 + c0, r[0]);
                tc::tmem_ld16(tmem + lane_off + 384 + c0 + 16, r[1]);
                tc::tmem_wait_ld();
                if (lane == 0) tc::bulk_wait_read<0>();
                __syncwarp();
                uint4* srow = (uint4*)(stg + lane * 128);
#pragma unroll
                for (int gi = 0; gi < 8; ++gi) {
                    const uint32_t* w = &r[gi >> 2][(gi & 3) * 4];
                    srow[gi ^ sw] = make_uint4(w[0], w[1], w[2], w[3]);
                }
                tc::fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tc::tma_store_2d(&mDK, g * kD + c0, krow, stg);
                    tc::bulk_commit();
                }
            }
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(acc_free);
        }
        if (lane == 0) tc::bulk_wait<0>();  // every store and reduction of this warp has completed
    }

    tc::fence_before_sync();
    __syncthreads();
    if (threadIdx.x == 0 && *abort_flag) atomicOr(a.status, QK_STATUS_TIMEOUT);
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, 512);
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
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)p;
    }
    return fn;
}

// 2-D map over [rows, cols] (row stride ld elements), box of box_x columns x box_y rows,
// 128-byte swizzle (box_x x element size = 128 bytes).
bool map2d(CUtensorMap* map, const void* base, bool f32, size_t cols, size_t rows, size_t ld, int box_x,
           int box_y) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * (f32 ? 4 : 2)};
    cuuint32_t box[2] = {(cuuint32_t)box_x, (cuuint32_t)box_y};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
              const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool al16(const void* p) { return ((uintptr_t)p & 15) == 0; }

}  // namespace

bool attn_bwd_supported(int d, int nq, int nkv, int T) { return d == kD && nq % nkv == 0 && T % kT == 0; }

// q, dO: [B T, nq d] bf16 (token-major); kvh: [2][B][nkv][T][d] bf16 (K then V);
// lse, D: [B nq T] fp32; dq: [B T, nq d] fp32, zero on entry (the kernel adds into it);
// dk: [B T, nkv d] fp32; dv: columns dv_col0 .. dv_col0 + nkv d of dv_base [B T, dv_ld] bf16.
int launch_attn_bwd(const bf16* q, const bf16* dO, const bf16* kvh, const float* lse, const float* D,
                    float* dq, float* dk, bf16* dv_base, int dv_ld, int dv_col0, int B, int T, int nq, int nkv,
                    int num_sms, uint32_t* status, cudaStream_t s) {
    static bool attr_set = false;
    if (!attr_set) {
        if (cudaFuncSetAttribute(attn_bwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem) !=
            cudaSuccess)
            return QK_ECUDA;
        attr_set = true;
    }
    const size_t M = (size_t)B * T;
    if (!al16(q) || !al16(dO) || !al16(kvh) || !al16(dq) || !al16(dk) || !al16(dv_base) || dv_ld % 8 ||
        dv_col0 % 64 || T % kT || M * nkv * 2 >= ((size_t)1 << 31))
        return QK_ESHAPE;
    CUtensorMap mq, mdo, mkv, mdq, mdk, mdv;
    if (!map2d(&mq, q, false, (size_t)nq * kD, M, (size_t)nq * kD, 64, 128) ||
        !map2d(&mdo, dO, false, (size_t)nq * kD, M, (size_t)nq * kD, 64, 128) ||
        !map2d(&mkv, kvh, false, kD, 2 * M * nkv, kD, 64, 128) ||
        !map2d(&mdq, dq, true, (size_t)nq * kD, M, (size_t)nq * kD, 32, 32) ||
        !map2d(&mdk, dk, true, (size_t)nkv * kD, M, (size_t)nkv * kD, 32, 32) ||
        !map2d(&mdv, dv_base, false, (size_t)dv_col0 + (size_t)nkv * kD, M, (size_t)dv_ld, 64, 32))
        return QK_ECUDA;
    Args a{B, T, nq, nkv, B * nkv * (T / kT), T / kT, lse, D, 1.f / sqrtf((float)kD), status};
    const int grid = a.n_items < num_sms ? a.n_items : num_sms;
    launch_k(attn_bwd_kernel, dim3(grid), dim3(kThreads), kSmem, s, mq, mdo, mkv, mdq, mdk, mdv, a, dv_col0);
    note_launch();
    return QK_OK;
}

}  // namespace qk
