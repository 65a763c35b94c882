// Causal GQA attention for prefill and teacher-forced scoring (bf16, d = 128) on
// the tcgen05 tensor cores with TMEM accumulators.
//
// Row r = b * T + t is the query at position p = start_b + t (start_b = start, or
// start_dev[b] when the rows start at different positions); it attends cache
// positions 0 .. p of its sequence (keys written by this call's QK-norm/RoPE
// kernel for positions >= start, by earlier calls below start).
//
// Persistent: one CTA per SM walks the work items (b, kv head, 128-query tile,
// query head of the group).  The (b, kv head) groups are taken in chunks small
// enough for the chunk's K/V to stay in L2; inside a chunk the longest query tile
// comes first, every (group, query head) pair of one tile before the next, the
// query heads of a group adjacent (their CTAs stream the same K/V tiles from L2 at
// about the same time).  The items are dealt to the CTAs in rounds of one item per
// CTA, the CTA order reversed every other round, so the CTAs' sums of work even out
// (work falls with the item index inside a chunk).  The
// rings, TMEM buffers and barrier phases run on across items, so the next item's
// Q and K/V copies overlap the current item's last tiles.  192 threads:
//   warp 0, one lane : TMA producer: the Q tile of each item, then 128-key K and
//                      V tiles into two 2-stage rings (the cache viewed as 2-D rows
//                      of 128 elements, two 64-column boxes per tile, 128-byte
//                      swizzle); a K stage is freed by its S product, a V stage by
//                      its P V product, and K runs one tile ahead of V;
//   warp 1, one lane : TMEM owner and MMA issuer:
//                        S_j = Q K_j^T  (M 128 queries, N 128 keys, K = d) into one
//                                        of two TMEM S buffers,
//                        O  += P_j V_j  (M 128, N = d, K 128 keys; V is the
//                                        MN-major B operand) into the TMEM O;
//                      issued as S_0, S_1, O+=P_0V_0, S_2, O+=P_1V_1, ... so the
//                      tensor cores compute S_{j+1} while row j is exponentiated;
//   warps 2..5       : softmax, one query row per thread (TMEM lane): read S_j,
//                      mask keys > p, online softmax in base 2, P_j in bf16 into
//                      a shared-memory buffer (two, alternating) in the K-major
//                      swizzled layout of an MMA operand; finally O / l to global.
// The running maximum is raised only when a row's new maximum exceeds it by more
// than 2^8 (then the row's O in TMEM and its sum are rescaled, after the previous
// P V product has landed); otherwise the stale maximum keeps every exponent
// <= 2^8, so P stays exact to bf16 and the sums cannot overflow.  V rows at or
// past the call's last written position are zeroed in shared memory (unwritten
// cache memory may hold NaN patterns; 0 x NaN would poison O).
//
// Every mbarrier wait is bounded; on a timeout the CTA records
// QK_STATUS_TIMEOUT, waits (bounded) for its copies and MMAs and exits without
// writing.
#include <algorithm>
#include <cuda.h>

#include "qk_internal.cuh"
#include "tc_ptx.cuh"

namespace qk {

namespace {

constexpr int kD = 128;
constexpr int kQT = 128;                 // queries per CTA (MMA M)
constexpr int kKT = 128;                 // keys per tile (MMA N of S, K of P V)
constexpr int kStages = 2;
constexpr int kBox = 128 * 128;          // one 64-column box of 128 rows (16 KB)
constexpr int kQBytes = 2 * kBox;        // Q tile: two boxes (d 0..63, 64..127)
constexpr int kKVBytes = 4 * kBox;       // K then V, two boxes each
constexpr int kPBytes = 2 * kBox;        // P tile: keys 0..63 and 64..127
constexpr int kOffKV = kQBytes;
constexpr int kOffP = kOffKV + kStages * kKVBytes;
constexpr int kOffBar = kOffP + 2 * kPBytes;
constexpr int kSmem = kOffBar + 256 + 1024;
static_assert(kSmem <= 232448, "shared memory per CTA");
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 512;      // S0 [0,128), S1 [128,256), O [256,384)
constexpr float kRescale = 8.f;          // raise the running max only past 2^8

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

// Work item `it` of a launch: chunks of `chunk` (b, kv head) groups (the last one
// may be shorter) in order; inside a chunk the query tiles longest first, inside a
// tile the chunk's groups in order, the group's query heads innermost.
struct Item {
    int b, g, h, q0;
};
__device__ __forceinline__ Item item_at(int it, int n_qt, int G, int nkv, int n_groups, int chunk) {
    const int per_chunk = chunk * n_qt * G;
    const int g0 = (it / per_chunk) * chunk, rem = it % per_chunk;
    const int per_tile = min(chunk, n_groups - g0) * G;
    const int k = rem % per_tile;
    const int bg = g0 + k / G;
    Item w;
    w.b = bg / nkv;
    w.g = bg % nkv;
    w.h = w.g * G + k % G;
    w.q0 = (n_qt - 1 - rem / per_tile) * kQT;
    return w;
}

// This CTA's item in round r (one item per CTA per round, the CTA order reversed on
// odd rounds), or -1 past the last item.
__device__ __forceinline__ int item_of(int r, int n_work) {
    const int c = (r & 1) ? (int)gridDim.x - 1 - (int)blockIdx.x : (int)blockIdx.x;
    const int it = r * (int)gridDim.x + c;
    return it < n_work ? it : -1;
}

// First position of row b (clamped into the cache; the cache-write kernel flags it).
__device__ __forceinline__ int row_start(const int32_t* start_dev, int start_all, int b, int max_seq,
                                         int T) {
    int st = start_dev ? start_dev[b] : start_all;
    return st < 0 ? 0 : (st > max_seq - T ? max_seq - T : st);
}

__device__ __forceinline__ int tiles_of(int start, int q0, int T) {
    return (start + min(q0 + kQT - 1, T - 1)) / kKT + 1;
}

__global__ void __launch_bounds__(kThreads, 1)
    attn_prefill_kernel(const __grid_constant__ CUtensorMap tmQ,
                        const __grid_constant__ CUtensorMap tmKV, int nq, int nkv,
                        KvPages kp, int start_all,
                        const int32_t* __restrict__ start_dev, int T, int n_work, int chunk,
                        bf16* __restrict__ o, float* __restrict__ lse, uint32_t* __restrict__ status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* sQ = smem;
    uint8_t* sKV = smem + kOffKV;
    uint8_t* sP = smem + kOffP;
    uint64_t* q_full = (uint64_t*)(smem + kOffBar);
    uint64_t* q_empty = q_full + 1;
    uint64_t* k_full = q_empty + 1;
    uint64_t* k_empty = k_full + kStages;
    uint64_t* v_full = k_empty + kStages;
    uint64_t* v_empty = v_full + kStages;
    uint64_t* s_full = v_empty + kStages;
    uint64_t* s_empty = s_full + 2;
    uint64_t* p_full = s_empty + 2;
    uint64_t* pv_done = p_full + 2;
    uint64_t* drain = pv_done + 2;
    uint32_t* tmem_slot = (uint32_t*)(drain + 1);
    volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int G = nq / nkv;
    const int n_qt = (T + kQT - 1) / kQT;
    const int n_groups = n_work / (n_qt * G);

    if (threadIdx.x == 0) {
        tc::mbar_init(q_full, 1);
        tc::mbar_init(q_empty, 1);
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(&k_full[s], 1);
            tc::mbar_init(&k_empty[s], 1);
            tc::mbar_init(&v_full[s], 1);
            tc::mbar_init(&v_empty[s], 1);
        }
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(&s_full[i], 1);
            tc::mbar_init(&s_empty[i], 4);
            tc::mbar_init(&p_full[i], 4);
            tc::mbar_init(&pv_done[i], 1);
        }
        tc::mbar_init(drain, 1);
        *abort_flag = 0;
        tc::fence_mbar_init();
        tc::tma_prefetch_desc(&tmQ);
        tc::tma_prefetch_desc(&tmKV);
    }
    if (warp == 1) tc::tmem_alloc(tmem_slot, kTmemCols);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;
    pdl_wait();  // q, K, V and the row starts come from the previous kernels
    const int v_off = kp.n_pages * nkv * kp.page;  // V's pool follows K's
    const int max_seq = kp.cap();                  // positions a row holds

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------ TMA producer
            // K tiles lead V tiles by one (S_{j+1} is computed before P_j V_j), and each
            // ring frees a stage as soon as its own product has read it.
            int k_armed[kStages] = {-1, -1}, v_armed[kStages] = {-1, -1};
            int q_armed = -1;
            bool ok = true;
            int gt = 0, n = 0;  // global tile and item counters of this CTA
            auto load_k = [&](int g, int r) -> bool {
                const int st = g % kStages;
                if (!tc::mbar_wait(&k_empty[st], (uint32_t)(((g / kStages) & 1) ^ 1), abort_flag)) return false;
                uint8_t* base = sKV + st * kKVBytes;
                tc::mbar_expect_tx(&k_full[st], 2 * kBox);
                tc::tma_load_2d(base, &tmKV, 0, r, &k_full[st]);
                tc::tma_load_2d(base + kBox, &tmKV, 64, r, &k_full[st]);
                k_armed[st] = (g / kStages) & 1;
                return true;
            };
            auto load_v = [&](int g, int r) -> bool {
                const int st = g % kStages;
                if (!tc::mbar_wait(&v_empty[st], (uint32_t)(((g / kStages) & 1) ^ 1), abort_flag)) return false;
                uint8_t* base = sKV + st * kKVBytes + 2 * kBox;
                tc::mbar_expect_tx(&v_full[st], 2 * kBox);
                tc::tma_load_2d(base, &tmKV, 0, v_off + r, &v_full[st]);
                tc::tma_load_2d(base + kBox, &tmKV, 64, v_off + r, &v_full[st]);
                v_armed[st] = (g / kStages) & 1;
                return true;
            };
            for (int it; ok && (it = item_of(n, n_work)) >= 0; ++n) {
                const Item w = item_at(it, n_qt, G, nkv, n_groups, chunk);
                const int start = row_start(start_dev, start_all, w.b, max_seq, T);
                const int n_kt = tiles_of(start, w.q0, T);
                // the row (in the cache view) of key tile j (paged: page % 128 == 0, so the
                // tile lies in one page; dense: the rows past the row's end are masked)
                auto tile_row = [&](int j) { return kv_row(kp, nkv, w.b, w.g, j * kKT, status); };
                // the Q buffer is free once every S MMA of the previous item has completed
                if (n > 0 && !tc::mbar_wait(q_empty, (uint32_t)((n - 1) & 1), abort_flag)) {
                    ok = false;
                    break;
                }
                tc::mbar_expect_tx(q_full, kQBytes);
                tc::tma_load_2d(sQ, &tmQ, w.h * kD, w.b * T + w.q0, q_full);
                tc::tma_load_2d(sQ + kBox, &tmQ, w.h * kD + 64, w.b * T + w.q0, q_full);
                q_armed = n & 1;
                for (int j = 0; j <= n_kt; ++j) {
                    if (j < n_kt && !load_k(gt + j, tile_row(j))) {
                        ok = false;
                        break;
                    }
                    if (j >= 1 && !load_v(gt + j - 1, tile_row(j - 1))) {
                        ok = false;
                        break;
                    }
                }
                gt += n_kt;
            }
            if (!ok) {  // abort path: let every copy this thread issued land before exit
                if (q_armed >= 0) tc::mbar_wait_drain(q_full, (uint32_t)q_armed);
                for (int s = 0; s < kStages; ++s) {
                    if (k_armed[s] >= 0) tc::mbar_wait_drain(&k_full[s], (uint32_t)k_armed[s]);
                    if (v_armed[s] >= 0) tc::mbar_wait_drain(&v_full[s], (uint32_t)v_armed[s]);
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ------------------------------------------------ MMA issuer
            constexpr uint32_t idesc_s = tc::idesc_bf16(128, kKT);
            constexpr uint32_t idesc_o = tc::idesc_bf16_bmn(128, kD);
            const uint32_t q_s = tc::smem_u32(sQ);
            bool ok = true, issued = false;
            int gt = 0, n = 0;
            for (int it; ok && (it = item_of(n, n_work)) >= 0; ++n) {
                const Item w = item_at(it, n_qt, G, nkv, n_groups, chunk);
                const int n_kt = tiles_of(row_start(start_dev, start_all, w.b, max_seq, T), w.q0, T);
                if (!tc::mbar_wait(q_full, (uint32_t)(n & 1), abort_flag)) {
                    ok = false;
                    break;
                }
                const int g0 = gt;  // global index of this item's tile 0
                for (int j = 0; j <= n_kt; ++j) {
                    if (j < n_kt) {
                        const int g = g0 + j, st = g % kStages;
                        if (!tc::mbar_wait(&k_full[st], (uint32_t)((g / kStages) & 1), abort_flag) ||
                            !tc::mbar_wait(&s_empty[g & 1], (uint32_t)(((g >> 1) & 1) ^ 1), abort_flag)) {
                            ok = false;
                            break;
                        }
                        tc::fence_after_sync();
                        const uint32_t k_s = tc::smem_u32(sKV + st * kKVBytes);
                        const uint32_t d_s = tmem_base + (uint32_t)((g & 1) * kKT);
#pragma unroll
                        for (int kk = 0; kk < kD / 16; ++kk) {
                            const uint32_t off = (uint32_t)((kk >> 2) * kBox + (kk & 3) * 32);
                            tc::mma_bf16(d_s, tc::sw128_desc(q_s + off), tc::sw128_desc(k_s + off),
                                         idesc_s, kk > 0 ? 1u : 0u);
                        }
                        issued = true;
                        tc::mma_commit(&s_full[g & 1]);
                        tc::mma_commit(&k_empty[st]);
                        if (j == n_kt - 1) tc::mma_commit(q_empty);  // last read of this Q
                    }
                    if (j >= 1) {
                        const int i = g0 + j - 1, st = i % kStages;
                        if (!tc::mbar_wait(&v_full[st], (uint32_t)((i / kStages) & 1), abort_flag) ||
                            !tc::mbar_wait(&p_full[i & 1], (uint32_t)((i >> 1) & 1), abort_flag)) {
                            ok = false;
                            break;
                        }
                        tc::fence_after_sync();
                        const uint32_t p_s = tc::smem_u32(sP + (i & 1) * kPBytes);
                        const uint32_t v_s = tc::smem_u32(sKV + st * kKVBytes + 2 * kBox);
#pragma unroll
                        for (int kk = 0; kk < kKT / 16; ++kk) {
                            const uint32_t aoff = (uint32_t)((kk >> 2) * kBox + (kk & 3) * 32);
                            tc::mma_bf16(tmem_base + 256, tc::sw128_desc(p_s + aoff),
                                         tc::sw128_desc_mn(v_s + kk * 16 * 128, kBox), idesc_o,
                                         (j > 1 || kk > 0) ? 1u : 0u);
                        }
                        tc::mma_commit(&pv_done[i & 1]);
                        tc::mma_commit(&v_empty[st]);
                    }
                }
                gt = g0 + n_kt;
            }
            if (!ok && issued) {  // abort path: wait for the MMAs in flight
                tc::mma_commit(drain);
                tc::mbar_wait_drain(drain, 0);
            }
        }
    } else {
        // ---------------------------------------------------- softmax (warps 2..5)
        const int qd = warp & 3;                 // TMEM lane quadrant of this warp
        const int row = qd * 32 + lane;          // query row of the tile = TMEM lane
        const uint32_t lane_off = (uint32_t)(qd * 32) << 16;
        const float c = rsqrtf((float)kD) * 1.4426950408889634f;  // 1/sqrt(d) in base 2
        bool ok = true;
        int gt = 0;
        for (int r = 0, it; ok && (it = item_of(r, n_work)) >= 0; ++r) {
            const Item w = item_at(it, n_qt, G, nkv, n_groups, chunk);
            const int start = row_start(start_dev, start_all, w.b, max_seq, T);
            const int n_kt = tiles_of(start, w.q0, T);
            const int kv_len = start + T;  // cache positions 0 .. kv_len-1 are written
            const int t = w.q0 + row;
            const int p = start + t;       // this row's position
            float m = -INFINITY, l = 0.f;  // running max (scaled, base 2) and sum
            for (int j = 0; j < n_kt; ++j, ++gt) {
                ok = tc::mbar_wait(&s_full[gt & 1], (uint32_t)((gt >> 1) & 1), abort_flag);
                ok = __all_sync(0xffffffffu, ok);
                if (!ok) break;
                tc::fence_after_sync();
                float x[kKT];
                const uint32_t s_t = tmem_base + lane_off + (uint32_t)((gt & 1) * kKT);
#pragma unroll
                for (int c0 = 0; c0 < kKT; c0 += 16) {
                    uint32_t r[16];
                    tc::tmem_ld16(s_t + c0, r);
#pragma unroll
                    for (int k = 0; k < 16; ++k) x[c0 + k] = __uint_as_float(r[k]);
                }
                tc::tmem_wait_ld();
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(&s_empty[gt & 1]);
                const int key0 = j * kKT;
                if (key0 + kKT - 1 > p) {  // diagonal tile: keys after p do not count
#pragma unroll
                    for (int k = 0; k < kKT; ++k) x[k] = key0 + k <= p ? x[k] : -INFINITY;
                }
                // row max of the raw scores with 8 independent chains, then scaled (c > 0)
                float mx8[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) mx8[k] = x[k];
#pragma unroll
                for (int k = 8; k < kKT; ++k) mx8[k & 7] = fmaxf(mx8[k & 7], x[k]);
                const float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                                       fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7]))) * c;
                // raise the running max only when exponents would exceed 2^kRescale
                const bool raise = mx > m + kRescale;
                float factor = 1.f;
                if (raise) {
                    factor = m == -INFINITY ? 0.f : tc::ex2_approx(m - mx);
                    m = mx;
                }
                if (j > 0 && __any_sync(0xffffffffu, raise)) {
                    // rescale this warp's rows of O once the previous P V product has landed
                    const int i = gt - 1;
                    ok = tc::mbar_wait(&pv_done[i & 1], (uint32_t)((i >> 1) & 1), abort_flag);
                    ok = __all_sync(0xffffffffu, ok);
                    if (!ok) break;
                    tc::fence_after_sync();
                    const uint32_t o_t = tmem_base + lane_off + 256;
#pragma unroll
                    for (int c0 = 0; c0 < kD; c0 += 64) {
                        uint32_t r[4][16];
#pragma unroll
                        for (int q = 0; q < 4; ++q) tc::tmem_ld16(o_t + c0 + 16 * q, r[q]);
                        tc::tmem_wait_ld();
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
#pragma unroll
                            for (int k = 0; k < 16; ++k)
                                r[q][k] = __float_as_uint(__uint_as_float(r[q][k]) * factor);
                            tc::tmem_st16(o_t + c0 + 16 * q, r[q]);
                        }
                    }
                    tc::tmem_wait_st();
                }
                // P_j = 2^(x c - m) in bf16 into buffer gt % 2 (free once the P V product of
                // global tile gt - 2 has landed); sums in 8 independent chains
                float sum8[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) sum8[k] = 0.f;
                uint32_t pk[kKT / 2];
                const float nm = -m;
#pragma unroll
                for (int k = 0; k < kKT; k += 2) {
                    const float e0 = tc::ex2_approx(fmaf(x[k], c, nm));
                    const float e1 = tc::ex2_approx(fmaf(x[k + 1], c, nm));
                    sum8[(k >> 1) & 7] += e0 + e1;
                    pk[k / 2] = pack2(e0, e1);
                }
                l = l * factor + (((sum8[0] + sum8[1]) + (sum8[2] + sum8[3])) +
                                  ((sum8[4] + sum8[5]) + (sum8[6] + sum8[7])));
                if (gt >= 2) {
                    const int i = gt - 2;
                    ok = tc::mbar_wait(&pv_done[i & 1], (uint32_t)((i >> 1) & 1), abort_flag);
                    ok = __all_sync(0xffffffffu, ok);
                    if (!ok) break;
                }
                uint8_t* pb = sP + (gt & 1) * kPBytes;
#pragma unroll
                for (int half = 0; half < 2; ++half) {
                    uint8_t* rb = pb + half * kBox + (row >> 3) * 1024 + (row & 7) * 128;
#pragma unroll
                    for (int ch = 0; ch < 8; ++ch) {
                        const int wd = half * 32 + ch * 4;
                        *reinterpret_cast<uint4*>(rb + ((ch ^ (row & 7)) << 4)) =
                            make_uint4(pk[wd], pk[wd + 1], pk[wd + 2], pk[wd + 3]);
                    }
                }
                if (key0 + kKT > kv_len) {
                    // last tile: zero the V rows of unwritten cache positions
                    const int st = gt % kStages;
                    ok = tc::mbar_wait(&v_full[st], (uint32_t)((gt / kStages) & 1), abort_flag);
                    ok = __all_sync(0xffffffffu, ok);
                    if (!ok) break;
                    uint8_t* vb = sKV + st * kKVBytes + 2 * kBox;
                    const int r0 = kv_len - key0 > 0 ? kv_len - key0 : 0;
                    for (int idx = threadIdx.x - 64; idx < (kKT - r0) * 16; idx += 128) {
                        const int rr = r0 + (idx >> 4), ch = idx & 15;
                        *reinterpret_cast<uint4*>(vb + (ch >> 3) * kBox + rr * 128 +
                                                  (((ch & 7) ^ (rr & 7)) << 4)) = make_uint4(0, 0, 0, 0);
                    }
                }
                tc::fence_proxy_async_smem();
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(&p_full[gt & 1]);
            }
            if (!ok) break;
            // O / l of this item once its last P V product has landed
            const int i = gt - 1;
            ok = tc::mbar_wait(&pv_done[i & 1], (uint32_t)((i >> 1) & 1), abort_flag);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            tc::fence_after_sync();
            const float inv = l > 0.f ? 1.f / l : 0.f;
            // log-sum-exp of the row's scaled scores: sum_k e^(s_k / sqrt(d)) = l 2^m
            if (lse && t < T) lse[((size_t)w.b * nq + w.h) * T + t] = (m + log2f(l)) * 0.6931471805599453f;
            const uint32_t o_t = tmem_base + lane_off + 256;
            bf16* orow = o + ((size_t)w.b * T + (t < T ? t : 0)) * (size_t)(nq * kD) + (size_t)w.h * kD;
#pragma unroll
            for (int c0 = 0; c0 < kD; c0 += 64) {
                uint32_t r[4][16];
#pragma unroll
                for (int q = 0; q < 4; ++q) tc::tmem_ld16(o_t + c0 + 16 * q, r[q]);
                tc::tmem_wait_ld();
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint32_t wv[8];
#pragma unroll
                    for (int k = 0; k < 8; ++k)
                        wv[k] = pack2(__uint_as_float(r[q][2 * k]) * inv, __uint_as_float(r[q][2 * k + 1]) * inv);
                    if (t < T) {
                        *reinterpret_cast<uint4*>(orow + c0 + 16 * q) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
                        *reinterpret_cast<uint4*>(orow + c0 + 16 * q + 8) = make_uint4(wv[4], wv[5], wv[6], wv[7]);
                    }
                }
            }
            // the next item's first P V product overwrites O only after its P is ready,
            // which these warps write after this readback
            tc::fence_before_sync();
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    if (threadIdx.x == 0 && *abort_flag) atomicOr(status, QK_STATUS_TIMEOUT);
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem_base, kTmemCols);
    }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// 2-D bf16 map over `rows` rows of `inner` elements (row stride ld elements), box of
// 64 elements x 128 rows, 128-byte swizzle, zero fill out of range.
bool make_map128(EncodeTiledFn fn, CUtensorMap* map, const void* base, size_t inner, size_t rows,
                 size_t ld) {
    cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {64, 128};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
              box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool attn_prefill_supported(int d, int nq, int nkv) { return d == kD && nq % nkv == 0; }

int launch_attn_prefill(const bf16* q, int q_ld, const void* k_layer, int nq, int nkv,
                        const KvPages& kp, int B, int T, int start,
                        const int32_t* start_dev, bf16* o, int num_sms,
                        uint32_t* status, cudaStream_t s, float* lse) {
    static bool attr_set = false;
    if (!attr_set) {
        if (cudaFuncSetAttribute(attn_prefill_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kSmem) != cudaSuccess)
            return QK_ECUDA;
        attr_set = true;
    }
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult qr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &qr) != cudaSuccess ||
        qr != cudaDriverEntryPointSuccess)
        return QK_ECUDA;
    if (kp.table && kp.page % kKT) return QK_ESHAPE;  // a paged tile must not cross a page
    const int max_seq = kp.cap();
    const size_t rows = 2 * (size_t)kp.n_pages * nkv * kp.page;
    if (rows >= ((size_t)1 << 31) || (size_t)B * T >= ((size_t)1 << 31)) return QK_ESHAPE;
    // q rows are 16-byte aligned (q_ld % 8 == 0) and every box starts at a multiple of 64
    if (q_ld % 8 || ((uintptr_t)q & 15)) return QK_EINVAL;
    CUtensorMap mq, mkv;
    if (!make_map128((EncodeTiledFn)fn, &mq, q, (size_t)q_ld, (size_t)B * T, (size_t)q_ld) ||
        !make_map128((EncodeTiledFn)fn, &mkv, k_layer, kD, rows, kD))
        return QK_ECUDA;
    const int n_qt = (T + kQT - 1) / kQT;
    const int n_work = B * nq * n_qt;
    const int grid = n_work < num_sms ? n_work : num_sms;
    // groups per chunk: a chunk's K and V (cache positions 0 .. start + T - 1, every
    // position when the rows' starts are on the device) within 32 MB of L2
    const size_t kv_len = start_dev ? (size_t)max_seq : (size_t)std::min(max_seq, start + T);
    const size_t group_bytes = 2 * kv_len * kD * sizeof(bf16);
    const int chunk = (int)std::min<size_t>((size_t)B * nkv, std::max<size_t>(1, ((size_t)32 << 20) / group_bytes));
    launch_k(attn_prefill_kernel, dim3(grid), dim3(kThreads), kSmem, s, mq, mkv, nq, nkv, kp, start,
             start_dev, T, n_work, chunk, o, lse, status);
    note_launch();
    return QK_OK;
}

}  // namespace qk
