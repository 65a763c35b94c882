// One work item of the split GQA decode attention over the bf16 KV cache, run
// by 128 threads (four warps); the decode attention kernel runs one item per CTA.
//
// Item (split, b, kvh): one decode token per row b; query head h = kvh * G + g
// (G = n_q / n_kv <= 8) attends cache positions 0 .. p(b).  The key tiles
// 0 .. p/64 of each (b, kvh) are cut evenly into n_split chunks at that row's
// position (the caller's `chunk` caps a chunk's length); the item streams its
// chunk through a 3-stage ring of 64-key K and V tiles loaded by TMA (128-byte
// swizzle, two 64-dim boxes per tile, one mbarrier per stage).  Each of the 4
// warps takes 16 keys of a tile and runs, on the tensor cores (mma.sync
// m16n8k16, bf16 in, fp32 out):
//   S[16 x 16] = Q_pad[16 x 128] * K^T   (rows 0..G-1 are the group's heads)
//   online softmax in base 2 over its keys (running max m, running sum l)
//   O[16 x 128] += P[16 x 16] * V[16 x 128]
// The 4 warps are merged in shared memory and the item writes an unnormalised
// partial (O, m, l) per head; the last item of a (row, kv head) to finish (an
// atomic ticket) merges the chunks of its heads:
//   o = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s,  M = max_s m_s,
// and resets the ticket.  Keys past p inside the last tile are masked to -inf in
// S, and their V rows are zeroed in shared memory before P*V (cache memory
// beyond p is unwritten and may hold NaN patterns; 0 * NaN would poison O).
//
// The ring's mbarrier phases continue across the items a CTA runs (`tiles`
// counts the tiles it has loaded so far; a CTA that runs one item passes 0).  Waits are bounded; on a timeout the
// item raises the abort flag, waits (bounded) for the copies it issued and
// returns -1 without writing its partial.  Otherwise it returns 1 if it wrote the
// (row, kv head) output (a single chunk, or the last chunk's merge), else 0.
#pragma once

#include <cuda.h>

#include "mma_sync.cuh"
#include "qk_internal.cuh"
#include "tc_ptx.cuh"

namespace qk {
namespace attn {

constexpr int kD = 128;          // head_dim
constexpr int kTileKeys = 64;    // keys per stage
constexpr int kStages = 3;
constexpr int kMergeChunks = 4;  // chunk partials per load batch of the final merge
constexpr int kHalfBytes = kTileKeys * 128;   // one 64-dim box: 64 rows x 128 B
constexpr int kTileBytes = 2 * kHalfBytes;    // K (or V) tile: dims 0..63 then 64..127
constexpr int kStageBytes = 2 * kTileBytes;   // K tile then V tile
constexpr int kRingBytes = kStages * kStageBytes;
// The warp-merge buffers ([4 warps][8 rows][128] O and [4][8][2] m, l) reuse the
// ring once every tile of the item has been consumed.
static_assert(4 * 8 * kD * 4 + 4 * 8 * 2 * 4 <= kRingBytes, "merge buffers");

struct Args {
    const bf16* q;
    int q_ld, nq, nkv;
    KvPages kp;        // cache layout (paged: page % 64 == 0, so a 64-key tile stays in its page)
    PosIndex pos;
    int chunk, n_split;
    float* part_o;     // [B nq][n_split][128]
    float2* part_ml;   // [B nq][n_split]
    int* tickets;      // [B nkv], zero on entry, zero again after the merge
    bf16* out;         // [B, nq * 128]
    uint32_t* status;
};

// Address of (key row, 16-byte chunk c) in a 64-key K or V tile.
__device__ __forceinline__ uint32_t tile_addr(uint32_t tile, int key, int c) {
    return ms::sw_addr<kTileKeys>(tile, key, c);
}

// Runs item (split, b, kvh) on 128 threads with thread index tid (0..127) and
// warp = tid / 32.  PAGED: the cache is paged (a.kp.table set); else dense.  ring: kRingBytes of 1024-aligned shared memory; full: its
// kStages mbarriers (count 1); tmKV: 3-D map of the caches ({128, rows, layers},
// K rows first, then V rows), z: the layer.  *last_s: a shared int.
template <bool PAGED>
__device__ __forceinline__ int decode_item(const Args& a, const CUtensorMap* tmKV, int z, int split,
                                            int b, int kvh, uint8_t* ring, uint64_t* full,
                                            int& tiles, volatile int* abort_flag, int* last_s,
                                            int tid) {
    using ms::ldsm_x4;
    using ms::ldsm_x4_t;
    using ms::mma16816;
    using ms::pack_bf16;
    const int nq = a.nq, nkv = a.nkv, cap = a.kp.cap();
    const int G = nq / nkv;
    const int warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, tig = lane & 3;
    float* red = (float*)ring;           // [4 warps][8 rows][128], after the key loop
    float* red_ml = red + 4 * 8 * kD;    // [4 warps][8 rows][2]

    int p = a.pos.pos_dev ? a.pos.pos_dev[b] : a.pos.start;
    if (p < 0 || p >= cap) p = p < 0 ? 0 : cap - 1;  // flagged by the cache-write kernel
    // The row's key tiles 0 .. p/64 are cut into n_split equal runs at this row's own
    // position; `chunk` caps a run at the cost model's length.
    const int n_tiles_b = p / kTileKeys + 1;
    const int per = min((n_tiles_b + a.n_split - 1) / a.n_split, a.chunk / kTileKeys);
    const int n_valid = (n_tiles_b + per - 1) / per;  // splits that hold keys
    const int k_begin = split * per * kTileKeys;
    if (split >= n_valid) return 0;  // nothing to attend in this split; the merge skips it
    const int k_end = min(k_begin + per * kTileKeys, p + 1);
    const int n_tiles = (k_end - k_begin + kTileKeys - 1) / kTileKeys;
    // V's pool follows K's in the 2-D view of a layer's cache; a dense cache's row b is
    // its page b, so the row of key k of (b, kvh) is row0 + k
    const int v_off = a.kp.n_pages * nkv * a.kp.page;
    const int row0 = (b * nkv + kvh) * a.kp.page;

    tc::bar128();  // the ring (and the previous item's merge buffers) is free
    auto issue = [&](int t) {
        const int st = (tiles + t) % kStages;
        uint8_t* base = ring + st * kStageBytes;
        const int r = PAGED ? kv_row(a.kp, nkv, b, kvh, k_begin + t * kTileKeys, a.status)
                            : row0 + k_begin + t * kTileKeys;  // the tile's first key
        tc::mbar_expect_tx(&full[st], kStageBytes);
        tc::tma_load_3d(base, tmKV, 0, r, z, &full[st]);
        tc::tma_load_3d(base + kHalfBytes, tmKV, 64, r, z, &full[st]);
        tc::tma_load_3d(base + kTileBytes, tmKV, 0, v_off + r, z, &full[st]);
        tc::tma_load_3d(base + kTileBytes + kHalfBytes, tmKV, 64, v_off + r, z, &full[st]);
    };
    int n_issued = 0;  // meaningful in thread 0 only
    if (tid == 0)
        for (; n_issued < kStages && n_issued < n_tiles; ++n_issued) issue(n_issued);

    // Q fragments (A operand, rows = heads of the group, padded to 16): a0a1 / a4a5
    // hold row g, dims 16ks + 2tig (+8); rows 8..15 are zero.
    uint32_t qa[8][2];
    {
        const bool valid = g < G;
        const bf16* qrow = a.q + (size_t)b * a.q_ld + (size_t)(kvh * G + (valid ? g : 0)) * kD;
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
            uint32_t lo = *reinterpret_cast<const uint32_t*>(qrow + 16 * ks + 2 * tig);
            uint32_t hi = *reinterpret_cast<const uint32_t*>(qrow + 16 * ks + 8 + 2 * tig);
            qa[ks][0] = valid ? lo : 0u;
            qa[ks][1] = valid ? hi : 0u;
        }
    }
    const float scale = rsqrtf((float)kD) * 1.4426950408889634f;  // 1/sqrt(d) * log2(e)
    float m_run = -INFINITY, l_run = 0.f;
    float o[16][4];
#pragma unroll
    for (int j = 0; j < 16; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;

    bool ok = true;
    int t_fail = n_tiles;
    for (int t = 0; t < n_tiles; ++t) {
        const int st = (tiles + t) % kStages;
        const uint32_t phase = (uint32_t)(((tiles + t) / kStages) & 1);
        bool got = tc::mbar_wait(&full[st], phase, abort_flag);
        if (!tc::bar128_and(got)) {
            ok = false;
            t_fail = t;
            break;
        }
        uint8_t* base = ring + st * kStageBytes;
        const int key0 = k_begin + t * kTileKeys;  // absolute position of the tile's first key
        if (key0 + kTileKeys - 1 > p) {
            // zero the V rows past p (16-byte stores over both boxes)
            for (int i = tid; i < kTileKeys * 16; i += 128) {
                const int key = i >> 4, c = i & 15;
                if (key0 + key > p)
                    *reinterpret_cast<uint4*>(base + kTileBytes + (c >> 3) * kHalfBytes + key * 128 +
                                              (((c & 7) ^ (key & 7)) << 4)) = make_uint4(0, 0, 0, 0);
            }
            tc::bar128();
        }
        const uint32_t kt = tc::smem_u32(base), vt = tc::smem_u32(base + kTileBytes);
        const int kw = warp * 16;  // this warp's 16 keys within the tile
        // ---- S = Q K^T for keys kw .. kw+15 (two n8 tiles)
        float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
            // matrices: (keys 0-7, dims lo), (keys 0-7, dims hi), (keys 8-15, lo), (keys 8-15, hi)
            const int mi = lane >> 3, r = lane & 7;
            const int key = kw + (mi >> 1) * 8 + r, c = 2 * ks + (mi & 1);
            uint32_t b00, b01, b10, b11;
            ldsm_x4(tile_addr(kt, key, c), b00, b01, b10, b11);
            const uint32_t qf[4] = {qa[ks][0], 0u, qa[ks][1], 0u};
            mma16816(s0, qf, b00, b01);
            mma16816(s1, qf, b10, b11);
        }
        // ---- online softmax (row g; rows 8..15 are padding)
        float sv[4] = {s0[0] * scale, s0[1] * scale, s1[0] * scale, s1[1] * scale};
        const int kk[4] = {kw + 2 * tig, kw + 2 * tig + 1, kw + 8 + 2 * tig, kw + 9 + 2 * tig};
#pragma unroll
        for (int i = 0; i < 4; ++i)
            if (key0 + kk[i] > p) sv[i] = -INFINITY;
        float mx = fmaxf(fmaxf(sv[0], sv[1]), fmaxf(sv[2], sv[3]));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        const float m_new = fmaxf(m_run, mx);
        float pv[4], ps = 0.f;
        if (m_new == -INFINITY) {  // every key so far masked (cannot happen for key 0 <= p)
            pv[0] = pv[1] = pv[2] = pv[3] = 0.f;
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                pv[i] = exp2f(sv[i] - m_new);
                ps += pv[i];
            }
        }
        ps += __shfl_xor_sync(0xffffffffu, ps, 1);
        ps += __shfl_xor_sync(0xffffffffu, ps, 2);
        const float corr = m_run == -INFINITY ? 0.f : exp2f(m_run - m_new);
        l_run = l_run * corr + ps;
        m_run = m_new;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            o[j][0] *= corr;
            o[j][1] *= corr;
        }
        // ---- O += P V: P as the A operand (rows 8..15 zero), V^T fragments via ldmatrix.trans
        const uint32_t pa[4] = {pack_bf16(pv[0], pv[1]), 0u, pack_bf16(pv[2], pv[3]), 0u};
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) {
            // matrices: (keys 0-7, dims 16jj..+7), (keys 8-15, same), (keys 0-7, dims 16jj+8..), (keys 8-15, ...)
            const int mi = lane >> 3, r = lane & 7;
            const int key = kw + (mi & 1) * 8 + r, c = 2 * jj + (mi >> 1);
            uint32_t v0, v1, v2, v3;
            ldsm_x4_t(tile_addr(vt, key, c), v0, v1, v2, v3);
            mma16816(o[2 * jj], pa, v0, v1);
            mma16816(o[2 * jj + 1], pa, v2, v3);
        }
        tc::bar128();  // every warp is done with this stage
        if (tid == 0 && n_issued < n_tiles) issue(n_issued++);
    }

    if (!ok) {
        if (tid == 0) {
            atomicOr(a.status, QK_STATUS_TIMEOUT);
            // let the copies issued for tiles not yet consumed land before returning
            for (int t = t_fail; t < n_issued; ++t)
                tc::mbar_wait_drain(&full[(tiles + t) % kStages],
                                    (uint32_t)(((tiles + t) / kStages) & 1));
        }
        return -1;
    }
    tiles += n_tiles;

    // ---- merge the 4 warps: row g (< 8) of each warp's O (dims 8j + 2tig, +1)
    if (g < 8) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            red[(warp * 8 + g) * kD + 8 * j + 2 * tig] = o[j][0];
            red[(warp * 8 + g) * kD + 8 * j + 2 * tig + 1] = o[j][1];
        }
        if (tig == 0) {
            red_ml[(warp * 8 + g) * 2] = m_run;
            red_ml[(warp * 8 + g) * 2 + 1] = l_run;
        }
    }
    tc::bar128();
    // thread -> (row gg, dim d): 128 threads cover one row's 128 dims; loop over the G rows
    for (int gg = 0; gg < G; ++gg) {
        const int d = tid;
        float M = -INFINITY;
        for (int w = 0; w < 4; ++w) M = fmaxf(M, red_ml[(w * 8 + gg) * 2]);
        float acc = 0.f, L = 0.f;
        for (int w = 0; w < 4; ++w) {
            const float mw = red_ml[(w * 8 + gg) * 2];
            const float f = mw == -INFINITY ? 0.f : exp2f(mw - M);
            acc += f * red[(w * 8 + gg) * kD + d];
            L += f * red_ml[(w * 8 + gg) * 2 + 1];
        }
        const size_t head = (size_t)b * nq + kvh * G + gg;
        if (n_valid == 1) {  // a single chunk is already the whole attention
            a.out[head * kD + d] = __float2bfloat16_rn(acc / L);
        } else {
            a.part_o[(head * a.n_split + split) * kD + d] = acc;
            if (d == 0) a.part_ml[head * a.n_split + split] = make_float2(M, L);
        }
    }
    if (n_valid == 1) return 1;
    // The last item of this (row, kv head) to finish merges the chunks' partials:
    //   o = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s,  M = max_s m_s,
    // then resets the ticket for the next layer.  The barrier orders every thread's
    // partial stores before thread 0's release; its acquire orders the merge's reads
    // after the other chunks' stores.
    tc::bar128();
    if (tid == 0) *last_s = tc::atom_add_acq_rel_gpu(&a.tickets[b * nkv + kvh], 1) == n_valid - 1;
    tc::bar128();
    if (!*last_s) return 0;
    // Online merge over the chunks in order, kMergeChunks at a time: every load of a
    // batch is issued before any is used, so a batch costs one L2 round trip.
    const int d = tid;
    float Mh[8], Ah[8], Lh[8];
#pragma unroll
    for (int gg = 0; gg < 8; ++gg) Mh[gg] = -INFINITY, Ah[gg] = 0.f, Lh[gg] = 0.f;
    for (int base = 0; base < n_valid; base += kMergeChunks) {
        float ov[8][kMergeChunks];
        float2 ml[8][kMergeChunks];
#pragma unroll
        for (int gg = 0; gg < 8; ++gg)
#pragma unroll
            for (int k = 0; k < kMergeChunks; ++k) {
                const bool v = gg < G && base + k < n_valid;
                const size_t i = ((size_t)b * nq + kvh * G + gg) * a.n_split + base + k;
                ov[gg][k] = v ? __ldcg(&a.part_o[i * kD + d]) : 0.f;
                ml[gg][k] = v ? __ldcg(&a.part_ml[i]) : make_float2(-INFINITY, 0.f);
            }
#pragma unroll
        for (int gg = 0; gg < 8; ++gg) {
            float Mn = Mh[gg];
#pragma unroll
            for (int k = 0; k < kMergeChunks; ++k) Mn = fmaxf(Mn, ml[gg][k].x);
            if (Mn == -INFINITY) continue;  // padding head
            const float sc = Mh[gg] == -INFINITY ? 0.f : exp2f(Mh[gg] - Mn);
            float A = Ah[gg] * sc, L = Lh[gg] * sc;
#pragma unroll
            for (int k = 0; k < kMergeChunks; ++k) {
                const float f = ml[gg][k].x == -INFINITY ? 0.f : exp2f(ml[gg][k].x - Mn);
                A += f * ov[gg][k];
                L += f * ml[gg][k].y;
            }
            Mh[gg] = Mn, Ah[gg] = A, Lh[gg] = L;
        }
    }
#pragma unroll
    for (int gg = 0; gg < 8; ++gg)
        if (gg < G) a.out[((size_t)b * nq + kvh * G + gg) * kD + d] = __float2bfloat16_rn(Ah[gg] / Lh[gg]);
    if (tid == 0) a.tickets[b * nkv + kvh] = 0;
    return 1;
}

}  // namespace attn
}  // namespace qk
