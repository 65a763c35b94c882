// Causal GQA attention for prefill and teacher-forced scoring (bf16, d = 128) on
// the tcgen05 tensor cores with TMEM accumulators.
//
// Row r = b * T + t is the query at position p = start_b + t (start_b = start, or
// start_dev[b] when the rows start at different positions); it attends cache
// positions 0 .. p of its sequence (keys written by this call's QK-norm/RoPE
// kernel for positions >= start, by earlier calls below start).
//
// One CTA per (b, kv head, 128-query tile, query head of the group); the query
// heads of a group are adjacent in the grid (so their CTAs stream the same K/V
// tiles from L2 at about the same time) and the longer query tiles of a group
// come first.  192 threads:
//   warp 0, one lane : TMA producer: the Q tile once, then 128-key K and V tiles
//                      into a 2-stage ring (the cache viewed as 2-D rows of 128
//                      elements, two 64-column boxes per tile, 128-byte swizzle);
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
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 512;      // S0 [0,128), S1 [128,256), O [256,384)
constexpr float kRescale = 8.f;          // raise the running max only past 2^8

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

__global__ void __launch_bounds__(kThreads, 1)
    attn_prefill_kernel(const __grid_constant__ CUtensorMap tmQ,
                        const __grid_constant__ CUtensorMap tmKV, int nq, int nkv,
                        int max_batch, int max_seq, int start_all,
                        const int32_t* __restrict__ start_dev, int T, bf16* __restrict__ o,
                        uint32_t* __restrict__ status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* sQ = smem;
    uint8_t* sKV = smem + kOffKV;
    uint8_t* sP = smem + kOffP;
    uint64_t* q_full = (uint64_t*)(smem + kOffBar);
    uint64_t* kv_full = q_full + 1;
    uint64_t* kv_empty = kv_full + kStages;
    uint64_t* s_full = kv_empty + kStages;
    uint64_t* s_empty = s_full + 2;
    uint64_t* p_full = s_empty + 2;
    uint64_t* pv_done = p_full + 2;
    uint64_t* drain = pv_done + 2;
    uint32_t* tmem_slot = (uint32_t*)(drain + 1);
    volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int G = nq / nkv;
    const int n_qt = (T + kQT - 1) / kQT;
    // grid order: (b, kv head) groups; inside, longest query tile first, heads innermost
    const int per_bg = n_qt * G;
    const int bg = blockIdx.x / per_bg, rem = blockIdx.x % per_bg;
    const int qt = n_qt - 1 - rem / G;
    const int b = bg / nkv, g = bg % nkv;
    const int h = g * G + rem % G;
    const int q0 = qt * kQT;
    int start = start_all;  // start_dev is read after the dependency wait below

    if (threadIdx.x == 0) {
        tc::mbar_init(q_full, 1);
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(&kv_full[s], 1);
            tc::mbar_init(&kv_empty[s], 1);
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
    pdl_wait();  // q, K and V come from the previous kernels
    if (start_dev) start = start_dev[b];
    // this row's first position (clamped into the cache; the cache-write kernel flags it)
    start = start < 0 ? 0 : (start > max_seq - T ? max_seq - T : start);
    const int kv_len = start + T;  // cache positions 0 .. kv_len-1 are written
    const int p_last = start + min(q0 + kQT - 1, T - 1);
    const int n_kt = p_last / kKT + 1;
    const int row0 = (b * nkv + g) * max_seq;
    const int v_off = max_batch * nkv * max_seq;

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------ TMA producer
            int armed[kStages] = {-1, -1};
            bool q_armed = true, ok = true;
            tc::mbar_expect_tx(q_full, kQBytes);
            tc::tma_load_2d(sQ, &tmQ, h * kD, b * T + q0, q_full);
            tc::tma_load_2d(sQ + kBox, &tmQ, h * kD + 64, b * T + q0, q_full);
            for (int j = 0; j < n_kt; ++j) {
                const int st = j % kStages;
                if (!tc::mbar_wait(&kv_empty[st], (uint32_t)(((j / kStages) & 1) ^ 1), abort_flag)) {
                    ok = false;
                    break;
                }
                uint8_t* base = sKV + st * kKVBytes;
                const int r = row0 + j * kKT;
                tc::mbar_expect_tx(&kv_full[st], kKVBytes);
                tc::tma_load_2d(base, &tmKV, 0, r, &kv_full[st]);
                tc::tma_load_2d(base + kBox, &tmKV, 64, r, &kv_full[st]);
                tc::tma_load_2d(base + 2 * kBox, &tmKV, 0, v_off + r, &kv_full[st]);
                tc::tma_load_2d(base + 3 * kBox, &tmKV, 64, v_off + r, &kv_full[st]);
                armed[st] = (j / kStages) & 1;
            }
            if (!ok) {  // abort path: let every copy this thread issued land before exit
                if (q_armed) tc::mbar_wait_drain(q_full, 0);
                for (int s = 0; s < kStages; ++s)
                    if (armed[s] >= 0) tc::mbar_wait_drain(&kv_full[s], (uint32_t)armed[s]);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ------------------------------------------------ MMA issuer
            constexpr uint32_t idesc_s = tc::idesc_bf16(128, kKT);
            constexpr uint32_t idesc_o = tc::idesc_bf16_bmn(128, kD);
            const uint32_t q_s = tc::smem_u32(sQ);
            bool ok = tc::mbar_wait(q_full, 0, abort_flag), issued = false;
            for (int j = 0; ok && j <= n_kt; ++j) {
                if (j < n_kt) {
                    const int st = j % kStages;
                    if (!tc::mbar_wait(&kv_full[st], (uint32_t)((j / kStages) & 1), abort_flag) ||
                        !tc::mbar_wait(&s_empty[j & 1], (uint32_t)(((j >> 1) & 1) ^ 1), abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc::fence_after_sync();
                    const uint32_t k_s = tc::smem_u32(sKV + st * kKVBytes);
                    const uint32_t d_s = tmem_base + (uint32_t)((j & 1) * kKT);
#pragma unroll
                    for (int kk = 0; kk < kD / 16; ++kk) {
                        const uint32_t off = (uint32_t)((kk >> 2) * kBox + (kk & 3) * 32);
                        tc::mma_bf16(d_s, tc::sw128_desc(q_s + off), tc::sw128_desc(k_s + off),
                                     idesc_s, kk > 0 ? 1u : 0u);
                    }
                    issued = true;
                    tc::mma_commit(&s_full[j & 1]);
                }
                if (j >= 1) {
                    const int i = j - 1, st = i % kStages;
                    if (!tc::mbar_wait(&p_full[i & 1], (uint32_t)((i >> 1) & 1), abort_flag)) {
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
                                     (i > 0 || kk > 0) ? 1u : 0u);
                    }
                    tc::mma_commit(&pv_done[i & 1]);
                    tc::mma_commit(&kv_empty[st]);
                }
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
        const int t = q0 + row;
        const int p = start + t;                 // this row's position
        const uint32_t lane_off = (uint32_t)(qd * 32) << 16;
        const float c = rsqrtf((float)kD) * 1.4426950408889634f;  // 1/sqrt(d) in base 2
        float m = -INFINITY, l = 0.f;
        bool ok = true;
        for (int j = 0; j < n_kt; ++j) {
            ok = tc::mbar_wait(&s_full[j & 1], (uint32_t)((j >> 1) & 1), abort_flag);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            tc::fence_after_sync();
            float x[kKT];
            const uint32_t s_t = tmem_base + lane_off + (uint32_t)((j & 1) * kKT);
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
            if (lane == 0) tc::mbar_arrive(&s_empty[j & 1]);
            const int key0 = j * kKT;
            float mx = -INFINITY;
            if (key0 + kKT - 1 > p) {  // diagonal tile: keys after p do not count
#pragma unroll
                for (int k = 0; k < kKT; ++k) {
                    x[k] = key0 + k <= p ? x[k] * c : -INFINITY;
                    mx = fmaxf(mx, x[k]);
                }
            } else {
#pragma unroll
                for (int k = 0; k < kKT; ++k) {
                    x[k] *= c;
                    mx = fmaxf(mx, x[k]);
                }
            }
            // raise the running max only when exponents would exceed 2^kRescale
            const bool raise = mx > m + kRescale;
            float factor = 1.f;
            if (raise) {
                factor = m == -INFINITY ? 0.f : tc::ex2_approx(m - mx);
                m = mx;
            }
            if (j > 0 && __any_sync(0xffffffffu, raise)) {
                // rescale this warp's rows of O once the previous P V product has landed
                const int i = j - 1;
                ok = tc::mbar_wait(&pv_done[i & 1], (uint32_t)((i >> 1) & 1), abort_flag);
                ok = __all_sync(0xffffffffu, ok);
                if (!ok) break;
                tc::fence_after_sync();
                const uint32_t o_t = tmem_base + lane_off + 256;
#pragma unroll
                for (int c0 = 0; c0 < kD; c0 += 16) {
                    uint32_t r[16];
                    tc::tmem_ld16(o_t + c0, r);
                    tc::tmem_wait_ld();
#pragma unroll
                    for (int k = 0; k < 16; ++k) r[k] = __float_as_uint(__uint_as_float(r[k]) * factor);
                    tc::tmem_st16(o_t + c0, r);
                }
                tc::tmem_wait_st();
            }
            l *= factor;
            // P_j = 2^(x - m) in bf16 into buffer j % 2 (free once P_{j-2} V_{j-2} landed)
            float sum = 0.f;
            uint32_t pk[kKT / 2];
#pragma unroll
            for (int k = 0; k < kKT; k += 2) {
                const float e0 = tc::ex2_approx(x[k] - m), e1 = tc::ex2_approx(x[k + 1] - m);
                sum += e0 + e1;
                pk[k / 2] = pack2(e0, e1);
            }
            l += sum;
            if (j >= 2) {
                const int i = j - 2;
                ok = tc::mbar_wait(&pv_done[i & 1], (uint32_t)((i >> 1) & 1), abort_flag);
                ok = __all_sync(0xffffffffu, ok);
                if (!ok) break;
            }
            uint8_t* pb = sP + (j & 1) * kPBytes;
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                uint8_t* rb = pb + half * kBox + (row >> 3) * 1024 + (row & 7) * 128;
#pragma unroll
                for (int ch = 0; ch < 8; ++ch) {
                    const int w = half * 32 + ch * 4;
                    *reinterpret_cast<uint4*>(rb + ((ch ^ (row & 7)) << 4)) =
                        make_uint4(pk[w], pk[w + 1], pk[w + 2], pk[w + 3]);
                }
            }
            if (key0 + kKT > kv_len) {
                // last tile: zero the V rows of unwritten cache positions
                const int st = j % kStages;
                ok = tc::mbar_wait(&kv_full[st], (uint32_t)((j / kStages) & 1), abort_flag);
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
            if (lane == 0) tc::mbar_arrive(&p_full[j & 1]);
        }
        if (ok) {
            const int i = n_kt - 1;
            ok = tc::mbar_wait(&pv_done[i & 1], (uint32_t)((i >> 1) & 1), abort_flag);
            ok = __all_sync(0xffffffffu, ok);
        }
        if (ok) {
            tc::fence_after_sync();
            const float inv = l > 0.f ? 1.f / l : 0.f;
            const uint32_t o_t = tmem_base + lane_off + 256;
            bf16* orow = o + ((size_t)b * T + (t < T ? t : 0)) * (size_t)(nq * kD) + (size_t)h * kD;
#pragma unroll
            for (int c0 = 0; c0 < kD; c0 += 16) {
                uint32_t r[16];
                tc::tmem_ld16(o_t + c0, r);
                tc::tmem_wait_ld();
                uint32_t w[8];
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    w[k] = pack2(__uint_as_float(r[2 * k]) * inv, __uint_as_float(r[2 * k + 1]) * inv);
                if (t < T) {
                    *reinterpret_cast<uint4*>(orow + c0) = make_uint4(w[0], w[1], w[2], w[3]);
                    *reinterpret_cast<uint4*>(orow + c0 + 8) = make_uint4(w[4], w[5], w[6], w[7]);
                }
            }
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
                        int max_batch, int max_seq, int B, int T, int start,
                        const int32_t* start_dev, bf16* o,
                        uint32_t* status, cudaStream_t s) {
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
    const size_t rows = 2 * (size_t)max_batch * nkv * max_seq;
    if (rows >= ((size_t)1 << 31) || (size_t)B * T >= ((size_t)1 << 31)) return QK_ESHAPE;
    // q rows are 16-byte aligned (q_ld % 8 == 0) and every box starts at a multiple of 64
    if (q_ld % 8 || ((uintptr_t)q & 15)) return QK_EINVAL;
    CUtensorMap mq, mkv;
    if (!make_map128((EncodeTiledFn)fn, &mq, q, (size_t)q_ld, (size_t)B * T, (size_t)q_ld) ||
        !make_map128((EncodeTiledFn)fn, &mkv, k_layer, kD, rows, kD))
        return QK_ECUDA;
    const int n_qt = (T + kQT - 1) / kQT;
    dim3 grid((unsigned)(B * nq * n_qt));
    launch_k(attn_prefill_kernel, grid, dim3(kThreads), kSmem, s, mq, mkv, nq, nkv, max_batch,
             max_seq, start, start_dev, T, o, status);
    note_launch();
    return QK_OK;
}

}  // namespace qk
