// Causal GQA attention for prefill and teacher-forced scoring (bf16, d = 128).
//
// Row r = b * T + t is the query at position p = start_b + t (start_b = start, or
// start_dev[b] when the rows start at different positions); it attends cache
// positions 0 .. p of its sequence (keys written by this call's QK-norm/RoPE
// kernel for positions >= start, by earlier calls below start).  One CTA per
// (64-query tile, b, query head), 4 warps of 16 queries.  The CTA walks the key
// tiles 0 .. (last query position)/64; K and V tiles of 64 keys arrive through
// a 2-stage TMA ring (the cache viewed as 2-D rows of 128 elements, two 64-dim
// boxes per tile, 128-byte swizzle).  Per warp and key tile, on the tensor
// cores (mma.sync m16n8k16, bf16 in, fp32 accumulate):
//   S[16 x 64] = Q[16 x 128] K^T;  mask keys > p;  online softmax in base 2
//   (running max and sum per query row);  O[16 x 128] += P[16 x 64] V[64 x 128]
// where P is re-used from the S accumulators as the A operand.  Query tiles run
// longest first (the grid is walked from the last tile).  V rows at or past the
// call's last written position are zeroed in shared memory (unwritten cache rows
// may hold NaN patterns; 0 * NaN would poison O).
//
// mbarrier waits are bounded; on a timeout the CTA records QK_STATUS_TIMEOUT,
// waits (bounded) for its copies and exits without writing.
#include <cuda.h>

#include "mma_sync.cuh"
#include "qk_internal.cuh"
#include "tc_ptx.cuh"

namespace qk {

namespace {

constexpr int kD = 128;
constexpr int kQT = 64;   // queries per CTA
constexpr int kKT = 64;   // keys per tile
constexpr int kStages = 2;
constexpr int kHalf = kKT * 128;        // one 64-dim box
constexpr int kTile = 2 * kHalf;        // K or V tile
constexpr int kStage = 2 * kTile;       // K then V
constexpr int kSmem = kStages * kStage + 1024 + 128;

using ms::ldsm_x4;
using ms::ldsm_x4_t;
using ms::mma16816;
using ms::pack_bf16;

__global__ void __launch_bounds__(128)
    attn_prefill_kernel(const __grid_constant__ CUtensorMap tmKV, const bf16* __restrict__ q,
                        int q_ld, int nq, int nkv, int max_batch, int max_seq, int start_all,
                        const int32_t* __restrict__ start_dev, int T, bf16* __restrict__ o,
                        uint32_t* __restrict__ status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t* full = (uint64_t*)(smem + kStages * kStage);
    volatile int* abort_flag = (volatile int*)(full + kStages);

    pdl_wait();
    const int n_qt = (T + kQT - 1) / kQT;
    const int qt = n_qt - 1 - blockIdx.x;
    const int b = blockIdx.y / nq, h = blockIdx.y % nq;
    const int kvh = h / (nq / nkv);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, tig = lane & 3;
    const int q0 = qt * kQT;
    // this row's first position (clamped into the cache; the cache-write kernel flags it)
    int start = start_dev ? start_dev[b] : start_all;
    start = start < 0 ? 0 : (start > max_seq - T ? max_seq - T : start);
    const int kv_len = start + T;  // cache positions 0 .. kv_len-1 are written
    const int p_last = start + min(q0 + kQT - 1, T - 1);
    const int n_kt = p_last / kKT + 1;
    const int row0 = (b * nkv + kvh) * max_seq;
    const int v_off = max_batch * nkv * max_seq;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) tc::mbar_init(&full[s], 1);
        *abort_flag = 0;
        tc::fence_mbar_init();
        tc::tma_prefetch_desc(&tmKV);
    }
    __syncthreads();
    auto issue = [&](int t) {
        const int st = t % kStages;
        uint8_t* base = smem + st * kStage;
        const int r = row0 + t * kKT;
        tc::mbar_expect_tx(&full[st], kStage);
        tc::tma_load_2d(base, &tmKV, 0, r, &full[st]);
        tc::tma_load_2d(base + kHalf, &tmKV, 64, r, &full[st]);
        tc::tma_load_2d(base + kTile, &tmKV, 0, v_off + r, &full[st]);
        tc::tma_load_2d(base + kTile + kHalf, &tmKV, 64, v_off + r, &full[st]);
    };
    int n_issued = 0;
    if (threadIdx.x == 0)
        for (; n_issued < kStages && n_issued < n_kt; ++n_issued) issue(n_issued);

    // Q fragments for rows (g, g+8) of this warp's 16 queries; rows past T are zero.
    const int ta = q0 + warp * 16 + g, tb = ta + 8;
    const int pa_pos = start + ta, pb_pos = start + tb;
    uint32_t qa[8][4];
    {
        const bf16* ra = q + ((size_t)b * T + min(ta, T - 1)) * q_ld + (size_t)h * kD;
        const bf16* rb = q + ((size_t)b * T + min(tb, T - 1)) * q_ld + (size_t)h * kD;
        const bool va = ta < T, vb = tb < T;
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
            const int c = 16 * ks + 2 * tig;
            qa[ks][0] = va ? *reinterpret_cast<const uint32_t*>(ra + c) : 0u;
            qa[ks][1] = vb ? *reinterpret_cast<const uint32_t*>(rb + c) : 0u;
            qa[ks][2] = va ? *reinterpret_cast<const uint32_t*>(ra + c + 8) : 0u;
            qa[ks][3] = vb ? *reinterpret_cast<const uint32_t*>(rb + c + 8) : 0u;
        }
    }
    const float scale = rsqrtf((float)kD) * 1.4426950408889634f;
    float m_a = -INFINITY, m_b = -INFINITY, l_a = 0.f, l_b = 0.f;
    float acc[16][4];
#pragma unroll
    for (int j = 0; j < 16; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;

    int t_fail = -1;
    for (int kt = 0; kt < n_kt; ++kt) {
        const int st = kt % kStages;
        bool got = tc::mbar_wait(&full[st], (uint32_t)((kt / kStages) & 1), abort_flag);
        if (!__syncthreads_and(got)) {
            t_fail = kt;
            break;
        }
        uint8_t* base = smem + st * kStage;
        const int key0 = kt * kKT;
        if (key0 + kKT > kv_len) {
            for (int i = threadIdx.x; i < kKT * 16; i += blockDim.x) {
                const int key = i >> 4, c = i & 15;
                if (key0 + key >= kv_len)
                    *reinterpret_cast<uint4*>(base + kTile + (c >> 3) * kHalf + key * 128 +
                                              (((c & 7) ^ (key & 7)) << 4)) = make_uint4(0, 0, 0, 0);
            }
            __syncthreads();
        }
        // Skip tiles entirely after this warp's last query (the diagonal of the earlier warps).
        const int warp_last = start + min(q0 + warp * 16 + 15, T - 1);
        if (key0 <= warp_last) {
            const uint32_t kt_s = tc::smem_u32(base), vt_s = tc::smem_u32(base + kTile);
            float s[8][4];
#pragma unroll
            for (int j = 0; j < 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
#pragma unroll
                for (int jp = 0; jp < 4; ++jp) {  // key n-tiles 2jp, 2jp+1
                    const int mi = lane >> 3, r = lane & 7;
                    const int key = 16 * jp + (mi >> 1) * 8 + r, c = 2 * ks + (mi & 1);
                    uint32_t b00, b01, b10, b11;
                    ldsm_x4(ms::sw_addr<kKT>(kt_s, key, c), b00, b01, b10, b11);
                    mma16816(s[2 * jp], qa[ks], b00, b01);
                    mma16816(s[2 * jp + 1], qa[ks], b10, b11);
                }
            }
            // mask and row maxima (row a = query ta, row b = query tb)
            float mxa = -INFINITY, mxb = -INFINITY;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int k0 = key0 + 8 * j + 2 * tig;
                s[j][0] = k0 <= pa_pos ? s[j][0] * scale : -INFINITY;
                s[j][1] = k0 + 1 <= pa_pos ? s[j][1] * scale : -INFINITY;
                s[j][2] = k0 <= pb_pos ? s[j][2] * scale : -INFINITY;
                s[j][3] = k0 + 1 <= pb_pos ? s[j][3] * scale : -INFINITY;
                mxa = fmaxf(mxa, fmaxf(s[j][0], s[j][1]));
                mxb = fmaxf(mxb, fmaxf(s[j][2], s[j][3]));
            }
            mxa = fmaxf(mxa, __shfl_xor_sync(0xffffffffu, mxa, 1));
            mxa = fmaxf(mxa, __shfl_xor_sync(0xffffffffu, mxa, 2));
            mxb = fmaxf(mxb, __shfl_xor_sync(0xffffffffu, mxb, 1));
            mxb = fmaxf(mxb, __shfl_xor_sync(0xffffffffu, mxb, 2));
            const float na = fmaxf(m_a, mxa), nb = fmaxf(m_b, mxb);
            const float ca = m_a == -INFINITY ? 0.f : exp2f(m_a - na);
            const float cb = m_b == -INFINITY ? 0.f : exp2f(m_b - nb);
            float sa = 0.f, sb = 0.f;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                s[j][0] = na == -INFINITY ? 0.f : exp2f(s[j][0] - na);
                s[j][1] = na == -INFINITY ? 0.f : exp2f(s[j][1] - na);
                s[j][2] = nb == -INFINITY ? 0.f : exp2f(s[j][2] - nb);
                s[j][3] = nb == -INFINITY ? 0.f : exp2f(s[j][3] - nb);
                sa += s[j][0] + s[j][1];
                sb += s[j][2] + s[j][3];
            }
            sa += __shfl_xor_sync(0xffffffffu, sa, 1);
            sa += __shfl_xor_sync(0xffffffffu, sa, 2);
            sb += __shfl_xor_sync(0xffffffffu, sb, 1);
            sb += __shfl_xor_sync(0xffffffffu, sb, 2);
            l_a = l_a * ca + sa;
            l_b = l_b * cb + sb;
            m_a = na;
            m_b = nb;
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                acc[j][0] *= ca;
                acc[j][1] *= ca;
                acc[j][2] *= cb;
                acc[j][3] *= cb;
            }
            // O += P V over 4 k-steps of 16 keys
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
                const uint32_t pa[4] = {pack_bf16(s[2 * kk][0], s[2 * kk][1]),
                                        pack_bf16(s[2 * kk][2], s[2 * kk][3]),
                                        pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]),
                                        pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3])};
#pragma unroll
                for (int jj = 0; jj < 8; ++jj) {
                    const int mi = lane >> 3, r = lane & 7;
                    const int key = 16 * kk + (mi & 1) * 8 + r, c = 2 * jj + (mi >> 1);
                    uint32_t v0, v1, v2, v3;
                    ldsm_x4_t(ms::sw_addr<kKT>(vt_s, key, c), v0, v1, v2, v3);
                    mma16816(acc[2 * jj], pa, v0, v1);
                    mma16816(acc[2 * jj + 1], pa, v2, v3);
                }
            }
        }
        __syncthreads();
        if (threadIdx.x == 0 && n_issued < n_kt) issue(n_issued++);
    }
    if (t_fail >= 0) {
        if (threadIdx.x == 0) {
            atomicOr(status, QK_STATUS_TIMEOUT);
            for (int t = t_fail; t < n_issued; ++t)
                tc::mbar_wait_drain(&full[t % kStages], (uint32_t)((t / kStages) & 1));
        }
        return;
    }
    const float ia = l_a > 0.f ? 1.f / l_a : 0.f, ib = l_b > 0.f ? 1.f / l_b : 0.f;
    bf16* oa = o + ((size_t)b * T + ta) * (size_t)(nq * kD) + (size_t)h * kD;
    bf16* ob = o + ((size_t)b * T + tb) * (size_t)(nq * kD) + (size_t)h * kD;
#pragma unroll
    for (int j = 0; j < 16; ++j) {
        const int c = 8 * j + 2 * tig;
        if (ta < T) *reinterpret_cast<uint32_t*>(oa + c) = pack_bf16(acc[j][0] * ia, acc[j][1] * ia);
        if (tb < T) *reinterpret_cast<uint32_t*>(ob + c) = pack_bf16(acc[j][2] * ib, acc[j][3] * ib);
    }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

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
    if (rows >= ((size_t)1 << 31)) return QK_ESHAPE;
    CUtensorMap map;
    cuuint64_t dims[2] = {(cuuint64_t)kD, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)kD * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)kKT};
    cuuint32_t estr[2] = {1, 1};
    if (((EncodeTiledFn)fn)(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(k_layer),
                            dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return QK_ECUDA;
    dim3 grid((T + kQT - 1) / kQT, B * nq);
    launch_k(attn_prefill_kernel, grid, dim3(128), kSmem, s, map, q, q_ld, nq, nkv, max_batch,
             max_seq, start, start_dev, T, o, status);
    note_launch();
    return QK_OK;
}

}  // namespace qk
