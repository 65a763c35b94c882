// GQA decode attention over the bf16 KV cache, split over the key sequence: the
// kernel (one work item per CTA; the item itself is attn::decode_item,
// attn_decode_core.cuh), its split model and its scratch layout.
#include <cuda.h>

#include "attn_decode_core.cuh"

namespace qk {

namespace {

using attn::kD;
using attn::kTileKeys;
constexpr int kSmem = attn::kRingBytes + 1024 + 256;

// PAGED: the cache is paged (one instance each, so the dense one pays no page lookup)
template <bool PAGED>
__global__ void __launch_bounds__(128)
    attn_decode_kernel(const __grid_constant__ CUtensorMap tmKV, const __grid_constant__ attn::Args a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t* full = (uint64_t*)(smem + attn::kRingBytes);
    volatile int* abort_flag = (volatile int*)(full + attn::kStages);
    int* last_s = (int*)(full + attn::kStages) + 1;

    pdl_wait();
    pdl_trigger();  // the next kernel may launch once every CTA of this grid is resident
    if (threadIdx.x == 0) {
        for (int s = 0; s < attn::kStages; ++s) tc::mbar_init(&full[s], 1);
        *abort_flag = 0;
        tc::fence_mbar_init();
        tc::tma_prefetch_desc(&tmKV);
    }
    __syncthreads();
    int tiles = 0;
    attn::decode_item<PAGED>(a, &tmKV, 0, blockIdx.x, blockIdx.y / a.nkv, blockIdx.y % a.nkv, smem, full,
                             tiles, abort_flag, last_s, threadIdx.x);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

}  // namespace

// Chunking of the key range into whole 64-key tiles.  With two resident CTAs
// per SM, the time is modelled as waves x (tiles per CTA + 1.5 tiles of fixed
// cost: prologue, pipeline fill, partial write and merge); the chunk with the
// lowest cost wins (ties go to the longer chunk).
void attn_decode_split(int B, int nkv, int max_seq, int num_sms, int* chunk, int* n_split) {
    const int pairs = B * nkv;
    const int n_tiles = (max_seq + kTileKeys - 1) / kTileKeys;
    const int slots = 2 * num_sms;
    int best_c = n_tiles;
    double best = 1e30;
    for (int c = n_tiles; c >= 1; --c) {
        const int splits = (n_tiles + c - 1) / c;
        const long ctas = (long)pairs * splits;
        const long waves = (ctas + slots - 1) / slots;
        const double cost = (double)waves * (c + 1.5);
        if (cost < best - 1e-9) {
            best = cost;
            best_c = c;
        }
    }
    *chunk = best_c * kTileKeys;
    *n_split = (n_tiles + best_c - 1) / best_c;
}

// Partials [B nq][n_split][128] fp32, (m, l) [B nq][n_split], then the merge tickets
// [B nkv] (int, must be zero before the first layer of a step: attn_decode_tickets).
size_t attn_decode_scratch_bytes(int B, int nq, int nkv, int max_seq, int num_sms) {
    int chunk, n_split;
    attn_decode_split(B, nkv, max_seq, num_sms, &chunk, &n_split);
    const size_t heads = (size_t)B * nq;
    return heads * n_split * (kD * sizeof(float) + sizeof(float2)) + (size_t)B * nkv * 4 + 256;
}

int* attn_decode_tickets(void* scratch, int B, int nq, int nkv, int max_seq, int num_sms) {
    int chunk, n_split;
    attn_decode_split(B, nkv, max_seq, num_sms, &chunk, &n_split);
    const size_t heads = (size_t)B * nq;
    return (int*)((char*)scratch + heads * n_split * (kD * sizeof(float) + sizeof(float2)));
}

void attn_scratch_parts(void* scratch, int B, int nq, int nkv, int max_seq, int num_sms, int n_split,
                        float** part_o, float2** part_ml, int** tickets) {
    const size_t heads = (size_t)B * nq;
    *part_o = (float*)scratch;
    *part_ml = (float2*)((char*)scratch + heads * n_split * kD * sizeof(float));
    *tickets = attn_decode_tickets(scratch, B, nq, nkv, max_seq, num_sms);
}

// 3-D map over the K / V caches of `layers` layers (layer stride layer_bytes): rows of
// 128 bf16 elements, K rows of a layer first, then its V rows; 64 x 64-row boxes,
// 128-byte swizzle.
bool make_kv_map(CUtensorMap* map, const void* k_layer0, const KvPages& kp, int nkv, int layers,
                 size_t layer_bytes) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult qr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &qr) != cudaSuccess ||
        qr != cudaDriverEntryPointSuccess)
        return false;
    const size_t rows = 2 * (size_t)kp.n_pages * nkv * kp.page;
    if (rows >= ((size_t)1 << 31)) return false;
    if (layers < 1) return false;
    if (layers == 1) layer_bytes = rows * kD * 2;
    cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)rows, (cuuint64_t)layers};
    cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)layer_bytes};
    cuuint32_t box[3] = {64, (cuuint32_t)kTileKeys, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return ((EncodeTiledFn)fn)(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(k_layer0),
                               dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool attn_decode_supported(int d, int nq, int nkv) { return d == kD && nq / nkv <= 8; }

int launch_attn_decode(const bf16* q, int q_ld, const void* k_layer, int nq, int nkv,
                       const KvPages& kp, int B, PosIndex pos, void* scratch,
                       bf16* o, int num_sms, uint32_t* status, cudaStream_t s) {
    static bool attr_set = false;
    if (!attr_set) {
        if (cudaFuncSetAttribute(attn_decode_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kSmem) != cudaSuccess ||
            cudaFuncSetAttribute(attn_decode_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kSmem) != cudaSuccess)
            return QK_ECUDA;
        attr_set = true;
    }
    CUtensorMap map;
    if (kp.table && kp.page % kTileKeys) return QK_ESHAPE;  // a paged tile must not cross a page
    if (!make_kv_map(&map, k_layer, kp, nkv, 1, 0)) return QK_ECUDA;
    attn::Args a;
    a.q = q;
    a.q_ld = q_ld;
    a.nq = nq;
    a.nkv = nkv;
    a.kp = kp;
    a.pos = pos;
    attn_decode_split(B, nkv, kp.cap(), num_sms, &a.chunk, &a.n_split);
    attn_scratch_parts(scratch, B, nq, nkv, kp.cap(), num_sms, a.n_split, &a.part_o, &a.part_ml,
                       &a.tickets);
    a.out = o;
    a.status = status;
    dim3 grid(a.n_split, B * nkv);
    if (kp.table)
        launch_k(attn_decode_kernel<true>, grid, dim3(128), kSmem, s, map, a);
    else
        launch_k(attn_decode_kernel<false>, grid, dim3(128), kSmem, s, map, a);
    note_launch(1);
    return QK_OK;
}

}  // namespace qk
