// Warp-level tensor-core helpers shared by the attention kernels: mma.sync
// m16n8k16 (bf16 in, fp32 accumulate), ldmatrix (plain and transposed), bf16
// packing, and addressing of K/V tiles that TMA wrote as two 64-column boxes
// of 128-byte-swizzled rows.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

namespace qk {
namespace ms {

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

// D[16x8] += A[16x16] (row-major fragment a0..a3) * B[16x8] (column fragment b0, b1).
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
        "{%8, %9}, {%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// A tile of `rows` 128-element bf16 rows stored by TMA as two boxes of 64 columns
// (box 0: columns 0..63, box 1: 64..127), each row 128 bytes with 128-byte
// swizzling.  Address of (row, 16-byte chunk c in 0..15); the tile base is
// 1024-byte aligned.
template <int ROWS>
__device__ __forceinline__ uint32_t sw_addr(uint32_t tile, int row, int c) {
    return tile + (uint32_t)((c >> 3) * (ROWS * 128) + row * 128 + (((c & 7) ^ (row & 7)) << 4));
}

}  // namespace ms
}  // namespace qk
