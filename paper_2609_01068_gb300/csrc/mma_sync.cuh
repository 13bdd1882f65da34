// Warp-level bf16 MMA (m16n8k16) and ldmatrix helpers for the attention kernels,
// plus the address of an element inside a TMA tile written with 128-byte
// swizzling (boxes of 64 bf16 columns, 1024-byte aligned).
#pragma once

#include "common.cuh"

namespace outlets {

OUTLETS_DEV void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}
OUTLETS_DEV void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}
// d += a * b, a: 16x16 bf16 (row), b: 16x8 bf16 (col), d: 16x8 f32
OUTLETS_DEV void mma_16816(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Byte offset of (row r, column d) in a tile made of 64-column boxes stacked
// along columns (box b holds columns [64b, 64b + 64), rows * 128 bytes each).
template <int ROWS>
OUTLETS_DEV uint32_t sw128_offset(int r, int d) {
  return static_cast<uint32_t>((d >> 6) * (ROWS * 128) + r * 128 + ((((d >> 3) & 7) ^ (r & 7)) << 4) +
                               (d & 7) * 2);
}

}  // namespace outlets
