// Warp-level fp16 tensor-core fragments (mma.sync m16n8k16) and cp.async helpers for the
// small contractions (LoRA down-projections, LoRA gradient reductions, attention tiles).
#pragma once
#include "common.cuh"

namespace mebp {

MEBP_DEV void ldsm_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
MEBP_DEV void ldsm_x4_t(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
// d += a * b  (A 16x16 row-major, B 16x8 "col", fp32 accumulate)
MEBP_DEV void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Lane address of an A fragment (rows r0..r0+15, k0..k0+15) from a row-major [row][k] tile.
MEBP_DEV uint32_t frag_a_addr(uint32_t base, int ld, int r0, int k0, int lane) {
  return base + 2u * static_cast<uint32_t>((r0 + (lane & 15)) * ld + k0 + ((lane >> 4) << 3));
}
// Lane address of an A fragment from a k-major [k][row] tile (use with ldsm_x4_t).
MEBP_DEV uint32_t frag_at_addr(uint32_t base, int ld, int r0, int k0, int lane) {
  return base + 2u * static_cast<uint32_t>((k0 + (lane & 7) + ((lane >> 4) << 3)) * ld + r0 + (((lane >> 3) & 1) << 3));
}
// Lane address of the B fragments of two n-tiles (n0..n0+15) from an [n][k] tile (ldsm_x4):
// r[0], r[1] = tile n0; r[2], r[3] = tile n0+8.
MEBP_DEV uint32_t frag_bn_addr(uint32_t base, int ld, int n0, int k0, int lane) {
  return base + 2u * static_cast<uint32_t>((n0 + (lane & 7) + ((lane >> 4) << 3)) * ld + k0 + (((lane >> 3) & 1) << 3));
}
// Lane address of the B fragments of two n-tiles from a [k][n] tile (ldsm_x4_t).
MEBP_DEV uint32_t frag_bk_addr(uint32_t base, int ld, int n0, int k0, int lane) {
  return base + 2u * static_cast<uint32_t>((k0 + (lane & 7) + (((lane >> 3) & 1) << 3)) * ld + n0 + ((lane >> 4) << 3));
}

MEBP_DEV void cp_async16(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(valid ? 16 : 0) : "memory");
}
MEBP_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
MEBP_DEV void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

}  // namespace mebp
