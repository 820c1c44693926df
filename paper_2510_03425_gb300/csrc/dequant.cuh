// Just-in-time decode of the 4-bit weight format into fp16 tensor-core operands.
//
// Format (Section 3, "Base model weights compression", read as symmetric INT4 with group 64
// and fp16 scales): element k of a row sits in nibble k of the row's packed bytes
// (low nibble = even k) as u = q + 8; deq = q * s, s = fp16 scale of the group.
//
// The operand must equal fp16_rne(q * s) bit for bit.  q * s is exact in fp32 (4-bit integer
// times an 11-bit significand), so one correctly rounded FMA that reaches it exactly and one
// RNE conversion give that value:
//   m   = float_from_bits(0x3F800000 | (u << p)) = 1 + u * 2^(p-23)     (exact, p in {8,12,16})
//   S_p = s * 2^(23-p),  C_p = -s * (2^(23-p) + 8)                      (both exact in fp32)
//   fma(m, S_p, C_p) = s * 2^(23-p) + u*s - s * 2^(23-p) - 8s = (u - 8) s  (exact -> no rounding)
// C_p is exact because 2^(23-p) + 8 has at most 13 significant bits for p >= 8 and s has 11.
// Each nibble is moved into bit position 8, 12 or 16 with at most one shift per word.
#pragma once
#include "common.cuh"

namespace mebp {

struct DeqConsts {
  float s8, c8, s12, c12, s16, c16;
};

MEBP_DEV DeqConsts deq_consts(float s) {
  DeqConsts c;
  c.s8 = s * 32768.0f;
  c.c8 = -(s * 32776.0f);
  c.s12 = s * 2048.0f;
  c.c12 = -(s * 2056.0f);
  c.s16 = s * 128.0f;
  c.c16 = -(s * 136.0f);
  return c;
}

MEBP_DEV float magic_nib(uint32_t w, uint32_t mask) { return __uint_as_float((w & mask) | 0x3F800000u); }

// 8 nibbles of `w` (element i at bits 4i..4i+3) -> 4 fp16x2 words, element 2i in the low half
// of out[i].
MEBP_DEV void dequant_word(uint32_t w, const DeqConsts& c, uint32_t (&out)[4]) {
  const uint32_t y = w << 8;   // nibbles 0,1 -> bits 8..11, 12..15
  const uint32_t z = w >> 12;  // nibbles 5,6,7 -> bits 8..11, 12..15, 16..19
  const float v0 = __fmaf_rn(magic_nib(y, 0x00000F00u), c.s8, c.c8);
  const float v1 = __fmaf_rn(magic_nib(y, 0x0000F000u), c.s12, c.c12);
  const float v2 = __fmaf_rn(magic_nib(w, 0x00000F00u), c.s8, c.c8);
  const float v3 = __fmaf_rn(magic_nib(w, 0x0000F000u), c.s12, c.c12);
  const float v4 = __fmaf_rn(magic_nib(w, 0x000F0000u), c.s16, c.c16);
  const float v5 = __fmaf_rn(magic_nib(z, 0x00000F00u), c.s8, c.c8);
  const float v6 = __fmaf_rn(magic_nib(z, 0x0000F000u), c.s12, c.c12);
  const float v7 = __fmaf_rn(magic_nib(z, 0x000F0000u), c.s16, c.c16);
  out[0] = pack_half2(v0, v1);
  out[1] = pack_half2(v2, v3);
  out[2] = pack_half2(v4, v5);
  out[3] = pack_half2(v6, v7);
}

// fp32 value of one element (used where the exact fp32 value is wanted, e.g. the embedding).
MEBP_DEV float dequant_f32(uint32_t u, float s) { return static_cast<float>(static_cast<int>(u) - 8) * s; }

}  // namespace mebp
