// Just-in-time decode of the 4-bit weight format into fp16 tensor-core operands.
//
// Format (Section 3, "Base model weights compression", read as symmetric INT4 with group 64
// and fp16 scales): u = q + 8 (offset binary).  Each run of 8 consecutive columns of a row is
// one little-endian 32-bit word: column 8w + 2j in bits 4j..4j+3 (low half-word), column
// 8w + 2j + 1 in bits 16 + 4j..16 + 4j + 3 (high half-word), j = 0..3.
//
// The operand must equal fp16_rne(q * s) bit for bit.  With that word order one mask selects
// an (even, odd) column pair already in operand order:
//   t   = ((w >> 4j) & 0x000F000F) | 0x64006400    fp16 pair (1024 + u_2j, 1024 + u_2j+1), exact
//   q   = t - (1032, 1032)                          exact small integers
//   out = q * (s, s)                                one IEEE fp16 multiplication = fp16_rne(q * s)
// i.e. 1 shift, 1 LOP3 and 2 half2 FP ops per two elements, and the scale is used as the
// fp16 bits it is stored in.  (The OR-into-the-mantissa conversion of small integers to fp16 is
// the published "magic number" method of Kim et al., 2022, "Who Says Elephants Can't Run".)
#pragma once
#include "common.cuh"

namespace mebp {

// (s, s) as an fp16x2 register from the stored scale bits.
MEBP_DEV uint32_t scale_pair(uint16_t s_bits) { return static_cast<uint32_t>(s_bits) * 0x00010001u; }

MEBP_DEV uint32_t hsub2_u32(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
MEBP_DEV uint32_t hmul2_u32(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// 8 nibbles of `w` -> 4 fp16x2 words: out[j] = (column 2j, column 2j+1) of the 8-column run.
MEBP_DEV void dequant_word(uint32_t w, uint32_t s2, uint32_t (&out)[4]) {
  constexpr uint32_t kMask = 0x000F000Fu, kMagic = 0x64006400u, kBias = 0x64086408u;  // 1024, 1032
  out[0] = hmul2_u32(hsub2_u32((w & kMask) | kMagic, kBias), s2);
  out[1] = hmul2_u32(hsub2_u32(((w >> 4) & kMask) | kMagic, kBias), s2);
  out[2] = hmul2_u32(hsub2_u32(((w >> 8) & kMask) | kMagic, kBias), s2);
  out[3] = hmul2_u32(hsub2_u32(((w >> 12) & kMask) | kMagic, kBias), s2);
}

// Nibble of column e (0..7) of a word, per the layout above.
MEBP_DEV uint32_t word_nibble(uint32_t w, int e) { return (w >> ((e & 1) * 16 + (e >> 1) * 4)) & 0xFu; }

// fp32 value of one element (the exact q * s, used by the embedding gather).
MEBP_DEV float dequant_f32(uint32_t u, float s) { return static_cast<float>(static_cast<int>(u) - 8) * s; }

}  // namespace mebp
