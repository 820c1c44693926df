// Compression (quantise + pack), debug decode and embedding gather-dequant kernels.
#include "dequant.cuh"
#include "kernels.h"

namespace mebp {

// One warp per (row, group of 64 columns).  Lane l writes byte l of the group: byte p of word
// w = l/4 packs columns (c_lo, c_hi) = 8w + {(0,2), (4,6), (1,3), (5,7)}[p] as
// (u_lo | u_hi << 4), the word layout of dequant.cuh.
// s = fp16_satfinite_rne(amax / 7) (IEEE fp32 division), q = clamp(rint(w / s), -7, 7), q = 0
// when s == 0, u = q + 8.
__global__ void compress_kernel(const float* __restrict__ W, int64_t rows, int64_t cols,
                                uint8_t* __restrict__ qpack, uint16_t* __restrict__ scales) {
  griddep_wait();
  griddep_launch();
  const int64_t groups = cols / 64;
  const int64_t gw = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (gw >= rows * groups) return;
  const int64_t r = gw / groups, g = gw % groups;
  const float* grp = W + r * cols + g * 64;
  const float2 pairv = reinterpret_cast<const float2*>(grp)[lane];  // columns 2l, 2l+1 for the max
  const float amax = warp_max(fmaxf(fabsf(pairv.x), fabsf(pairv.y)));
  const int wi = lane >> 2, pos = lane & 3;
  const int c_lo = 8 * wi + ((pos & 1) ? 4 : 0) + ((pos & 2) ? 1 : 0);
  const float2 w = make_float2(grp[c_lo], grp[c_lo + 2]);
  const float sq = __fdiv_rn(amax, 7.0f);
  uint16_t sbits;
  asm("cvt.rn.satfinite.f16.f32 %0, %1;" : "=h"(sbits) : "f"(sq));
  const float s = __half2float(__ushort_as_half(sbits));
  int q0 = 0, q1 = 0;
  if (s != 0.0f) {
    q0 = static_cast<int>(fminf(fmaxf(rintf(__fdiv_rn(w.x, s)), -7.0f), 7.0f));
    q1 = static_cast<int>(fminf(fmaxf(rintf(__fdiv_rn(w.y, s)), -7.0f), 7.0f));
  }
  qpack[r * (cols / 2) + g * 32 + lane] = static_cast<uint8_t>((q0 + 8) | ((q1 + 8) << 4));
  if (lane == 0) scales[g * rows + r] = sbits;
}

// Decode every 8-column word with the GEMM's operand transform.
__global__ void decode_kernel(const uint8_t* __restrict__ qpack, const uint16_t* __restrict__ scales, int64_t rows,
                              int64_t cols, uint16_t* __restrict__ out) {
  griddep_wait();
  griddep_launch();
  const int64_t words_per_row = cols / 8;
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= rows * words_per_row) return;
  const int64_t r = i / words_per_row, j = i % words_per_row;
  const uint32_t w = reinterpret_cast<const uint32_t*>(qpack + r * (cols / 2))[j];
  uint32_t o[4];
  dequant_word(w, scale_pair(scales[(j / 8) * rows + r]), o);
  reinterpret_cast<uint4*>(out + r * cols)[j] = make_uint4(o[0], o[1], o[2], o[3]);
}

// x0[t, :] = scale * deq(E)[ids[t], :] in fp32 (exact for scale 1).  One warp per token, 8 elements
// per lane-step.
__global__ void embed_kernel(const uint8_t* __restrict__ qpack, const uint16_t* __restrict__ scales, int64_t V,
                             int64_t D, const int32_t* __restrict__ ids, int64_t T, float* __restrict__ x0,
                             int* err, float scale) {
  griddep_wait();
  griddep_launch();
  const int64_t t = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (t >= T) return;
  const int32_t id = ids[t];
  float* dst = x0 + t * D;
  if (id < 0 || id >= V) {
    for (int64_t k = lane * 4; k < D; k += 128) *reinterpret_cast<float4*>(dst + k) = make_float4(0, 0, 0, 0);
    if (lane == 0) flag_error(err, kErrDevice);
    return;
  }
  const uint32_t* row = reinterpret_cast<const uint32_t*>(qpack + static_cast<int64_t>(id) * (D / 2));
  for (int64_t j = lane; j < D / 8; j += 32) {
    const uint32_t w = row[j];
    const float s = __half2float(__ushort_as_half(scales[(j / 8) * V + id]));
    float v[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = dequant_f32(word_nibble(w, e), s) * scale;
    reinterpret_cast<float4*>(dst + j * 8)[0] = make_float4(v[0], v[1], v[2], v[3]);
    reinterpret_cast<float4*>(dst + j * 8)[1] = make_float4(v[4], v[5], v[6], v[7]);
  }
}

void launch_compress(const float* W, int64_t rows, int64_t cols, uint8_t* qpack, uint16_t* scales, cudaStream_t st) {
  const int64_t warps = rows * (cols / 64);
  const int64_t blocks = (warps * 32 + 255) / 256;
  launch_k(compress_kernel, static_cast<unsigned>(blocks), 256, 0, st, W, rows, cols, qpack, scales);
}

void launch_decode(const uint8_t* qpack, const uint16_t* scales, int64_t rows, int64_t cols, uint16_t* out,
                   cudaStream_t st) {
  const int64_t n = rows * (cols / 8);
  launch_k(decode_kernel, static_cast<unsigned>((n + 255) / 256), 256, 0, st, qpack, scales, rows, cols, out);
}

void launch_embed(const uint8_t* qpack, const uint16_t* scales, int64_t V, int64_t D, const int32_t* ids, int64_t T,
                  float* x0, int* err, float scale, cudaStream_t st) {
  const int64_t blocks = (T * 32 + 255) / 256;
  launch_k(embed_kernel, static_cast<unsigned>(blocks), 256, 0, st, qpack, scales, V, D, ids, T, x0, err, scale);
}

}  // namespace mebp
