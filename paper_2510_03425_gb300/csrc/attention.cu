// Causal grouped-query attention of the decoder block: the pieces around the tcgen05 kernels of
// attention_tc.cu and the choice of their launch mode.
//
//   forward : o = softmax(q k^T / sqrt(hd) + mask) v, per (sequence, query head); query head h
//             reads key/value head h / (H/KV); lse = log-sum-exp of each score row.  mask: query i
//             sees key j iff j <= i and, with a sliding window W > 0 (the local layers of Gemma3),
//             i - j < W.  Grids under one wave split each query tile's key blocks over a cluster.
//   backward: dP = dO v^T, dS = P (dP - D) with D = rowsum(dO o) (dvec_kernel below),
//             dq = dS k / sqrt(hd), dk = dS^T q / sqrt(hd), dv = P^T dO, dk and dv summed over the
//             query heads of a group.  Grids that fill the GPU: dK/dV and dQ kernels write dqkv
//             directly.  Smaller grids: split items write fp32 partials to a workspace and
//             bwd_finish_kernel below sums them in a fixed order and applies the inverse RoPE.
//             Deterministic, no atomics.
// q, k, v live in the fused projection buffer [T, (H + 2 KV) hd] (q heads, k heads, v heads);
// token t = b*S + s.
#include "common.cuh"
#include "kernels.h"

namespace mebp {
namespace attn {

// dvec[b, h, s] = sum_d dO[t, h, d] * o[t, h, d]
__global__ void dvec_kernel(const uint16_t* __restrict__ o, const uint16_t* __restrict__ dout, int64_t ldo, int B,
                            int S, int H, int HD, float* __restrict__ dvec) {
  griddep_wait();
  griddep_launch();
  const int64_t w = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (w >= static_cast<int64_t>(B) * S * H) return;
  const int h = static_cast<int>(w % H);
  const int64_t t = w / H;
  const uint32_t* a = reinterpret_cast<const uint32_t*>(o + t * ldo + h * HD);
  const uint32_t* d = reinterpret_cast<const uint32_t*>(dout + t * ldo + h * HD);
  float s = 0.0f;
  for (int i = lane; i < HD / 2; i += 32) {
    const uint32_t x = a[i], y = d[i];
    s += h2_lo(x) * h2_lo(y) + h2_hi(x) * h2_hi(y);
  }
  s = warp_sum(s);
  if (lane == 0) {
    const int64_t b = t / S, sidx = t % S;
    dvec[(b * H + h) * S + sidx] = s;
  }
}

// The split backward's partials: slots of [64 rows][hd] floats, slot ((b * nb + 64-row block) * H
// + query head) * P + part, for dK (already / sqrt(hd)), dV and dQ (/ sqrt(hd)).
struct BwdArgs {
  int S, H, KV, B;
  uint16_t* dqkv;
  int64_t ld;
  int P;
  float *wk, *wv, *wq;
};

// dqkv from the split partials: dQ = sum over parts; dK, dV = sum over the group's query heads and
// parts (fixed order); q and k then rotated back by their RoPE angle when cs != null (the VJP of
// the rotation: (d1, d2) -> (d1 c + d2 s, d2 c - d1 s)).  One thread per (token, head slot, pair j).
constexpr int kFinishMax = 16;  // partials per element: query heads per kv head (<= 8) x parts (<= 2)
template <int HD>
__global__ void bwd_finish_kernel(const BwdArgs a, const float2* __restrict__ cs) {
  griddep_wait();
  griddep_launch();
  constexpr int HALF = HD / 2;
  const int H = a.H, KV = a.KV, S = a.S, P = a.P, nh = H + 2 * KV, grp = H / KV;
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  const int64_t T = static_cast<int64_t>(a.B) * S;
  if (i >= T * nh * HALF) return;
  const int j = static_cast<int>(i % HALF);
  const int64_t r1 = i / HALF;
  const int slot_h = static_cast<int>(r1 % nh);
  const int64_t t = r1 / nh;
  const int b = static_cast<int>(t / S), pos = static_cast<int>(t % S);
  const int blk = pos / 64, row = pos % 64, nb = (S + 63) / 64;
  const float* base;
  int h0, hn;
  if (slot_h < H) {
    base = a.wq; h0 = slot_h; hn = 1;
  } else if (slot_h < H + KV) {
    base = a.wk; h0 = (slot_h - H) * grp; hn = grp;
  } else {
    base = a.wv; h0 = (slot_h - H - KV) * grp; hn = grp;
  }
  // all loads first (up to kFinishMax independent L2 reads in flight), then the sums in
  // (head, part) order
  const int n = hn * P;
  const float* pp0 = base + ((static_cast<int64_t>(b) * nb + blk) * H + h0) * P * (64 * HD) + row * HD + j;
  float v1[kFinishMax], v2[kFinishMax];
#pragma unroll
  for (int k = 0; k < kFinishMax; ++k) {
    v1[k] = k < n ? __ldcg(pp0 + static_cast<int64_t>(k) * (64 * HD)) : 0.0f;
    v2[k] = k < n ? __ldcg(pp0 + static_cast<int64_t>(k) * (64 * HD) + HALF) : 0.0f;
  }
  float x1 = 0.0f, x2 = 0.0f;
#pragma unroll
  for (int k = 0; k < kFinishMax; ++k) {
    x1 += v1[k];
    x2 += v2[k];
  }
  if (cs && slot_h < H + KV) {
    const float2 c = cs[static_cast<int64_t>(pos) * HALF + j];
    const float y1 = x1 * c.x + x2 * c.y, y2 = x2 * c.x - x1 * c.y;
    x1 = y1;
    x2 = y2;
  }
  uint16_t* dst = a.dqkv + t * a.ld + static_cast<int64_t>(slot_h) * HD;
  dst[j] = f_to_h(x1);
  dst[j + HALF] = f_to_h(x2);
}

}  // namespace attn

int launch_attn_fwd(const uint16_t* qkv, int64_t ld, int B, int S, int H, int KV, int hd, uint16_t* o, int64_t ldo,
                    float* lse, int window, int* err, cudaStream_t st) {
  return launch_attn_fwd_tc(qkv, ld, B, S, H, KV, hd, o, ldo, lse, window, err, st);
}

bool launch_attn_bwd(const uint16_t* qkv, int64_t ld, const uint16_t* o, const uint16_t* dout, int64_t ldo,
                     const float* lse, int B, int S, int H, int KV, int hd, float* dvec, uint16_t* dqkv, int window,
                     const float2* rope_cs, float* ws, int64_t ws_floats, int* err, cudaStream_t st) {
  const int64_t nw = static_cast<int64_t>(B) * S * H;
  launch_k(attn::dvec_kernel, static_cast<unsigned>((nw * 32 + 255) / 256), 256, 0, st, o, dout, ldo, B, S, H, hd,
           dvec);
  // Direct mode when the dK/dV grid (128-key blocks x kv heads x sequences x column halves at
  // hd 256) fills the GPU (Gemma3-4B shape: 1024 CTAs).  Below that each of its CTAs would loop
  // over every query head of its group and every query block, so the work is split into
  // (query head, part) items instead, summed by the finish kernel.
  const int64_t kv_tiles = static_cast<int64_t>((S + 127) / 128) * KV * B * (hd == 256 ? 2 : 1);
  // query blocks of a head split in P parts: two at hd 64 / 128, one at hd 256 (measured per
  // step: Gemma3-1B shape, hd 256, 1024 tokens, 13.19 ms with one part, 13.56 with two;
  // Qwen2.5-0.5B shape, hd 64, 512 tokens, 5.44 with two, 5.48 with one)
  const int P = hd == 256 ? 1 : 2;
  const int nb = (S + 63) / 64;
  const int64_t part_floats = static_cast<int64_t>(B) * nb * H * P * 64 * hd;  // per array
  if (kv_tiles < 152 && ws && 3 * part_floats <= ws_floats && (H / KV) * P <= attn::kFinishMax) {
    launch_attn_bwd_tc(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, hd, dqkv, window, P, ws, ws + part_floats,
                       ws + 2 * part_floats, err, st);
    const attn::BwdArgs a{S, H, KV, B, dqkv, ld, P, ws, ws + part_floats, ws + 2 * part_floats};
    const int64_t n = static_cast<int64_t>(B) * S * (H + 2 * KV) * (hd / 2);
    const unsigned grid = static_cast<unsigned>((n + 255) / 256);
    if (hd == 64) launch_k(attn::bwd_finish_kernel<64>, grid, 256, 0, st, a, rope_cs);
    else if (hd == 128) launch_k(attn::bwd_finish_kernel<128>, grid, 256, 0, st, a, rope_cs);
    else launch_k(attn::bwd_finish_kernel<256>, grid, 256, 0, st, a, rope_cs);
    return true;  // the finish kernel applied the inverse RoPE (when rope_cs != null)
  }
  launch_attn_bwd_tc(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, hd, dqkv, window, 0, nullptr, nullptr, nullptr, err,
                     st);
  return false;  // the caller applies the inverse RoPE
}

}  // namespace mebp
