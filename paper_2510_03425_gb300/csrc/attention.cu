// Causal grouped-query attention of the decoder block, forward and backward, as tiled
// warp-level tensor-core kernels (mma.sync m16n8k16, fp16 in / fp32 accumulate).
//
//   forward : o = softmax(q k^T / sqrt(hd) + mask) v, per (sequence, query head); query head h
//             reads key/value head h / (H/KV).  Saves lse = log-sum-exp of each score row.
//             mask: query i sees key j iff j <= i and, with a sliding window W > 0 (the local
//             layers of Gemma3), i - j < W; key blocks wholly outside the window are skipped.
//   backward: dP = dO v^T, dS = P (dP - rowsum(dO o)), dq = dS k / sqrt(hd),
//             dk = dS^T q / sqrt(hd), dv = P^T dO; dk, dv summed over the query heads of a
//             group.  P is recomputed from q, k and lse.  Large grids: dk/dv items (key block,
//             kv head, looping over the group's query heads) and dq items (query block, head)
//             write dqkv directly.  Small grids: dk/dv items per query head and dq items, each
//             cut into interleaved parts, write fp32 partials; a finish kernel sums them in a
//             fixed order (and applies the inverse RoPE).  Deterministic, no atomics.
// q, k, v live in the fused projection buffer [T, (H + 2 KV) hd] (q heads, k heads, v heads);
// token t = b*S + s.
#include "kernels.h"
#include "mma.cuh"

namespace mebp {
namespace attn {

constexpr int BQ = 64, BKV = 64;
constexpr float kLog2e = 1.4426950408889634f;

// 64 rows x HD columns into shared memory (row pitch HD + 8), NT threads cooperating; rows past S
// are zero-filled.
template <int HD, int NT = 128>
__device__ __forceinline__ void load_tile(uint16_t* dst, const uint16_t* base, int64_t ld, int64_t tok0, int r0,
                                          int S, int col, int tid) {
  constexpr int LD = HD + 8, CH = HD / 8;
  for (int c = tid; c < 64 * CH; c += NT) {
    const int r = c / CH, cc = c % CH;
    const bool v = r0 + r < S;
    const uint16_t* src = v ? base + (tok0 + r0 + r) * ld + col + cc * 8 : base;
    cp_async16(smem_u32(dst + r * LD + cc * 8), src, v);
  }
}

// S (16 rows of this warp x 64 columns) = A_rows . B_rows^T over HD, both row-major [row][d] in smem.
template <int HD>
__device__ __forceinline__ void qk_tile(float (&s)[8][4], uint32_t abase, uint32_t bbase, int warp, int lane) {
  constexpr int LD = HD + 8;
#pragma unroll
  for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.0f;
#pragma unroll
  for (int kk = 0; kk < HD; kk += 16) {
    uint32_t a[4];
    ldsm_x4(a, frag_a_addr(abase, LD, warp * 16, kk, lane));
#pragma unroll
    for (int nt = 0; nt < 8; nt += 2) {
      uint32_t b[4];
      ldsm_x4(b, frag_bn_addr(bbase, LD, nt * 8, kk, lane));
      mma16816(s[nt], a, b[0], b[1]);
      mma16816(s[nt + 1], a, b[2], b[3]);
    }
  }
}

// acc (16 x NC*8) += P (16 x 64, accumulator layout) . B[64][d0 .. d0 + NC*8) with B row-major [k][d].
template <int HD, int NC>
__device__ __forceinline__ void pv_tile(float (&acc)[NC][4], const float (&p)[8][4], uint32_t bbase, int d0,
                                        int lane) {
  constexpr int LD = HD + 8;
#pragma unroll
  for (int kq = 0; kq < 4; ++kq) {
    uint32_t a[4];
    a[0] = pack_half2(p[2 * kq][0], p[2 * kq][1]);
    a[1] = pack_half2(p[2 * kq][2], p[2 * kq][3]);
    a[2] = pack_half2(p[2 * kq + 1][0], p[2 * kq + 1][1]);
    a[3] = pack_half2(p[2 * kq + 1][2], p[2 * kq + 1][3]);
#pragma unroll
    for (int dt = 0; dt < NC; dt += 2) {
      uint32_t b[4];
      ldsm_x4_t(b, frag_bk_addr(bbase, LD, d0 + dt * 8, kq * 16, lane));
      mma16816(acc[dt], a, b[0], b[1]);
      mma16816(acc[dt + 1], a, b[2], b[3]);
    }
  }
}

// ------------------------------------------------------------------------------------ forward
// One CTA per (query block of 64 rows, head, sequence) with NWG warp-groups of four warps (warp r
// of a group owns query rows 16 r .. 16 r + 15).  Warp-group g takes key blocks kb_first + g,
// kb_first + g + NWG, ... with its own online softmax, and the groups' (max, sum, o) are merged
// through shared memory at the end: NWG = 2 on grids of less than one CTA per SM doubles the warps
// per scheduler and halves the serial key-block steps of the longest query block.  NB key/value
// buffers per group: 2 overlaps the next round's loads with this one; 1 saves shared memory.
// WIN: sliding-window layer (window W); key blocks wholly before the window are skipped.  (Masking
// only the blocks a mask cuts measured slower than masking every block.)
// C = 2: a query block's key blocks are shared by a cluster of two CTAs (grid.x = query blocks x 2,
// rank = blockIdx.x % 2), key block i of the list going to group i % NWG of CTA (i / NWG) % 2; each
// CTA merges its groups, then CTA r merges rows 32 r .. 32 r + 31 of both CTAs' (max, sum, o)
// through distributed shared memory.  For grids whose doubled size still fits one CTA per SM.
template <int HD, int NB, bool WIN, int NWG, int C = 1>
__global__ void __launch_bounds__(128 * NWG, 1) fwd_kernel(const uint16_t* __restrict__ qkv, int64_t ld, int S,
                                                           int H, int KV, uint16_t* __restrict__ o, int64_t ldo,
                                                           float* __restrict__ lse, int W) {
  griddep_wait();
  griddep_launch();
  constexpr int LD = HD + 8, NO = HD / 8, NT = 128 * NWG, TILE = BQ * LD;
  extern __shared__ __align__(16) uint16_t sm[];
  uint16_t* qs = sm;  // then per buffer slot and group: K, V
  auto ks = [&](int buf, int g) { return qs + (1 + 2 * (buf * NWG + g)) * TILE; };
  auto vs = [&](int buf, int g) { return qs + (2 + 2 * (buf * NWG + g)) * TILE; };
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int wg = warp >> 2, wr = warp & 3;
  // C = 1: grid (H, B, query blocks), the longest (last) query blocks launched first;
  // C > 1: grid (query blocks x C, H, B), a cluster's CTAs adjacent in x
  const int crank = C > 1 ? static_cast<int>(blockIdx.x) % C : 0;
  const int qb = C > 1 ? static_cast<int>(blockIdx.x) / C : static_cast<int>(gridDim.z - 1 - blockIdx.z);
  const int h = C > 1 ? blockIdx.y : blockIdx.x, b = C > 1 ? blockIdx.z : blockIdx.y;
  const int kvh = h / (H / KV);
  const int64_t tok0 = static_cast<int64_t>(b) * S;
  const int q0 = qb * BQ;
  const float sc = kLog2e * rsqrtf(static_cast<float>(HD));
  // visible key blocks: kb_first .. qb (window: from the first block inside it)
  const int kb_first = WIN ? max(0, q0 - W + 1) / BKV : 0;
  const int nrounds = (qb - kb_first + C * NWG) / (C * NWG);
  // key block of group g of this CTA in round t
  auto kb_of = [&](int t, int g) { return kb_first + (t * C + crank) * NWG + g; };
  auto fetch = [&](int t, int buf) {  // the key/value blocks of round t, one per group
#pragma unroll
    for (int g = 0; g < NWG; ++g) {
      const int kb = kb_of(t, g);
      if (kb > qb) break;
      load_tile<HD, NT>(ks(buf, g), qkv, ld, tok0, kb * BKV, S, (H + kvh) * HD, tid);
      load_tile<HD, NT>(vs(buf, g), qkv, ld, tok0, kb * BKV, S, (H + KV + kvh) * HD, tid);
    }
  };
  load_tile<HD, NT>(qs, qkv, ld, tok0, q0, S, h * HD, tid);
  if (NB == 2) fetch(0, 0);
  cp_async_commit();

  float oacc[NO][4];
#pragma unroll
  for (int i = 0; i < NO; ++i) oacc[i][0] = oacc[i][1] = oacc[i][2] = oacc[i][3] = 0.0f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.0f, 0.0f};
  const int ra = q0 + wr * 16 + (lane >> 2);

  for (int t = 0; t < nrounds; ++t) {
    const int buf = NB == 2 ? t & 1 : 0;
    if (NB == 1) {
      fetch(t, 0);
      cp_async_commit();
      cp_async_wait<0>();
    } else if (t + 1 < nrounds) {
      fetch(t + 1, buf ^ 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const int kb = kb_of(t, wg);
    if (kb <= qb) {  // uniform over the warp-group
      const int k0 = kb * BKV;
      float s[8][4];
      qk_tile<HD>(s, smem_u32(qs), smem_u32(ks(buf, wg)), wr, lane);
#pragma unroll
      for (int nt = 0; nt < 8; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int col = k0 + nt * 8 + 2 * (lane & 3) + (e & 1);
          const int row = ra + ((e >> 1) << 3);
          s[nt][e] = (col > row || col >= S || (WIN && row - col >= W)) ? -INFINITY : s[nt][e] * sc;
        }
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        float mx = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) mx = fmaxf(mx, fmaxf(s[nt][2 * i], s[nt][2 * i + 1]));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        const float mnew = fmaxf(mrow[i], mx);
        const float alpha = (mnew == -INFINITY) ? 1.0f : exp2f(mrow[i] - mnew);
        float rs = 0.0f;
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
          const float p0 = (mnew == -INFINITY) ? 0.0f : exp2f(s[nt][2 * i] - mnew);
          const float p1 = (mnew == -INFINITY) ? 0.0f : exp2f(s[nt][2 * i + 1] - mnew);
          s[nt][2 * i] = p0;
          s[nt][2 * i + 1] = p1;
          rs += p0 + p1;
        }
        rs += __shfl_xor_sync(0xffffffffu, rs, 1);
        rs += __shfl_xor_sync(0xffffffffu, rs, 2);
        lrow[i] = lrow[i] * alpha + rs;
        mrow[i] = mnew;
#pragma unroll
        for (int dt = 0; dt < NO; ++dt) {
          oacc[dt][2 * i] *= alpha;
          oacc[dt][2 * i + 1] *= alpha;
        }
      }
      pv_tile<HD, NO>(oacc, s, smem_u32(vs(buf, wg)), 0, lane);
    }
    __syncthreads();  // every warp is done with this slot before it is refilled
  }

  const int c = 2 * (lane & 3);
  if constexpr (NWG > 1) {
    // groups 1 .. NWG-1 park (o, m, l) in the idle tile buffers; group 0 merges them in group
    // order and writes
    constexpr int LDO = HD + 4, PART = 64 * LDO + 128;  // floats per parked group
    static_assert((NWG - 1) * PART * 4 <= (1 + 2 * NB * NWG) * TILE * 2, "merge buffers fit");
    float* park = reinterpret_cast<float*>(sm);
    if (wg > 0) {
      float* op = park + (wg - 1) * PART;
      float2* ml = reinterpret_cast<float2*>(op + 64 * LDO);
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const int rl = wr * 16 + (lane >> 2) + 8 * i;
#pragma unroll
        for (int dt = 0; dt < NO; ++dt)
          *reinterpret_cast<float2*>(op + rl * LDO + dt * 8 + c) = make_float2(oacc[dt][2 * i], oacc[dt][2 * i + 1]);
        if ((lane & 3) == 0) ml[rl] = make_float2(mrow[i], lrow[i]);
      }
    }
    __syncthreads();
    if (C == 1 && wg > 0) return;  // (with a cluster every thread stays for its barriers)
#pragma unroll
    for (int g = 1; g < NWG; ++g) {
      if (wg > 0) break;
      const float* op = park + (g - 1) * PART;
      const float2* ml = reinterpret_cast<const float2*>(op + 64 * LDO);
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const int rl = wr * 16 + (lane >> 2) + 8 * i;
        const float2 p = ml[rl];
        const float M = fmaxf(mrow[i], p.x);
        const float a0 = mrow[i] == -INFINITY ? 0.0f : exp2f(mrow[i] - M);
        const float a1 = p.x == -INFINITY ? 0.0f : exp2f(p.x - M);
        lrow[i] = a0 * lrow[i] + a1 * p.y;
        mrow[i] = M;
#pragma unroll
        for (int dt = 0; dt < NO; ++dt) {
          const float2 q = *reinterpret_cast<const float2*>(op + rl * LDO + dt * 8 + c);
          oacc[dt][2 * i] = a0 * oacc[dt][2 * i] + a1 * q.x;
          oacc[dt][2 * i + 1] = a0 * oacc[dt][2 * i + 1] + a1 * q.y;
        }
      }
    }
  }
  if constexpr (C > 1) {
    // group 0 of each CTA parks the CTA's (o, m, l) in its own shared memory; CTA r then merges
    // rows r * 64/C .. of all C CTAs through distributed shared memory in rank order
    constexpr int LDO = HD + 4, RPC = 64 / C, C4 = HD / 4;
    static_assert(64 * LDO * 4 + 64 * 16 <= (1 + 2 * NB * NWG) * TILE * 2, "cluster merge buffers fit");
    __syncthreads();  // the group merge has read the parked groups
    float* op = reinterpret_cast<float*>(sm);
    float4* ml = reinterpret_cast<float4*>(op + 64 * LDO);
    if (wg == 0) {
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const int rl = wr * 16 + (lane >> 2) + 8 * i;
#pragma unroll
        for (int dt = 0; dt < NO; ++dt)
          *reinterpret_cast<float2*>(op + rl * LDO + dt * 8 + c) = make_float2(oacc[dt][2 * i], oacc[dt][2 * i + 1]);
        if ((lane & 3) == 0) ml[rl] = make_float4(mrow[i], lrow[i], 0.0f, 0.0f);
      }
    }
    cluster_sync_all();
    const uint32_t op_u = smem_u32(op), ml_u = smem_u32(ml);
    for (int e = tid; e < RPC * C4; e += NT) {
      const int rl = crank * RPC + e / C4, cc = (e % C4) * 4;
      const int row = q0 + rl;
      float mj[C], lj[C];
      float M = -INFINITY;
#pragma unroll
      for (int j = 0; j < C; ++j) {
        const float4 v = ld_dsmem_f4(dsmem_addr(ml_u + rl * 16, j));
        mj[j] = v.x;
        lj[j] = v.y;
        M = fmaxf(M, v.x);
      }
      float L = 0.0f;
      float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
      for (int j = 0; j < C; ++j) {
        const float w = mj[j] == -INFINITY ? 0.0f : exp2f(mj[j] - M);
        L += w * lj[j];
        const float4 q = ld_dsmem_f4(dsmem_addr(op_u + (rl * LDO + cc) * 4, j));
        acc.x += w * q.x; acc.y += w * q.y; acc.z += w * q.z; acc.w += w * q.w;
      }
      if (row < S) {
        const float inv = 1.0f / L;
        *reinterpret_cast<uint2*>(o + (tok0 + row) * ldo + h * HD + cc) =
            make_uint2(pack_half2(acc.x * inv, acc.y * inv), pack_half2(acc.z * inv, acc.w * inv));
        if (cc == 0) lse[(static_cast<int64_t>(b) * H + h) * S + row] = (M + log2f(L)) / kLog2e;
      }
    }
    cluster_sync_all();  // no CTA leaves while its partials are being read
    return;
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int row = ra + 8 * i;
    if (row >= S) continue;
    const float inv = 1.0f / lrow[i];
    uint16_t* orow = o + (tok0 + row) * ldo + h * HD;
#pragma unroll
    for (int dt = 0; dt < NO; ++dt)
      *reinterpret_cast<uint32_t*>(orow + dt * 8 + c) = pack_half2(oacc[dt][2 * i] * inv, oacc[dt][2 * i + 1] * inv);
    if ((lane & 3) == 0) lse[(static_cast<int64_t>(b) * H + h) * S + row] = (mrow[i] + log2f(lrow[i])) / kLog2e;
  }
}

// ------------------------------------------------------------------------------------ backward
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

struct BwdArgs {
  const uint16_t* qkv;
  int64_t ld;
  const uint16_t* dout;
  int64_t ldo;
  const float* lse;
  const float* dvec;
  int S, H, KV, B;
  int W;  // sliding window (0 = none)
  uint16_t* dqkv;
  // split mode: every item cut into P parts, fp32 partials [slot][64][HD] (slots of dK, dV: (b, key
  // block, query head, part); of dQ: (b, query block, head, part))
  int P = 1;
  float *wk = nullptr, *wv = nullptr, *wq = nullptr;
};

// dK, dV of key block kb, output columns d0 .. d0 + DC, accumulated over the (head, query block)
// pairs that see the block — heads h_first .. h_first + h_count - 1, query blocks kb .. — taking
// pairs it0, it0 + dit, ... of that list.  PART: write the fp32 sums (dK already scaled by
// 1/sqrt(hd)) to pk / pv [64][HD]; else write fp16 into dqkv.
template <int HD, int DC, bool PART, bool WIN>
__device__ __forceinline__ void dkdv_run(const BwdArgs& a, int b, int kb, int kvh, int h_first, int h_count, int d0,
                                         int it0, int dit, float* pk, float* pv, uint16_t* sm) {
  constexpr int LD = HD + 8, NC = DC / 8;
  const int S = a.S, H = a.H, KV = a.KV;
  uint16_t* ks = sm;
  uint16_t* vs = ks + BKV * LD;
  // two (Q, dO, lse, dvec) buffers: the next query block loads while this one is used
  auto qs = [&](int buf) { return vs + (1 + 2 * buf) * BQ * LD; };
  auto dos = [&](int buf) { return vs + (2 + 2 * buf) * BQ * LD; };
  auto lse_s = [&](int buf) { return reinterpret_cast<float*>(vs + 5 * BQ * LD) + buf * 2 * BQ; };
  auto dv_s = [&](int buf) { return lse_s(buf) + BQ; };
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t tok0 = static_cast<int64_t>(b) * S;
  const int k0 = kb * BKV;
  const float sc = kLog2e * rsqrtf(static_cast<float>(HD));

  float dk[NC][4], dv[NC][4];
#pragma unroll
  for (int i = 0; i < NC; ++i) {
    dk[i][0] = dk[i][1] = dk[i][2] = dk[i][3] = 0.0f;
    dv[i][0] = dv[i][1] = dv[i][2] = dv[i][3] = 0.0f;
  }
  const int key_a = k0 + warp * 16 + (lane >> 2);
  const int nqb = (S + BQ - 1) / BQ;
  // query blocks kb .. qb_end-1 see this key block (with a window, queries < k0 + BKV - 1 + W)
  const int qb_end = WIN ? min(nqb, (k0 + BKV - 1 + a.W - 1) / BQ + 1) : nqb;
  const int per_head = qb_end - kb;
  const int n_all = h_count * per_head;
  const int n_it = it0 < n_all ? (n_all - it0 + dit - 1) / dit : 0;
  auto fetch = [&](int i, int buf, bool with_dvec) {
    const int it = it0 + i * dit;
    const int h = h_first + it / per_head, q0 = (kb + it % per_head) * BQ;
    load_tile<HD>(qs(buf), a.qkv, a.ld, tok0, q0, S, h * HD, tid);
    load_tile<HD>(dos(buf), a.dout, a.ldo, tok0, q0, S, h * HD, tid);
    for (int r = tid; r < BQ; r += 128) {
      const int q = q0 + r;
      const int64_t li = (static_cast<int64_t>(b) * H + h) * S + q;
      lse_s(buf)[r] = q < S ? __ldcg(a.lse + li) * kLog2e : 0.0f;  // L2 only: may run before the wait
      if (with_dvec) dv_s(buf)[r] = q < S ? a.dvec[li] : 0.0f;
    }
  };
  // q, k, v, lse (the forward) and dO (two kernels back) are complete when this kernel starts;
  // dvec comes from the kernel right before: the first tiles load before the wait
  if (n_it > 0) {
    load_tile<HD>(ks, a.qkv, a.ld, tok0, k0, S, (H + kvh) * HD, tid);
    load_tile<HD>(vs, a.qkv, a.ld, tok0, k0, S, (H + KV + kvh) * HD, tid);
    fetch(0, 0, false);
  }
  cp_async_commit();
  griddep_wait();
  if (n_it > 0) {
    const int h = h_first + it0 / per_head, q0 = (kb + it0 % per_head) * BQ;
    for (int r = tid; r < BQ; r += 128) {
      const int q = q0 + r;
      dv_s(0)[r] = q < S ? a.dvec[(static_cast<int64_t>(b) * H + h) * S + q] : 0.0f;
    }
  }

  for (int i = 0; i < n_it; ++i) {
    const int buf = i & 1;
    const int it = it0 + i * dit;
    const int q0 = (kb + it % per_head) * BQ;
    if (i + 1 < n_it) {
      fetch(i + 1, buf ^ 1, true);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const float* lsb = lse_s(buf);
    const float* dvb = dv_s(buf);
    // P^T (16 keys x 64 queries)
    float pt[8][4];
    qk_tile<HD>(pt, smem_u32(ks), smem_u32(qs(buf)), warp, lane);
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = key_a + ((e >> 1) << 3);
        const int qi = nt * 8 + 2 * (lane & 3) + (e & 1);
        const int q = q0 + qi;
        const bool vis = key <= q && q < S && key < S && (!WIN || q - key < a.W);
        pt[nt][e] = vis ? exp2f(pt[nt][e] * sc - lsb[qi]) : 0.0f;
      }
    // dV += P^T dO
    pv_tile<HD, NC>(dv, pt, smem_u32(dos(buf)), d0, lane);
    // dP^T = V dO^T ; dS^T = P^T (dP^T - dvec)
    float dpt[8][4];
    qk_tile<HD>(dpt, smem_u32(vs), smem_u32(dos(buf)), warp, lane);
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int qi = nt * 8 + 2 * (lane & 3) + (e & 1);
        dpt[nt][e] = pt[nt][e] * (dpt[nt][e] - dvb[qi]);
      }
    // dK += dS^T Q
    pv_tile<HD, NC>(dk, dpt, smem_u32(qs(buf)), d0, lane);
    __syncthreads();  // every warp is done with this buffer before it is refilled
  }

  const float inv = rsqrtf(static_cast<float>(HD));
  const int c = 2 * (lane & 3);
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int kr = warp * 16 + (lane >> 2) + 8 * i;
    if (PART) {
#pragma unroll
      for (int dt = 0; dt < NC; ++dt) {
        __stcg(reinterpret_cast<float2*>(pk + kr * HD + d0 + dt * 8 + c),
               make_float2(dk[dt][2 * i] * inv, dk[dt][2 * i + 1] * inv));
        __stcg(reinterpret_cast<float2*>(pv + kr * HD + d0 + dt * 8 + c), make_float2(dv[dt][2 * i], dv[dt][2 * i + 1]));
      }
    } else {
      const int key = k0 + kr;
      if (key >= S) continue;
      uint16_t* krow = a.dqkv + (tok0 + key) * a.ld + (H + kvh) * HD + d0;
      uint16_t* vrow = a.dqkv + (tok0 + key) * a.ld + (H + KV + kvh) * HD + d0;
#pragma unroll
      for (int dt = 0; dt < NC; ++dt) {
        *reinterpret_cast<uint32_t*>(krow + dt * 8 + c) = pack_half2(dk[dt][2 * i] * inv, dk[dt][2 * i + 1] * inv);
        *reinterpret_cast<uint32_t*>(vrow + dt * 8 + c) = pack_half2(dv[dt][2 * i], dv[dt][2 * i + 1]);
      }
    }
  }
}

// dQ of query block qb and head h, output columns d0 .. d0 + DC, from the key blocks kb_first + it0,
// kb_first + it0 + dit, ... <= qb.  PART: fp32 (scaled by 1/sqrt(hd)) into pq [64][HD]; else fp16.
template <int HD, int DC, bool PART, bool WIN>
__device__ __forceinline__ void dq_run(const BwdArgs& a, int b, int qb, int h, int d0, int it0, int dit, float* pq,
                                       uint16_t* sm) {
  constexpr int LD = HD + 8, NC = DC / 8;
  const int S = a.S, H = a.H, KV = a.KV;
  uint16_t* qs = sm;
  uint16_t* dos = qs + BQ * LD;
  // two (K, V) buffers: the next key block loads while this one is used
  auto ks = [&](int buf) { return dos + (1 + 2 * buf) * BQ * LD; };
  auto vs = [&](int buf) { return dos + (2 + 2 * buf) * BQ * LD; };
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int kvh = h / (H / KV);
  const int64_t tok0 = static_cast<int64_t>(b) * S;
  const int q0 = qb * BQ;
  const float sc = kLog2e * rsqrtf(static_cast<float>(HD));
  const int kb_first = WIN ? max(0, q0 - a.W + 1) / BKV : 0;  // first key block inside the window
  const int n_all = qb - kb_first + 1;
  const int n_it = it0 < n_all ? (n_all - it0 + dit - 1) / dit : 0;

  if (n_it > 0) {
    const int k0 = (kb_first + it0) * BKV;
    load_tile<HD>(qs, a.qkv, a.ld, tok0, q0, S, h * HD, tid);
    load_tile<HD>(dos, a.dout, a.ldo, tok0, q0, S, h * HD, tid);
    load_tile<HD>(ks(0), a.qkv, a.ld, tok0, k0, S, (H + kvh) * HD, tid);
    load_tile<HD>(vs(0), a.qkv, a.ld, tok0, k0, S, (H + KV + kvh) * HD, tid);
  }
  cp_async_commit();
  const int ra = q0 + warp * 16 + (lane >> 2);
  float lse2[2], dvv[2];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int row = ra + 8 * i;
    lse2[i] = row < S ? __ldcg(a.lse + (static_cast<int64_t>(b) * H + h) * S + row) * kLog2e : 0.0f;
  }
  griddep_wait();  // dvec comes from the kernel right before (the tiles above are older)
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int row = ra + 8 * i;
    dvv[i] = row < S ? a.dvec[(static_cast<int64_t>(b) * H + h) * S + row] : 0.0f;
  }
  float dq[NC][4];
#pragma unroll
  for (int i = 0; i < NC; ++i) dq[i][0] = dq[i][1] = dq[i][2] = dq[i][3] = 0.0f;

  for (int i = 0; i < n_it; ++i) {
    const int k0 = (kb_first + it0 + i * dit) * BKV, buf = i & 1;
    if (i + 1 < n_it) {
      const int k1 = k0 + dit * BKV;
      load_tile<HD>(ks(buf ^ 1), a.qkv, a.ld, tok0, k1, S, (H + kvh) * HD, tid);
      load_tile<HD>(vs(buf ^ 1), a.qkv, a.ld, tok0, k1, S, (H + KV + kvh) * HD, tid);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    float p[8][4];
    qk_tile<HD>(p, smem_u32(qs), smem_u32(ks(buf)), warp, lane);
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int col = k0 + nt * 8 + 2 * (lane & 3) + (e & 1);
        const int ii = e >> 1;
        const int row = ra + 8 * ii;
        const bool vis = col <= row && col < S && row < S && (!WIN || row - col < a.W);
        p[nt][e] = vis ? exp2f(p[nt][e] * sc - lse2[ii]) : 0.0f;
      }
    float dp[8][4];
    qk_tile<HD>(dp, smem_u32(dos), smem_u32(vs(buf)), warp, lane);
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) dp[nt][e] = p[nt][e] * (dp[nt][e] - dvv[e >> 1]);
    pv_tile<HD, NC>(dq, dp, smem_u32(ks(buf)), d0, lane);
    __syncthreads();  // every warp is done with this buffer before it is refilled
  }
  const float inv = rsqrtf(static_cast<float>(HD));
  const int c = 2 * (lane & 3);
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    if (PART) {
      const int rl = warp * 16 + (lane >> 2) + 8 * i;
#pragma unroll
      for (int dt = 0; dt < NC; ++dt)
        __stcg(reinterpret_cast<float2*>(pq + rl * HD + d0 + dt * 8 + c),
               make_float2(dq[dt][2 * i] * inv, dq[dt][2 * i + 1] * inv));
    } else {
      const int row = ra + 8 * i;
      if (row >= S) continue;
      uint16_t* qrow = a.dqkv + (tok0 + row) * a.ld + h * HD + d0;
#pragma unroll
      for (int dt = 0; dt < NC; ++dt)
        *reinterpret_cast<uint32_t*>(qrow + dt * 8 + c) = pack_half2(dq[dt][2 * i] * inv, dq[dt][2 * i + 1] * inv);
    }
  }
}

// Large grids: dK/dV with one CTA per (key block, kv head) looping over the group's query heads,
// then dQ with one CTA per (query block, head), as two launches writing dqkv directly.
template <int HD, int DC, bool WIN>
__global__ void __launch_bounds__(128, 1) dkdv_kernel(const BwdArgs a) {
  griddep_launch();  // the item functions wait (after issuing the loads of older data)
  extern __shared__ __align__(16) uint16_t sm[];
  constexpr int NCH = HD / DC;
  const int grp = a.H / a.KV;
  // key block slowest-varying: the longest items (key block 0 sees every query block) first
  const int per = a.KV * a.B * NCH;
  const int kb = blockIdx.x / per;
  int rest = blockIdx.x % per;
  const int kvh = rest % a.KV;
  rest /= a.KV;
  const int b = rest / NCH, d0 = (rest % NCH) * DC;
  dkdv_run<HD, DC, false, WIN>(a, b, kb, kvh, kvh * grp, grp, d0, 0, 1, nullptr, nullptr, sm);
}
template <int HD, int DC, bool WIN>
__global__ void __launch_bounds__(128, 1) dq_kernel(const BwdArgs a) {
  griddep_launch();  // the item functions wait (after issuing the loads of older data)
  extern __shared__ __align__(16) uint16_t sm[];
  constexpr int NCH = HD / DC;
  const int nqb = (a.S + BQ - 1) / BQ;
  // query block slowest-varying, last first: the longest items first
  const int per = a.H * a.B * NCH;
  const int qb = nqb - 1 - static_cast<int>(blockIdx.x) / per;
  int rest = blockIdx.x % per;
  const int h = rest % a.H;
  rest /= a.H;
  const int b = rest / NCH, d0 = (rest % NCH) * DC;
  dq_run<HD, DC, false, WIN>(a, b, qb, h, d0, 0, 1, nullptr, sm);
}

// Small grids: one launch of dK/dV items (key block, query head) and dQ items (query block, head),
// each cut into P interleaved parts, longest first: group L holds the dK/dV items of key block L and
// the dQ items of query block nqb-1-L (both see nqb-L blocks).  Partials go to the workspace;
// bwd_finish_kernel sums them.
template <int HD, int DC, bool WIN>
__global__ void __launch_bounds__(128, 1) bwd_split_kernel(const BwdArgs a) {
  griddep_launch();  // the item functions wait (after issuing the loads of older data)
  extern __shared__ __align__(16) uint16_t sm[];
  constexpr int NCH = HD / DC;
  const int H = a.H, P = a.P, nb = (a.S + BQ - 1) / BQ;
  const int G = H * a.B * NCH * P;
  const int L = blockIdx.x / (2 * G), rem = blockIdx.x % (2 * G);
  int r = rem % G;
  const int p = r % P;
  r /= P;
  const int d0 = (r % NCH) * DC;
  r /= NCH;
  const int h = r % H, b = r / H;
  if (rem < G) {
    const int kb = L;
    const int64_t slot = ((static_cast<int64_t>(b) * nb + kb) * H + h) * P + p;
    dkdv_run<HD, DC, true, WIN>(a, b, kb, h / (H / a.KV), h, 1, d0, p, P, a.wk + slot * (64 * HD),
                                a.wv + slot * (64 * HD), sm);
  } else {
    const int qb = nb - 1 - L;
    const int64_t slot = ((static_cast<int64_t>(b) * nb + qb) * H + h) * P + p;
    dq_run<HD, DC, true, WIN>(a, b, qb, h, d0, p, P, a.wq + slot * (64 * HD), sm);
  }
}

// dqkv from the split partials: dQ = sum over parts; dK, dV = sum over the group's query heads and
// parts (fixed order); q and k then rotated back by their RoPE angle when cs != null (the VJP of
// the rotation: (d1, d2) -> (d1 c + d2 s, d2 c - d1 s)).  One thread per (token, head slot, pair j).
constexpr int kFinishMax = 16;  // partials per element: query heads per kv head (<= 8) x parts (2)
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

template <int HD, int NB, bool WIN, int NWG, int C = 1>
void fwd_launch_g(const uint16_t* qkv, int64_t ld, int B, int S, int H, int KV, uint16_t* o, int64_t ldo, float* lse,
                  int W, cudaStream_t st) {
  constexpr int smem = (1 + 2 * NB * NWG) * 64 * (HD + 8) * 2;  // Q, NB x NWG x (K, V)
  static_assert(smem <= 232448, "attention forward shared memory");
  static bool init = false;
  if (!init) {
    cudaFuncSetAttribute(fwd_kernel<HD, NB, WIN, NWG, C>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    init = true;
  }
  const dim3 grid = C > 1 ? dim3((S + BQ - 1) / BQ * C, H, B) : dim3(H, B, (S + BQ - 1) / BQ);
  if (C == 1) launch_k(fwd_kernel<HD, NB, WIN, NWG, C>, grid, 128 * NWG, smem, st, qkv, ld, S, H, KV, o, ldo, lse, W);
  else
    launch_k_cluster(fwd_kernel<HD, NB, WIN, NWG, C>, grid, 128 * NWG, smem, st, dim3(C, 1, 1), qkv, ld, S, H, KV, o,
                     ldo, lse, W);
}

// Grids of at most one CTA per SM: several warp-groups per CTA — four at head_dim 64 when the
// sequence has at least four query blocks (512 threads, 128 registers each), else two
// (single-buffered at head_dim 256, for shared memory).  Measured at 512 tokens, 14 heads, hd 64:
// 16.5 us with one group, 11.9 with two, 9.8 with four.  Larger grids: one group, double-buffered,
// except at head_dim 256 with more than two waves, where the single-buffered kernel fits two CTAs
// per SM and hides the loads better.
template <int HD, bool WIN>
void fwd_launch_w(const uint16_t* qkv, int64_t ld, int B, int S, int H, int KV, uint16_t* o, int64_t ldo, float* lse,
                  int W, cudaStream_t st) {
  const int nqb = (S + BQ - 1) / BQ;
  const int64_t ctas = static_cast<int64_t>(nqb) * H * B;
  if constexpr (HD == 64) {
    if (ctas <= 152 && nqb >= 4) return fwd_launch_g<HD, 2, WIN, 4>(qkv, ld, B, S, H, KV, o, ldo, lse, W, st);
  }
  // hd 128 / 256 on grids of at most half the SMs: also split the key blocks over a CTA pair
  if (HD != 64 && ctas <= 76 && nqb > 1)
    return fwd_launch_g<HD, HD == 256 ? 1 : 2, WIN, 2, 2>(qkv, ld, B, S, H, KV, o, ldo, lse, W, st);
  if (ctas <= 152 && nqb > 1) fwd_launch_g<HD, HD == 256 ? 1 : 2, WIN, 2>(qkv, ld, B, S, H, KV, o, ldo, lse, W, st);
  else if (HD == 256 && ctas > 2 * 152) fwd_launch_g<HD, 1, WIN, 1>(qkv, ld, B, S, H, KV, o, ldo, lse, W, st);
  else fwd_launch_g<HD, 2, WIN, 1>(qkv, ld, B, S, H, KV, o, ldo, lse, W, st);
}
template <int HD>
void fwd_launch(const uint16_t* qkv, int64_t ld, int B, int S, int H, int KV, uint16_t* o, int64_t ldo, float* lse,
                int W, cudaStream_t st) {
  if (W > 0) fwd_launch_w<HD, true>(qkv, ld, B, S, H, KV, o, ldo, lse, W, st);
  else fwd_launch_w<HD, false>(qkv, ld, B, S, H, KV, o, ldo, lse, 0, st);
}

// Returns true when the split mode ran (which also applied the inverse RoPE when cs != null).
template <int HD, int DC, bool WIN>
bool bwd_launch_w(const uint16_t* qkv, int64_t ld, const uint16_t* dout, int64_t ldo, const float* lse,
                  const float* dvec, int B, int S, int H, int KV, int W, uint16_t* dqkv, const float2* cs, float* ws,
                  int64_t ws_floats, cudaStream_t st) {
  constexpr int smem = 6 * 64 * (HD + 8) * 2 + 4 * 64 * 4;  // 6 tiles (2 of them double-buffered) + lse, dvec x 2
  static_assert(smem <= 232448, "attention backward shared memory");
  static bool init = false;
  if (!init) {
    cudaFuncSetAttribute(bwd_split_kernel<HD, DC, WIN>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    cudaFuncSetAttribute(dkdv_kernel<HD, DC, WIN>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    cudaFuncSetAttribute(dq_kernel<HD, DC, WIN>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    init = true;
  }
  constexpr int NCH = HD / DC, P = 2;
  const int nb = (S + BKV - 1) / BKV;
  BwdArgs a{qkv, ld, dout, ldo, lse, dvec, S, H, KV, B, W, dqkv};
  const int64_t n_grouped = static_cast<int64_t>(nb) * KV * B * NCH;
  const int64_t part_floats = static_cast<int64_t>(B) * nb * H * P * 64 * HD;  // per array
  if (n_grouped < 2 * 152 && ws && 3 * part_floats <= ws_floats && (H / KV) * P <= kFinishMax) {
    a.P = P;
    a.wk = ws;
    a.wv = ws + part_floats;
    a.wq = ws + 2 * part_floats;
    launch_k(bwd_split_kernel<HD, DC, WIN>, dim3(static_cast<unsigned>(2LL * nb * H * B * NCH * P)), 128, smem, st,
             a);
    const int64_t n = static_cast<int64_t>(B) * S * (H + 2 * KV) * (HD / 2);
    launch_k(bwd_finish_kernel<HD>, static_cast<unsigned>((n + 255) / 256), 256, 0, st, a, cs);
    return true;
  }
  launch_k(dkdv_kernel<HD, DC, WIN>, dim3(static_cast<unsigned>(n_grouped)), 128, smem, st, a);
  launch_k(dq_kernel<HD, DC, WIN>, dim3(static_cast<unsigned>(static_cast<int64_t>(nb) * H * B * NCH)), 128, smem, st,
           a);
  return false;
}
template <int HD, int DC>
bool bwd_launch(const uint16_t* qkv, int64_t ld, const uint16_t* dout, int64_t ldo, const float* lse,
                const float* dvec, int B, int S, int H, int KV, int W, uint16_t* dqkv, const float2* cs, float* ws,
                int64_t ws_floats, cudaStream_t st) {
  if (W > 0)
    return bwd_launch_w<HD, DC, true>(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, W, dqkv, cs, ws, ws_floats, st);
  return bwd_launch_w<HD, DC, false>(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, 0, dqkv, cs, ws, ws_floats, st);
}

}  // namespace attn

// Grids of at least this many 128-query tiles run the tcgen05 kernels (attention_tc.cu); smaller
// ones keep the warp-level kernels above, which split the keys of a query block over several
// warp-groups or a CTA pair (measured: tcgen05 595 TFLOP/s at the Gemma3-4B shape, 36.1 -> 15.5 ms
// per step; at 56 tiles, Qwen2.5-0.5B, 0.68 ms warp-level against 0.97 ms tcgen05).
constexpr int64_t kTcMinTiles = 64;

int launch_attn_fwd(const uint16_t* qkv, int64_t ld, int B, int S, int H, int KV, int hd, uint16_t* o, int64_t ldo,
                    float* lse, int window, int* err, cudaStream_t st) {
  const int64_t tiles = static_cast<int64_t>((S + 127) / 128) * H * B;
  if (tiles >= kTcMinTiles) return launch_attn_fwd_tc(qkv, ld, B, S, H, KV, hd, o, ldo, lse, window, err, st);
  const int W = window >= S ? 0 : window;  // a window covering the sequence is plain causal
  if (hd == 64) attn::fwd_launch<64>(qkv, ld, B, S, H, KV, o, ldo, lse, W, st);
  else if (hd == 128) attn::fwd_launch<128>(qkv, ld, B, S, H, KV, o, ldo, lse, W, st);
  else attn::fwd_launch<256>(qkv, ld, B, S, H, KV, o, ldo, lse, W, st);
  return cudaGetLastError() == cudaSuccess ? MEBP_OK : MEBP_ERR_CUDA;
}

bool launch_attn_bwd(const uint16_t* qkv, int64_t ld, const uint16_t* o, const uint16_t* dout, int64_t ldo,
                     const float* lse, int B, int S, int H, int KV, int hd, float* dvec, uint16_t* dqkv, int window,
                     const float2* rope_cs, float* ws, int64_t ws_floats, int* err, cudaStream_t st) {
  const int W = window >= S ? 0 : window;
  const int64_t nw = static_cast<int64_t>(B) * S * H;
  launch_k(attn::dvec_kernel, static_cast<unsigned>((nw * 32 + 255) / 256), 256, 0, st, o, dout, ldo, B, S, H, hd,
           dvec);
  // tcgen05 dK/dV and dQ when the dK/dV grid (128-key blocks x kv heads x sequences x column
  // halves at hd 256) fills the GPU: Gemma3-4B shape 108 -> 51 ms per step; below that its CTAs
  // each loop over too many query blocks, and the warp-level kernels split the work instead
  const int64_t kv_tiles = static_cast<int64_t>((S + 127) / 128) * KV * B * (hd == 256 ? 2 : 1);
  if (kv_tiles >= 152) {
    launch_attn_bwd_tc(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, hd, dqkv, window, err, st);
    return false;  // the caller applies the inverse RoPE
  }
  if (hd == 64)
    return attn::bwd_launch<64, 64>(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, W, dqkv, rope_cs, ws, ws_floats, st);
  if (hd == 128)
    return attn::bwd_launch<128, 128>(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, W, dqkv, rope_cs, ws, ws_floats, st);
  return attn::bwd_launch<256, 128>(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, W, dqkv, rope_cs, ws, ws_floats, st);
}

}  // namespace mebp
