// Causal grouped-query attention forward on 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
//   o = softmax(q k^T / sqrt(hd) + mask) v per (sequence, query head); query head h reads key/value
//   head h / (H/KV); lse = log-sum-exp of each score row (natural log), kept for the backward.
//   mask: query i sees key j iff j <= i and, with a sliding window W > 0 (Gemma3's local layers),
//   i - j < W; key blocks wholly outside the window are skipped.
//
// One CTA per (128 queries, head, sequence), 224 threads:
//   warps 0-3  softmax: thread r owns query row r (TMEM lane r) — reads its score row from TMEM,
//              keeps the running max m and sum l, writes the fp16 probabilities P to shared memory
//              (the A operand of P v) and at the end normalises its row of O out of TMEM;
//   warp 4     TMA: the query tile once, then the key tiles of every visible key block;
//   warp 5     TMA: the value tiles;
//   warp 6     tcgen05.mma issuer and TMEM owner: S_j = Q K_j^T into one of two TMEM score buffers,
//              then O += P_{j-1} V_{j-1} into the TMEM accumulator, so the tensor cores compute the
//              next scores while the softmax warps work on the current ones.
// q, k and v are read from the fused projection buffer [T, (H + 2 KV) hd] (q heads, k heads, v
// heads) through one 3-D tensor map {columns, positions, sequences}: tiles past the end of a
// sequence are zero-filled, never read from the next one.
//
// Online softmax with a lazy rescale: a row's reference max moves (and O, l are rescaled) only
// when a new block raises the row max by more than 2^8 over it, so most blocks touch O not at all;
// the probabilities stay below 2^8 (exact in fp16's range) and the final O / l is unchanged.
// Every wait is bounded (device error word, CTA abort flag); copies in flight are drained and
// TMEM is freed before a CTA exits.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"

namespace mebp {
namespace atc {

constexpr int BQ = 128, BKV = 128;
constexpr int FWD_THREADS = 224;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRescale = 8.0f;  // log2 units

template <int HD>
struct Fwd {
  // keys per block (64 at hd 256, with two K/V stages and two P buffers, measured 7 % slower than
  // 128 with one of each: more blocks, more hand-offs)
  static constexpr int BK = BKV;
  static constexpr int NST = HD == 256 ? 1 : (HD == 128 ? 2 : 3);  // key ring = value ring depth
  static constexpr int NP = HD == 256 ? 1 : 2;                      // probability buffers
  static constexpr int NCH = HD / 64;                               // 64-column (128-byte) chunks
  static constexpr int Q_BYTES = BQ * HD * 2;
  static constexpr int KV_BYTES = BK * HD * 2;
  static constexpr int P_BYTES = BQ * BK * 2;
  static constexpr int Q_OFF = 0;
  static constexpr int K_OFF = Q_OFF + Q_BYTES;
  static constexpr int V_OFF = K_OFF + NST * KV_BYTES;
  static constexpr int P_OFF = V_OFF + NST * KV_BYTES;
  static constexpr int BAR_OFF = P_OFF + NP * P_BYTES;
  static constexpr int SMEM = BAR_OFF + 256 + 1024;
  static constexpr uint32_t TM_O = 0, TM_S = 256;  // TMEM columns: O [0, HD), scores 256 + BK b
};

// CL > 1 (grids under one wave): the key blocks of a query tile are dealt round-robin to the CL
// CTAs of a cluster; each keeps its own (m, l, O) and the cluster merges them through
// distributed shared memory, CTA c normalising and writing rows c*128/CL .. (c+1)*128/CL - 1.
template <int HD, bool WIN, int CL>
__global__ void __launch_bounds__(FWD_THREADS, 1)
    fwd_tc_kernel(const __grid_constant__ CUtensorMap tm, const __grid_constant__ CUtensorMap tmkv, int S, int H, int KV,
                  uint16_t* __restrict__ o, int64_t ldo, float* __restrict__ lse, int W, int* err) {
  using C = Fwd<HD>;
  constexpr int BKV = C::BK;  // keys per block in this kernel
  constexpr int NST = C::NST, NP = C::NP;
  static_assert(C::SMEM <= 232448, "shared memory");
  static_assert(C::SMEM > 232448 / 2, "one CTA per SM (512 TMEM columns each)");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* qfull = reinterpret_cast<uint64_t*>(sm + C::BAR_OFF);
  uint64_t* kfull = qfull + 1;
  uint64_t* kempty = kfull + NST;
  uint64_t* vfull = kempty + NST;
  uint64_t* vempty = vfull + NST;
  uint64_t* sfull = vempty + NST;  // [2]
  uint64_t* pfull = sfull + 2;     // [NP]
  uint64_t* pvdone = pfull + NP;   // [NP]
  uint64_t* ofull = pvdone + NP;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(ofull + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = static_cast<int>(blockIdx.x) / CL, crank = static_cast<int>(blockIdx.x) % CL, b = blockIdx.y;
  const int qb = static_cast<int>(gridDim.z) - 1 - static_cast<int>(blockIdx.z);  // longest rows first
  const int kvh = h / (H / KV);
  const int q0 = qb * BQ;
  const int kend = min(S, q0 + BQ);                          // keys below kend are seen by some row
  const int kb0 = WIN ? max(0, q0 - W + 1) / BKV : 0;        // first key block inside the window
  const int nkb_all = (kend + BKV - 1) / BKV - kb0;
  const int nkb = (nkb_all - crank + CL - 1) / CL;           // this CTA's blocks: crank, crank + CL, ...
  auto kblock = [&](int j) { return kb0 + crank + j * CL; };

  if (threadIdx.x == 0) {
    mbar_init(qfull, 1);
    for (int s = 0; s < NST; ++s) {
      mbar_init(&kfull[s], 1);
      mbar_init(&kempty[s], 1);
      mbar_init(&vfull[s], 1);
      mbar_init(&vempty[s], 1);
    }
    for (int i = 0; i < 2; ++i) mbar_init(&sfull[i], 1);
    for (int i = 0; i < NP; ++i) {
      mbar_init(&pfull[i], 4);  // one arrival per softmax warp
      mbar_init(&pvdone[i], 1);
    }
    mbar_init(ofull, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 6) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  griddep_wait();  // q, k, v come from the kernel right before (RoPE)
  griddep_launch();

  if (warp == 4) {
    // ---------------------------------------------------------------- query + key tiles
    if (lane == 0) {
      tma_prefetch_desc(&tm);
      tma_prefetch_desc(&tmkv);
      mbar_arrive_expect_tx(qfull, C::Q_BYTES);
      for (int c = 0; c < C::NCH; ++c) tma_load_3d(sm + C::Q_OFF + c * BQ * 128, &tm, qfull, h * HD + c * 64, q0, b);
      int issued = 0;
      for (int j = 0; j < nkb; ++j) {
        const int s = j % NST;
        if (j >= NST && !mbar_wait(&kempty[s], ((j / NST) & 1) ^ 1, abort_flag, err)) break;
        mbar_arrive_expect_tx(&kfull[s], C::KV_BYTES);
        for (int c = 0; c < C::NCH; ++c)
          tma_load_3d(sm + C::K_OFF + s * C::KV_BYTES + c * BKV * 128, &tmkv, &kfull[s], (H + kvh) * HD + c * 64,
                      kblock(j) * BKV, b);
        issued = j + 1;
      }
      int dummy = 0;  // never leave with copies in flight
      mbar_wait(qfull, 0, &dummy, err);
      for (int j = (issued > NST ? issued - NST : 0); j < issued; ++j)
        mbar_wait(&kfull[j % NST], (j / NST) & 1, &dummy, err);
    }
  } else if (warp == 5) {
    // ---------------------------------------------------------------- value tiles
    if (lane == 0) {
      int issued = 0;
      for (int j = 0; j < nkb; ++j) {
        const int s = j % NST;
        if (j >= NST && !mbar_wait(&vempty[s], ((j / NST) & 1) ^ 1, abort_flag, err)) break;
        mbar_arrive_expect_tx(&vfull[s], C::KV_BYTES);
        for (int c = 0; c < C::NCH; ++c)
          tma_load_3d(sm + C::V_OFF + s * C::KV_BYTES + c * BKV * 128, &tmkv, &vfull[s],
                      (H + KV + kvh) * HD + c * 64, kblock(j) * BKV, b);
        issued = j + 1;
      }
      int dummy = 0;
      for (int j = (issued > NST ? issued - NST : 0); j < issued; ++j)
        mbar_wait(&vfull[j % NST], (j / NST) & 1, &dummy, err);
    }
  } else if (warp == 6) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t id_s = idesc_f16_f32(BQ, BKV, false);  // S = Q K^T: both K-major
      constexpr uint32_t id_o = idesc_f16_f32(BQ, HD, true);    // O += P V: V is N(hd)-major
      bool ok = mbar_wait(qfull, 0, abort_flag, err);
      const uint32_t q_addr = smem_u32(sm + C::Q_OFF);
      for (int j = 0; ok && j <= nkb; ++j) {
        if (j < nkb) {
          const int s = j % NST;
          if (!(ok = mbar_wait(&kfull[s], (j / NST) & 1, abort_flag, err))) break;
          tc_fence_after();
          const uint32_t k_addr = smem_u32(sm + C::K_OFF + s * C::KV_BYTES);
          const uint32_t ts = tmem + C::TM_S + (j & 1) * BKV;
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk) {
            const uint32_t off = (kk >> 2) * (BQ * 128) + (kk & 3) * 32;  // 64-column chunk, k16 slice
            const uint32_t koff = (kk >> 2) * (BKV * 128) + (kk & 3) * 32;
            tc_mma_f16(ts, smem_desc_sw128(q_addr + off, 16, 1024), smem_desc_sw128(k_addr + koff, 16, 1024), id_s,
                       kk > 0 ? 1u : 0u);
          }
          tc_commit(&sfull[j & 1]);
          tc_commit(&kempty[s]);
        }
        if (j >= 1) {
          const int i = j - 1, p = i % NP, s = i % NST;
          if (!(ok = mbar_wait(&pfull[p], (i / NP) & 1, abort_flag, err))) break;
          if (!(ok = mbar_wait(&vfull[s], (i / NST) & 1, abort_flag, err))) break;
          tc_fence_after();
          const uint32_t p_addr = smem_u32(sm + C::P_OFF + p * C::P_BYTES);
          const uint32_t v_addr = smem_u32(sm + C::V_OFF + s * C::KV_BYTES);
#pragma unroll
          for (int kk = 0; kk < BKV / 16; ++kk) {
            const uint32_t poff = (kk >> 2) * (BQ * 128) + (kk & 3) * 32;
            // V [keys][hd]: 64-column chunks BKV*128 bytes apart (LBO), 16 key rows per k16 slice
            tc_mma_f16(tmem + C::TM_O, smem_desc_sw128(p_addr + poff, 16, 1024),
                       smem_desc_sw128(v_addr + kk * 16 * 128, BKV * 128, 1024), id_o, (i > 0 || kk > 0) ? 1u : 0u);
          }
          tc_commit(&pvdone[p]);
          tc_commit(&vempty[s]);
        }
      }
      tc_commit(ofull);
    }
  } else {
    // ---------------------------------------------------------------- softmax (warps 0-3)
    const int r = 32 * warp + lane, row = q0 + r;
    const uint32_t lane_off = static_cast<uint32_t>(32 * warp) << 16;
    const float sc = kLog2e * rsqrtf(static_cast<float>(HD));
    float m_used = -INFINITY, l = 0.0f;
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      ok = __all_sync(0xffffffffu, mbar_wait(&sfull[j & 1], (j >> 1) & 1, abort_flag, err));
      if (!ok) break;
      tc_fence_after();
      // pass 1: the row max of this block (scores scaled to log2 units, masked)
      const int k0 = kblock(j) * BKV;
      const uint32_t ts = tmem + lane_off + C::TM_S + (j & 1) * BKV;
      auto masked = [&](float (&t)[32], int c) {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int key = k0 + 32 * c + i;
          const bool vis = key <= row && (!WIN || row - key < W);
          t[i] = vis ? t[i] * sc : -INFINITY;
        }
      };
      float mx = -INFINITY;
#pragma unroll 1
      for (int c = 0; c < BKV / 32; ++c) {
        float t[32];
        tmem_ld32(ts + 32 * c, t);
        masked(t, c);
#pragma unroll
        for (int i = 0; i < 32; ++i) mx = fmaxf(mx, t[i]);
      }
      const float m_new = fmaxf(m_used, mx);
      const bool need = m_new > m_used + kRescale;
      if (__any_sync(0xffffffffu, need)) {
        const float alpha = need ? exp2f(m_used - m_new) : 1.0f;  // 0 when m_used = -inf
        if (j > 0) {  // O holds the blocks before j once P_{j-1} V_{j-1} has retired
          const int i = j - 1;
          ok = __all_sync(0xffffffffu, mbar_wait(&pvdone[i % NP], (i / NP) & 1, abort_flag, err));
          if (!ok) break;
          tc_fence_after();
#pragma unroll 1
          for (int c = 0; c < HD / 32; ++c) {
            float t[32];
            tmem_ld32(tmem + lane_off + C::TM_O + 32 * c, t);
#pragma unroll
            for (int e = 0; e < 32; ++e) t[e] *= alpha;
            tmem_st32(tmem + lane_off + C::TM_O + 32 * c, t);
          }
        }
        if (need) {
          l *= alpha;
          m_used = m_new;
        }
      }
      // the probability buffer is free once P_{j-NP} V_{j-NP} has retired
      if (j >= NP) {
        const int i = j - NP;
        ok = __all_sync(0xffffffffu, mbar_wait(&pvdone[i % NP], (i / NP) & 1, abort_flag, err));
        if (!ok) break;
      }
      // pass 2: probabilities against the reference max, written as the fp16 A operand of P V
      uint8_t* prow = sm + C::P_OFF + (j % NP) * C::P_BYTES + r * 128;
      float rs = 0.0f;
      const bool live = m_used != -INFINITY;
#pragma unroll 1
      for (int c = 0; c < BKV / 32; ++c) {
        float t[32];
        tmem_ld32(ts + 32 * c, t);
        masked(t, c);
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          t[i] = live ? exp2f(t[i] - m_used) : 0.0f;
          rs += t[i];
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {  // 8 keys per 16-byte unit; 8 units per 128-byte chunk row
          const int u = 4 * c + q, ch = u >> 3, w = u & 7;
          *reinterpret_cast<uint4*>(prow + ch * (BQ * 128) + ((w ^ (r & 7)) << 4)) =
              make_uint4(pack_half2(t[8 * q], t[8 * q + 1]), pack_half2(t[8 * q + 2], t[8 * q + 3]),
                         pack_half2(t[8 * q + 4], t[8 * q + 5]), pack_half2(t[8 * q + 6], t[8 * q + 7]));
        }
      }
      l += rs;
      fence_proxy_async_smem();  // the MMA (async proxy) reads P
      tc_fence_before();         // the score reads (and O rescale) are ordered before the arrival
      __syncwarp();
      if (lane == 0) mbar_arrive(&pfull[j % NP]);
    }
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(ofull, 0, abort_flag, err));
    tc_fence_after();
    if (CL > 1) {
      // park the unnormalised row of O and (m, l) in this CTA's shared memory (every load and
      // MMA of the CTA has completed, so the tiles are free); a CTA without key blocks parks zeros
      float* po = reinterpret_cast<float*>(sm) + r * (HD + 4);
#pragma unroll 1
      for (int c = 0; c < HD / 32; ++c) {
        float t[32];
        tmem_ld32(tmem + lane_off + C::TM_O + 32 * c, t);
#pragma unroll
        for (int i = 0; i < 8; ++i)
          *reinterpret_cast<float4*>(po + 32 * c + 4 * i) =
              (ok && nkb > 0) ? make_float4(t[4 * i], t[4 * i + 1], t[4 * i + 2], t[4 * i + 3])
                              : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
      }
      reinterpret_cast<float4*>(sm + BQ * (HD + 4) * 4)[r] =
          make_float4((ok && nkb > 0) ? m_used : -INFINITY, (ok && nkb > 0) ? l : 0.0f, 0.0f, 0.0f);
    } else if (ok) {
      const float inv = l > 0.0f ? 1.0f / l : 0.0f;
      const int64_t tok = static_cast<int64_t>(b) * S + row;
#pragma unroll 1
      for (int c = 0; c < HD / 32; ++c) {
        float t[32];
        tmem_ld32(tmem + lane_off + C::TM_O + 32 * c, t);
        if (row < S) {
          uint4* dst = reinterpret_cast<uint4*>(o + tok * ldo + h * HD + 32 * c);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            dst[i] = make_uint4(pack_half2(t[8 * i] * inv, t[8 * i + 1] * inv),
                                pack_half2(t[8 * i + 2] * inv, t[8 * i + 3] * inv),
                                pack_half2(t[8 * i + 4] * inv, t[8 * i + 5] * inv),
                                pack_half2(t[8 * i + 6] * inv, t[8 * i + 7] * inv));
        }
      }
      if (row < S) lse[(static_cast<int64_t>(b) * H + h) * S + row] = (m_used + log2f(l)) / kLog2e;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 6) {
    if (lane == 0) {  // every MMA has retired before TMEM is freed
      int dummy = 0;
      mbar_wait(ofull, 0, &dummy, err);
    }
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
  if constexpr (CL > 1) {
    // every thread of every CTA of the cluster passes both barriers (no wait above is unbounded)
    cluster_sync_all();
    constexpr int RPC = BQ / CL, C4 = HD / 4;
    const uint32_t o_base = smem_u32(sm), ml_base = smem_u32(sm + BQ * (HD + 4) * 4);
    for (int e = threadIdx.x; e < RPC * C4; e += FWD_THREADS) {
      const int rl = crank * RPC + e / C4, cc = (e % C4) * 4, row = q0 + rl;
      float mj[CL], lj[CL];
      float Mx = -INFINITY;
#pragma unroll
      for (int j = 0; j < CL; ++j) {
        const float4 v = ld_dsmem_f4(dsmem_addr(ml_base + rl * 16, j));
        mj[j] = v.x;
        lj[j] = v.y;
        Mx = fmaxf(Mx, v.x);
      }
      float L = 0.0f;
      float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
      for (int j = 0; j < CL; ++j) {
        if (mj[j] == -INFINITY) continue;
        const float w = exp2f(mj[j] - Mx);
        L += w * lj[j];
        const float4 q = ld_dsmem_f4(dsmem_addr(o_base + (rl * (HD + 4) + cc) * 4, j));
        acc.x += w * q.x; acc.y += w * q.y; acc.z += w * q.z; acc.w += w * q.w;
      }
      if (row < S) {
        const float inv = L > 0.0f ? 1.0f / L : 0.0f;
        *reinterpret_cast<uint2*>(o + (static_cast<int64_t>(b) * S + row) * ldo + h * HD + cc) =
            make_uint2(pack_half2(acc.x * inv, acc.y * inv), pack_half2(acc.z * inv, acc.w * inv));
        if (cc == 0) lse[(static_cast<int64_t>(b) * H + h) * S + row] = (Mx + log2f(L)) / kLog2e;
      }
    }
    cluster_sync_all();  // no CTA leaves while its partials are being read
  }
}

template <int HD, bool WIN, int CL>
int fwd_launch_cl(const CUtensorMap& tm, const CUtensorMap& tmkv, int B, int S, int H, int KV, uint16_t* o,
                  int64_t ldo, float* lse, int W, int* err, cudaStream_t st) {
  using C = Fwd<HD>;
  static_assert(BQ * (HD + 4) * 4 + BQ * 16 <= C::BAR_OFF, "parked O and (m, l) fit below the barriers");
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(fwd_tc_kernel<HD, WIN, CL>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM) !=
        cudaSuccess) {
      cudaGetLastError();
      return MEBP_ERR_CUDA;
    }
    attr = true;
  }
  const dim3 grid(H * CL, B, (S + BQ - 1) / BQ);
  if (CL == 1)
    launch_k(fwd_tc_kernel<HD, WIN, CL>, grid, FWD_THREADS, C::SMEM, st, tm, tmkv, S, H, KV, o, ldo, lse, W, err);
  else
    launch_k_cluster(fwd_tc_kernel<HD, WIN, CL>, grid, FWD_THREADS, C::SMEM, st, dim3(CL, 1, 1), tm, tmkv, S, H, KV, o,
                     ldo, lse, W, err);
  return cudaGetLastError() == cudaSuccess ? MEBP_OK : MEBP_ERR_CUDA;
}

template <int HD, bool WIN>
int fwd_launch(const uint16_t* qkv, int64_t ld, int B, int S, int H, int KV, uint16_t* o, int64_t ldo, float* lse,
               int W, int* err, cudaStream_t st) {
  CUtensorMap tm, tmkv;
  // {columns of the fused projection buffer, positions, sequences}: 64 x 128 x 1 boxes for the
  // query tile, 64 x BK x 1 for key / value blocks
  const uint64_t seq = static_cast<uint64_t>(S) * ld * 2;
  int rc = make_tmap_3d(&tm, qkv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, ld, S, B, ld * 2, seq, 64, BQ, 1,
                        CU_TENSOR_MAP_SWIZZLE_128B);
  if (!rc)
    rc = make_tmap_3d(&tmkv, qkv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, ld, S, B, ld * 2, seq, 64, Fwd<HD>::BK, 1,
                      CU_TENSOR_MAP_SWIZZLE_128B);
  if (rc) return rc;
  // grids under one wave whose longest query tiles see at least 8 key blocks share each tile's
  // key blocks among a cluster of 2 or 4 CTAs (Gemma3-1B shape, 1024 tokens).  With fewer blocks
  // the cluster merge costs more than the shorter chain saves (Qwen2.5-0.5B shape, 512 tokens:
  // 5.36 ms per step without the split, 5.44 with pairs).
  const int64_t tiles = static_cast<int64_t>((S + BQ - 1) / BQ) * H * B;
  const int nkb_max = (S + Fwd<HD>::BK - 1) / Fwd<HD>::BK;
  if (tiles * 4 <= 152 && nkb_max >= 8)
    return fwd_launch_cl<HD, WIN, 4>(tm, tmkv, B, S, H, KV, o, ldo, lse, W, err, st);
  if (tiles * 2 <= 152 && nkb_max >= 8)
    return fwd_launch_cl<HD, WIN, 2>(tm, tmkv, B, S, H, KV, o, ldo, lse, W, err, st);
  return fwd_launch_cl<HD, WIN, 1>(tm, tmkv, B, S, H, KV, o, ldo, lse, W, err, st);
}

// ================================================================================== backward
// dP = dO v^T, dS = P (dP - D) with D = rowsum(dO o) (dvec_kernel), P recomputed from q, k and the
// forward's lse; dq = dS k / sqrt(hd), dk = dS^T q / sqrt(hd), dv = P^T dO, dk and dv summed over
// the query heads of a group.  Two kernels write dqkv directly (no atomics, deterministic):
//  * dkdv_tc_kernel: one CTA per (128 keys, kv head, sequence[, half of the head columns at
//    hd 256]); the key and value tiles stay in shared memory while the CTA loops over the
//    group's query heads and the query blocks (64 queries) that see its keys: S^T = K Q^T and
//    dP^T = V dO^T into one of two TMEM buffers, the four "softmax" warps (thread = key row)
//    turn them into P^T and dS^T (fp16, shared memory), then dV += P^T dO and dK += dS^T Q
//    accumulate in TMEM.
//  * dq_tc_kernel: one CTA per (128 queries, head, sequence) looping over key blocks of 64:
//    S = Q K^T and dP = dO V^T, dS from the thread's own row (lse, D), dQ += dS K in TMEM.
// With a single operand stage (hd 256) the MMA warp issues the accumulation of block j-1 before
// the scores of block j (the stage is reused); otherwise the scores of block j go first so the
// tensor cores run while the softmax warps work.
constexpr int BWD_THREADS = 192;  // warps 0-3 elementwise + epilogue, 4 TMA, 5 MMA
// Queries per dK/dV iteration and keys per dQ iteration.  (At hd 256 the resident 128-row tiles,
// K and V or Q and dO, take 128 KB and leave room for one operand stage of 64-row blocks; 32-row
// blocks with two stages measured 18 % slower: more iterations, more hand-offs.)  The P^T / dS^T /
// dS tiles have 128-byte rows (64 columns).
template <int HD>
constexpr int bwd_block() { return 64; }

// Split mode (grids under one wave): a dK/dV item is one (128 keys, query head, part) and takes
// every P-th query block of that head; a dQ item is one (128 queries, head, part) and takes every
// P-th key block.  Items write fp32 partials (dK and dQ already times 1/sqrt(hd)) into slots of
// [64 rows][hd] floats indexed ((b * nb64 + 64-row block) * H + query head) * P + part, which the
// finish kernel sums over parts and the query heads of a group.  P == 0: direct mode.
struct SplitOut {
  int P;
  float *wk, *wv, *wq;
};

template <int HD>
struct DkDv {
  // hd 256: V lives in TMEM as the A operand of dP^T = V dO^T (tcgen05 reads A from TMEM), which
  // frees its 64 KB of shared memory for a second (Q, dO) stage; V lands in that stage's slot once
  // and the elementwise warps copy it row by row into TMEM before the loop.
  static constexpr bool VT = HD == 256;
  static constexpr int QB = bwd_block<HD>();       // queries per iteration
  static constexpr int DC = HD == 256 ? 128 : HD;  // output columns per CTA
  static constexpr int NCOL = HD / DC;
  static constexpr int NS = HD == 256 ? 2 : (HD == 128 ? 3 : 4);  // (Q, dO) stages
  static constexpr int NPB = HD == 256 ? 1 : 2;                   // (P^T, dS^T) buffers
  static constexpr int NSB = VT ? 1 : 2;                          // S^T / dP^T buffers in TMEM
  static constexpr int NCH = HD / 64;
  static constexpr int KV_BYTES = BKV * HD * 2;   // one of K, V
  static constexpr int Q_BYTES = QB * HD * 2;     // one of Q_i, dO_i
  static constexpr int P_BYTES = BKV * 64 * 2;    // one of P^T, dS^T (128-byte rows)
  static constexpr int K_OFF = 0, V_OFF = KV_BYTES;  // (V_OFF unused when VT)
  static constexpr int Q_OFF = VT ? KV_BYTES : 2 * KV_BYTES;  // stage s: Q at Q_OFF + 2 s Q_BYTES, dO after it
  static constexpr int V_LAND = Q_OFF + 2 * Q_BYTES;          // VT: V passes through stage 1
  static constexpr int P_OFF = Q_OFF + NS * 2 * Q_BYTES;      // buffer p: P^T, then dS^T
  static constexpr int VEC_OFF = P_OFF + NPB * 2 * P_BYTES;   // [2][2][64] floats: lse*log2e, D
  static constexpr int BAR_OFF = VEC_OFF + 2 * 2 * 64 * 4;
  static constexpr int SMEM = BAR_OFF + 256 + 1024;
  // S^T / dP^T buffer b: TM_S + 128 b (+64); V (VT): 256 fp16 per key row packed in 128 columns
  static constexpr uint32_t TM_DK = 0, TM_DV = DC, TM_V = 256, TM_S = VT ? 384 : 256;
  static_assert(!VT || 2 * Q_BYTES == KV_BYTES, "V fits the second stage");
};

// tcgen05.mma with the A operand in TMEM (K-major: TMEM lane = row of A, each 32-bit column two
// consecutive K elements): D[tmem] (+)= A[a_tmem] * B[smem desc]^T.
__device__ __forceinline__ void tc_mma_f16_ta(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                              uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// One dK/dV item: item = (((kb * B + b) * heads + head) * NCOL + col) * P + part, heads = KV (direct,
// P = 1) or H (split).
template <int HD, bool WIN>
__device__ __forceinline__ void dkdv_body(const CUtensorMap& tmKV, const CUtensorMap& tmQ, const CUtensorMap& tmDO,
                                          int S, int H, int KV, const float* __restrict__ lse,
                                          const float* __restrict__ dvec, uint16_t* __restrict__ dqkv, int64_t ld,
                                          int W, int* err, const SplitOut& so, int item, int B) {
  using C = DkDv<HD>;
  constexpr int NS = C::NS, NPB = C::NPB, DC = C::DC, BQB = C::QB, NSB = C::NSB;
  constexpr bool VT = C::VT;
  static_assert(C::SMEM <= 232448, "shared memory");
  static_assert(C::SMEM > 232448 / 2, "one CTA per SM (512 TMEM columns each)");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* kvfull = reinterpret_cast<uint64_t*>(sm + C::BAR_OFF);
  uint64_t* qfull = kvfull + 1;    // [NS]
  uint64_t* qempty = qfull + NS;   // [NS]
  uint64_t* sfull = qempty + NS;   // [2]
  uint64_t* sfree = sfull + 2;     // [2]
  uint64_t* pready = sfree + 2;    // [NPB]
  uint64_t* pdone = pready + NPB;  // [NPB]
  uint64_t* dfull = pdone + NPB;
  uint64_t* vready = dfull + 1;    // [2] the lse / D vectors of an iteration are in shared memory
  uint64_t* vland = vready + 2;    // VT: V landed in stage 1's slot
  uint64_t* vmoved = vland + 1;    // VT: V copied into TMEM (stage 1's slot is free again)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(vmoved + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* vec = reinterpret_cast<float*>(sm + C::VEC_OFF);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // direct: blockIdx.x = ((kb * B + b) * KV + kvh) * NCOL + col; split: (((kb * B + b) * H + h) * NCOL +
  // col) * P + p; key block slowest and first (the longest items)
  const bool split = so.P > 0;
  const int P = split ? so.P : 1;
  const int heads = split ? H : KV;
  int t = item;
  const int part = t % P;
  t /= P;
  const int col = t % C::NCOL;
  t /= C::NCOL;
  const int hsel = t % heads;
  t /= heads;
  const int b = t % B, kb = t / B;
  const int grp = H / KV;
  const int kvh = split ? hsel / grp : hsel;
  const int h_first = split ? hsel : kvh * grp;
  const int c0 = col * DC;
  const int k0 = kb * BKV;
  const int nqb = (S + BQB - 1) / BQB;
  const int qb_first = k0 / BQB;
  const int qb_end = WIN ? min(nqb, (k0 + BKV - 1 + W - 1) / BQB + 1) : nqb;
  const int per_head = qb_end - qb_first;
  const int n_all = split ? per_head : grp * per_head;
  const int n_it = part < n_all ? (n_all - part + P - 1) / P : 0;
  auto g_of = [&](int j) { return part + j * P; };  // iteration j covers (head, query block) number g

  if (threadIdx.x == 0) {
    mbar_init(kvfull, 1);
    for (int s = 0; s < NS; ++s) {
      mbar_init(&qfull[s], 1);
      mbar_init(&qempty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sfull[i], 1);
      mbar_init(&sfree[i], 4);
    }
    for (int i = 0; i < NPB; ++i) {
      mbar_init(&pready[i], 4);
      mbar_init(&pdone[i], 1);
    }
    mbar_init(dfull, 1);
    for (int i = 0; i < 2; ++i) mbar_init(&vready[i], 128);
    mbar_init(vland, 1);
    mbar_init(vmoved, 4);  // one arrival per elementwise warp
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 5) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  griddep_wait();  // dvec comes from the kernel right before
  griddep_launch();

  if (warp == 4) {
    if (lane == 0) {
      tma_prefetch_desc(&tmKV);
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmDO);
      mbar_arrive_expect_tx(kvfull, (VT ? 1 : 2) * C::KV_BYTES);
      if (VT) mbar_arrive_expect_tx(vland, C::KV_BYTES);
      for (int c = 0; c < C::NCH; ++c) {
        tma_load_3d(sm + C::K_OFF + c * BKV * 128, &tmKV, kvfull, (H + kvh) * HD + c * 64, k0, b);
        if (VT) tma_load_3d(sm + C::V_LAND + c * BKV * 128, &tmKV, vland, (H + KV + kvh) * HD + c * 64, k0, b);
        else tma_load_3d(sm + C::V_OFF + c * BKV * 128, &tmKV, kvfull, (H + KV + kvh) * HD + c * 64, k0, b);
      }
      int issued = 0;
      bool v_out = !VT;  // stage 1's slot holds V until the elementwise warps have moved it
      for (int it = 0; it < n_it; ++it) {
        const int s = it % NS;
        if (it >= NS && !mbar_wait(&qempty[s], ((it / NS) & 1) ^ 1, abort_flag, err)) break;
        if (!v_out && s == 1) {
          if (!mbar_wait(vmoved, 0, abort_flag, err)) break;
          v_out = true;
        }
        const int g = g_of(it), hh = h_first + g / per_head, q0 = (qb_first + g % per_head) * BQB;
        uint8_t* qs = sm + C::Q_OFF + s * 2 * C::Q_BYTES;
        mbar_arrive_expect_tx(&qfull[s], 2 * C::Q_BYTES);
        for (int c = 0; c < C::NCH; ++c) {
          tma_load_3d(qs + c * BQB * 128, &tmQ, &qfull[s], hh * HD + c * 64, q0, b);
          tma_load_3d(qs + C::Q_BYTES + c * BQB * 128, &tmDO, &qfull[s], hh * HD + c * 64, q0, b);
        }
        issued = it + 1;
      }
      int dummy = 0;  // never leave with copies in flight
      mbar_wait(kvfull, 0, &dummy, err);
      if (VT) mbar_wait(vland, 0, &dummy, err);
      for (int it = (issued > NS ? issued - NS : 0); it < issued; ++it)
        mbar_wait(&qfull[it % NS], (it / NS) & 1, &dummy, err);
    }
  } else if (warp == 5) {
    if (lane == 0) {
      constexpr uint32_t id_s = idesc_f16_f32(BKV, BQB, false);  // S^T = K Q^T, dP^T = V dO^T
      constexpr uint32_t id_a = idesc_f16_f32(BKV, DC, true);    // dV += P^T dO, dK += dS^T Q (N-major B)
      bool ok = mbar_wait(kvfull, 0, abort_flag, err);
      const uint32_t k_addr = smem_u32(sm + C::K_OFF), v_addr = smem_u32(sm + C::V_OFF);
      auto scores = [&](int j) -> bool {
        const int s = j % NS, bf = j % NSB;
        if (!mbar_wait(&qfull[s], (j / NS) & 1, abort_flag, err)) return false;
        if (j >= NSB && !mbar_wait(&sfree[bf], ((j / NSB) & 1) ^ 1, abort_flag, err)) return false;
        if (VT && j == 0 && !mbar_wait(vmoved, 0, abort_flag, err)) return false;  // V is in TMEM
        tc_fence_after();
        const uint32_t q_addr = smem_u32(sm + C::Q_OFF + s * 2 * C::Q_BYTES), do_addr = q_addr + C::Q_BYTES;
        const uint32_t ts = tmem + C::TM_S + 128 * bf;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint32_t ka = (kk >> 2) * (BKV * 128) + (kk & 3) * 32, qa = (kk >> 2) * (BQB * 128) + (kk & 3) * 32;
          tc_mma_f16(ts, smem_desc_sw128(k_addr + ka, 16, 1024), smem_desc_sw128(q_addr + qa, 16, 1024), id_s,
                     kk > 0 ? 1u : 0u);
          if (VT)  // 16 hd elements of V = 8 TMEM columns
            tc_mma_f16_ta(ts + 64, tmem + C::TM_V + 8 * kk, smem_desc_sw128(do_addr + qa, 16, 1024), id_s,
                          kk > 0 ? 1u : 0u);
          else
            tc_mma_f16(ts + 64, smem_desc_sw128(v_addr + ka, 16, 1024), smem_desc_sw128(do_addr + qa, 16, 1024), id_s,
                       kk > 0 ? 1u : 0u);
        }
        tc_commit(&sfull[bf]);
        return true;
      };
      auto accumulate = [&](int i) -> bool {
        const int p = i % NPB, s = i % NS;
        if (!mbar_wait(&pready[p], (i / NPB) & 1, abort_flag, err)) return false;
        tc_fence_after();
        const uint32_t q_addr = smem_u32(sm + C::Q_OFF + s * 2 * C::Q_BYTES), do_addr = q_addr + C::Q_BYTES;
        const uint32_t pt = smem_u32(sm + C::P_OFF + p * 2 * C::P_BYTES), dst = pt + C::P_BYTES;
        const uint32_t cb = (c0 / 64) * (BQB * 128);  // first 64-column chunk of this CTA's columns
#pragma unroll
        for (int kk = 0; kk < BQB / 16; ++kk) {
          const uint64_t bq = smem_desc_sw128(q_addr + cb + kk * 16 * 128, BQB * 128, 1024);
          const uint64_t bo = smem_desc_sw128(do_addr + cb + kk * 16 * 128, BQB * 128, 1024);
          const uint32_t acc = (i > 0 || kk > 0) ? 1u : 0u;
          tc_mma_f16(tmem + C::TM_DV, smem_desc_sw128(pt + kk * 32, 16, 1024), bo, id_a, acc);
          tc_mma_f16(tmem + C::TM_DK, smem_desc_sw128(dst + kk * 32, 16, 1024), bq, id_a, acc);
        }
        tc_commit(&pdone[p]);
        tc_commit(&qempty[s]);
        return true;
      };
      for (int j = 0; ok && j <= n_it; ++j) {
        if (NS == 1) {
          if (j >= 1 && !(ok = accumulate(j - 1))) break;
          if (j < n_it && !(ok = scores(j))) break;
        } else {
          if (j < n_it && !(ok = scores(j))) break;
          if (j >= 1 && !(ok = accumulate(j - 1))) break;
        }
      }
      tc_commit(dfull);
    }
  } else {
    // ---------------------------------------------------------------- P^T, dS^T (warps 0-3)
    const int r = threadIdx.x, kr = k0 + r;
    const uint32_t lane_off = static_cast<uint32_t>(32 * warp) << 16;
    const float sc = kLog2e * rsqrtf(static_cast<float>(HD));
    // thread r < 64 carries lse * log2e of query q0 + r, thread r >= 64 D of query q0 + r - 64;
    // the value of iteration j + 1 is loaded while iteration j runs
    auto vec_load = [&](int j) -> float {
      const int g = g_of(j), hh = h_first + g / per_head, q = (qb_first + g % per_head) * BQB + (r % BQB);
      const int64_t li = (static_cast<int64_t>(b) * H + hh) * S + q;
      return (q < S && r < 2 * BQB) ? (r < BQB ? lse[li] * kLog2e : dvec[li]) : 0.0f;
    };
    float vnext = n_it > 0 ? vec_load(0) : 0.0f;
    bool ok = true;
    if (VT) {
      // thread r copies key row r of V from stage 1's slot (128-byte swizzled chunks of 64 columns)
      // into TMEM lane r: the 16-byte unit u of chunk c (columns 64 c + 8 u ..) is TMEM columns
      // 32 c + 4 u .. + 3 (two fp16 per column)
      ok = __all_sync(0xffffffffu, mbar_wait(vland, 0, abort_flag, err));
      if (ok) {
#pragma unroll 1
        for (int c = 0; c < C::NCH; ++c) {
          float w[32];
          const uint8_t* row = sm + C::V_LAND + c * BKV * 128 + r * 128;
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const uint4 x = *reinterpret_cast<const uint4*>(row + ((u ^ (r & 7)) << 4));
            w[4 * u] = __uint_as_float(x.x);
            w[4 * u + 1] = __uint_as_float(x.y);
            w[4 * u + 2] = __uint_as_float(x.z);
            w[4 * u + 3] = __uint_as_float(x.w);
          }
          tmem_st32(tmem + lane_off + C::TM_V + 32 * c, w);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(vmoved);  // also after an abort: the waiters do not sit out their limit
    }
    for (int j = 0; ok && j < n_it; ++j) {
      const int q0 = (qb_first + g_of(j) % per_head) * BQB;
      float* lv = vec + (j & 1) * 2 * 64;  // [BQB] lse * log2e, then [BQB] D
      if (r < 2 * BQB) lv[r] = vnext;
      if (j + 1 < n_it) vnext = vec_load(j + 1);
      // every thread of the four warps has written its entry (and, by the same token, finished
      // reading this buffer two iterations ago): a bounded mbarrier, never a named barrier, so an
      // aborting warp cannot leave the others waiting
      mbar_arrive(&vready[j & 1]);
      ok = __all_sync(0xffffffffu, mbar_wait(&vready[j & 1], (j >> 1) & 1, abort_flag, err));
      if (!ok) break;
      ok = __all_sync(0xffffffffu, mbar_wait(&sfull[j % NSB], (j / NSB) & 1, abort_flag, err));
      if (!ok) break;
      tc_fence_after();
      const uint32_t ts = tmem + lane_off + C::TM_S + 128 * (j % NSB);
      float sv[BQB], dp[BQB];
      if constexpr (BQB == 64) {
        tmem_ld64(ts, sv);
        tmem_ld64(ts + 64, dp);
      } else {
        tmem_ld32(ts, sv);
        tmem_ld32(ts + 64, dp);
      }
      tc_fence_before();  // the score buffer may be overwritten once every warp has read it
      __syncwarp();
      if (lane == 0) mbar_arrive(&sfree[j % NSB]);
#pragma unroll
      for (int e = 0; e < BQB; ++e) {
        const int q = q0 + e;
        const bool vis = kr <= q && q < S && kr < S && (!WIN || q - kr < W);
        const float pv = vis ? exp2f(sv[e] * sc - lv[e]) : 0.0f;
        sv[e] = pv;
        dp[e] = pv * (dp[e] - lv[BQB + e]);
      }
      if (j >= NPB) {  // the P^T / dS^T buffer is free once the products of block j - NPB retired
        const int i = j - NPB;
        ok = __all_sync(0xffffffffu, mbar_wait(&pdone[i % NPB], (i / NPB) & 1, abort_flag, err));
        if (!ok) break;
      }
      uint8_t* prow = sm + C::P_OFF + (j % NPB) * 2 * C::P_BYTES + r * 128;
#pragma unroll
      for (int qd = 0; qd < BQB / 8; ++qd) {  // 8 queries per 16-byte unit
        const int off = (qd ^ (r & 7)) << 4;
        *reinterpret_cast<uint4*>(prow + off) =
            make_uint4(pack_half2(sv[8 * qd], sv[8 * qd + 1]), pack_half2(sv[8 * qd + 2], sv[8 * qd + 3]),
                       pack_half2(sv[8 * qd + 4], sv[8 * qd + 5]), pack_half2(sv[8 * qd + 6], sv[8 * qd + 7]));
        *reinterpret_cast<uint4*>(prow + C::P_BYTES + off) =
            make_uint4(pack_half2(dp[8 * qd], dp[8 * qd + 1]), pack_half2(dp[8 * qd + 2], dp[8 * qd + 3]),
                       pack_half2(dp[8 * qd + 4], dp[8 * qd + 5]), pack_half2(dp[8 * qd + 6], dp[8 * qd + 7]));
      }
      fence_proxy_async_smem();  // the MMA (async proxy) reads P^T and dS^T
      __syncwarp();
      if (lane == 0) mbar_arrive(&pready[j % NPB]);
    }
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(dfull, 0, abort_flag, err));
    tc_fence_after();
    if (ok && split) {
      // fp32 partials of this (head, part); an item without query blocks writes zeros
      const float inv = rsqrtf(static_cast<float>(HD));
      const int nb64 = (S + 63) / 64;
      const int64_t slot = ((static_cast<int64_t>(b) * nb64 + 2 * kb + r / 64) * H + hsel) * P + part;
      float* pk = so.wk + slot * (64 * HD) + (r % 64) * HD + c0;
      float* pv = so.wv + slot * (64 * HD) + (r % 64) * HD + c0;
#pragma unroll 1
      for (int c = 0; c < DC / 32; ++c) {
        float dk[32], dv[32];
        tmem_ld32(tmem + lane_off + C::TM_DK + 32 * c, dk);
        tmem_ld32(tmem + lane_off + C::TM_DV + 32 * c, dv);
        if (kr < S) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const bool z = n_it == 0;
            __stcg(reinterpret_cast<float4*>(pk + 32 * c + 4 * i),
                   z ? make_float4(0.0f, 0.0f, 0.0f, 0.0f)
                     : make_float4(dk[4 * i] * inv, dk[4 * i + 1] * inv, dk[4 * i + 2] * inv, dk[4 * i + 3] * inv));
            __stcg(reinterpret_cast<float4*>(pv + 32 * c + 4 * i),
                   z ? make_float4(0.0f, 0.0f, 0.0f, 0.0f)
                     : make_float4(dv[4 * i], dv[4 * i + 1], dv[4 * i + 2], dv[4 * i + 3]));
          }
        }
      }
    } else if (ok) {
      const float inv = rsqrtf(static_cast<float>(HD));
      const int64_t tok = static_cast<int64_t>(b) * S + kr;
      // every key block below S is seen by at least its own query block, so n_it >= 1
#pragma unroll 1
      for (int c = 0; c < DC / 32; ++c) {
        float dk[32], dv[32];
        tmem_ld32(tmem + lane_off + C::TM_DK + 32 * c, dk);
        tmem_ld32(tmem + lane_off + C::TM_DV + 32 * c, dv);
        if (kr < S) {
          uint4* pk = reinterpret_cast<uint4*>(dqkv + tok * ld + (H + kvh) * HD + c0 + 32 * c);
          uint4* pv = reinterpret_cast<uint4*>(dqkv + tok * ld + (H + KV + kvh) * HD + c0 + 32 * c);
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            pk[i] = make_uint4(pack_half2(dk[8 * i] * inv, dk[8 * i + 1] * inv),
                               pack_half2(dk[8 * i + 2] * inv, dk[8 * i + 3] * inv),
                               pack_half2(dk[8 * i + 4] * inv, dk[8 * i + 5] * inv),
                               pack_half2(dk[8 * i + 6] * inv, dk[8 * i + 7] * inv));
            pv[i] = make_uint4(pack_half2(dv[8 * i], dv[8 * i + 1]), pack_half2(dv[8 * i + 2], dv[8 * i + 3]),
                               pack_half2(dv[8 * i + 4], dv[8 * i + 5]), pack_half2(dv[8 * i + 6], dv[8 * i + 7]));
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    if (lane == 0) {
      int dummy = 0;
      mbar_wait(dfull, 0, &dummy, err);
    }
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int HD>
struct Dq {
  // hd 256: dO lives in TMEM as the A operand of dP = dO V^T (as V does in the dK/dV kernel),
  // freeing 64 KB for a second (K, V) stage; dO lands in that stage's slot once and the dS warps
  // copy it row by row into TMEM before the loop.
  static constexpr bool DT = HD == 256;
  static constexpr int QB = bwd_block<HD>();                      // keys per iteration
  static constexpr int NS = HD == 256 ? 2 : (HD == 128 ? 3 : 4);  // (K_j, V_j) stages
  static constexpr int NPB = 2;                                   // dS buffers
  static constexpr int NSB = DT ? 1 : 2;                          // S / dP buffers in TMEM
  static constexpr int NCH = HD / 64;
  static constexpr int Q_BYTES = BQ * HD * 2;    // one of Q, dO
  static constexpr int K_BYTES = QB * HD * 2;    // one of K_j, V_j
  static constexpr int P_BYTES = BQ * 64 * 2;    // one dS buffer (128-byte rows)
  static constexpr int Q_OFF = 0, DO_OFF = Q_BYTES;  // (DO_OFF unused when DT)
  static constexpr int K_OFF = DT ? Q_BYTES : 2 * Q_BYTES;  // stage s: K at K_OFF + 2 s K_BYTES, V after it
  static constexpr int D_LAND = K_OFF + 2 * K_BYTES;        // DT: dO passes through stage 1
  static constexpr int P_OFF = K_OFF + NS * 2 * K_BYTES;
  static constexpr int BAR_OFF = P_OFF + NPB * P_BYTES;
  static constexpr int SMEM = BAR_OFF + 256 + 1024;
  // S / dP buffer b: TM_S + 128 b (+64); dO (DT): 256 fp16 per query row packed in 128 columns
  static constexpr uint32_t TM_DQ = 0, TM_DO = 256, TM_S = DT ? 384 : 256;
  static_assert(!DT || 2 * K_BYTES == Q_BYTES, "dO fits the second stage");
};

// One dQ item: x = head * P + part, sequence b, query tile nqb - 1 - z (the longest first).
template <int HD, bool WIN>
__device__ __forceinline__ void dq_body(const CUtensorMap& tmQ, const CUtensorMap& tmKV, const CUtensorMap& tmDO,
                                        int S, int H, int KV, const float* __restrict__ lse,
                                        const float* __restrict__ dvec, uint16_t* __restrict__ dqkv, int64_t ld,
                                        int W, int* err, const SplitOut& so, int x, int b, int z) {
  using C = Dq<HD>;
  constexpr int NS = C::NS, NPB = C::NPB, BQB = C::QB, NSB = C::NSB;
  constexpr bool DT = C::DT;
  static_assert(C::SMEM <= 232448, "shared memory");
  static_assert(C::SMEM > 232448 / 2, "one CTA per SM (512 TMEM columns each)");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* qfull = reinterpret_cast<uint64_t*>(sm + C::BAR_OFF);
  uint64_t* kfull = qfull + 1;    // [NS]
  uint64_t* kempty = kfull + NS;  // [NS]
  uint64_t* sfull = kempty + NS;  // [2]
  uint64_t* sfree = sfull + 2;    // [2]
  uint64_t* pready = sfree + 2;   // [NPB]
  uint64_t* pdone = pready + NPB; // [NPB]
  uint64_t* dfull = pdone + NPB;
  uint64_t* dland = dfull + 1;    // DT: dO landed in stage 1's slot
  uint64_t* dmoved = dland + 1;   // DT: dO copied into TMEM (stage 1's slot is free again)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(dmoved + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool split = so.P > 0;
  const int P = split ? so.P : 1;
  const int h = x / P, part = x % P;
  const int qb = (S + BQ - 1) / BQ - 1 - z;  // longest rows first
  const int kvh = h / (H / KV);
  const int q0 = qb * BQ;
  const int kend = min(S, q0 + BQ);
  const int kb0 = WIN ? max(0, q0 - W + 1) / BQB : 0;
  const int nkb_all = (kend + BQB - 1) / BQB - kb0;
  const int nkb = part < nkb_all ? (nkb_all - part + P - 1) / P : 0;  // key blocks part, part + P, ...
  auto kblock = [&](int j) { return kb0 + part + j * P; };

  if (threadIdx.x == 0) {
    mbar_init(qfull, 1);
    for (int s = 0; s < NS; ++s) {
      mbar_init(&kfull[s], 1);
      mbar_init(&kempty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sfull[i], 1);
      mbar_init(&sfree[i], 4);
    }
    for (int i = 0; i < NPB; ++i) {
      mbar_init(&pready[i], 4);
      mbar_init(&pdone[i], 1);
    }
    mbar_init(dfull, 1);
    mbar_init(dland, 1);
    mbar_init(dmoved, 4);  // one arrival per dS warp
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 5) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  griddep_wait();  // dvec comes from the kernel right before
  griddep_launch();

  if (warp == 4) {
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmKV);
      tma_prefetch_desc(&tmDO);
      mbar_arrive_expect_tx(qfull, (DT ? 1 : 2) * C::Q_BYTES);
      if (DT) mbar_arrive_expect_tx(dland, C::Q_BYTES);
      for (int c = 0; c < C::NCH; ++c) {
        tma_load_3d(sm + C::Q_OFF + c * BQ * 128, &tmQ, qfull, h * HD + c * 64, q0, b);
        if (DT) tma_load_3d(sm + C::D_LAND + c * BQ * 128, &tmDO, dland, h * HD + c * 64, q0, b);
        else tma_load_3d(sm + C::DO_OFF + c * BQ * 128, &tmDO, qfull, h * HD + c * 64, q0, b);
      }
      int issued = 0;
      bool d_out = !DT;  // stage 1's slot holds dO until the dS warps have moved it
      for (int j = 0; j < nkb; ++j) {
        const int s = j % NS;
        if (j >= NS && !mbar_wait(&kempty[s], ((j / NS) & 1) ^ 1, abort_flag, err)) break;
        if (!d_out && s == 1) {
          if (!mbar_wait(dmoved, 0, abort_flag, err)) break;
          d_out = true;
        }
        uint8_t* ks = sm + C::K_OFF + s * 2 * C::K_BYTES;
        mbar_arrive_expect_tx(&kfull[s], 2 * C::K_BYTES);
        for (int c = 0; c < C::NCH; ++c) {
          tma_load_3d(ks + c * BQB * 128, &tmKV, &kfull[s], (H + kvh) * HD + c * 64, kblock(j) * BQB, b);
          tma_load_3d(ks + C::K_BYTES + c * BQB * 128, &tmKV, &kfull[s], (H + KV + kvh) * HD + c * 64,
                      kblock(j) * BQB, b);
        }
        issued = j + 1;
      }
      int dummy = 0;
      mbar_wait(qfull, 0, &dummy, err);
      if (DT) mbar_wait(dland, 0, &dummy, err);
      for (int j = (issued > NS ? issued - NS : 0); j < issued; ++j)
        mbar_wait(&kfull[j % NS], (j / NS) & 1, &dummy, err);
    }
  } else if (warp == 5) {
    if (lane == 0) {
      constexpr uint32_t id_s = idesc_f16_f32(BQ, BQB, false);  // S = Q K^T, dP = dO V^T
      constexpr uint32_t id_q = idesc_f16_f32(BQ, HD, true);    // dQ += dS K (K is N(hd)-major)
      bool ok = mbar_wait(qfull, 0, abort_flag, err);
      const uint32_t q_addr = smem_u32(sm + C::Q_OFF), do_addr = smem_u32(sm + C::DO_OFF);
      auto scores = [&](int j) -> bool {
        const int s = j % NS, bf = j % NSB;
        if (!mbar_wait(&kfull[s], (j / NS) & 1, abort_flag, err)) return false;
        if (j >= NSB && !mbar_wait(&sfree[bf], ((j / NSB) & 1) ^ 1, abort_flag, err)) return false;
        if (DT && j == 0 && !mbar_wait(dmoved, 0, abort_flag, err)) return false;  // dO is in TMEM
        tc_fence_after();
        const uint32_t k_addr = smem_u32(sm + C::K_OFF + s * 2 * C::K_BYTES), v_addr = k_addr + C::K_BYTES;
        const uint32_t ts = tmem + C::TM_S + 128 * bf;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint32_t qa = (kk >> 2) * (BQ * 128) + (kk & 3) * 32, ka = (kk >> 2) * (BQB * 128) + (kk & 3) * 32;
          tc_mma_f16(ts, smem_desc_sw128(q_addr + qa, 16, 1024), smem_desc_sw128(k_addr + ka, 16, 1024), id_s,
                     kk > 0 ? 1u : 0u);
          if (DT)  // 16 hd elements of dO = 8 TMEM columns
            tc_mma_f16_ta(ts + 64, tmem + C::TM_DO + 8 * kk, smem_desc_sw128(v_addr + ka, 16, 1024), id_s,
                          kk > 0 ? 1u : 0u);
          else
            tc_mma_f16(ts + 64, smem_desc_sw128(do_addr + qa, 16, 1024), smem_desc_sw128(v_addr + ka, 16, 1024),
                       id_s, kk > 0 ? 1u : 0u);
        }
        tc_commit(&sfull[bf]);
        return true;
      };
      auto accumulate = [&](int i) -> bool {
        const int p = i % NPB, s = i % NS;
        if (!mbar_wait(&pready[p], (i / NPB) & 1, abort_flag, err)) return false;
        tc_fence_after();
        const uint32_t k_addr = smem_u32(sm + C::K_OFF + s * 2 * C::K_BYTES);
        const uint32_t ds = smem_u32(sm + C::P_OFF + p * C::P_BYTES);
#pragma unroll
        for (int kk = 0; kk < BQB / 16; ++kk)
          tc_mma_f16(tmem + C::TM_DQ, smem_desc_sw128(ds + kk * 32, 16, 1024),
                     smem_desc_sw128(k_addr + kk * 16 * 128, BQB * 128, 1024), id_q, (i > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&pdone[p]);
        tc_commit(&kempty[s]);
        return true;
      };
      for (int j = 0; ok && j <= nkb; ++j) {
        if (NS == 1) {
          if (j >= 1 && !(ok = accumulate(j - 1))) break;
          if (j < nkb && !(ok = scores(j))) break;
        } else {
          if (j < nkb && !(ok = scores(j))) break;
          if (j >= 1 && !(ok = accumulate(j - 1))) break;
        }
      }
      tc_commit(dfull);
    }
  } else {
    // ---------------------------------------------------------------- dS (warps 0-3)
    const int r = threadIdx.x, row = q0 + r;
    const uint32_t lane_off = static_cast<uint32_t>(32 * warp) << 16;
    const float sc = kLog2e * rsqrtf(static_cast<float>(HD));
    const int64_t li = (static_cast<int64_t>(b) * H + h) * S + row;
    const float l2 = row < S ? lse[li] * kLog2e : 0.0f;
    const float dr = row < S ? dvec[li] : 0.0f;
    bool ok = true;
    if (DT) {
      // thread r copies query row r of dO from stage 1's slot into TMEM lane r (as V in dK/dV)
      ok = __all_sync(0xffffffffu, mbar_wait(dland, 0, abort_flag, err));
      if (ok) {
#pragma unroll 1
        for (int c = 0; c < C::NCH; ++c) {
          float w[32];
          const uint8_t* src = sm + C::D_LAND + c * BQ * 128 + r * 128;
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const uint4 x = *reinterpret_cast<const uint4*>(src + ((u ^ (r & 7)) << 4));
            w[4 * u] = __uint_as_float(x.x);
            w[4 * u + 1] = __uint_as_float(x.y);
            w[4 * u + 2] = __uint_as_float(x.z);
            w[4 * u + 3] = __uint_as_float(x.w);
          }
          tmem_st32(tmem + lane_off + C::TM_DO + 32 * c, w);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(dmoved);  // also after an abort: the waiters do not sit out their limit
    }
    for (int j = 0; ok && j < nkb; ++j) {
      ok = __all_sync(0xffffffffu, mbar_wait(&sfull[j % NSB], (j / NSB) & 1, abort_flag, err));
      if (!ok) break;
      if (j >= NPB) {
        const int i = j - NPB;
        ok = __all_sync(0xffffffffu, mbar_wait(&pdone[i % NPB], (i / NPB) & 1, abort_flag, err));
        if (!ok) break;
      }
      tc_fence_after();
      const uint32_t ts = tmem + lane_off + C::TM_S + 128 * (j % NSB);
      uint8_t* drow = sm + C::P_OFF + (j % NPB) * C::P_BYTES + r * 128;
      const int k0 = kblock(j) * BQB;
      {
        float sv[BQB], dp[BQB];
        if constexpr (BQB == 64) {
          tmem_ld64(ts, sv);
          tmem_ld64(ts + 64, dp);
        } else {
          tmem_ld32(ts, sv);
          tmem_ld32(ts + 64, dp);
        }
        tc_fence_before();  // the score buffer may be overwritten once every warp has read it
        __syncwarp();
        if (lane == 0) mbar_arrive(&sfree[j % NSB]);
#pragma unroll
        for (int e = 0; e < BQB; ++e) {
          const int key = k0 + e;
          const bool vis = key <= row && row < S && (!WIN || row - key < W);
          const float pv = vis ? exp2f(sv[e] * sc - l2) : 0.0f;
          dp[e] = pv * (dp[e] - dr);
        }
#pragma unroll
        for (int kd = 0; kd < BQB / 8; ++kd)
          *reinterpret_cast<uint4*>(drow + ((kd ^ (r & 7)) << 4)) =
              make_uint4(pack_half2(dp[8 * kd], dp[8 * kd + 1]), pack_half2(dp[8 * kd + 2], dp[8 * kd + 3]),
                         pack_half2(dp[8 * kd + 4], dp[8 * kd + 5]), pack_half2(dp[8 * kd + 6], dp[8 * kd + 7]));
      }
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&pready[j % NPB]);
    }
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(dfull, 0, abort_flag, err));
    tc_fence_after();
    if (ok && split) {
      const float inv = rsqrtf(static_cast<float>(HD));
      const int nb64 = (S + 63) / 64;
      const int64_t slot = ((static_cast<int64_t>(b) * nb64 + 2 * qb + r / 64) * H + h) * P + part;
      float* pq = so.wq + slot * (64 * HD) + (r % 64) * HD;
#pragma unroll 1
      for (int c = 0; c < HD / 32; ++c) {
        float t[32];
        tmem_ld32(tmem + lane_off + C::TM_DQ + 32 * c, t);
        if (row < S) {
#pragma unroll
          for (int i = 0; i < 8; ++i)
            __stcg(reinterpret_cast<float4*>(pq + 32 * c + 4 * i),
                   nkb == 0 ? make_float4(0.0f, 0.0f, 0.0f, 0.0f)
                            : make_float4(t[4 * i] * inv, t[4 * i + 1] * inv, t[4 * i + 2] * inv, t[4 * i + 3] * inv));
        }
      }
    } else if (ok) {
      const float inv = rsqrtf(static_cast<float>(HD));
      const int64_t tok = static_cast<int64_t>(b) * S + row;
#pragma unroll 1
      for (int c = 0; c < HD / 32; ++c) {
        float t[32];
        tmem_ld32(tmem + lane_off + C::TM_DQ + 32 * c, t);
        if (row < S) {
          uint4* dst = reinterpret_cast<uint4*>(dqkv + tok * ld + h * HD + 32 * c);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            dst[i] = make_uint4(pack_half2(t[8 * i] * inv, t[8 * i + 1] * inv),
                                pack_half2(t[8 * i + 2] * inv, t[8 * i + 3] * inv),
                                pack_half2(t[8 * i + 4] * inv, t[8 * i + 5] * inv),
                                pack_half2(t[8 * i + 6] * inv, t[8 * i + 7] * inv));
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    if (lane == 0) {
      int dummy = 0;
      mbar_wait(dfull, 0, &dummy, err);
    }
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int HD, bool WIN>
__global__ void __launch_bounds__(BWD_THREADS, 1)
    dkdv_tc_kernel(const __grid_constant__ CUtensorMap tmKV, const __grid_constant__ CUtensorMap tmQ,
                   const __grid_constant__ CUtensorMap tmDO, int S, int H, int KV, const float* __restrict__ lse,
                   const float* __restrict__ dvec, uint16_t* __restrict__ dqkv, int64_t ld, int W, int* err,
                   const SplitOut so, int B) {
  dkdv_body<HD, WIN>(tmKV, tmQ, tmDO, S, H, KV, lse, dvec, dqkv, ld, W, err, so, blockIdx.x, B);
}

template <int HD, bool WIN>
__global__ void __launch_bounds__(BWD_THREADS, 1)
    dq_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKV,
                 const __grid_constant__ CUtensorMap tmDO, int S, int H, int KV, const float* __restrict__ lse,
                 const float* __restrict__ dvec, uint16_t* __restrict__ dqkv, int64_t ld, int W, int* err,
                 const SplitOut so) {
  dq_body<HD, WIN>(tmQ, tmKV, tmDO, S, H, KV, lse, dvec, dqkv, ld, W, err, so, blockIdx.x, blockIdx.y, blockIdx.z);
}

// Split mode as one launch: group L holds the dK/dV items of key tile L and the dQ items of query
// tile nqb - 1 - L (both see nqb - L tiles of the other kind), groups in order, so the longest
// items of both kinds start first and the two kinds run side by side.
template <int HD, bool WIN>
__global__ void __launch_bounds__(BWD_THREADS, 1)
    bwd_split_tc_kernel(const __grid_constant__ CUtensorMap kv128, const __grid_constant__ CUtensorMap q64,
                        const __grid_constant__ CUtensorMap do64, const __grid_constant__ CUtensorMap q128,
                        const __grid_constant__ CUtensorMap kv64, const __grid_constant__ CUtensorMap do128, int S,
                        int H, int KV, const float* __restrict__ lse, const float* __restrict__ dvec,
                        uint16_t* __restrict__ dqkv, int64_t ld, int W, int* err, const SplitOut so, int B) {
  const int nd = B * H * DkDv<HD>::NCOL * so.P, nq = H * so.P * B;
  const int L = static_cast<int>(blockIdx.x) / (nd + nq), r = static_cast<int>(blockIdx.x) % (nd + nq);
  if (r < nd)
    dkdv_body<HD, WIN>(kv128, q64, do64, S, H, KV, lse, dvec, dqkv, ld, W, err, so, L * nd + r, B);
  else
    dq_body<HD, WIN>(q128, kv64, do128, S, H, KV, lse, dvec, dqkv, ld, W, err, so, (r - nd) % (H * so.P),
                     (r - nd) / (H * so.P), L);
}

template <int HD, bool WIN>
int bwd_launch(const uint16_t* qkv, int64_t ld, const uint16_t* dout, int64_t ldo, const float* lse,
               const float* dvec, int B, int S, int H, int KV, int W, uint16_t* dqkv, int* err, const SplitOut& so,
               cudaStream_t st) {
  constexpr int SPLIT_SMEM = DkDv<HD>::SMEM > Dq<HD>::SMEM ? DkDv<HD>::SMEM : Dq<HD>::SMEM;
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(dkdv_tc_kernel<HD, WIN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             DkDv<HD>::SMEM) != cudaSuccess ||
        cudaFuncSetAttribute(dq_tc_kernel<HD, WIN>, cudaFuncAttributeMaxDynamicSharedMemorySize, Dq<HD>::SMEM) !=
            cudaSuccess ||
        cudaFuncSetAttribute(bwd_split_tc_kernel<HD, WIN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             SPLIT_SMEM) != cudaSuccess) {
      cudaGetLastError();
      return MEBP_ERR_CUDA;
    }
    attr = true;
  }
  const uint64_t seq_q = static_cast<uint64_t>(S) * ld * 2, seq_o = static_cast<uint64_t>(S) * ldo * 2;
  constexpr int QB = bwd_block<HD>();  // box rows of the 32 / 64-row operand blocks
  CUtensorMap kv128, q64, do64, q128, kv64, do128;
  int rc;
  if ((rc = make_tmap_3d(&kv128, qkv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, ld, S, B, ld * 2, seq_q, 64, BKV, 1,
                         CU_TENSOR_MAP_SWIZZLE_128B)) ||
      (rc = make_tmap_3d(&q64, qkv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, ld, S, B, ld * 2, seq_q, 64, QB, 1,
                         CU_TENSOR_MAP_SWIZZLE_128B)) ||
      (rc = make_tmap_3d(&do64, dout, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, ldo, S, B, ldo * 2, seq_o, 64, QB, 1,
                         CU_TENSOR_MAP_SWIZZLE_128B)) ||
      (rc = make_tmap_3d(&q128, qkv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, ld, S, B, ld * 2, seq_q, 64, BQ, 1,
                         CU_TENSOR_MAP_SWIZZLE_128B)) ||
      (rc = make_tmap_3d(&kv64, qkv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, ld, S, B, ld * 2, seq_q, 64, QB, 1,
                         CU_TENSOR_MAP_SWIZZLE_128B)) ||
      (rc = make_tmap_3d(&do128, dout, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, ldo, S, B, ldo * 2, seq_o, 64, BQ, 1,
                         CU_TENSOR_MAP_SWIZZLE_128B)))
    return rc;
  const int nkb = (S + BKV - 1) / BKV;
  if (so.P > 0) {  // 128-key and 128-query tiles pair up group by group (nkb of each)
    const int64_t n = static_cast<int64_t>(nkb) * (B * H * DkDv<HD>::NCOL * so.P + H * so.P * B);
    launch_k(bwd_split_tc_kernel<HD, WIN>, dim3(static_cast<unsigned>(n)), BWD_THREADS, SPLIT_SMEM, st, kv128, q64,
             do64, q128, kv64, do128, S, H, KV, lse, dvec, dqkv, ld, W, err, so, B);
  } else {
    const int64_t n_dkdv = static_cast<int64_t>(nkb) * B * KV * DkDv<HD>::NCOL;
    launch_k(dkdv_tc_kernel<HD, WIN>, dim3(static_cast<unsigned>(n_dkdv)), BWD_THREADS, DkDv<HD>::SMEM, st, kv128,
             q64, do64, S, H, KV, lse, dvec, dqkv, ld, W, err, so, B);
    launch_k(dq_tc_kernel<HD, WIN>, dim3(H, B, (S + BQ - 1) / BQ), BWD_THREADS, Dq<HD>::SMEM, st, q128, kv64, do128,
             S, H, KV, lse, dvec, dqkv, ld, W, err, so);
  }
  return cudaGetLastError() == cudaSuccess ? MEBP_OK : MEBP_ERR_CUDA;
}

}  // namespace atc

int launch_attn_fwd_tc(const uint16_t* qkv, int64_t ld, int B, int S, int H, int KV, int hd, uint16_t* o, int64_t ldo,
                       float* lse, int window, int* err, cudaStream_t st) {
  const int W = window >= S ? 0 : window;  // a window covering the sequence is plain causal
  if (ld % 64 || ldo % 8) return MEBP_ERR_INVALID_ARG;
  switch (hd) {
    case 64: return W ? atc::fwd_launch<64, true>(qkv, ld, B, S, H, KV, o, ldo, lse, W, err, st)
                      : atc::fwd_launch<64, false>(qkv, ld, B, S, H, KV, o, ldo, lse, 0, err, st);
    case 128: return W ? atc::fwd_launch<128, true>(qkv, ld, B, S, H, KV, o, ldo, lse, W, err, st)
                       : atc::fwd_launch<128, false>(qkv, ld, B, S, H, KV, o, ldo, lse, 0, err, st);
    case 256: return W ? atc::fwd_launch<256, true>(qkv, ld, B, S, H, KV, o, ldo, lse, W, err, st)
                       : atc::fwd_launch<256, false>(qkv, ld, B, S, H, KV, o, ldo, lse, 0, err, st);
    default: return MEBP_ERR_UNSUPPORTED;
  }
}

}  // namespace mebp

namespace mebp {
int launch_attn_bwd_tc(const uint16_t* qkv, int64_t ld, const uint16_t* dout, int64_t ldo, const float* lse,
                       const float* dvec, int B, int S, int H, int KV, int hd, uint16_t* dqkv, int window, int parts,
                       float* wk, float* wv, float* wq, int* err, cudaStream_t st) {
  const int W = window >= S ? 0 : window;
  if (ld % 64 || ldo % 64) return MEBP_ERR_INVALID_ARG;
  const atc::SplitOut so{parts, wk, wv, wq};
  switch (hd) {
    case 64: return W ? atc::bwd_launch<64, true>(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, W, dqkv, err, so, st)
                      : atc::bwd_launch<64, false>(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, 0, dqkv, err, so, st);
    case 128: return W ? atc::bwd_launch<128, true>(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, W, dqkv, err, so, st)
                       : atc::bwd_launch<128, false>(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, 0, dqkv, err, so, st);
    case 256: return W ? atc::bwd_launch<256, true>(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, W, dqkv, err, so, st)
                       : atc::bwd_launch<256, false>(qkv, ld, dout, ldo, lse, dvec, B, S, H, KV, 0, dqkv, err, so, st);
    default: return MEBP_ERR_UNSUPPORTED;
  }
}
}  // namespace mebp
