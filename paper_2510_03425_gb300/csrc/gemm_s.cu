// Narrow-tile fused dequant-GEMM for few-token (latency-bound) projections: the computation of
// gemm.cu (Algorithm 1's LazyLoadAndDecompressWeights fused into the mainloop, bit-exact fp16
// operand decode, fp32 TMEM accumulation, the rank-r LoRA block as extra K steps) on 128 x 64
// output tiles.  At a few hundred tokens the 128 x 256 tiles leave most SMs idle; instead of
// splitting K (partial tiles plus a reduction), the narrow tiles give every SM its own tile and
// a K loop whose per-step MMA is short, so the loop runs at the pace of its barrier hand-offs.
//
// 192 threads: warps 0-3 decode (two threads per weight row) and then run the epilogue (warp w
// reads TMEM lanes 32w ..), warp 4 issues TMA, warp 5 issues tcgen05.mma and owns the 64-column
// TMEM allocation.  About 100 KB of shared memory: two CTAs per SM.  Every wait is bounded (2 s)
// with a CTA abort flag and the device error word; copies and MMAs are drained before exit.
#include <cudaTypedefs.h>

#include "dequant.cuh"
#include "kernels.h"

namespace mebp {
namespace gemms {

constexpr int BM = 128, BN = 64, BK = 64;
constexpr int CONV = 4;
constexpr int TMA_WARP = CONV, MMA_WARP = CONV + 1;
constexpr int THREADS = (CONV + 2) * 32;
constexpr int A_BYTES = BM * BK * 2;
constexpr int P_BYTES = BN * BK / 2;
constexpr int S_BYTES = 128;
constexpr int B_BYTES = BN * BK * 2;
constexpr uint32_t TMEM_COLS = 64;
// Shared-memory layout for KCH chunks of 64 K per pipeline stage: a TMA slot holds KCH activation
// tiles, then KCH packed weight tiles, then KCH scale rows; a decode slot holds KCH decoded tiles.
// KCH = 1: four TMA slots and three decode slots, two CTAs per SM.  KCH = 2 (grids of at most one
// CTA per SM): half as many stages, so half the barrier hand-offs for the same K.
template <int KCH>
struct Lay {
  static constexpr int TSTG = KCH == 1 ? 4 : 3, BSTG = KCH == 1 ? 3 : 2;
  static constexpr int A_OFF = 0, P_OFF = KCH * A_BYTES, S_OFF = P_OFF + KCH * P_BYTES;
  static constexpr int T_STRIDE = (S_OFF + KCH * S_BYTES + 1023) / 1024 * 1024;
  static constexpr int B_SLOT = KCH * B_BYTES;
  static constexpr int B_BASE = TSTG * T_STRIDE;
  static constexpr int BAR_OFF = B_BASE + BSTG * B_SLOT;
  static constexpr int SMEM = BAR_OFF + 512 + 1024;
};
static_assert(2 * Lay<1>::SMEM <= 232448, "two CTAs per SM");
static_assert(Lay<2>::SMEM <= 232448, "one CTA per SM");

struct Params {
  int M, N, K;
  int kx_steps, kx;
  const uint16_t* Bx;
  int64_t ldbx;
  int epi;  // EPI_F16 or EPI_F32
  void* C;
  int64_t ldc;
  const float* R;
  int64_t ldr;
  float alpha;
  int* err;
};

// FWD: packed tile [64 rows][32 B], scales [64]; thread t: row r = t >> 1, words 4h .. 4h+3
// (h = t & 1) -> chunks 4h .. 4h+3 of row r of the K-major SW128 tile (chunk j at j ^ (r&7)).
__device__ __forceinline__ void convert_fwd(const uint8_t* pk, const uint8_t* sc, uint8_t* bt, int t) {
  const int r = t >> 1, h = t & 1;
  const uint4 p = reinterpret_cast<const uint4*>(pk + r * 32)[h];
  const uint32_t s2 = scale_pair(reinterpret_cast<const uint16_t*>(sc)[r]);
  uint8_t* row = bt + r * 128;
  const uint32_t words[4] = {p.x, p.y, p.z, p.w};
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    const int j = 4 * h + w;
    uint32_t o[4];
    dequant_word(words[w], s2, o);
    *reinterpret_cast<uint4*>(row + ((j ^ (r & 7)) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// TRANS: packed tile [64 k-rows][32 B] (64 output columns), scales [64 k-rows] (one group).
// Thread t: row k = t & 63, packed chunk c = t >> 6 (columns 32c .. 32c+31) -> chunks 4c .. 4c+3
// of row k of the MN-major SW128 atom (64 columns x 64 k-rows, chunk j at j ^ (k&7)).
__device__ __forceinline__ void convert_trans(const uint8_t* pk, const uint8_t* sc, uint8_t* bt, int t) {
  const int k = t & 63, c = t >> 6;
  const uint4 p = *reinterpret_cast<const uint4*>(pk + k * 32 + c * 16);
  const uint32_t s2 = scale_pair(reinterpret_cast<const uint16_t*>(sc)[k]);
  uint8_t* row = bt + k * 128;
  const uint32_t words[4] = {p.x, p.y, p.z, p.w};
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    const int j = 4 * c + w;
    uint32_t o[4];
    dequant_word(words[w], s2, o);
    *reinterpret_cast<uint4*>(row + ((j ^ (k & 7)) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// LoRA block e: the 64-wide slice of B_x into the B slot (zero outside [0, kx) x [0, N)).
template <bool TRANS>
__device__ __forceinline__ void copy_lora_b(const Params& p, int e, int n0, uint8_t* bt, int t) {
  const uint4 zero = make_uint4(0, 0, 0, 0);
  if (!TRANS) {  // K-major: row r = output column n0 + r, chunk j = 8 rank columns
    const int r = t >> 1, h = t & 1, n = n0 + r;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const int j = 4 * h + w;
      const int col = e * 64 + 8 * j;
      uint4 v = zero;
      if (n < p.N && col < p.kx) v = *reinterpret_cast<const uint4*>(p.Bx + static_cast<int64_t>(n) * p.ldbx + col);
      *reinterpret_cast<uint4*>(bt + r * 128 + ((j ^ (r & 7)) << 4)) = v;
    }
  } else {       // MN-major: row k of the rank axis, columns 32c .. 32c+31 of the tile
    const int k = t & 63, c = t >> 6;
    const int rr = e * 64 + k;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const int j = 4 * c + w;
      const int col = n0 + 8 * j;
      uint4 v = zero;
      if (rr < p.kx && col < p.N) v = *reinterpret_cast<const uint4*>(p.Bx + static_cast<int64_t>(rr) * p.ldbx + col);
      *reinterpret_cast<uint4*>(bt + k * 128 + ((j ^ (k & 7)) << 4)) = v;
    }
  }
}

// Warp w: output row m0 + 32w + lane, the tile's 64 columns.
__device__ __forceinline__ void epilogue(const Params& p, uint32_t tmem, int warp, int lane, int m0, int n0) {
  const int row = m0 + 32 * warp + lane;
  const uint32_t tb = tmem + (static_cast<uint32_t>(32 * warp) << 16);
  uint32_t bad = 0;  // an fp16 output overflowed (or is NaN)
#pragma unroll 1
  for (int cc = 0; cc < 2; ++cc) {
    float v[32];
    tmem_ld32(tb + 32 * cc, v);
    const int c0 = n0 + 32 * cc;
    if (row >= p.M || c0 >= p.N) continue;
    if (p.epi == EPI_F16) {
      uint4* dst = reinterpret_cast<uint4*>(static_cast<uint16_t*>(p.C) + static_cast<int64_t>(row) * p.ldc + c0);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint4 o = make_uint4(pack_half2(v[8 * i], v[8 * i + 1]), pack_half2(v[8 * i + 2], v[8 * i + 3]),
                                   pack_half2(v[8 * i + 4], v[8 * i + 5]), pack_half2(v[8 * i + 6], v[8 * i + 7]));
        bad |= h2_nonfinite(o.x) | h2_nonfinite(o.y) | h2_nonfinite(o.z) | h2_nonfinite(o.w);
        dst[i] = o;
      }
    } else {  // EPI_F32 (+ residual, which may alias C)
      float4* dst = reinterpret_cast<float4*>(static_cast<float*>(p.C) + static_cast<int64_t>(row) * p.ldc + c0);
      const float4* res = p.R ? reinterpret_cast<const float4*>(p.R + static_cast<int64_t>(row) * p.ldr + c0) : nullptr;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        float4 o = make_float4(p.alpha * v[4 * i], p.alpha * v[4 * i + 1], p.alpha * v[4 * i + 2],
                               p.alpha * v[4 * i + 3]);
        if (res) {
          const float4 r = res[i];
          o.x += r.x; o.y += r.y; o.z += r.z; o.w += r.w;
        }
        dst[i] = o;
      }
    }
  }
  if (bad) flag_error(p.err, kErrNonFinite);
}

template <bool TRANS, int KCH>
__global__ void __launch_bounds__(THREADS, KCH == 1 ? 2 : 1)
    dequant_gemm_narrow(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmP,
                        const __grid_constant__ CUtensorMap tmS, const __grid_constant__ CUtensorMap tmAx,
                        const Params p) {
  using L = Lay<KCH>;
  constexpr int TSTG = L::TSTG, BSTG = L::BSTG, T_STRIDE = L::T_STRIDE, B_BASE = L::B_BASE;
  constexpr int A_OFF = L::A_OFF, P_OFF = L::P_OFF, S_OFF = L::S_OFF;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* wfull = reinterpret_cast<uint64_t*>(smem + L::BAR_OFF);  // packed weights + scales landed
  uint64_t* afull = wfull + TSTG;                                  // activation tile landed
  uint64_t* empty = afull + TSTG;                                  // MMA done with the TMA slot
  uint64_t* bfull = empty + TSTG;                                  // decoded tile ready
  uint64_t* bempty = bfull + BSTG;                                 // MMA done with the B slot
  uint64_t* accf = bempty + BSTG;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accf + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  griddep_launch();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * BM;
  // chunks of 64 K: main ones, then the LoRA block's (each up to four k16 steps); stage it holds
  // chunks it*KCH .. of the main sequence (it < num_main), then of the LoRA sequence
  const int nch_main = p.K / BK, nch_lora = (p.kx_steps + 3) / 4;
  const int num_main = (nch_main + KCH - 1) / KCH;
  const int total = num_main + (nch_lora + KCH - 1) / KCH;
  auto stage_chunks = [&](int it) {
    return it < num_main ? min(KCH, nch_main - it * KCH) : min(KCH, nch_lora - (it - num_main) * KCH);
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < TSTG; ++s) {
      mbar_init(&wfull[s], 1);
      mbar_init(&afull[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < BSTG; ++b) {
      mbar_init(&bfull[b], CONV);
      mbar_init(&bempty[b], 1);
    }
    mbar_init(accf, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == MMA_WARP) tmem_alloc(tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == TMA_WARP) {
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmP);
      tma_prefetch_desc(&tmS);
      auto load_w = [&](int it) {
        const int s = it % TSTG, nch = stage_chunks(it);
        uint8_t* st = smem + s * T_STRIDE;
        mbar_arrive_expect_tx(&wfull[s], nch * (P_BYTES + S_BYTES));
        for (int c = 0; c < nch; ++c) {
          const int kc = it * KCH + c;
          if (!TRANS) {
            tma_load_2d(st + P_OFF + c * P_BYTES, &tmP, &wfull[s], kc * (BK / 2), n0);  // packed [N, K/2]
            tma_load_2d(st + S_OFF + c * S_BYTES, &tmS, &wfull[s], n0, kc);             // scales [K/64, N]
          } else {
            tma_load_2d(st + P_OFF + c * P_BYTES, &tmP, &wfull[s], n0 / 2, kc * BK);    // packed [K, N/2]
            tma_load_2d(st + S_OFF + c * S_BYTES, &tmS, &wfull[s], kc * BK, n0 / 64);   // scales [N/64, K]
          }
        }
      };
      // The packed weights are never written by a kernel of the same call (and the first kernel
      // of a call is a normal launch), so the first slots' weights load before the wait.
      int w_issued = 0, a_issued = 0;
      for (; w_issued < min(TSTG, num_main); ++w_issued) load_w(w_issued);
      griddep_wait();
      for (int it = 0; it < total; ++it) {
        const int s = it % TSTG;
        if (it >= TSTG && !mbar_wait(&empty[s], ((it / TSTG) & 1) ^ 1, abort_flag, p.err)) break;
        if (it < num_main && it >= w_issued) load_w(w_issued++);
        uint8_t* st = smem + s * T_STRIDE;
        const int nch = stage_chunks(it);
        mbar_arrive_expect_tx(&afull[s], nch * A_BYTES);
        for (int c = 0; c < nch; ++c) {
          if (it < num_main) tma_load_2d(st + A_OFF + c * A_BYTES, &tmA, &afull[s], (it * KCH + c) * BK, m0);
          else tma_load_2d(st + A_OFF + c * A_BYTES, &tmAx, &afull[s], ((it - num_main) * KCH + c) * BK, m0);
        }
        a_issued = it + 1;
      }
      int dummy = 0;
      for (int i = (w_issued > TSTG ? w_issued - TSTG : 0); i < w_issued; ++i)
        mbar_wait(&wfull[i % TSTG], (i / TSTG) & 1, &dummy, p.err);
      for (int i = (a_issued > TSTG ? a_issued - TSTG : 0); i < a_issued; ++i)
        mbar_wait(&afull[i % TSTG], (i / TSTG) & 1, &dummy, p.err);
    }
  } else if (warp == MMA_WARP) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f16_f32(BM, BN, TRANS);
      for (int it = 0; it < total; ++it) {
        const int s = it % TSTG, b = it % BSTG;
        if (!mbar_wait(&afull[s], (it / TSTG) & 1, abort_flag, p.err)) break;
        if (!mbar_wait(&bfull[b], (it / BSTG) & 1, abort_flag, p.err)) break;
        tc_fence_after();
        // the stage's first-slice descriptors; later k16 slices advance the start-address field,
        // later chunks start one tile further (A: A_BYTES, B: B_BYTES)
        const uint64_t ad0 = smem_desc_sw128(smem_u32(smem + s * T_STRIDE + A_OFF), 16, 1024);
        const uint64_t bd0 = TRANS ? smem_desc_sw128(smem_u32(smem + B_BASE + b * L::B_SLOT), 8192, 1024)
                                   : smem_desc_sw128(smem_u32(smem + B_BASE + b * L::B_SLOT), 16, 1024);
        constexpr uint64_t A_K16 = 32 >> 4, B_K16 = (TRANS ? 2048 : 32) >> 4;
        constexpr uint64_t A_CH = A_BYTES >> 4, B_CH = B_BYTES >> 4;
        const int nch = stage_chunks(it);
        if (it < num_main && nch == KCH) {
#pragma unroll
          for (int c = 0; c < KCH; ++c)
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc_mma_f16(tmem, ad0 + c * A_CH + kk * A_K16, bd0 + c * B_CH + kk * B_K16, idesc,
                         (it > 0 || c > 0 || kk > 0) ? 1u : 0u);
        } else {
          for (int c = 0; c < nch; ++c) {
            const int nk = it < num_main ? 4 : min(4, p.kx_steps - 4 * ((it - num_main) * KCH + c));
            for (int kk = 0; kk < nk; ++kk)
              tc_mma_f16(tmem, ad0 + c * A_CH + kk * A_K16, bd0 + c * B_CH + kk * B_K16, idesc,
                         (it > 0 || c > 0 || kk > 0) ? 1u : 0u);
          }
        }
        tc_commit(&empty[s]);
        tc_commit(&bempty[b]);
      }
      tc_commit(accf);
    }
  } else {
    // converters, then the epilogue
    const int t = threadIdx.x;  // 0 .. 127
    for (int it = 0; it < total; ++it) {
      const int s = it % TSTG, b = it % BSTG;
      if (!mbar_wait(&bempty[b], ((it / BSTG) & 1) ^ 1, abort_flag, p.err)) break;
      uint8_t* bt = smem + B_BASE + b * L::B_SLOT;
      const int nch = stage_chunks(it);
      if (it < num_main) {
        if (!mbar_wait(&wfull[s], (it / TSTG) & 1, abort_flag, p.err)) break;
        const uint8_t* st = smem + s * T_STRIDE;
        for (int c = 0; c < nch; ++c) {
          if (TRANS) convert_trans(st + P_OFF + c * P_BYTES, st + S_OFF + c * S_BYTES, bt + c * B_BYTES, t);
          else convert_fwd(st + P_OFF + c * P_BYTES, st + S_OFF + c * S_BYTES, bt + c * B_BYTES, t);
        }
      } else {
        griddep_wait();  // the LoRA operand comes from an earlier kernel
        for (int c = 0; c < nch; ++c) copy_lora_b<TRANS>(p, (it - num_main) * KCH + c, n0, bt + c * B_BYTES, t);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bfull[b]);
    }
    griddep_wait();
    const bool acc_ok = __all_sync(0xffffffffu, mbar_wait(accf, 0, abort_flag, p.err));
    tc_fence_after();
    if (acc_ok && total > 0) epilogue(p, tmem, warp, lane, m0, n0);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == MMA_WARP) {
    if (lane == 0) {  // the accumulator is complete (or every issued MMA has retired) before TMEM is freed
      int dummy = 0;
      mbar_wait(accf, 0, &dummy, p.err);
    }
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

}  // namespace gemms

namespace {
template <bool TRANS, int KCH>
int launch_s(dim3 grid, const CUtensorMap& tA, const CUtensorMap& tP, const CUtensorMap& tS, const CUtensorMap& tAx,
             const gemms::Params& p, cudaStream_t st) {
  constexpr int smem = gemms::Lay<KCH>::SMEM;
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(gemms::dequant_gemm_narrow<TRANS, KCH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             smem) != cudaSuccess)
      return MEBP_ERR_CUDA;
    attr = true;
  }
  if (launch_k(gemms::dequant_gemm_narrow<TRANS, KCH>, grid, dim3(gemms::THREADS), smem, st, tA, tP, tS, tAx, p) !=
      cudaSuccess)
    return MEBP_ERR_CUDA;
  return MEBP_OK;
}
}  // namespace

int launch_dequant_gemm_narrow(const GemmArgs& g, cudaStream_t st) {
  using namespace gemms;
  if (g.epi != EPI_F16 && g.epi != EPI_F32) return MEBP_ERR_INVALID_ARG;
  CUtensorMap tA, tP, tS, tAx;
  int rc;
  if ((rc = make_tmap_2d(&tA, g.A, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, g.K, g.M, g.lda * 2, 64, BM,
                         CU_TENSOR_MAP_SWIZZLE_128B)))
    return rc;
  if (!g.trans) {
    if ((rc = make_tmap_2d(&tP, g.qpack, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, g.K / 2, g.N, g.K / 2, 32, BN,
                           CU_TENSOR_MAP_SWIZZLE_NONE)))
      return rc;
    if ((rc = make_tmap_2d(&tS, g.scales, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, g.N, g.K / 64, g.scale_pitch * 2, BN, 1,
                           CU_TENSOR_MAP_SWIZZLE_NONE)))
      return rc;
  } else {
    if ((rc = make_tmap_2d(&tP, g.qpack, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, g.N / 2, g.K, g.N / 2, BN / 2, 64,
                           CU_TENSOR_MAP_SWIZZLE_NONE)))
      return rc;
    if ((rc = make_tmap_2d(&tS, g.scales, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, g.K, g.N / 64, g.scale_pitch * 2, 64, 1,
                           CU_TENSOR_MAP_SWIZZLE_NONE)))
      return rc;
  }
  Params p{};
  if (g.Ax && g.kx > 0) {
    if ((g.kx % 16) || (reinterpret_cast<uintptr_t>(g.Bx) & 15) || (g.ldbx % 8)) return MEBP_ERR_INVALID_ARG;
    p.kx_steps = static_cast<int>(g.kx / 16);
    if ((rc = make_tmap_2d(&tAx, g.Ax, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, g.kx, g.M, g.ldax * 2, 64, BM,
                           CU_TENSOR_MAP_SWIZZLE_128B)))
      return rc;
    p.Bx = static_cast<const uint16_t*>(g.Bx);
    p.ldbx = g.ldbx;
    p.kx = static_cast<int>(g.kx);
  } else {
    tAx = tA;
  }
  p.M = static_cast<int>(g.M);
  p.N = static_cast<int>(g.N);
  p.K = static_cast<int>(g.K);
  p.epi = g.epi;
  p.C = g.C;
  p.ldc = g.ldc;
  p.R = g.R;
  p.ldr = g.ldr;
  p.alpha = g.alpha;
  p.err = g.err;
  const dim3 grid(static_cast<unsigned>(g.N / BN), static_cast<unsigned>((g.M + BM - 1) / BM));
  // grids of at most one CTA per SM take two K chunks per stage
  if (static_cast<int64_t>(grid.x) * grid.y <= 152)
    rc = g.trans ? launch_s<true, 2>(grid, tA, tP, tS, tAx, p, st) : launch_s<false, 2>(grid, tA, tP, tS, tAx, p, st);
  else
    rc = g.trans ? launch_s<true, 1>(grid, tA, tP, tS, tAx, p, st) : launch_s<false, 1>(grid, tA, tP, tS, tAx, p, st);
  if (rc) return rc;
  return cudaGetLastError() == cudaSuccess ? MEBP_OK : MEBP_ERR_CUDA;
}

}  // namespace mebp
