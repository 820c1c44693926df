// LoRA-gradient reductions at large token counts on 5th-generation tensor cores:
//   C_j[p, q] (+)= mult * sum_m P[m, p] Q[m, j r + q]     p < Pw, q < r, j < nq
// i.e. dB_t = dY_t^T U_t and dA_t = dU_t^T X of LoRA targets (Section 3: only the LoRA weights are
// trained; Algorithm 1 returns their gradients), P being the wide operand (a column slice of dY, or
// the block input X, [M, Pw]) and Q the rank-wide one ([M, nq r]).  nq > 1 when several targets
// read the same P (dA of q, k and v all read the normed block input): P is then read once for all.
//
// The token axis is the contraction, so both operands enter the MMA "MN-major": P's columns are
// the MMA's M (128 per accumulator), Q's columns its N.  A CTA owns NA x 128 columns of P (NA
// accumulators of 128 x QW fp32 in TMEM, QW = nq r) and one split of the tokens; a three-stage TMA
// ring brings 64 tokens per stage: the P tile as 2 NA boxes of 64 columns (128-byte swizzle) and the
// Q tile as one or two boxes, each one swizzle atom wide (64 columns: 128-byte, 32: 64-byte, 16:
// 32-byte swizzle).  The kernel streams P from HBM once and is bound by HBM bandwidth; two stages
// ahead (up to 144 KB) keep enough bytes in flight per SM.  The token splits of a column block run
// as one thread-block cluster: every CTA parks its fp32 partial in its own (then idle) ring, and
// CTA z adds rows z/S .. (z+1)/S of all S partials over distributed shared memory in split order
// and writes C: deterministic, no workspace and no second kernel.  The host picks the cluster size
// so that all clusters are resident at once.  (The
// warp-level kernel it replaces at these sizes issued one 16-byte copy, with its address
// arithmetic, per thread and chunk, and ran instruction-bound at half the HBM bandwidth.)
//
// CTA: warps 0-3 epilogue (warp w reads TMEM lanes 32w .. 32w+31 = P columns), warp 4 TMA, warp 5
// MMA and TMEM owner.  Every wait is bounded; copies in flight are drained and TMEM is freed
// before the CTA exits.
#include <cudaTypedefs.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace mebp {
namespace ttc {

constexpr int BT = 64, THREADS = 192, STG = 3;  // tokens per stage
constexpr int kMaxNq = 3;

// Q tile pieces: one box per swizzle atom (QW = 96 is 64 + 32 columns).
template <int QW>
struct QPieces {
  static constexpr int N = QW == 96 ? 2 : 1;
  static constexpr int W0 = QW == 96 ? 64 : QW, W1 = QW == 96 ? 32 : 0;
};

template <int NA, int QW>
struct Layout {
  static constexpr int P_BYTES = NA * 128 * BT * 2;  // 2 NA boxes of 64 columns x 64 tokens
  static constexpr int Q_BYTES = QW * BT * 2;
  static constexpr int STRIDE = (P_BYTES + Q_BYTES + 1023) / 1024 * 1024;
  static constexpr int BAR_OFF = STG * STRIDE;
  static constexpr int SMEM = BAR_OFF + 256 + 1024;
  static constexpr int COLS = NA * QW;
  static constexpr int LDQ = QW + 4;  // floats per row of a parked partial (conflict-free float4 rows)
  static_assert(NA * 128 * LDQ * 4 <= BAR_OFF, "the partial fits in the idle ring");
  static constexpr uint32_t TMEM_COLS = COLS <= 32 ? 32 : COLS <= 64 ? 64 : COLS <= 128 ? 128 : COLS <= 256 ? 256 : 512;
};

// Shared-memory descriptor (SM100 format, version 1) with a given layout type: 2 = 128-byte,
// 4 = 64-byte, 6 = 32-byte swizzle.  lbo / sbo are byte offsets (multiples of 16).
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo, uint32_t layout) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= 1ull << 46;
  d |= static_cast<uint64_t>(layout) << 61;
  return d;
}
__host__ __device__ constexpr uint32_t swz_layout(int width) { return width == 64 ? 2u : (width == 32 ? 4u : 6u); }

// 16 consecutive fp32 columns of this warp's 32 TMEM lanes -> 16 registers per thread.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

struct Out {
  float* C[kMaxNq];       // C_j[p * sp + q * sq] (+)= mult * sum
  int r;                  // columns of Q per target
  int64_t sp, sq;
  int accumulate;
  const float* mult;
};

// grid (ceil(Pw / (128 NA)), S), cluster (1, S, 1); split z covers tokens [z m_per_split, ...)
// (a multiple of 64).
template <int NA, int QW>
__global__ void __launch_bounds__(THREADS, 1)
    tall_tc_kernel(const __grid_constant__ CUtensorMap tmP, const __grid_constant__ CUtensorMap tmQ0,
                   const __grid_constant__ CUtensorMap tmQ1, int64_t M, int Pw, int64_t m_per_split, Out o,
                   int* err) {
  using Ly = Layout<NA, QW>;
  using QP = QPieces<QW>;
  static_assert(QW == 16 || QW == 32 || QW == 64 || QW == 96, "Q tile of whole swizzle atoms");
  static_assert(Ly::SMEM <= 232448, "shared memory");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Ly::BAR_OFF);
  uint64_t* empty = full + STG;
  uint64_t* accf = empty + STG;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accf + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int p0 = static_cast<int>(blockIdx.x) * NA * 128;
  const int64_t mb = static_cast<int64_t>(blockIdx.y) * m_per_split;
  const int64_t me = min(M, mb + m_per_split);
  const int nst = me > mb ? static_cast<int>((me - mb + BT - 1) / BT) : 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STG; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accf, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 5) tmem_alloc(tmem_slot, Ly::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  griddep_wait();  // P and Q come from earlier kernels
  griddep_launch();

  if (warp == 4) {
    if (lane == 0) {
      tma_prefetch_desc(&tmP);
      tma_prefetch_desc(&tmQ0);
      if (QP::N > 1) tma_prefetch_desc(&tmQ1);
      int issued = 0;
      for (int it = 0; it < nst; ++it) {
        const int s = it % STG;
        if (it >= STG && !mbar_wait(&empty[s], ((it / STG) & 1) ^ 1, abort_flag, err)) break;
        uint8_t* st = smem + s * Ly::STRIDE;
        const int m = static_cast<int>(mb + static_cast<int64_t>(it) * BT);
        mbar_arrive_expect_tx(&full[s], Ly::P_BYTES + Ly::Q_BYTES);
        for (int j = 0; j < 2 * NA; ++j) tma_load_2d(st + j * 8192, &tmP, &full[s], p0 + 64 * j, m);
        tma_load_2d(st + Ly::P_BYTES, &tmQ0, &full[s], 0, m);
        if (QP::N > 1) tma_load_2d(st + Ly::P_BYTES + BT * QP::W0 * 2, &tmQ1, &full[s], 0, m);
        issued = it + 1;
      }
      int dummy = 0;  // never leave with copies in flight
      for (int it = (issued > STG ? issued - STG : 0); it < issued; ++it)
        mbar_wait(&full[it % STG], (it / STG) & 1, &dummy, err);
    }
  } else if (warp == 5) {
    if (lane == 0) {
      // M = 128 columns of P, N = a Q piece, both operands MN-major (bits 15 and 16)
      constexpr uint32_t id0 = idesc_f16_f32(128, QP::W0, true) | (1u << 15);
      constexpr uint32_t id1 = idesc_f16_f32(128, QP::N > 1 ? QP::W1 : 16, true) | (1u << 15);
      constexpr uint32_t rb0 = QP::W0 * 2, rb1 = QP::W1 * 2;  // bytes per token row of each piece
      for (int it = 0; it < nst; ++it) {
        const int s = it % STG;
        if (!mbar_wait(&full[s], (it / STG) & 1, abort_flag, err)) break;
        tc_fence_after();
        const uint32_t sa = smem_u32(smem + s * Ly::STRIDE);
        const uint32_t q0 = sa + Ly::P_BYTES, q1 = q0 + BT * rb0;
#pragma unroll
        for (int kk = 0; kk < BT / 16; ++kk) {  // 16 tokens per MMA: 2048 bytes of P, 16 rows of Q
          const uint64_t bd0 = smem_desc(q0 + kk * 16 * rb0, 8 * rb0, 8 * rb0, swz_layout(QP::W0));
          const uint64_t bd1 = smem_desc(q1 + kk * 16 * rb1, 8 * rb1, 8 * rb1, swz_layout(QP::W1));
#pragma unroll
          for (int a = 0; a < NA; ++a) {
            const uint64_t ad = smem_desc(sa + a * 16384 + kk * 2048, 8192, 1024, 2);
            const uint32_t acc = (it > 0 || kk > 0) ? 1u : 0u;
            tc_mma_f16(tmem + a * QW, ad, bd0, id0, acc);
            if (QP::N > 1) tc_mma_f16(tmem + a * QW + QP::W0, ad, bd1, id1, acc);
          }
        }
        tc_commit(&empty[s]);
      }
      tc_commit(accf);
    }
  } else {
    // epilogue: thread = column p of each accumulator; this split's partial into the idle ring
    // (row a 128 + 32 w + lane at LDQ floats: the TMA drain and accf mean the ring is quiet)
    const bool ok = __all_sync(0xffffffffu, mbar_wait(accf, 0, abort_flag, err));
    tc_fence_after();
#pragma unroll 1
    for (int a = 0; a < NA; ++a) {
      float* row = reinterpret_cast<float*>(smem) + (128 * a + 32 * warp + lane) * Ly::LDQ;
#pragma unroll 1
      for (int c0 = 0; c0 < QW; c0 += 16) {
        float v[16];
        if (ok && nst > 0) {
          tmem_ld16(tmem + (static_cast<uint32_t>(32 * warp) << 16) + a * QW + c0, v);
        } else {
#pragma unroll
          for (int i = 0; i < 16; ++i) v[i] = 0.0f;
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
          *reinterpret_cast<float4*>(row + c0 + 4 * i) = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    if (lane == 0) {  // every issued MMA has retired before TMEM is freed
      int dummy = 0;
      mbar_wait(accf, 0, &dummy, err);
    }
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, Ly::TMEM_COLS);
  }
  // Every thread of every CTA of the cluster passes both barriers.  CTA z sums rows
  // [z rpc, (z + 1) rpc) of the S partials (S = cluster size) in split order.
  const int S = static_cast<int>(gridDim.y);
  if (S > 1) cluster_sync_all();
  else __syncthreads();
  {
    const int z = static_cast<int>(blockIdx.y);
    const int nrow = NA * 128, rpc = (nrow + S - 1) / S;
    const int r0 = z * rpc, r1 = min(nrow, r0 + rpc);
    constexpr int C4 = QW / 4;
    const float mu = o.mult ? *o.mult : 1.0f;
    const uint32_t base = smem_u32(smem);
    for (int i = threadIdx.x; i < (r1 - r0) * C4; i += THREADS) {
      const int rr = r0 + i / C4, q = (i % C4) * 4, p = p0 + rr;
      if (p >= Pw) continue;
      const uint32_t off = base + (rr * Ly::LDQ + q) * 4;
      float4 sum = S > 1 ? ld_dsmem_f4(dsmem_addr(off, 0))
                         : *reinterpret_cast<const float4*>(smem + (rr * Ly::LDQ + q) * 4);
      for (int j = 1; j < S; ++j) {
        const float4 v = ld_dsmem_f4(dsmem_addr(off, j));
        sum.x += v.x; sum.y += v.y; sum.z += v.z; sum.w += v.w;
      }
      const int t = q / o.r, qq = q % o.r;  // target, column within it (r is a multiple of 4)
      float* c = (t == 0 ? o.C[0] : (t == 1 ? o.C[1] : o.C[2])) + p * o.sp + qq * o.sq;
      const float s4[4] = {sum.x, sum.y, sum.z, sum.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float* d = c + e * o.sq;
        *d = o.accumulate ? *d + mu * s4[e] : mu * s4[e];
      }
    }
  }
  if (S > 1) cluster_sync_all();  // no CTA leaves while its partial is being read
}

template <int NA, int QW>
bool set_attr() {
  static int state = 0;  // 0 unknown, 1 ok, -1 failed
  if (state == 0) {
    const bool ok = cudaFuncSetAttribute(tall_tc_kernel<NA, QW>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Layout<NA, QW>::SMEM) == cudaSuccess &&
                    cudaFuncSetAttribute(tall_tc_kernel<NA, QW>, cudaFuncAttributeNonPortableClusterSizeAllowed, 0) ==
                        cudaSuccess;
    if (!ok) cudaGetLastError();
    state = ok ? 1 : -1;
  }
  return state > 0;
}

// Clusters of S CTAs (along y) of this variant that can be resident at once (0: none).  Queried
// once per S.
template <int NA, int QW>
int max_clusters(int S) {
  static int cache[9] = {-1, -1, -1, -1, -1, -1, -1, -1, -1};
  if (S < 1 || S > 8) return 0;
  if (cache[S] < 0) {
    int n = 0;
    if (set_attr<NA, QW>()) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(1, S, 1);
      cfg.blockDim = dim3(THREADS);
      cfg.dynamicSmemBytes = Layout<NA, QW>::SMEM;
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = 1;
      at[0].val.clusterDim.y = S;
      at[0].val.clusterDim.z = 1;
      cfg.attrs = at;
      cfg.numAttrs = 1;
      if (cudaOccupancyMaxActiveClusters(&n, tall_tc_kernel<NA, QW>, &cfg) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
      }
    }
    cache[S] = n;
  }
  return cache[S];
}

// The largest split count S <= 8 (each split at least four 64-token stages) whose gx clusters are
// all resident at once; 0 when none fits.
template <int NA, int QW>
int plan(int Pw, int64_t M, int* gx_out) {
  const int gx = (Pw + NA * 128 - 1) / (NA * 128);
  *gx_out = gx;
  const int smax = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(8, M / (4 * BT))));
  for (int S = smax; S >= 1; --S)
    if (gx <= max_clusters<NA, QW>(S)) return S;
  return 0;
}

template <int NA, int QW>
int launch(const uint16_t* P, int64_t ldp, const uint16_t* Q, int64_t ldq, int64_t M, int Pw, int r, float* const* C,
           int64_t ldc, bool accumulate, const float* mult, int S, int* err, cudaStream_t st) {
  using QP = QPieces<QW>;
  CUtensorMap tP, tQ0, tQ1;
  int rc;
  if ((rc = make_tmap_2d(&tP, P, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, Pw, M, ldp * 2, 64, BT,
                         CU_TENSOR_MAP_SWIZZLE_128B)))
    return rc;
  auto swz = [](int w) {
    return w == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : (w == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B);
  };
  if ((rc = make_tmap_2d(&tQ0, Q, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, QP::W0, M, ldq * 2, QP::W0, BT, swz(QP::W0))))
    return rc;
  tQ1 = tQ0;
  if (QP::N > 1 &&
      (rc = make_tmap_2d(&tQ1, Q + QP::W0, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, QP::W1, M, ldq * 2, QP::W1, BT,
                         swz(QP::W1))))
    return rc;
  const int gx = (Pw + NA * 128 - 1) / (NA * 128);
  int64_t mps = (M + S - 1) / S;
  mps = (mps + BT - 1) / BT * BT;
  Out o{};
  for (int j = 0; j < QW / r && j < kMaxNq; ++j) o.C[j] = C[j];
  o.r = r;
  o.sp = ldc > 0 ? ldc : 1;
  o.sq = ldc > 0 ? 1 : -ldc;
  o.accumulate = accumulate ? 1 : 0;
  o.mult = mult;
  launch_k_cluster(tall_tc_kernel<NA, QW>, dim3(static_cast<unsigned>(gx), static_cast<unsigned>(S)), dim3(THREADS),
                   Layout<NA, QW>::SMEM, st, dim3(1, S, 1), tP, tQ0, tQ1, M, Pw, mps, o, err);
  return cudaGetLastError() == cudaSuccess ? MEBP_OK : MEBP_ERR_CUDA;
}

// Pick the variant (accumulators per CTA) that keeps the most SMs busy in one wave of clusters,
// preferring more accumulators per CTA (fewer CTAs re-reading the same Q rows) on a tie.
template <int QW>
int launch_best(const uint16_t* P, int64_t ldp, const uint16_t* Q, int64_t ldq, int64_t M, int Pw, int r,
                float* const* C, int64_t ldc, bool accumulate, const float* mult, int* err, cudaStream_t st) {
  int gx4 = 0, gx2 = 0, gx1 = 0;
  const int s4 = QW <= 64 ? plan<QW <= 64 ? 4 : 2, QW>(Pw, M, &gx4) : 0;
  const int s2 = plan<2, QW>(Pw, M, &gx2);
  const int s1 = plan<1, QW>(Pw, M, &gx1);
  const int c4 = s4 * gx4, c2 = s2 * gx2, c1 = s1 * gx1;
  if (QW <= 64 && c4 > 0 && c4 >= c2 && c4 >= c1)
    return launch<QW <= 64 ? 4 : 2, QW>(P, ldp, Q, ldq, M, Pw, r, C, ldc, accumulate, mult, s4, err, st);
  if (c2 > 0 && c2 >= c1) return launch<2, QW>(P, ldp, Q, ldq, M, Pw, r, C, ldc, accumulate, mult, s2, err, st);
  if (c1 > 0) return launch<1, QW>(P, ldp, Q, ldq, M, Pw, r, C, ldc, accumulate, mult, s1, err, st);
  return MEBP_ERR_UNSUPPORTED;
}

}  // namespace ttc

int launch_tall_tc(const uint16_t* P, int64_t ldp, const uint16_t* Q, int64_t ldq, int64_t M, int Pw, int nq, int r,
                   float* const* C, int64_t ldc, bool accumulate, const float* mult, int* err, cudaStream_t st) {
  if (M <= 0 || Pw <= 0) return MEBP_OK;
  const int qw = nq * r;
  if (Pw % 64 || nq < 1 || nq > ttc::kMaxNq || r % 16 || (qw != 16 && qw != 32 && qw != 64 && qw != 96))
    return MEBP_ERR_UNSUPPORTED;
  switch (qw) {
    case 16: return ttc::launch_best<16>(P, ldp, Q, ldq, M, Pw, r, C, ldc, accumulate, mult, err, st);
    case 32: return ttc::launch_best<32>(P, ldp, Q, ldq, M, Pw, r, C, ldc, accumulate, mult, err, st);
    case 64: return ttc::launch_best<64>(P, ldp, Q, ldq, M, Pw, r, C, ldc, accumulate, mult, err, st);
    default: return ttc::launch_best<96>(P, ldp, Q, ldq, M, Pw, r, C, ldc, accumulate, mult, err, st);
  }
}

}  // namespace mebp
