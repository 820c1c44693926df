// Rank-r LoRA down-projections at large token counts on 5th-generation tensor cores:
//   out[M, J] = alpha * X[M, K] . W[J, K]^T      (U_s = s X A^T, and dU = s dY B in the backward)
// J is the padded width of the concatenated rank axis (16 .. 96).  The kernel streams X from HBM
// once, so it is bound by HBM bandwidth: a deep TMA ring keeps enough bytes in flight per SM (the
// whole X tile of a stage is 16 KB), tcgen05.mma (M = 128, N = J) accumulates in TMEM, and the
// four epilogue warps convert the fp32 result to fp16.  When the 128-row tiles alone would leave
// many SMs idle, K is split over a thread-block cluster and the fp32 partial tiles are summed
// through distributed shared memory in split order (deterministic, no workspace).
//
// CTA: warps 0-3 epilogue (warp w reads TMEM lanes 32w .. 32w+31, i.e. tile rows), warp 4 issues
// TMA, warp 5 issues MMA and owns the TMEM allocation.  Every wait is bounded; TMA copies in
// flight are drained and TMEM is freed before the CTA exits.
#include <cudaTypedefs.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace mebp {
namespace skt {

constexpr int BM = 128, BK = 64, STG = 6, THREADS = 192;
constexpr int X_BYTES = BM * BK * 2;  // one 128 x 64 fp16 tile of X (16 KB)

template <int J>
struct Layout {
  static constexpr int W_BYTES = J * BK * 2;
  static constexpr int STRIDE = (X_BYTES + W_BYTES + 1023) / 1024 * 1024;
  static constexpr int BAR_OFF = STG * STRIDE;
  static constexpr int SMEM = BAR_OFF + 256 + 1024;  // + barriers + alignment slack
  static constexpr int LDP = J + 4;                  // floats per row of a parked partial tile
};

template <int J>
__global__ void __launch_bounds__(THREADS, 1)
    skinny_tc_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW, int M, int K,
                     float alpha, uint16_t* __restrict__ out, int64_t ldo, int kt_split, int* err) {
  using Ly = Layout<J>;
  static_assert(J % 16 == 0 && J >= 16 && J <= 128, "MMA N");
  static_assert(BM * Ly::LDP * 4 <= Ly::BAR_OFF, "partial tile fits in the idle ring");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Ly::BAR_OFF);
  uint64_t* empty = full + STG;
  uint64_t* accf = empty + STG;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accf + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = blockIdx.x * BM;
  const int nk_all = K / BK;
  const int kt0 = blockIdx.y * kt_split;
  const int nk = max(0, min(nk_all, kt0 + kt_split) - kt0);
  const bool split = gridDim.y > 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STG; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accf, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 5) tmem_alloc(tmem_slot, 128);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // X and W may both come from the kernel right before (a single linear builds W just before)
  griddep_wait();
  griddep_launch();

  if (warp == 4) {
    if (lane == 0) {
      tma_prefetch_desc(&tmX);
      tma_prefetch_desc(&tmW);
      int issued = 0;
      for (int it = 0; it < nk; ++it) {
        const int s = it % STG;
        if (it >= STG && !mbar_wait(&empty[s], ((it / STG) & 1) ^ 1, abort_flag, err)) break;
        uint8_t* st = smem + s * Ly::STRIDE;
        mbar_arrive_expect_tx(&full[s], X_BYTES + Ly::W_BYTES);
        tma_load_2d(st, &tmX, &full[s], (kt0 + it) * BK, m0);
        tma_load_2d(st + X_BYTES, &tmW, &full[s], (kt0 + it) * BK, 0);
        issued = it + 1;
      }
      // never leave with copies in flight
      int dummy = 0;
      for (int it = (issued > STG ? issued - STG : 0); it < issued; ++it)
        mbar_wait(&full[it % STG], (it / STG) & 1, &dummy, err);
    }
  } else if (warp == 5) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f16_f32(BM, J, false);
      for (int it = 0; it < nk; ++it) {
        const int s = it % STG;
        if (!mbar_wait(&full[s], (it / STG) & 1, abort_flag, err)) break;
        tc_fence_after();
        const uint32_t sa = smem_u32(smem + s * Ly::STRIDE);
        const uint64_t ad = smem_desc_sw128(sa, 16, 1024), bd = smem_desc_sw128(sa + X_BYTES, 16, 1024);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)  // k16 slices: +32 bytes in the 128-byte swizzled rows
          tc_mma_f16(tmem, ad + kk * 2, bd + kk * 2, idesc, (it > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&empty[s]);
      }
      tc_commit(accf);
    }
  } else {
    // epilogue: thread = tile row 32 w + lane
    const int r = 32 * warp + lane;
    const bool ok = __all_sync(0xffffffffu, mbar_wait(accf, 0, abort_flag, err)) && nk > 0;
    tc_fence_after();
    const uint32_t tb = tmem + (static_cast<uint32_t>(32 * warp) << 16);
    if (!split) {
      const int64_t row = m0 + r;
#pragma unroll
      for (int c0 = 0; c0 < J; c0 += 32) {
        float v[32];
        if (ok) {
          tmem_ld32(tb + c0, v);
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = 0.0f;
        }
        if (row < M) {
          uint4* dst = reinterpret_cast<uint4*>(out + row * ldo + c0);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            if (c0 + 8 * i < J)
              dst[i] = make_uint4(pack_half2(alpha * v[8 * i], alpha * v[8 * i + 1]),
                                  pack_half2(alpha * v[8 * i + 2], alpha * v[8 * i + 3]),
                                  pack_half2(alpha * v[8 * i + 4], alpha * v[8 * i + 5]),
                                  pack_half2(alpha * v[8 * i + 6], alpha * v[8 * i + 7]));
        }
      }
    } else {
      // park the fp32 partial tile in this CTA's (idle) ring: row r at r * LDP floats
      float* part = reinterpret_cast<float*>(smem) + r * Ly::LDP;
#pragma unroll
      for (int c0 = 0; c0 < J; c0 += 32) {
        float v[32];
        if (ok) {
          tmem_ld32(tb + c0, v);
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = 0.0f;
        }
#pragma unroll
        for (int i = 0; i < 8; ++i)
          if (c0 + 4 * i < J)
            *reinterpret_cast<float4*>(part + c0 + 4 * i) = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
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
    tmem_dealloc(tmem, 128);
  }
  if (split) {  // every thread of every CTA of the cluster passes both barriers
    cluster_sync_all();
    const int S = gridDim.y, z = blockIdx.y;
    const int rpc = (BM + S - 1) / S;
    const int r0 = z * rpc, r1 = min(BM, r0 + rpc);
    constexpr int C4 = J / 4;
    const uint32_t base = smem_u32(smem);
    for (int i = threadIdx.x; i < (r1 - r0) * C4; i += THREADS) {
      const int rr = r0 + i / C4, cc = (i % C4) * 4;
      const int64_t row = m0 + rr;
      if (row >= M) continue;
      const uint32_t off = base + (rr * Ly::LDP + cc) * 4;
      float4 v[8];
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (j < S) v[j] = ld_dsmem_f4(dsmem_addr(off, j));
      float4 sum = v[0];
#pragma unroll
      for (int j = 1; j < 8; ++j)
        if (j < S) {
          sum.x += v[j].x; sum.y += v[j].y; sum.z += v[j].z; sum.w += v[j].w;
        }
      *reinterpret_cast<uint2*>(out + row * ldo + cc) =
          make_uint2(pack_half2(alpha * sum.x, alpha * sum.y), pack_half2(alpha * sum.z, alpha * sum.w));
    }
    cluster_sync_all();  // no CTA leaves while its partial is being read
  }
}

template <int J>
int launch(const uint16_t* X, int64_t ldx, int64_t M, int64_t K, const uint16_t* W, int64_t ldw, float alpha,
           uint16_t* out, int64_t ldo, int* err, cudaStream_t st) {
  using Ly = Layout<J>;
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(skinny_tc_kernel<J>, cudaFuncAttributeMaxDynamicSharedMemorySize, Ly::SMEM) !=
        cudaSuccess) {
      cudaGetLastError();
      return MEBP_ERR_CUDA;
    }
    attr = true;
  }
  CUtensorMap tX, tW;
  int rc;
  if ((rc = make_tmap_2d(&tX, X, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, K, M, ldx * 2, BK, BM,
                         CU_TENSOR_MAP_SWIZZLE_128B)))
    return rc;
  if ((rc = make_tmap_2d(&tW, W, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, K, J, ldw * 2, BK, J, CU_TENSOR_MAP_SWIZZLE_128B)))
    return rc;
  const int gx = static_cast<int>((M + BM - 1) / BM);
  const int nk = static_cast<int>(K / BK);
  // Split K over a cluster (<= 8) when the row tiles leave more than a quarter of the 152 SMs
  // idle: each split keeps >= 4 K tiles, at most one CTA per SM in total.
  int splits = 1;
  if (gx < 114) splits = std::max(1, std::min({8, nk / 4, 152 / gx}));
  const int kt_split = (nk + splits - 1) / splits;
  splits = std::max(1, (nk + kt_split - 1) / kt_split);
  launch_k_cluster(skinny_tc_kernel<J>, dim3(gx, splits), THREADS, Ly::SMEM, st, dim3(1, splits, 1), tX, tW,
                   static_cast<int>(M), static_cast<int>(K), alpha, out, ldo, kt_split, err);
  return cudaGetLastError() == cudaSuccess ? MEBP_OK : MEBP_ERR_CUDA;
}

}  // namespace skt

int launch_skinny_tc(const uint16_t* X, int64_t ldx, int64_t M, int64_t K, const uint16_t* W, int64_t ldw,
                     float alpha, uint16_t* out, int64_t ldo, int* err, cudaStream_t st) {
  if (M <= 0) return MEBP_OK;
  if (K % skt::BK || K <= 0) return MEBP_ERR_INVALID_ARG;
  switch (ldo) {
    case 16: return skt::launch<16>(X, ldx, M, K, W, ldw, alpha, out, ldo, err, st);
    case 32: return skt::launch<32>(X, ldx, M, K, W, ldw, alpha, out, ldo, err, st);
    case 48: return skt::launch<48>(X, ldx, M, K, W, ldw, alpha, out, ldo, err, st);
    case 64: return skt::launch<64>(X, ldx, M, K, W, ldw, alpha, out, ldo, err, st);
    case 80: return skt::launch<80>(X, ldx, M, K, W, ldw, alpha, out, ldo, err, st);
    case 96: return skt::launch<96>(X, ldx, M, K, W, ldw, alpha, out, ldo, err, st);
    default: return MEBP_ERR_UNSUPPORTED;
  }
}

}  // namespace mebp
