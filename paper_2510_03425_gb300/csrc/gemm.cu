// Fused dequant-in-the-mainloop GEMM on 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
//   FWD   : C[M, N] = A[M, K] * deq(W)^T      W packed [N, K]  (Y = X W^T of a linear layer)
//   TRANS : C[M, N] = A[M, K] * deq(W)        W packed [K, N]  (dX = dY W, the input gradient)
//   plus an optional extra K-block  A_x[M, Kx] * B_x^T  that carries the rank-r LoRA product
//   (FWD: A_x = s X A^T, B_x = B [N, Kx];  TRANS: A_x = s dY B, B_x = A [Kx, N]).
//
// This is the decompression of Algorithm 1's LazyLoadAndDecompressWeights fused into the GEMM:
// TMA brings the packed 4-bit tile and its fp16 scales into shared memory, eight converter
// warps turn them into the fp16 operand (bit-exact fp16_rne(q*s), see dequant.cuh) in the
// 128-byte-swizzled layout tcgen05 reads, one thread issues tcgen05.mma into fp32 TMEM
// accumulators, and the same eight warps run the epilogue out of TMEM.
//
// CTA: 320 threads.  warps 0-7 convert + epilogue, warp 8 issues TMA, warp 9 issues MMA and
// owns the TMEM allocation.  Tile (128*NACC) x 256 x 64: NACC 128-row A tiles share every
// decoded 256-row B tile (NACC = 2 halves the decode work per flop and fills all 512 TMEM
// columns).  3-stage smem ring.  Small grids split K over blockIdx.z into fp32 partial tiles
// that a second kernel sums in a fixed order and finishes with the real epilogue.
#include <cudaTypedefs.h>

#include <algorithm>

#include "dequant.cuh"
#include "kernels.h"

namespace mebp {
namespace gemm {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 3, THREADS = 320;
constexpr int B_BYTES = BN * BK * 2, A_BYTES = BM * BK * 2, P_BYTES = BN * BK / 2, S_BYTES = 512;

// Shared-memory stage layout for NACC accumulators (all tiles 1024-byte aligned).
template <int NACC>
struct Layout {
  static constexpr int B_OFF = 0;                                   // fp16 B: 256 x 64
  static constexpr int A_OFF = B_BYTES;                             // fp16 A: NACC x 128 x 64
  static constexpr int P_OFF = A_OFF + NACC * A_BYTES;              // packed nibbles
  static constexpr int S_OFF = P_OFF + P_BYTES;                     // fp16 scales
  static constexpr int STRIDE = (S_OFF + S_BYTES + 1023) / 1024 * 1024;
  static constexpr int BAR_OFF = STAGES * STRIDE;
  static constexpr int SMEM = BAR_OFF + 256 + 1024;                 // + barriers + alignment slack
  static constexpr uint32_t TMEM_COLS = 256 * NACC;
};
static_assert(Layout<2>::SMEM <= 232448, "shared memory budget");

enum { EPI_PARTIAL = 100 };  // split-K: fp32 partial tile into Params::C + z * M * ldc

struct Params {
  int M, N, K;
  int kx_steps;        // 16-wide MMA steps of the extra (LoRA) block; 0 = none
  int kt_split;        // main 64-wide K tiles per split (blockIdx.z)
  int epi;             // GemmEpi or EPI_PARTIAL
  void* C;
  int64_t ldc;
  const float* R;      // fp32 residual / accumulation source (EPI_F32), may alias C
  int64_t ldr;
  float alpha;         // EPI_F32: C = alpha * acc (+ R)
  // LM-head epilogues
  const int32_t* targets;  // [M]
  int col_offset;          // global vocabulary index of GEMM column 0
  int n_valid;             // GEMM columns >= n_valid are outside the vocabulary
  float* part;             // EPI_LSE: float2 [M, nparts]
  int nparts;
  float* zt;               // EPI_LSE: target logit [M]
  const float* lse;        // EPI_CEGRAD: [M]
  const float* ce_w;       // EPI_CEGRAD: device scalar weight of a valid row
  int* err;
};

__device__ __forceinline__ int mbar_phase(int it) { return (it / STAGES) & 1; }

// ---------------------------------------------------------------------------------- convert
// FWD: packed tile [256 rows][32 B] (plain), scales [256]; thread t converts row t (one group)
// into the K-major SW128 B tile (row t at t*128 B, 16-byte chunk j stored at chunk j ^ (t&7)).
template <int NACC>
__device__ __forceinline__ void convert_fwd(uint8_t* stage, int t) {
  using Ly = Layout<NACC>;
  const uint4* src = reinterpret_cast<const uint4*>(stage + Ly::P_OFF + t * 32);
  const uint4 p0 = src[0], p1 = src[1];
  const uint32_t s2 = scale_pair(reinterpret_cast<const uint16_t*>(stage + Ly::S_OFF)[t]);
  uint8_t* row = stage + Ly::B_OFF + t * 128;
  const uint32_t words[8] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    uint32_t o[4];
    dequant_word(words[j], s2, o);
    *reinterpret_cast<uint4*>(row + ((j ^ (t & 7)) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// TRANS: packed tile [64 k-rows][128 B] loaded with the 128-byte swizzle (chunk c of row k at
// chunk c ^ (k&7)), scales [4 groups][64 k-rows].  Thread t: group g = t/64 (64 output
// columns), row k = t%64; its 8 words become chunks 0..7 of row k of MN-major atom g
// (atom = 64 columns x 64 k-rows, 128 B per k-row, chunk c stored at c ^ (k&7)).
template <int NACC>
__device__ __forceinline__ void convert_trans(uint8_t* stage, int t) {
  using Ly = Layout<NACC>;
  const int g = t >> 6, k = t & 63;
  const uint8_t* prow = stage + Ly::P_OFF + k * 128;
  const uint4 p0 = *reinterpret_cast<const uint4*>(prow + (((2 * g) ^ (k & 7)) << 4));
  const uint4 p1 = *reinterpret_cast<const uint4*>(prow + (((2 * g + 1) ^ (k & 7)) << 4));
  const uint32_t s2 = scale_pair(reinterpret_cast<const uint16_t*>(stage + Ly::S_OFF)[g * 64 + k]);
  uint8_t* row = stage + Ly::B_OFF + g * 8192 + k * 128;
  const uint32_t words[8] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    uint32_t o[4];
    dequant_word(words[j], s2, o);
    *reinterpret_cast<uint4*>(row + ((j ^ (k & 7)) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// ---------------------------------------------------------------------------------- epilogue
// NACC = 1: warp w owns TMEM lanes 32*(w&3) .. +31 (tile rows) and columns 128*(w>>2) .. +127.
// NACC = 2: warp w owns lanes 32*(w&3) .. +31 of accumulator w>>2 (tile rows 128*(w>>2) + ...)
//           and all 256 columns.
template <int NACC>
__device__ __forceinline__ void epilogue(const Params& p, uint32_t tmem, int warp, int lane, int m0, int n0) {
  const int q = warp & 3, h = warp >> 2;
  constexpr int NCH = (NACC == 2) ? 8 : 4;  // 32-column chunks per thread
  const int row = m0 + (NACC == 2 ? 128 * h : 0) + 32 * q + lane;
  const bool row_ok = row < p.M;
  const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * q) << 16) + (NACC == 2 ? 256 * h : 128 * h);
  const int cbase = n0 + (NACC == 2 ? 0 : 128 * h);  // first GEMM column of this thread's range

  if (p.epi == EPI_LSE) {
    float mx = -INFINITY, sum = 0.0f, zt = 0.0f;
    bool has_t = false;
    const int tgt = row_ok ? p.targets[row] - p.col_offset : -1;
#pragma unroll 1
    for (int cc = 0; cc < NCH; ++cc) {
      float v[32];
      tmem_ld32(tbase + 32 * cc, v);
      const int c0 = cbase + 32 * cc;
      float cm = -INFINITY;
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        if (c0 + i < p.n_valid) cm = fmaxf(cm, v[i]);
        if (c0 + i == tgt) { zt = v[i]; has_t = true; }
      }
      if (cm > -INFINITY) {
        const float nm = fmaxf(mx, cm);
        float acc = 0.0f;
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (c0 + i < p.n_valid) acc += __expf(v[i] - nm);
        sum = sum * __expf(mx - nm) + acc;
        mx = nm;
      }
    }
    if (row_ok) {
      float2* pr = reinterpret_cast<float2*>(p.part) + static_cast<int64_t>(row) * p.nparts + blockIdx.x * 2;
      if (NACC == 2) {
        pr[0] = make_float2(mx, sum);
        pr[1] = make_float2(-INFINITY, 0.0f);
      } else {
        pr[h] = make_float2(mx, sum);
      }
      if (has_t) p.zt[row] = zt;
    }
    return;
  }

  if (p.epi == EPI_CEGRAD) {
    const float lse = row_ok ? p.lse[row] : 0.0f;
    const int tgt = row_ok ? p.targets[row] : -1;
    const float w = (tgt >= 0) ? *p.ce_w : 0.0f;
    const int tl = tgt - p.col_offset;
    uint16_t* C = static_cast<uint16_t*>(p.C);
#pragma unroll 1
    for (int cc = 0; cc < NCH; ++cc) {
      float v[32];
      tmem_ld32(tbase + 32 * cc, v);
      const int c0 = cbase + 32 * cc;
      if (!row_ok || c0 >= p.N) continue;
      uint32_t o[16];
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        float a = (c0 + i < p.n_valid) ? __expf(v[i] - lse) * w : 0.0f;
        float b = (c0 + i + 1 < p.n_valid) ? __expf(v[i + 1] - lse) * w : 0.0f;
        if (c0 + i == tl) a -= w;
        if (c0 + i + 1 == tl) b -= w;
        o[i / 2] = pack_half2(a, b);
      }
      uint4* dst = reinterpret_cast<uint4*>(C + static_cast<int64_t>(row) * p.ldc + c0);
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (c0 + 8 * i < p.N) dst[i] = make_uint4(o[4 * i], o[4 * i + 1], o[4 * i + 2], o[4 * i + 3]);
    }
    return;
  }

  float* Cp = static_cast<float*>(p.C);
  if (p.epi == EPI_PARTIAL) Cp += static_cast<int64_t>(blockIdx.z) * p.M * p.ldc;
#pragma unroll 1
  for (int cc = 0; cc < NCH; ++cc) {
    float v[32];
    tmem_ld32(tbase + 32 * cc, v);
    const int c0 = cbase + 32 * cc;
    if (!row_ok || c0 >= p.N) continue;
    if (p.epi == EPI_F16) {
      uint16_t* C = static_cast<uint16_t*>(p.C);
      uint4* dst = reinterpret_cast<uint4*>(C + static_cast<int64_t>(row) * p.ldc + c0);
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (c0 + 8 * i < p.N)
          dst[i] = make_uint4(pack_half2(v[8 * i], v[8 * i + 1]), pack_half2(v[8 * i + 2], v[8 * i + 3]),
                              pack_half2(v[8 * i + 4], v[8 * i + 5]), pack_half2(v[8 * i + 6], v[8 * i + 7]));
    } else {  // EPI_F32 (+ residual) or EPI_PARTIAL
      const bool part = p.epi == EPI_PARTIAL;
      const float al = part ? 1.0f : p.alpha;
      float4* dst = reinterpret_cast<float4*>(Cp + static_cast<int64_t>(row) * p.ldc + c0);
      const float4* res =
          (!part && p.R) ? reinterpret_cast<const float4*>(p.R + static_cast<int64_t>(row) * p.ldr + c0) : nullptr;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        if (c0 + 4 * i >= p.N) break;
        float4 o = make_float4(al * v[4 * i], al * v[4 * i + 1], al * v[4 * i + 2], al * v[4 * i + 3]);
        if (res) {
          const float4 r = res[i];
          o.x += r.x; o.y += r.y; o.z += r.z; o.w += r.w;
        }
        dst[i] = o;
      }
    }
  }
}

// ---------------------------------------------------------------------------------- kernel
template <bool TRANS, int NACC>
__global__ void __launch_bounds__(THREADS, 1)
    dequant_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmP,
                        const __grid_constant__ CUtensorMap tmS, const __grid_constant__ CUtensorMap tmAx,
                        const __grid_constant__ CUtensorMap tmBx, const Params p) {
  using Ly = Layout<NACC>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Ly::BAR_OFF);
  uint64_t* conv = full + STAGES;
  uint64_t* empty = conv + STAGES;
  uint64_t* accf = empty + STAGES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accf + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * BM * NACC;
  // K range of this split: main tiles [kt0, kt1); the LoRA block rides with the last split.
  const int num_k = p.K / BK;
  const int kt0 = blockIdx.z * p.kt_split;
  const int kt1 = min(num_k, kt0 + p.kt_split);
  const int num_main = max(0, kt1 - kt0);
  const bool last_split = blockIdx.z == gridDim.z - 1;
  const int num_x = last_split ? (p.kx_steps + 3) / 4 : 0;
  const int total = num_main + num_x;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&conv[s], 8);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accf, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 9) tmem_alloc(tmem_slot, Ly::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 8) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmP);
      tma_prefetch_desc(&tmS);
      int issued = 0;
      for (int it = 0; it < total; ++it) {
        const int s = it % STAGES;
        if (!mbar_wait(&empty[s], mbar_phase(it) ^ 1, abort_flag, p.err)) break;
        uint8_t* st = smem + s * Ly::STRIDE;
        if (it < num_main) {
          const int kt = kt0 + it;
          mbar_arrive_expect_tx(&full[s], NACC * A_BYTES + P_BYTES + S_BYTES);
          tma_load_2d(st + Ly::A_OFF, &tmA, &full[s], kt * BK, m0);
          if (!TRANS) {
            tma_load_2d(st + Ly::P_OFF, &tmP, &full[s], kt * (BK / 2), n0);  // packed [N, K/2]
            tma_load_2d(st + Ly::S_OFF, &tmS, &full[s], n0, kt);             // scales [K/64, N]
          } else {
            tma_load_2d(st + Ly::P_OFF, &tmP, &full[s], n0 / 2, kt * BK);    // packed [K, N/2]
            tma_load_2d(st + Ly::S_OFF, &tmS, &full[s], kt * BK, n0 / 64);   // scales [N/64, K]
          }
        } else {
          const int e = it - num_main;
          mbar_arrive_expect_tx(&full[s], NACC * A_BYTES + B_BYTES);
          tma_load_2d(st + Ly::A_OFF, &tmAx, &full[s], e * BK, m0);
          if (!TRANS) {
            tma_load_2d(st + Ly::B_OFF, &tmBx, &full[s], e * BK, n0);        // B_x [N, Kx], K-major
          } else {
#pragma unroll
            for (int a = 0; a < 4; ++a)                                        // B_x [Kx, N], MN-major atoms
              tma_load_2d(st + Ly::B_OFF + a * 8192, &tmBx, &full[s], n0 + 64 * a, e * BK);
          }
        }
        issued = it + 1;
      }
      // Never leave the CTA with copies in flight: wait (bounded) for the last stages issued.
      for (int it = (issued > STAGES ? issued - STAGES : 0); it < issued; ++it) {
        int dummy = 0;
        mbar_wait(&full[it % STAGES], mbar_phase(it), &dummy, p.err);
      }
    }
  } else if (warp == 9) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f16_f32(BM, BN, TRANS);
      for (int it = 0; it < total; ++it) {
        const int s = it % STAGES;
        if (!mbar_wait(&full[s], mbar_phase(it), abort_flag, p.err)) break;
        if (!mbar_wait(&conv[s], mbar_phase(it), abort_flag, p.err)) break;
        tc_fence_after();
        uint8_t* st = smem + s * Ly::STRIDE;
        const uint32_t a_base = smem_u32(st + Ly::A_OFF), b_base = smem_u32(st + Ly::B_OFF);
        const int nk = (it < num_main) ? 4 : min(4, p.kx_steps - 4 * (it - num_main));
        for (int kk = 0; kk < nk; ++kk) {
          const uint64_t bd = TRANS ? smem_desc_sw128(b_base + kk * 2048, 8192, 1024)
                                    : smem_desc_sw128(b_base + kk * 32, 16, 1024);
#pragma unroll
          for (int a = 0; a < NACC; ++a) {
            const uint64_t ad = smem_desc_sw128(a_base + a * A_BYTES + kk * 32, 16, 1024);
            tc_mma_f16(tmem + 256 * a, ad, bd, idesc, (it > 0 || kk > 0) ? 1u : 0u);
          }
        }
        tc_commit(&empty[s]);
      }
      tc_commit(accf);
    }
  } else {
    // ------------------------------------------------------------ converters, then epilogue
    const int t = threadIdx.x;  // 0..255
    for (int it = 0; it < total; ++it) {
      const int s = it % STAGES;
      if (!mbar_wait(&full[s], mbar_phase(it), abort_flag, p.err)) break;
      if (it < num_main) {
        uint8_t* st = smem + s * Ly::STRIDE;
        if (TRANS) convert_trans<NACC>(st, t);
        else convert_fwd<NACC>(st, t);
        fence_proxy_async_smem();
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&conv[s]);
    }
    if (mbar_wait(accf, 0, abort_flag, p.err)) {
      tc_fence_after();
      if (total > 0) epilogue<NACC>(p, tmem, warp, lane, m0, n0);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    if (lane == 0) {  // the accumulator is complete (or every issued MMA has retired) before TMEM is freed
      int dummy = 0;
      mbar_wait(accf, 0, &dummy, p.err);
    }
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, Ly::TMEM_COLS);
  }
}

// Split-K finish: C = epilogue(sum_z part[z]) in split order.  EPI_F32: alpha * sum (+ R); EPI_F16.
__global__ void splitk_reduce_kernel(const float* __restrict__ part, int splits, int M, int N, int epi, void* C,
                                     int64_t ldc, const float* R, int64_t ldr, float alpha) {
  const int64_t n4 = static_cast<int64_t>(M) * (N / 4);
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= n4) return;
  const int64_t row = i / (N / 4), c = (i % (N / 4)) * 4;
  const int64_t stride = static_cast<int64_t>(M) * N;
  float4 s = make_float4(0, 0, 0, 0);
  for (int z = 0; z < splits; ++z) {
    const float4 v = *reinterpret_cast<const float4*>(part + z * stride + row * N + c);
    s.x += v.x; s.y += v.y; s.z += v.z; s.w += v.w;
  }
  if (epi == EPI_F16) {
    *reinterpret_cast<uint2*>(static_cast<uint16_t*>(C) + row * ldc + c) =
        make_uint2(pack_half2(s.x, s.y), pack_half2(s.z, s.w));
    return;
  }
  float4 o = make_float4(alpha * s.x, alpha * s.y, alpha * s.z, alpha * s.w);
  if (R) {
    const float4 r = *reinterpret_cast<const float4*>(R + row * ldr + c);
    o.x += r.x; o.y += r.y; o.z += r.z; o.w += r.w;
  }
  *reinterpret_cast<float4*>(static_cast<float*>(C) + row * ldc + c) = o;
}

}  // namespace gemm

// ------------------------------------------------------------------------------------ host side
static PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void* f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  }
  return fn;
}

// 2-D tiled tensor map: dims {d0 (inner), d1}, row pitch in bytes, box {b0, b1}.
int make_tmap_2d(CUtensorMap* m, const void* base, CUtensorMapDataType dt, int elem_bytes, uint64_t d0, uint64_t d1,
                 uint64_t pitch_bytes, uint32_t b0, uint32_t b1, CUtensorMapSwizzle swz) {
  auto enc = get_encode();
  if (!enc) return MEBP_ERR_CUDA;
  if ((reinterpret_cast<uintptr_t>(base) & 15) || (pitch_bytes & 15) || ((b0 * elem_bytes) & 15))
    return MEBP_ERR_INVALID_ARG;
  cuuint64_t dims[2] = {d0, d1};
  cuuint64_t strides[1] = {pitch_bytes};
  cuuint32_t box[2] = {b0, b1};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(m, dt, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? MEBP_OK : MEBP_ERR_INVALID_ARG;
}

int gemm_smem_bytes() { return gemm::Layout<2>::SMEM; }

namespace {
template <bool TRANS, int NACC>
int launch_variant(dim3 grid, const CUtensorMap& tA, const CUtensorMap& tP, const CUtensorMap& tS,
                   const CUtensorMap& tAx, const CUtensorMap& tBx, const gemm::Params& p, cudaStream_t st) {
  using Ly = gemm::Layout<NACC>;
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(gemm::dequant_gemm_kernel<TRANS, NACC>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             Ly::SMEM) != cudaSuccess)
      return MEBP_ERR_CUDA;
    attr = true;
  }
  count_launch();
  gemm::dequant_gemm_kernel<TRANS, NACC><<<grid, gemm::THREADS, Ly::SMEM, st>>>(tA, tP, tS, tAx, tBx, p);
  return MEBP_OK;
}
}  // namespace

int launch_dequant_gemm(const GemmArgs& g, cudaStream_t st) {
  using namespace gemm;
  if (g.M <= 0 || g.N <= 0) return MEBP_OK;
  if (g.K % 64 || g.N % 64 || g.K <= 0) return MEBP_ERR_INVALID_ARG;
  // Two 128-row accumulators per CTA once M is large enough to fill the GPU with 256-row tiles.
  const int nacc = (g.M >= 2048) ? 2 : 1;
  const int bm = BM * nacc;

  CUtensorMap tA, tP, tS, tAx, tBx;
  int rc;
  // A: fp16 [M, K], row pitch lda elements.
  if ((rc = make_tmap_2d(&tA, g.A, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, g.K, g.M, g.lda * 2, 64, bm,
                         CU_TENSOR_MAP_SWIZZLE_128B)))
    return rc;
  if (!g.trans) {
    // packed [N, K/2] bytes, scales [K/64, N] (pitch = scale_pitch elements)
    if ((rc = make_tmap_2d(&tP, g.qpack, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, g.K / 2, g.N, g.K / 2, 32, BN,
                           CU_TENSOR_MAP_SWIZZLE_NONE)))
      return rc;
    if ((rc = make_tmap_2d(&tS, g.scales, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, g.N, g.K / 64, g.scale_pitch * 2, BN, 1,
                           CU_TENSOR_MAP_SWIZZLE_NONE)))
      return rc;
  } else {
    // packed [K, N/2] bytes, scales [N/64, K]
    if ((rc = make_tmap_2d(&tP, g.qpack, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, g.N / 2, g.K, g.N / 2, 128, 64,
                           CU_TENSOR_MAP_SWIZZLE_128B)))
      return rc;
    if ((rc = make_tmap_2d(&tS, g.scales, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, g.K, g.N / 64, g.scale_pitch * 2, 64, 4,
                           CU_TENSOR_MAP_SWIZZLE_NONE)))
      return rc;
  }
  int kx_steps = 0;
  if (g.Ax && g.kx > 0) {
    kx_steps = static_cast<int>((g.kx + 15) / 16);
    if ((rc = make_tmap_2d(&tAx, g.Ax, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, g.kx, g.M, g.ldax * 2, 64, bm,
                           CU_TENSOR_MAP_SWIZZLE_128B)))
      return rc;
    if (!g.trans) {
      if ((rc = make_tmap_2d(&tBx, g.Bx, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, g.kx, g.N, g.ldbx * 2, 64, BN,
                             CU_TENSOR_MAP_SWIZZLE_128B)))
        return rc;
    } else {
      if ((rc = make_tmap_2d(&tBx, g.Bx, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, g.N, g.kx, g.ldbx * 2, 64, 64,
                             CU_TENSOR_MAP_SWIZZLE_128B)))
        return rc;
    }
  } else {
    tAx = tA;
    tBx = tA;
  }
  Params p{};
  p.M = static_cast<int>(g.M);
  p.N = static_cast<int>(g.N);
  p.K = static_cast<int>(g.K);
  p.kx_steps = kx_steps;
  p.epi = g.epi;
  p.C = g.C;
  p.ldc = g.ldc;
  p.R = g.R;
  p.ldr = g.ldr;
  p.alpha = g.alpha;
  p.targets = g.targets;
  p.col_offset = g.col_offset;
  p.n_valid = g.n_valid > 0 ? g.n_valid : static_cast<int>(g.N);
  p.part = g.part;
  p.nparts = g.nparts;
  p.zt = g.zt;
  p.lse = g.lse;
  p.ce_w = g.ce_w;
  p.err = g.err;

  const int tiles_n = static_cast<int>((g.N + BN - 1) / BN), tiles_m = static_cast<int>((g.M + bm - 1) / bm);
  const int num_k = static_cast<int>(g.K / BK);
  // Split K when the output tiles cannot fill the GPU (152 SMs, one CTA each) and each split
  // keeps >= 4 K tiles; partial tiles go to the caller's workspace.
  int splits = 1;
  const int grid_mn = tiles_n * tiles_m;
  if ((g.epi == EPI_F32 || g.epi == EPI_F16) && g.split_ws && grid_mn < 120 && num_k >= 8) {
    splits = std::min({num_k / 4, (2 * 152 + grid_mn - 1) / grid_mn, 16});
    const int64_t need = g.M * g.N;
    while (splits > 1 && splits * need > g.split_ws_floats) --splits;
  }
  const int kt_split = (num_k + splits - 1) / splits;
  splits = (num_k + kt_split - 1) / kt_split;
  p.kt_split = kt_split;
  if (splits > 1) {
    p.epi = EPI_PARTIAL;
    p.C = g.split_ws;
    p.ldc = g.N;
  }
  dim3 grid(tiles_n, tiles_m, splits);
  if (g.trans)
    rc = nacc == 2 ? launch_variant<true, 2>(grid, tA, tP, tS, tAx, tBx, p, st)
                   : launch_variant<true, 1>(grid, tA, tP, tS, tAx, tBx, p, st);
  else
    rc = nacc == 2 ? launch_variant<false, 2>(grid, tA, tP, tS, tAx, tBx, p, st)
                   : launch_variant<false, 1>(grid, tA, tP, tS, tAx, tBx, p, st);
  if (rc) return rc;
  if (splits > 1) {
    const int64_t n4 = g.M * (g.N / 4);
    count_launch();
    splitk_reduce_kernel<<<static_cast<unsigned>((n4 + 255) / 256), 256, 0, st>>>(
        g.split_ws, splits, static_cast<int>(g.M), static_cast<int>(g.N), g.epi, g.C, g.ldc, g.R, g.ldr, g.alpha);
  }
  return cudaGetLastError() == cudaSuccess ? MEBP_OK : MEBP_ERR_CUDA;
}

}  // namespace mebp
