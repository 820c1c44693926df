// LoRA kernels (Section 3: only LoRA weights are trainable; the compressed base is frozen).
//
//  * skinny_gemm:  U_s = s * X A^T  (and dU = s * dY B) — the rank-r down-projections whose
//    fp16 result feeds the fused GEMM's extra K-block.  HBM-bound on X.
//  * tall_reduce:  dB = dY^T U_s and dA = dU^T X — reductions over all T tokens, done as
//    warp-level tensor-core tiles over a token split, then summed in a fixed order
//    (deterministic; no floating-point atomics).
//  * lora_shadow:  fp16 operand copies of the fp32 masters, with the targets of a fused
//    linear (q|k|v or gate|up) laid side by side along the rank axis:
//      A_cat [kx, K]  rows ro_t .. ro_t+r-1 = A_t
//      B_cat [N, kx]  block-diagonal: rows of target t, columns ro_t .. ro_t+r-1 = B_t
//      Bt_cat [kx, N] = B_cat^T
#include <algorithm>

#include "kernels.h"
#include "mma.cuh"

namespace mebp {

// ------------------------------------------------------------------------------------ skinny
// CTA (blockIdx.x, blockIdx.y): rows m0 .. m0+63, K tiles of split blockIdx.y.  With more than
// one split (gridDim.y > 1) the splits of a row block form one cluster: each parks its fp32
// partial [64][JR] in shared memory and CTA z sums rows z*ceil(64/S) .. of all S partials over
// distributed shared memory in split order (deterministic).
template <int NT>
__global__ void __launch_bounds__(128) skinny_gemm_kernel(const uint16_t* __restrict__ X, int64_t ldx, int64_t M,
                                                          int64_t K, const uint16_t* __restrict__ W, int64_t ldw,
                                                          float alpha, uint16_t* __restrict__ out, int64_t ldo,
                                                          int kt_split) {
  griddep_wait();
  griddep_launch();
  constexpr int BMs = 64, BKs = 64, LDS = BKs + 8, JR = NT * 8, LDP = JR + 4;
  constexpr int XS_BYTES = 2 * BMs * LDS * 2, WS_BYTES = 2 * JR * LDS * 2;
  static_assert(BMs * LDP * 4 <= XS_BYTES + WS_BYTES, "partial fits in the staging buffers");
  __shared__ __align__(16) uint8_t smraw[XS_BYTES + WS_BYTES];
  uint16_t (*xs)[BMs * LDS] = reinterpret_cast<uint16_t (*)[BMs * LDS]>(smraw);
  uint16_t (*ws)[JR * LDS] = reinterpret_cast<uint16_t (*)[JR * LDS]>(smraw + XS_BYTES);
  float* part = reinterpret_cast<float*>(smraw);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t m0 = static_cast<int64_t>(blockIdx.x) * BMs;
  float acc[NT][4];
#pragma unroll
  for (int i = 0; i < NT; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.0f;

  auto load = [&](int stage, int64_t k0) {
    for (int c = tid; c < BMs * 8; c += 128) {
      const int r = c >> 3, cc = c & 7;
      const int64_t gm = m0 + r;
      const bool v = gm < M;
      cp_async16(smem_u32(&xs[stage][r * LDS + cc * 8]), X + (v ? gm : 0) * ldx + k0 + cc * 8, v);
    }
    for (int c = tid; c < JR * 8; c += 128) {
      const int r = c >> 3, cc = c & 7;
      cp_async16(smem_u32(&ws[stage][r * LDS + cc * 8]), W + r * ldw + k0 + cc * 8, true);
    }
    cp_async_commit();
  };
  const int nk_all = static_cast<int>(K / BKs);
  const int kt0 = blockIdx.y * kt_split;
  const int nk = max(0, min(nk_all, kt0 + kt_split) - kt0);
  if (nk > 0) load(0, static_cast<int64_t>(kt0) * BKs);
  for (int kt = 0; kt < nk; ++kt) {
    if (kt + 1 < nk) {
      load((kt + 1) & 1, static_cast<int64_t>(kt0 + kt + 1) * BKs);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const int s = kt & 1;
    const uint32_t xb = smem_u32(xs[s]), wb = smem_u32(ws[s]);
#pragma unroll
    for (int kk = 0; kk < BKs; kk += 16) {
      uint32_t a[4];
      ldsm_x4(a, frag_a_addr(xb, LDS, warp * 16, kk, lane));
#pragma unroll
      for (int nt = 0; nt < NT; nt += 2) {
        uint32_t b[4];
        ldsm_x4(b, frag_bn_addr(wb, LDS, nt * 8, kk, lane));
        mma16816(acc[nt], a, b[0], b[1]);
        mma16816(acc[nt + 1], a, b[2], b[3]);
      }
    }
    __syncthreads();
  }
  const int r = lane >> 2, c = (lane & 3) * 2;
  if (gridDim.y == 1) {
    const int64_t row0 = m0 + warp * 16 + r;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int col = nt * 8 + c;
      if (row0 < M)
        *reinterpret_cast<uint32_t*>(out + row0 * ldo + col) = pack_half2(alpha * acc[nt][0], alpha * acc[nt][1]);
      if (row0 + 8 < M)
        *reinterpret_cast<uint32_t*>(out + (row0 + 8) * ldo + col) =
            pack_half2(alpha * acc[nt][2], alpha * acc[nt][3]);
    }
    return;
  }
  // split K: partial tile into own shared memory (the staging buffers are idle after the loop)
  const int pr = warp * 16 + r;
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    *reinterpret_cast<float2*>(part + pr * LDP + nt * 8 + c) = make_float2(acc[nt][0], acc[nt][1]);
    *reinterpret_cast<float2*>(part + (pr + 8) * LDP + nt * 8 + c) = make_float2(acc[nt][2], acc[nt][3]);
  }
  cluster_sync_all();
  const int S = gridDim.y, z = blockIdx.y;
  const int rpc = (BMs + S - 1) / S;
  const int r0 = z * rpc, r1 = min(BMs, r0 + rpc);
  constexpr int C4 = JR / 4;
  const uint32_t base = smem_u32(part);
  for (int i = tid; i < (r1 - r0) * C4; i += 128) {
    const int rr = r0 + i / C4, cc = (i % C4) * 4;
    const int64_t row = m0 + rr;
    if (row >= M) continue;
    const uint32_t off = base + (rr * LDP + cc) * 4;
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

// Few tokens: one CTA per 16 rows holding the rows' whole K slab and all of W in shared memory
// (one load, no pipeline), the four warps each taking a quarter of the k16 steps; the four fp32
// partials are summed in warp order through shared memory.  No cluster, no second barrier round.
template <int NT>
__global__ void __launch_bounds__(128) skinny_slab_kernel(const uint16_t* __restrict__ X, int64_t ldx, int64_t M,
                                                          int K, const uint16_t* __restrict__ W, int64_t ldw,
                                                          float alpha, uint16_t* __restrict__ out, int64_t ldo) {
  griddep_wait();  // W may come from the kernel right before (a single linear builds its shadow first)
  griddep_launch();
  constexpr int JR = NT * 8, LDR = JR + 4;
  extern __shared__ __align__(16) uint8_t sm[];
  const int LDS = K + 8;
  uint16_t* xs = reinterpret_cast<uint16_t*>(sm);
  uint16_t* ws = xs + 16 * LDS;
  float* red = reinterpret_cast<float*>(ws + JR * LDS);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t m0 = static_cast<int64_t>(blockIdx.x) * 16;
  const int kc = K / 8;
  for (int c = tid; c < JR * kc; c += 128) {
    const int r = c / kc, cc = c % kc;
    cp_async16(smem_u32(ws + r * LDS + cc * 8), W + r * ldw + cc * 8, true);
  }
  for (int c = tid; c < 16 * kc; c += 128) {
    const int r = c / kc, cc = c % kc;
    const int64_t gm = m0 + r;
    const bool v = gm < M;
    cp_async16(smem_u32(xs + r * LDS + cc * 8), X + (v ? gm : 0) * ldx + cc * 8, v);
  }
  cp_async_commit();
  cp_async_wait<0>();
  __syncthreads();
  float acc[NT][4];
#pragma unroll
  for (int i = 0; i < NT; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.0f;
  const int nks = K / 16, ks0 = warp * nks / 4, ks1 = (warp + 1) * nks / 4;
  const uint32_t xb = smem_u32(xs), wb = smem_u32(ws);
  for (int ks = ks0; ks < ks1; ++ks) {
    uint32_t a[4];
    ldsm_x4(a, frag_a_addr(xb, LDS, 0, ks * 16, lane));
#pragma unroll
    for (int nt = 0; nt < NT; nt += 2) {
      uint32_t b[4];
      ldsm_x4(b, frag_bn_addr(wb, LDS, nt * 8, ks * 16, lane));
      mma16816(acc[nt], a, b[0], b[1]);
      mma16816(acc[nt + 1], a, b[2], b[3]);
    }
  }
  const int r = lane >> 2, c = (lane & 3) * 2;
  float* rw = red + warp * 16 * LDR;
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    *reinterpret_cast<float2*>(rw + r * LDR + nt * 8 + c) = make_float2(acc[nt][0], acc[nt][1]);
    *reinterpret_cast<float2*>(rw + (r + 8) * LDR + nt * 8 + c) = make_float2(acc[nt][2], acc[nt][3]);
  }
  __syncthreads();
  for (int i = tid; i < 16 * JR; i += 128) {
    const int rr = i / JR, col = i % JR;
    const int64_t row = m0 + rr;
    if (row >= M) continue;
    const float s = red[rr * LDR + col] + red[16 * LDR + rr * LDR + col] + red[32 * LDR + rr * LDR + col] +
                    red[48 * LDR + rr * LDR + col];
    out[row * ldo + col] = f_to_h(alpha * s);
  }
}

template <int NT>
int64_t skinny_slab_smem(int64_t K) {
  return (16 + NT * 8) * (K + 8) * 2 + 4 * 16 * (NT * 8 + 4) * 4;
}

// The slab kernel when the token count is short and the slab fits; true if it was launched.
template <int NT>
bool skinny_slab_launch(const uint16_t* X, int64_t ldx, int64_t M, int64_t K, const uint16_t* W, int64_t ldw,
                        float alpha, uint16_t* out, int64_t ldo, cudaStream_t st) {
  const int64_t smem = skinny_slab_smem<NT>(K);
  if (M > 1024 || smem > 200 * 1024 || K % 16) return false;
  static int64_t set = 0;
  if (smem > set) {
    if (cudaFuncSetAttribute(skinny_slab_kernel<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem)) != cudaSuccess) {
      cudaGetLastError();
      return false;
    }
    set = smem;
  }
  launch_k(skinny_slab_kernel<NT>, static_cast<unsigned>((M + 15) / 16), 128, static_cast<size_t>(smem), st, X, ldx,
           M, static_cast<int>(K), W, ldw, alpha, out, ldo);
  return true;
}

// Token counts above this stream X through the tcgen05 kernel (skinny_tc.cu): with the warp-level
// kernel's two small cp.async stages per CTA the X pass ran at under a tenth of HBM bandwidth at
// 16384 tokens.
constexpr int64_t kSkinnyTcMinM = 1024;

template <int NT>
void skinny_launch(const uint16_t* X, int64_t ldx, int64_t M, int64_t K, const uint16_t* W, int64_t ldw, float alpha,
                   uint16_t* out, int64_t ldo, cudaStream_t st, int* err) {
  if (M > kSkinnyTcMinM && K % 64 == 0 && ldx % 8 == 0 && ldw % 8 == 0 &&
      !((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(W)) & 15)) {
    launch_skinny_tc(X, ldx, M, K, W, ldw, alpha, out, ldo, err, st);
    return;
  }
  if (skinny_slab_launch<NT>(X, ldx, M, K, W, ldw, alpha, out, ldo, st)) return;
  const int gx = static_cast<int>((M + 63) / 64);
  const int nk = static_cast<int>(K / 64);
  // Split K over a cluster when the row blocks alone leave most of the SMs idle: up to 8 splits
  // of >= 2 K tiles, at most ~2 CTAs per SM in total.
  int splits = 1;
  if (gx < 152) splits = std::max(1, std::min({8, nk / 2, (2 * 152) / gx}));
  const int kt_split = (nk + splits - 1) / splits;
  splits = std::max(1, (nk + kt_split - 1) / kt_split);
  launch_k_cluster(skinny_gemm_kernel<NT>, dim3(gx, splits), 128, 0, st, dim3(1, splits, 1), X, ldx, M, K, W, ldw,
                   alpha, out, ldo, kt_split);
}

void launch_skinny_gemm(const uint16_t* X, int64_t ldx, int64_t M, int64_t K, const uint16_t* W, int64_t ldw, int J,
                        float alpha, uint16_t* out, int64_t ldo, cudaStream_t st, int* err) {
  (void)J;  // W holds ldo rows (zero beyond the used ranks), so every output column is written
  if (M <= 0) return;
  switch (ldo) {
    case 16: skinny_launch<2>(X, ldx, M, K, W, ldw, alpha, out, ldo, st, err); break;
    case 32: skinny_launch<4>(X, ldx, M, K, W, ldw, alpha, out, ldo, st, err); break;
    case 48: skinny_launch<6>(X, ldx, M, K, W, ldw, alpha, out, ldo, st, err); break;
    case 64: skinny_launch<8>(X, ldx, M, K, W, ldw, alpha, out, ldo, st, err); break;
    default: skinny_launch<12>(X, ldx, M, K, W, ldw, alpha, out, ldo, st, err); break;
  }
}

// ------------------------------------------------------------------------------------ tall reduce
// Direct output of a single-split reduction: C[p * sp + q * sq] (+)= mult * sum.
struct Direct {
  float* C;
  int64_t sp, sq;
  int accumulate;
  const float* mult;
};

// part[z][p][q] = sum_{m in split z} P[m, p] Q[m, q]   (p < Pw, q < Qw).  NS-stage cp.async
// pipeline over the token axis (three stages measured slower than two at 16384 tokens: fewer
// CTAs fit on an SM).
template <int NQ, int NS = 2>
__global__ void __launch_bounds__(128) tall_reduce_kernel(const uint16_t* __restrict__ P, int64_t ldp,
                                                          const uint16_t* __restrict__ Q, int64_t ldq, int64_t M,
                                                          int Pw, int Qw, int64_t m_per_split,
                                                          float* __restrict__ part, Direct dw) {
  griddep_wait();
  griddep_launch();
  constexpr int BP = 64, BMr = 64, QT = NQ * 8, LDP = BP + 8, LDQ = QT + 8;
  __shared__ __align__(16) uint16_t ps[NS][BMr * LDP];
  __shared__ __align__(16) uint16_t qs[NS][BMr * LDQ];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int p0 = blockIdx.x * BP, q0 = blockIdx.y * QT;
  const int64_t mb = static_cast<int64_t>(blockIdx.z) * m_per_split;
  const int64_t me = min(M, mb + m_per_split);
  float acc[NQ][4];
#pragma unroll
  for (int i = 0; i < NQ; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.0f;

  auto load = [&](int stage, int64_t m) {
    for (int c = tid; c < BMr * 8; c += 128) {
      const int r = c >> 3, cc = c & 7;
      const bool v = (m + r < me) && (p0 + cc * 8 < Pw);
      const uint16_t* src = v ? P + (m + r) * ldp + p0 + cc * 8 : P;
      cp_async16(smem_u32(&ps[stage][r * LDP + cc * 8]), src, v);
    }
    for (int c = tid; c < BMr * NQ; c += 128) {
      const int r = c / NQ, cc = c % NQ;
      const bool v = (m + r < me) && (q0 + cc * 8 < Qw);
      const uint16_t* src = v ? Q + (m + r) * ldq + q0 + cc * 8 : Q;
      cp_async16(smem_u32(&qs[stage][r * LDQ + cc * 8]), src, v);
    }
  };
  const int64_t ntile = (me - mb + BMr - 1) / BMr;
#pragma unroll
  for (int st = 0; st < NS - 1; ++st) {  // one commit group per stage, empty past the end
    if (st < ntile) load(st, mb + st * BMr);
    cp_async_commit();
  }
  for (int64_t it = 0; it < ntile; ++it) {
    if (it + NS - 1 < ntile) load(static_cast<int>((it + NS - 1) % NS), mb + (it + NS - 1) * BMr);
    cp_async_commit();
    cp_async_wait<NS - 1>();  // the group of tile it has landed
    __syncthreads();
    const int s = static_cast<int>(it % NS);
    const uint32_t pb = smem_u32(ps[s]), qb = smem_u32(qs[s]);
#pragma unroll
    for (int kk = 0; kk < BMr; kk += 16) {
      uint32_t a[4];
      ldsm_x4_t(a, frag_at_addr(pb, LDP, warp * 16, kk, lane));
#pragma unroll
      for (int nq = 0; nq < NQ; nq += 2) {
        uint32_t b[4];
        ldsm_x4_t(b, frag_bk_addr(qb, LDQ, nq * 8, kk, lane));
        mma16816(acc[nq], a, b[0], b[1]);
        mma16816(acc[nq + 1], a, b[2], b[3]);
      }
    }
    __syncthreads();
  }
  const int r = lane >> 2, c = (lane & 3) * 2;
  const int pr = p0 + warp * 16 + r;
  if (dw.C) {  // a single split: finish here (C (+)= mult * sum)
    const float mu = dw.mult ? *dw.mult : 1.0f;
#pragma unroll
    for (int nq = 0; nq < NQ; ++nq) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int pp = pr + ((e >> 1) << 3), qq = q0 + nq * 8 + c + (e & 1);
        if (pp >= Pw || qq >= Qw) continue;
        float* dst = dw.C + pp * dw.sp + qq * dw.sq;
        *dst = dw.accumulate ? *dst + mu * acc[nq][e] : mu * acc[nq][e];
      }
    }
    return;
  }
  float* out = part + static_cast<int64_t>(blockIdx.z) * Pw * Qw;
#pragma unroll
  for (int nq = 0; nq < NQ; ++nq) {
    const int qc = q0 + nq * 8 + c;
    if (qc >= Qw) continue;
    if (pr < Pw) *reinterpret_cast<float2*>(out + static_cast<int64_t>(pr) * Qw + qc) = make_float2(acc[nq][0], acc[nq][1]);
    if (pr + 8 < Pw)
      *reinterpret_cast<float2*>(out + static_cast<int64_t>(pr + 8) * Qw + qc) = make_float2(acc[nq][2], acc[nq][3]);
  }
}

// C[p * sp + q * sq] (+)= mult * sum_z part[z][p][q]  in split order.
__global__ void split_sum_kernel(const float* __restrict__ part, int splits, int Pw, int Qw, float* __restrict__ C,
                                 int64_t sp, int64_t sq, int accumulate, const float* __restrict__ mult) {
  griddep_wait();
  griddep_launch();
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  const int64_t n = static_cast<int64_t>(Pw) * Qw;
  if (i >= n) return;
  float s = 0.0f;
  for (int z = 0; z < splits; ++z) s += part[z * n + i];
  if (mult) s *= *mult;
  const int64_t p = i / Qw, q = i % Qw;
  float* dst = C + p * sp + q * sq;
  *dst = accumulate ? *dst + s : s;
}

void launch_split_sum(const float* part, int splits, int Pw, int Qw, float* C, int64_t sp, int64_t sq, bool accumulate,
                      const float* mult, cudaStream_t st) {
  const int64_t n = static_cast<int64_t>(Pw) * Qw;
  launch_k(split_sum_kernel, static_cast<unsigned>((n + 255) / 256), 256, 0, st, part, splits, Pw, Qw, C, sp, sq,
           accumulate ? 1 : 0, mult);
}

// Token counts from this on take the tcgen05 kernel (tall_tc.cu) where the shapes allow.
constexpr int64_t kTallTcMinM = 2048;

bool tall_tc_takes(int64_t M, int Pw, int nq, int r) {
  const int qw = nq * r;
  return M >= kTallTcMinM && Pw % 64 == 0 && r % 16 == 0 && (qw == 16 || qw == 32 || qw == 64 || qw == 96);
}

int launch_tall_reduce_multi(const uint16_t* P, int64_t ldp, const uint16_t* Q, int64_t ldq, int64_t M, int Pw,
                             int nq, int r, float* const* C, int64_t ldc, bool accumulate, const float* mult,
                             float* scratch, int64_t scratch_floats, int* err, cudaStream_t st) {
  if (Pw <= 0 || M <= 0) return MEBP_OK;
  if (tall_tc_takes(M, Pw, nq, r) && ldp % 8 == 0 && ldq % 8 == 0 &&
      !((reinterpret_cast<uintptr_t>(P) | reinterpret_cast<uintptr_t>(Q)) & 15)) {
    const int rc = launch_tall_tc(P, ldp, Q, ldq, M, Pw, nq, r, C, ldc, accumulate, mult, err, st);
    if (rc != MEBP_ERR_UNSUPPORTED) return rc;
  }
  for (int j = 0; j < nq; ++j) {  // one target at a time (the tensor-core kernel where it takes one)
    const int rc = nq > 1 ? launch_tall_reduce_multi(P, ldp, Q + j * r, ldq, M, Pw, 1, r, C + j, ldc, accumulate, mult,
                                                     scratch, scratch_floats, err, st)
                          : launch_tall_reduce(P, ldp, Q, ldq, M, Pw, r, C[0], ldc, accumulate, mult, scratch,
                                               scratch_floats, err, st);
    if (rc) return rc;
  }
  return MEBP_OK;
}

int64_t tall_reduce_scratch_floats(int64_t M, int Pw, int Qw) {
  (void)M;
  return static_cast<int64_t>(Pw) * Qw * 16;
}

// C is written with strides (sp, sq) = (ldc, 1) for ldc > 0, and (1, -ldc) for ldc < 0
// (transposed output).
int launch_tall_reduce(const uint16_t* P, int64_t ldp, const uint16_t* Q, int64_t ldq, int64_t M, int Pw, int Qw,
                       float* C, int64_t ldc, bool accumulate, const float* mult, float* scratch,
                       int64_t scratch_floats, int* err, cudaStream_t st) {
  (void)err;
  if (Pw <= 0 || Qw <= 0) return MEBP_OK;
  if ((Pw % 8) || (Qw % 8) || Qw > 96) return MEBP_ERR_UNSUPPORTED;
  const int nq = Qw <= 32 ? 4 : (Qw <= 64 ? 8 : 12);
  const int gx = (Pw + 63) / 64, gy = (Qw + nq * 8 - 1) / (nq * 8);
  int64_t splits = (4 * 152 + gx * gy - 1) / (gx * gy);
  splits = std::min<int64_t>(splits, std::max<int64_t>(1, M / 1024));  // short token ranges: one pass, no second kernel
  splits = std::min<int64_t>(splits, scratch_floats / (static_cast<int64_t>(Pw) * Qw));
  if (splits < 1) return MEBP_ERR_INVALID_ARG;
  int64_t mps = (M + splits - 1) / splits;
  mps = (mps + 63) / 64 * 64;
  splits = std::max<int64_t>(1, (M + mps - 1) / mps);
  dim3 grid(gx, gy, static_cast<unsigned>(splits));
  const int64_t sp = ldc > 0 ? ldc : 1, sq = ldc > 0 ? 1 : -ldc;
  Direct dw{nullptr, sp, sq, accumulate ? 1 : 0, mult};
  if (splits == 1) dw.C = C;
  switch (nq) {
    case 4: launch_k(tall_reduce_kernel<4>, grid, 128, 0, st, P, ldp, Q, ldq, M, Pw, Qw, mps, scratch, dw); break;
    case 8: launch_k(tall_reduce_kernel<8>, grid, 128, 0, st, P, ldp, Q, ldq, M, Pw, Qw, mps, scratch, dw); break;
    default: launch_k(tall_reduce_kernel<12>, grid, 128, 0, st, P, ldp, Q, ldq, M, Pw, Qw, mps, scratch, dw); break;
  }
  if (dw.C) return MEBP_OK;
  const int64_t n = static_cast<int64_t>(Pw) * Qw;
  launch_k(split_sum_kernel, static_cast<unsigned>((n + 255) / 256), 256, 0, st, scratch, static_cast<int>(splits), Pw,
           Qw, C, sp, sq, accumulate ? 1 : 0, mult);
  return MEBP_OK;
}

// Several single-pass reductions in one launch (the LoRA gradients of a block at short token
// counts, where each alone is a handful of CTAs): CTA -> (problem, 64-row block of its output).
// Three-stage cp.async pipeline over the token axis; C (+)= mult * sum, written directly.
__global__ void __launch_bounds__(128) tall_reduce_batched_kernel(const TallBatch b) {
  griddep_wait();
  griddep_launch();
  constexpr int NQ = 4, BP = 64, BMr = 64, QT = NQ * 8, LDP = BP + 8, LDQ = QT + 8, NS = 3;
  __shared__ __align__(16) uint16_t ps[NS][BMr * LDP];
  __shared__ __align__(16) uint16_t qs[NS][BMr * LDQ];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // this CTA's problem (fields read with compile-time indices: no local-memory copy)
  int idx = blockIdx.x, pi = 0;
#pragma unroll
  for (int i = 0; i < kTallMaxProbs; ++i)
    if (i < b.n && pi == i && idx >= b.p[i].ctas) {
      idx -= b.p[i].ctas;
      pi = i + 1;
    }
  TallProb pr;
#pragma unroll
  for (int i = 0; i < kTallMaxProbs; ++i)
    if (i == pi) pr = b.p[i];
  const int Pw = pr.Pw, Qw = pr.Qw;
  const int p0 = idx * BP;
  const int64_t M = b.M;
  float acc[NQ][4];
#pragma unroll
  for (int i = 0; i < NQ; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.0f;
  auto load = [&](int stage, int64_t m) {
    for (int c = tid; c < BMr * 8; c += 128) {
      const int r = c >> 3, cc = c & 7;
      const bool v = (m + r < M) && (p0 + cc * 8 < Pw);
      const uint16_t* src = v ? pr.P + (m + r) * pr.ldp + p0 + cc * 8 : pr.P;
      cp_async16(smem_u32(&ps[stage][r * LDP + cc * 8]), src, v);
    }
    for (int c = tid; c < BMr * NQ; c += 128) {
      const int r = c / NQ, cc = c % NQ;
      const bool v = (m + r < M) && (cc * 8 < Qw);
      const uint16_t* src = v ? pr.Q + (m + r) * pr.ldq + cc * 8 : pr.Q;
      cp_async16(smem_u32(&qs[stage][r * LDQ + cc * 8]), src, v);
    }
  };
  const int64_t ntile = (M + BMr - 1) / BMr;
#pragma unroll
  for (int st = 0; st < NS - 1; ++st) {
    if (st < ntile) load(st, st * BMr);
    cp_async_commit();
  }
  for (int64_t it = 0; it < ntile; ++it) {
    if (it + NS - 1 < ntile) load(static_cast<int>((it + NS - 1) % NS), (it + NS - 1) * BMr);
    cp_async_commit();
    cp_async_wait<NS - 1>();
    __syncthreads();
    const int s = static_cast<int>(it % NS);
    const uint32_t pb = smem_u32(ps[s]), qb = smem_u32(qs[s]);
#pragma unroll
    for (int kk = 0; kk < BMr; kk += 16) {
      uint32_t a[4];
      ldsm_x4_t(a, frag_at_addr(pb, LDP, warp * 16, kk, lane));
#pragma unroll
      for (int nq = 0; nq < NQ; nq += 2) {
        uint32_t bb[4];
        ldsm_x4_t(bb, frag_bk_addr(qb, LDQ, nq * 8, kk, lane));
        mma16816(acc[nq], a, bb[0], bb[1]);
        mma16816(acc[nq + 1], a, bb[2], bb[3]);
      }
    }
    __syncthreads();
  }
  const float mu = b.mult ? *b.mult : 1.0f;
  const int r = lane >> 2, c = (lane & 3) * 2;
  const int prow = p0 + warp * 16 + r;
#pragma unroll
  for (int nq = 0; nq < NQ; ++nq)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int pp = prow + ((e >> 1) << 3), qq = nq * 8 + c + (e & 1);
      if (pp >= Pw || qq >= Qw) continue;
      float* dst = pr.C + pp * pr.sp + qq * pr.sq;
      *dst = pr.acc ? *dst + mu * acc[nq][e] : mu * acc[nq][e];
    }
}

bool tall_batch_add(TallBatch& b, const uint16_t* P, int64_t ldp, const uint16_t* Q, int64_t ldq, int Pw, int Qw,
                    float* C, int64_t ldc, bool accumulate) {
  if (b.n >= kTallMaxProbs || Pw <= 0 || Qw <= 0 || Qw > 32 || (Pw % 8) || (Qw % 8)) return false;
  TallProb& p = b.p[b.n++];
  p.P = P; p.ldp = ldp; p.Q = Q; p.ldq = ldq; p.Pw = Pw; p.Qw = Qw; p.C = C;
  p.sp = ldc > 0 ? ldc : 1;
  p.sq = ldc > 0 ? 1 : -ldc;
  p.acc = accumulate ? 1 : 0;
  p.ctas = (Pw + 63) / 64;
  return true;
}

void launch_tall_reduce_batched(const TallBatch& b, cudaStream_t st) {
  int ctas = 0;
  for (int i = 0; i < b.n; ++i) ctas += b.p[i].ctas;
  if (ctas > 0) launch_k(tall_reduce_batched_kernel, static_cast<unsigned>(ctas), 128, 0, st, b);
}

// ------------------------------------------------------------------------------------ shadows
// Per-layer LoRA masters of one fused linear (up to 3 targets side by side).
struct ShadowTable {
  const float* A[kShadowMaxLayers][3];
  const float* B[kShadowMaxLayers][3];
  int ro[3];     // rank offset of target t in the concatenated rank axis
  int no[3];     // first output row of target t
  int nl[3];     // output rows of target t
  int nt;
};

// Layer blockIdx.y: A_cat [kx, K], B_cat [N, kx], Bt_cat [kx, N] at offsets layer * (stride_a,
// stride_b, stride_b).
__global__ void lora_shadow_kernel(ShadowTable a, int r, int K, int N, int kx, uint16_t* __restrict__ A_cat,
                                   uint16_t* __restrict__ B_cat, uint16_t* __restrict__ Bt_cat, int64_t stride_a,
                                   int64_t stride_b) {
  griddep_wait();
  griddep_launch();
  const int layer = blockIdx.y;
  const float* const* As = a.A[layer];
  const float* const* Bs = a.B[layer];
  A_cat += layer * stride_a;
  B_cat += layer * stride_b;
  Bt_cat += layer * stride_b;
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  const int64_t na = static_cast<int64_t>(kx) * K, nb = static_cast<int64_t>(N) * kx;
  if (i < na) {
    const int j = static_cast<int>(i / K), k = static_cast<int>(i % K);
    float v = 0.0f;
    for (int t = 0; t < a.nt; ++t)
      if (j >= a.ro[t] && j < a.ro[t] + r) v = As[t][static_cast<int64_t>(j - a.ro[t]) * K + k];
    A_cat[i] = f_to_h(v);
  }
  if (i < nb) {
    const int n = static_cast<int>(i / kx), j = static_cast<int>(i % kx);
    float v = 0.0f;
    for (int t = 0; t < a.nt; ++t)
      if (j >= a.ro[t] && j < a.ro[t] + r && n >= a.no[t] && n < a.no[t] + a.nl[t])
        v = Bs[t][static_cast<int64_t>(n - a.no[t]) * r + (j - a.ro[t])];
    const uint16_t b = f_to_h(v);
    B_cat[i] = b;
    Bt_cat[static_cast<int64_t>(j) * N + n] = b;
  }
}

void launch_lora_shadow_layers(int n_layers, const float* const* A, const float* const* B, int nt,
                               const int* ranks_off, const int* n_off, const int* n_len, int r, int K, int N, int kx,
                               uint16_t* A_cat, uint16_t* B_cat, uint16_t* Bt_cat, int64_t stride_a, int64_t stride_b,
                               cudaStream_t st) {
  const int64_t n = std::max(static_cast<int64_t>(kx) * K, static_cast<int64_t>(N) * kx);
  for (int l0 = 0; l0 < n_layers; l0 += kShadowMaxLayers) {
    const int nl_batch = std::min(kShadowMaxLayers, n_layers - l0);
    ShadowTable a{};
    a.nt = nt;
    for (int t = 0; t < nt && t < 3; ++t) {
      a.ro[t] = ranks_off[t];
      a.no[t] = n_off[t];
      a.nl[t] = n_len[t];
      for (int l = 0; l < nl_batch; ++l) {
        a.A[l][t] = A[(l0 + l) * 3 + t];
        a.B[l][t] = B[(l0 + l) * 3 + t];
      }
    }
    launch_k(lora_shadow_kernel, dim3(static_cast<unsigned>((n + 255) / 256), static_cast<unsigned>(nl_batch)), 256,
             0, st, a, r, K, N, kx, A_cat + l0 * stride_a, B_cat + l0 * stride_b, Bt_cat + l0 * stride_b, stride_a,
             stride_b);
  }
}

void launch_lora_shadow(const float* const* A, const float* const* B, int nt, const int* ranks_off, const int* n_off,
                        const int* n_len, int r, int K, int N, int kx, uint16_t* A_cat, uint16_t* B_cat,
                        uint16_t* Bt_cat, cudaStream_t st) {
  const float* Al[3] = {nullptr, nullptr, nullptr};
  const float* Bl[3] = {nullptr, nullptr, nullptr};
  for (int t = 0; t < nt && t < 3; ++t) {
    Al[t] = A[t];
    Bl[t] = B[t];
  }
  launch_lora_shadow_layers(1, Al, Bl, nt, ranks_off, n_off, n_len, r, K, N, kx, A_cat, B_cat, Bt_cat, 0, 0, st);
}

}  // namespace mebp
