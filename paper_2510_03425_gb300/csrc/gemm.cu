// Fused dequant-in-the-mainloop GEMM on 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
//   FWD   : C[M, N] = A[M, K] * deq(W)^T      W packed [N, K]  (Y = X W^T of a linear layer)
//   TRANS : C[M, N] = A[M, K] * deq(W)        W packed [K, N]  (dX = dY W, the input gradient)
//   plus an optional extra K-block  A_x[M, Kx] * B_x^T  that carries the rank-r LoRA product
//   (FWD: A_x = s X A^T, B_x = B [N, Kx];  TRANS: A_x = s dY B, B_x = A [Kx, N]).
//
// This is the decompression of Algorithm 1's LazyLoadAndDecompressWeights fused into the GEMM:
// TMA brings the packed 4-bit tile and its fp16 scales into shared memory, sixteen converter
// warps turn them into the fp16 operand (bit-exact fp16_rne(q*s), see dequant.cuh) in the
// 128-byte-swizzled layout tcgen05 reads, one thread issues tcgen05.mma into fp32 TMEM
// accumulators, and the same sixteen warps run the epilogue out of TMEM.
//
// CTA: 16 (NACC 1) or 8 (NACC 2) converter warps that also run the epilogue, then one warp that
// issues TMA and one that issues MMA and owns the TMEM allocation.  Tile (128*NACC) x 256 x 64: NACC 128-row A tiles share every
// decoded 256-row B tile (NACC = 2 halves the decode work per flop and fills all 512 TMEM
// columns).  Two shared-memory rings: a TMA ring (A tile(s) + packed nibbles + scales, with
// separate barriers for the weight half and the activation half, so weights can be fetched and
// decoded before the previous kernel has finished) and a ring of decoded B tiles written by the
// converters (which also copy the LoRA B tile there).  Small grids split K over a thread-block
// cluster along z and reduce the fp32 partial tiles through distributed shared memory
// (deterministic, no workspace, no extra launch).
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstdint>

#include "dequant.cuh"
#include "kernels.h"

namespace mebp {
namespace gemm {

constexpr int BM = 128, BN = 256, BK = 64;
// Decode + epilogue warps: 16 (two threads per decoded row) when one 128-row accumulator uses
// each decoded tile, so the decode keeps pace with the tensor pipe; 8 with two accumulators,
// where the decode is not the limit and fewer warps compete with the MMA-issuing thread.
template <int NACC>
struct Warps {
  static constexpr int CONV = NACC == 1 ? 16 : 8;
  static constexpr int TPR = CONV / 8;  // converter threads per decoded 256-row tile row
  static constexpr int CONV_THREADS = CONV * 32;
  static constexpr int TMA = CONV, MMA = CONV + 1;
  static constexpr int THREADS = CONV_THREADS + 64;
};
constexpr int B_BYTES = BN * BK * 2, A_BYTES = BM * BK * 2, P_BYTES = BN * BK / 2, S_BYTES = 512;

// Shared-memory layout for NACC accumulators (tiles 1024-byte aligned).
template <int NACC>
struct Layout {
  static constexpr int TSTG = NACC == 1 ? 4 : 3;                    // TMA ring depth
  // decoded-B ring depth: three slots let the decode of a step start two steps ahead of its MMAs
  // (with two accumulators two slots measured 2-4 % slower; a TMA slot traded for a fourth, 20 %)
  static constexpr int BSTG = 3;
  static constexpr int A_OFF = 0;                                   // fp16 A: NACC x 128 x 64
  static constexpr int P_OFF = NACC * A_BYTES;                      // packed nibbles
  static constexpr int S_OFF = P_OFF + P_BYTES;                     // fp16 scales
  static constexpr int T_STRIDE = (S_OFF + S_BYTES + 1023) / 1024 * 1024;
  static constexpr int B_BASE = TSTG * T_STRIDE;                    // decoded fp16 B ring
  static constexpr int BAR_OFF = B_BASE + BSTG * B_BYTES;
  static constexpr int SMEM = BAR_OFF + 512 + 1024;                 // + barriers + alignment slack
  static constexpr uint32_t TMEM_COLS = 256 * NACC;
};
static_assert(Layout<1>::SMEM <= 232448 && Layout<2>::SMEM <= 232448, "shared memory budget");
// One CTA per SM (no two GEMM CTAs ever share an SM's TMEM), and the split-K partial tile fits in
// the idle rings.
static_assert(Layout<1>::SMEM > 232448 / 2 && Layout<2>::SMEM > 232448 / 2, "one CTA per SM");
static_assert(Layout<1>::BAR_OFF >= BM * BN * 4, "partial tile fits below the barriers");
static_assert(Layout<1>::BAR_OFF >= Warps<1>::CONV * 8192 && Layout<2>::BAR_OFF >= Warps<2>::CONV * 8192,
              "epilogue staging slots fit below the barriers");

struct Params {
  int M, N, K;
  int kx_steps;        // 16-wide MMA steps of the extra (LoRA) block; 0 = none
  int kx;              // LoRA block width (columns of A_x / B_x, multiple of 16)
  const uint16_t* Bx;  // LoRA B operand (FWD [N, kx], TRANS [kx, N]), row pitch ldbx
  int64_t ldbx;
  int kt_split;        // main 64-wide K tiles per split (blockIdx.z)
  int m_group;         // > 0: grouped tile order over a 1-D grid (see the host), else (n, m) = blockIdx
  int tiles_m, tiles_n;
  int epi;             // GemmEpi
  void* C;
  int64_t ldc;
  const float* R;      // fp32 residual / accumulation source (EPI_F32), may alias C
  int64_t ldr;
  float alpha;         // EPI_F32: C = alpha * acc (+ R)
  // LM-head epilogues
  const int32_t* targets;  // [M]
  int col_offset;          // global vocabulary index of GEMM column 0
  int n_valid;             // GEMM columns >= n_valid are outside the vocabulary
  float* lse_part;         // EPI_LSE: float2 [M, nparts]
  int nparts;
  float* zt;               // EPI_LSE: target logit [M]
  const float* lse;        // EPI_CEGRAD: [M]
  const float* ce_w;       // EPI_CEGRAD: device scalar weight of a valid row
  void* C2;                // EPI_GLU: gate and up outputs (fp16), or null
  int64_t ldc2;
  int glu_half;            // EPI_GLU: rows of the gate half of the fused weight
  int act;                 // EPI_GLU: activation
  int64_t zstride;         // > 0: K split through memory (no cluster): CTA z stores its fp32 partial
                           // tile with the EPI_F32 epilogue at C + z * zstride
  int* err;
};

// ---------------------------------------------------------------------------------- convert
// TPR converter threads per decoded row (1 or 2): thread t handles part h of its row's 8 words.
// FWD: packed tile [256 rows][32 B] (plain), scales [256]; row r = t / TPR goes to the K-major
// SW128 B tile (row r at r*128 B, 16-byte chunk j stored at chunk j ^ (r&7)).
template <int TPR>
__device__ __forceinline__ void convert_fwd(const uint8_t* pk, const uint8_t* sc, uint8_t* bt, int t) {
  constexpr int NW = 8 / TPR;
  const int r = t / TPR, h = t % TPR;
  const uint4* src = reinterpret_cast<const uint4*>(pk + r * 32) + h * (NW / 4);
  uint32_t words[NW];
#pragma unroll
  for (int i = 0; i < NW / 4; ++i) {
    const uint4 p = src[i];
    words[4 * i] = p.x; words[4 * i + 1] = p.y; words[4 * i + 2] = p.z; words[4 * i + 3] = p.w;
  }
  const uint32_t s2 = scale_pair(reinterpret_cast<const uint16_t*>(sc)[r]);
  uint8_t* row = bt + r * 128;
#pragma unroll
  for (int w = 0; w < NW; ++w) {
    const int j = NW * h + w;
    uint32_t o[4];
    dequant_word(words[w], s2, o);
    *reinterpret_cast<uint4*>(row + ((j ^ (r & 7)) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// TRANS: packed tile [64 k-rows][128 B] loaded with the 128-byte swizzle (chunk c of row k at
// chunk c ^ (k&7)), scales [4 groups][64 k-rows].  Thread t: row k = t & 63, group g =
// (t >> 6) & 3 (64 output columns), part h = t >> 8; packed chunks 2g .. 2g+1 (part h of them)
// become chunks of row k of MN-major atom g (atom = 64 columns x 64 k-rows, 128 B per k-row,
// chunk c stored at c ^ (k&7)).  Consecutive threads take consecutive k: conflict-free.
template <int TPR>
__device__ __forceinline__ void convert_trans(const uint8_t* pk, const uint8_t* sc, uint8_t* bt, int t) {
  constexpr int NW = 8 / TPR;
  const int k = t & 63, g = (t >> 6) & 3, h = t >> 8;
  const uint8_t* prow = pk + k * 128;
  uint32_t words[NW];
#pragma unroll
  for (int i = 0; i < NW / 4; ++i) {
    const int c = 2 * g + h * (NW / 4) + i;
    const uint4 p = *reinterpret_cast<const uint4*>(prow + ((c ^ (k & 7)) << 4));
    words[4 * i] = p.x; words[4 * i + 1] = p.y; words[4 * i + 2] = p.z; words[4 * i + 3] = p.w;
  }
  const uint32_t s2 = scale_pair(reinterpret_cast<const uint16_t*>(sc)[g * 64 + k]);
  uint8_t* row = bt + g * 8192 + k * 128;
#pragma unroll
  for (int w = 0; w < NW; ++w) {
    const int j = NW * h + w;
    uint32_t o[4];
    dequant_word(words[w], s2, o);
    *reinterpret_cast<uint4*>(row + ((j ^ (k & 7)) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// LoRA block e: copy the 64-wide slice of B_x into the B slot in the layout the MMA reads,
// zero outside [0, kx) x [0, N).  The operand is a few tens of KB and stays in L2.
template <bool TRANS, int TPR>
__device__ __forceinline__ void copy_lora_b(const Params& p, int e, int n0, uint8_t* bt, int t) {
  constexpr int NW = 8 / TPR;
  const uint4 zero = make_uint4(0, 0, 0, 0);
  if (!TRANS) {  // K-major: row r, chunk j = 8 columns of the rank axis
    const int r = t / TPR, h = t % TPR;
    // EPI_GLU: tile rows 0-127 are gate rows n0/2 + r, rows 128-255 the up rows glu_half + n0/2 + r - 128
    const int n = p.epi != EPI_GLU ? n0 + r : (r < BN / 2 ? n0 / 2 + r : p.glu_half + n0 / 2 + r - BN / 2);
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      const int j = NW * h + w;
      const int col = e * 64 + 8 * j;
      uint4 v = zero;
      if (n < p.N && col < p.kx) v = *reinterpret_cast<const uint4*>(p.Bx + static_cast<int64_t>(n) * p.ldbx + col);
      *reinterpret_cast<uint4*>(bt + r * 128 + ((j ^ (r & 7)) << 4)) = v;
    }
  } else {       // MN-major: atom g (64 output columns), row k of the rank axis
    const int k = t & 63, g = (t >> 6) & 3, h = t >> 8;
    const int rr = e * 64 + k;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      const int c = NW * h + w;
      const int col = n0 + 64 * g + 8 * c;
      uint4 v = zero;
      if (rr < p.kx && col < p.N) v = *reinterpret_cast<const uint4*>(p.Bx + static_cast<int64_t>(rr) * p.ldbx + col);
      *reinterpret_cast<uint4*>(bt + g * 8192 + k * 128 + ((c ^ (k & 7)) << 4)) = v;
    }
  }
}

// ---------------------------------------------------------------------------------- epilogue
// Warp w reads TMEM lanes 32*(w&3) .. +31 (a warp may only touch its lane quarter); the warps
// of a quarter split the NACC x 256 accumulator columns into column groups cg = w >> 2:
// NACC = 1 (16 warps): columns 64*cg .. +63 of the single accumulator;
// NACC = 2 (8 warps):  accumulator cg (tile rows 128*cg + ...), all 256 columns.
// Stored outputs go through the warp's 8 KB slot `stage` of shared memory (the rings are idle
// once the accumulator is final), 64 columns per round.  tcgen05.ld hands each thread one row, so
// written straight to global memory every store instruction would touch 32 rows (32 lines); that
// made the epilogue a quarter of a CTA's life.  Phase 1: thread = row writes its values to the
// slot, 16-byte chunk c of row r at chunk c ^ (r & 7) within its 128-byte half (no bank
// conflicts).  Phase 2: the warp copies the slot out with consecutive lanes on consecutive chunks
// of a row, so each instruction writes (and, for the residual, reads) whole 128-byte lines.
template <bool TRANS, int NACC>
__device__ __forceinline__ void epilogue(const Params& p, uint32_t tmem, int warp, int lane, int m0, int n0,
                                         uint8_t* stage) {
  const int q = warp & 3, cg = warp >> 2;
  constexpr int NCG = Warps<NACC>::CONV / 4;            // column groups
  constexpr int COLS = NACC * 256 / NCG;                // columns per group
  constexpr int NCH = COLS / 32;                        // 32-column chunks per thread
  static_assert(COLS <= 256 && 256 % COLS == 0, "a column group stays in one accumulator");
  const int acc = (cg * COLS) / 256;
  const int col0 = (cg * COLS) % 256;
  const int row = m0 + 128 * acc + 32 * q + lane;
  const bool row_ok = row < p.M;
  const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * q) << 16) + 256 * acc + col0;
  const int cbase = n0 + col0;  // first GEMM column of this thread's range

  if (!TRANS && p.epi == EPI_LSE) {  // the LM-head epilogues run on forward GEMMs only
    float mx = -INFINITY, sum = 0.0f, zt = 0.0f;
    bool has_t = false;
    const int tgt = row_ok ? p.targets[row] - p.col_offset : -1;
    auto chunk = [&](const uint32_t (&r)[32], int cc) {
      float v[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
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
    };
    static_assert(NCH % 2 == 0, "chunks are processed in pairs");
    uint32_t ra[32];
    if constexpr (NACC == 2) {  // the TMEM loads run one chunk ahead of the arithmetic
      uint32_t rb[32];
      tmem_ld32_issue(tbase, ra);
#pragma unroll 1
      for (int cc = 0; cc < NCH; cc += 2) {
        tmem_wait_ld32(ra);
        tmem_ld32_issue(tbase + 32 * (cc + 1), rb);
        chunk(ra, cc);
        tmem_wait_ld32(rb);
        if (cc + 2 < NCH) tmem_ld32_issue(tbase + 32 * (cc + 2), ra);
        chunk(rb, cc + 1);
      }
    } else {  // 96 registers a thread: one load at a time
#pragma unroll 1
      for (int cc = 0; cc < NCH; ++cc) {
        tmem_ld32_issue(tbase + 32 * cc, ra);
        tmem_wait_ld32(ra);
        chunk(ra, cc);
      }
    }
    if (row_ok) {  // four (max, sum) parts per 256-column tile and row; unused parts are empty
      float2* pr = reinterpret_cast<float2*>(p.lse_part) + static_cast<int64_t>(row) * p.nparts + (n0 / BN) * 4;
      constexpr int GPR = 256 / COLS;      // column groups per row (1 or 4)
      const int part = col0 / COLS;
      pr[part] = make_float2(mx, sum);
      if (GPR == 1)
        for (int k = 1; k < 4; ++k) pr[k] = make_float2(-INFINITY, 0.0f);
      if (has_t) p.zt[row] = zt;
    }
    return;
  }

  {
    if (!TRANS && p.epi == EPI_GLU) {
      // The accumulator holds the gate (columns 0-127) and up (128-255) pre-activations of hidden
      // units j0 .. j0 + 127, j0 = n0 / 2.  NACC = 2: the warp takes all 128 units of its
      // accumulator; NACC = 1: column group cg takes units 32 cg .. +31 (gate and up columns of
      // the same units, not the group's own 64 columns).  Per round of 32 units: gate and up
      // rounded to fp16 (the values the unfused path stores), m = act(gate) up from those, as the
      // GLU kernel computes it (bit-identical), all three staged at 64 bytes per row (16-byte chunk
      // c of row r at chunk c ^ ((r >> 1) & 3): conflict-free) and written out 8 rows per
      // instruction.
      const int j0 = n0 / 2, row0 = row - lane;
      const int u_beg = col0 / 2, u_end = u_beg + COLS / 2;
      const uint32_t tacc = tmem + (static_cast<uint32_t>(32 * q) << 16) + 256 * acc;
      // slots of 2 KB in the staging area: m at +0, gate at +2048, up at +4096
      const int nout = p.C2 ? 3 : 1;
      uint32_t bad = 0;
#pragma unroll 1
      for (int u0 = u_beg; u0 < u_end; u0 += 32) {
        const int j = j0 + u0;
        if (j >= p.glu_half) break;  // warp-uniform
        float gv[32], uv[32];
        {  // both loads in flight at once
          uint32_t rg[32], ru[32];
          tmem_ld32x2(tacc + u0, tacc + 128 + u0, rg, ru);
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            gv[i] = __uint_as_float(rg[i]);
            uv[i] = __uint_as_float(ru[i]);
          }
        }
#pragma unroll
        for (int c = 0; c < 4; ++c) {  // 8 units per 16-byte chunk
          uint32_t mo[4], go[4], uo[4];
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int e = 8 * c + 2 * k;
            go[k] = pack_half2(gv[e], gv[e + 1]);
            uo[k] = pack_half2(uv[e], uv[e + 1]);
            mo[k] = pack_half2(act_f(h2_lo(go[k]), p.act) * h2_lo(uo[k]), act_f(h2_hi(go[k]), p.act) * h2_hi(uo[k]));
            if (row_ok) bad |= h2_exp_probe(mo[k]) | (p.C2 ? h2_exp_probe(go[k]) | h2_exp_probe(uo[k]) : 0u);
          }
          const int off = lane * 64 + ((c ^ ((lane >> 1) & 3)) << 4);
          *reinterpret_cast<uint4*>(stage + off) = make_uint4(mo[0], mo[1], mo[2], mo[3]);
          if (p.C2) {
            *reinterpret_cast<uint4*>(stage + 2048 + off) = make_uint4(go[0], go[1], go[2], go[3]);
            *reinterpret_cast<uint4*>(stage + 4096 + off) = make_uint4(uo[0], uo[1], uo[2], uo[3]);
          }
        }
        __syncwarp();
        const int c = lane & 3;
#pragma unroll 1
        for (int o = 0; o < nout; ++o) {
          uint16_t* dst = o == 0 ? static_cast<uint16_t*>(p.C) + j
                                 : static_cast<uint16_t*>(p.C2) + (o == 1 ? j : p.glu_half + j);
          const int64_t ld = o == 0 ? p.ldc : p.ldc2;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int rr = 8 * i + (lane >> 2), r = row0 + rr;
            const uint4 v = *reinterpret_cast<const uint4*>(stage + o * 2048 + rr * 64 + ((c ^ ((rr >> 1) & 3)) << 4));
            if (r < p.M) *reinterpret_cast<uint4*>(dst + static_cast<int64_t>(r) * ld + 8 * c) = v;
          }
        }
        __syncwarp();  // the slots are rewritten by the next round
      }
      if (bad & kH2Bad) flag_error(p.err, kErrNonFinite);
      return;
    }
  }

  // EPI_F16, EPI_CEGRAD (fp16 rows of 128 bytes per round) and EPI_F32 (fp32, 256 bytes)
  const bool f32 = p.epi == EPI_F32, ce = !TRANS && p.epi == EPI_CEGRAD;
  const float lse = (ce && row_ok) ? p.lse[row] : 0.0f;
  const int tgt = (ce && row_ok) ? p.targets[row] : -1;
  const float cw = (tgt >= 0) ? *p.ce_w : 0.0f;
  const int tl = tgt - p.col_offset;
  const int row0 = row - lane;
  uint32_t bad = 0;  // OR of h2_exp_probe over the fp16 outputs (an overflow or NaN sets kH2Bad bits)
  // Phase 1 for one 32-column chunk: half hh of round rd (first column c0 of the round).
  auto stage32 = [&](float (&v)[32], int hh, int c0) {
    if (f32) {
      uint8_t* srow = stage + lane * 256;
#pragma unroll
      for (int jj = 0; jj < 8; ++jj) {
        const int j = 8 * hh + jj;
        *reinterpret_cast<float4*>(srow + (((j & 8) | ((j ^ lane) & 7)) << 4)) =
            make_float4(p.alpha * v[4 * jj], p.alpha * v[4 * jj + 1], p.alpha * v[4 * jj + 2], p.alpha * v[4 * jj + 3]);
      }
    } else {
      if (ce) {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int col = c0 + 32 * hh + i;
          float a = (col < p.n_valid) ? __expf(v[i] - lse) * cw : 0.0f;
          if (col == tl) a -= cw;
          v[i] = a;
        }
      }
      uint8_t* srow = stage + lane * 128;
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        const int j = 4 * hh + jj;
        const uint4 o = make_uint4(pack_half2(v[8 * jj], v[8 * jj + 1]), pack_half2(v[8 * jj + 2], v[8 * jj + 3]),
                                   pack_half2(v[8 * jj + 4], v[8 * jj + 5]), pack_half2(v[8 * jj + 6], v[8 * jj + 7]));
        if (!ce && row_ok) bad |= h2_exp_probe(o.x) | h2_exp_probe(o.y) | h2_exp_probe(o.z) | h2_exp_probe(o.w);
        *reinterpret_cast<uint4*>(srow + (((j ^ lane) & 7) << 4)) = o;
      }
    }
  };
#pragma unroll 1
  for (int rd = 0; rd < COLS / 64; ++rd) {
    const int c0 = cbase + 64 * rd;
    if (c0 >= p.N) break;  // warp-uniform (N is a multiple of 64)
    // ---- phase 1: this thread's row into the slot.  Forward GEMMs with fp16 outputs: both
    // 32-column loads of the round in flight at once (loading one round ahead as well needs more
    // than the 168 registers a thread has); otherwise one load at a time (the transposed kernel,
    // without the forward-only paths, stays at 106 registers: with them compiled in, at 168, it
    // ran 2-4 % slower)
    if (f32 || TRANS) {
#pragma unroll 1
      for (int hh = 0; hh < 2; ++hh) {
        float v[32];
        tmem_ld32(tbase + 64 * rd + 32 * hh, v);
        stage32(v, hh, c0);
      }
    } else {
      uint32_t ra[32], rb[32];
      tmem_ld32x2(tbase + 64 * rd, tbase + 64 * rd + 32, ra, rb);
      float v[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(ra[i]);
      stage32(v, 0, c0);
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(rb[i]);
      stage32(v, 1, c0);
    }
    __syncwarp();
    // ---- phase 2: whole lines out (rows past M skipped)
    if (f32) {
      float* C = static_cast<float*>(p.C) + blockIdx.z * p.zstride;
      const int c = lane & 15;
#pragma unroll 4
      for (int i = 0; i < 16; ++i) {
        const int rr = 2 * i + (lane >> 4), r = row0 + rr;
        float4 o = *reinterpret_cast<const float4*>(stage + rr * 256 + (((c & 8) | ((c ^ rr) & 7)) << 4));
        if (r < p.M) {
          if (p.R) {
            const float4 res = *reinterpret_cast<const float4*>(p.R + static_cast<int64_t>(r) * p.ldr + c0 + 4 * c);
            o.x += res.x; o.y += res.y; o.z += res.z; o.w += res.w;
          }
          *reinterpret_cast<float4*>(C + static_cast<int64_t>(r) * p.ldc + c0 + 4 * c) = o;
        }
      }
    } else {
      uint16_t* C = static_cast<uint16_t*>(p.C);
      const int c = lane & 7;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int rr = 4 * i + (lane >> 3), r = row0 + rr;
        const uint4 o = *reinterpret_cast<const uint4*>(stage + rr * 128 + (((c ^ rr) & 7) << 4));
        if (r < p.M) *reinterpret_cast<uint4*>(C + static_cast<int64_t>(r) * p.ldc + c0 + 8 * c) = o;
      }
    }
    __syncwarp();  // the slot is rewritten by the next round
  }
  if (bad & kH2Bad) flag_error(p.err, kErrNonFinite);
}

// ---------------------------------------------------------------------------------- split-K
// The splits of one output tile run as one thread-block cluster along z.  Each CTA parks its fp32
// accumulator tile in its own shared memory (the rings are idle once the accumulator is final):
// row r at r * 1 KB, 16-byte chunk c at chunk c ^ (r & 31), conflict-free for the row-per-thread
// writes and the chunk-per-thread reads.  After a cluster barrier CTA z sums rows
// [z * ceil(128/S), ...) of all S partials over distributed shared memory in split order
// (deterministic) and applies the epilogue.
__device__ __forceinline__ void stash_partial(uint32_t tmem, bool valid, int warp, int lane, uint8_t* smem) {
  static_assert(Warps<1>::CONV == 16, "one-accumulator kernels stash with 16 warps of 64 columns");
  const int q = warp & 3, cg = warp >> 2;
  const int r = 32 * q + lane;
  const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * q) << 16) + 64 * cg;
  uint8_t* row = smem + r * 1024;
#pragma unroll 1
  for (int cc = 0; cc < 2; ++cc) {
    float v[32];
    if (valid) {
      tmem_ld32(tbase + 32 * cc, v);
    } else {
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = 0.0f;
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int c = 16 * cg + 8 * cc + i;
      *reinterpret_cast<float4*>(row + ((c ^ (r & 31)) << 4)) =
          make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
    }
  }
}

__device__ __forceinline__ void split_reduce(const Params& p, const uint8_t* smem, int m0, int n0) {
  const int S = gridDim.z, z = blockIdx.z;
  const int rpc = (BM + S - 1) / S;
  const int r0 = z * rpc, r1 = min(BM, r0 + rpc);
  const uint32_t base = smem_u32(smem);
  for (int i = threadIdx.x; i < (r1 - r0) * 64; i += Warps<1>::THREADS) {
    const int r = r0 + (i >> 6), c = i & 63;
    const int64_t row = m0 + r, col = n0 + 4 * c;
    if (row >= p.M || col >= p.N) continue;
    const uint32_t off = base + r * 1024 + ((c ^ (r & 31)) << 4);
    float4 v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (j < S) v[j] = ld_dsmem_f4(dsmem_addr(off, j));
    float4 s = v[0];
#pragma unroll
    for (int j = 1; j < 8; ++j)
      if (j < S) {
        s.x += v[j].x; s.y += v[j].y; s.z += v[j].z; s.w += v[j].w;
      }
    if (p.epi == EPI_F16) {
      const uint2 o = make_uint2(pack_half2(s.x, s.y), pack_half2(s.z, s.w));
      if (h2_nonfinite(o.x) | h2_nonfinite(o.y)) flag_error(p.err, kErrNonFinite);
      *reinterpret_cast<uint2*>(static_cast<uint16_t*>(p.C) + row * p.ldc + col) = o;
    } else {
      float4 o = make_float4(p.alpha * s.x, p.alpha * s.y, p.alpha * s.z, p.alpha * s.w);
      if (p.R) {
        const float4 rr = *reinterpret_cast<const float4*>(p.R + row * p.ldr + col);
        o.x += rr.x; o.y += rr.y; o.z += rr.z; o.w += rr.w;
      }
      *reinterpret_cast<float4*>(static_cast<float*>(p.C) + row * p.ldc + col) = o;
    }
  }
}

// A K split through memory: partial tiles [S][M][N] (fp32, pitch N, split z at z * zstride) are
// summed in split order (deterministic) and given the epilogue the split replaced: C = alpha *
// sum (+ R, which may alias C) in fp32, or the sum rounded to fp16 with the overflow check.  One
// thread per 4 columns.
__global__ void ksplit_sum_kernel(const float* __restrict__ part, int S, int64_t zstride, int M, int N, float alpha,
                                  const float* R, int64_t ldr, void* C, int64_t ldc, int f16, int* err) {
  griddep_wait();  // the partials come from the GEMM right before
  griddep_launch();
  const int nq = N / 4;
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= static_cast<int64_t>(M) * nq) return;
  const int64_t row = i / nq, col = 4 * (i % nq);
  const float* src = part + row * N + col;
  float4 s = *reinterpret_cast<const float4*>(src);
  for (int z = 1; z < S; ++z) {
    const float4 v = *reinterpret_cast<const float4*>(src + z * zstride);
    s.x += v.x; s.y += v.y; s.z += v.z; s.w += v.w;
  }
  if (f16) {
    const uint2 o = make_uint2(pack_half2(s.x, s.y), pack_half2(s.z, s.w));
    if (h2_nonfinite(o.x) | h2_nonfinite(o.y)) flag_error(err, kErrNonFinite);
    *reinterpret_cast<uint2*>(static_cast<uint16_t*>(C) + row * ldc + col) = o;
  } else {
    float4 o = make_float4(alpha * s.x, alpha * s.y, alpha * s.z, alpha * s.w);
    if (R) {
      const float4 rr = *reinterpret_cast<const float4*>(R + row * ldr + col);
      o.x += rr.x; o.y += rr.y; o.z += rr.z; o.w += rr.w;
    }
    *reinterpret_cast<float4*>(static_cast<float*>(C) + row * ldc + col) = o;
  }
}

// ---------------------------------------------------------------------------------- kernel
// Launched with programmatic stream serialization: the prologue and the weight loads and decodes
// of the first ring slots overlap the previous kernel; everything that reads an activation or
// writes memory waits in griddep_wait() first.
template <bool TRANS, int NACC>
__global__ void __launch_bounds__(Warps<NACC>::THREADS, 1)
    dequant_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmP,
                        const __grid_constant__ CUtensorMap tmS, const __grid_constant__ CUtensorMap tmAx,
                        const Params p) {
  using Ly = Layout<NACC>;
  using Wp = Warps<NACC>;
  constexpr int TSTG = Ly::TSTG, BSTG = Ly::BSTG;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* wfull = reinterpret_cast<uint64_t*>(smem + Ly::BAR_OFF);  // TMA ring: packed W + scales landed
  uint64_t* afull = wfull + TSTG;                                      // TMA ring: A tile landed
  uint64_t* empty = afull + TSTG;                                      // TMA ring: MMA done with slot
  uint64_t* bfull = empty + TSTG;                                      // B ring: tile decoded
  uint64_t* bempty = bfull + BSTG;                                     // B ring: MMA done with slot
  uint64_t* accf = bempty + BSTG;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accf + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  griddep_launch();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int n_tile = blockIdx.x, m_tile = blockIdx.y;
  if (p.m_group > 0) {  // groups of m_group row tiles, row-fastest within a group
    const int per = p.m_group * p.tiles_n, g = static_cast<int>(blockIdx.x) / per, idx = static_cast<int>(blockIdx.x) % per;
    const int rows = min(p.m_group, p.tiles_m - g * p.m_group);
    m_tile = g * p.m_group + idx % rows;
    n_tile = idx / rows;
  }
  const int n0 = n_tile * BN, m0 = m_tile * BM * NACC;
  // K range of this split: main tiles [kt0, kt1); the LoRA block rides with the last split.
  const int num_k = p.K / BK;
  const int kt0 = blockIdx.z * p.kt_split;
  const int kt1 = min(num_k, kt0 + p.kt_split);
  const int num_main = max(0, kt1 - kt0);
  const bool split = gridDim.z > 1 && p.zstride == 0;  // cluster split: NACC == 1 only (host)
  const bool last_split = blockIdx.z == gridDim.z - 1;
  const int num_x = last_split ? (p.kx_steps + 3) / 4 : 0;
  const int total = num_main + num_x;

  if (threadIdx.x == 0) {
    for (int s = 0; s < TSTG; ++s) {
      mbar_init(&wfull[s], 1);
      mbar_init(&afull[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < BSTG; ++b) {
      mbar_init(&bfull[b], Wp::CONV);
      mbar_init(&bempty[b], 1);
    }
    mbar_init(accf, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == Wp::MMA) tmem_alloc(tmem_slot, Ly::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == Wp::TMA) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmP);
      tma_prefetch_desc(&tmS);
      auto load_w = [&](int it) {
        const int s = it % TSTG, kt = kt0 + it;
        uint8_t* st = smem + s * Ly::T_STRIDE;
        mbar_arrive_expect_tx(&wfull[s], P_BYTES + S_BYTES);
        if (!TRANS && p.epi == EPI_GLU) {  // 128 gate rows, then the matching 128 up rows
          const int j0 = n0 / 2;
          tma_load_2d(st + Ly::P_OFF, &tmP, &wfull[s], kt * (BK / 2), j0);
          tma_load_2d(st + Ly::P_OFF + (BN / 2) * (BK / 2), &tmP, &wfull[s], kt * (BK / 2), p.glu_half + j0);
          tma_load_2d(st + Ly::S_OFF, &tmS, &wfull[s], j0, kt);
          tma_load_2d(st + Ly::S_OFF + BN, &tmS, &wfull[s], p.glu_half + j0, kt);  // BN / 2 fp16 scales
        } else if (!TRANS) {
          tma_load_2d(st + Ly::P_OFF, &tmP, &wfull[s], kt * (BK / 2), n0);  // packed [N, K/2]
          tma_load_2d(st + Ly::S_OFF, &tmS, &wfull[s], n0, kt);             // scales [K/64, N]
        } else {
          tma_load_2d(st + Ly::P_OFF, &tmP, &wfull[s], n0 / 2, kt * BK);    // packed [K, N/2]
          tma_load_2d(st + Ly::S_OFF, &tmS, &wfull[s], kt * BK, n0 / 64);   // scales [N/64, K]
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
        uint8_t* st = smem + s * Ly::T_STRIDE;
        mbar_arrive_expect_tx(&afull[s], NACC * A_BYTES);
        if (it < num_main) tma_load_2d(st + Ly::A_OFF, &tmA, &afull[s], (kt0 + it) * BK, m0);
        else tma_load_2d(st + Ly::A_OFF, &tmAx, &afull[s], (it - num_main) * BK, m0);
        a_issued = it + 1;
      }
      // Never leave the CTA with copies in flight: wait (bounded) for the last loads issued.
      int dummy = 0;
      for (int it = (w_issued > TSTG ? w_issued - TSTG : 0); it < w_issued; ++it)
        mbar_wait(&wfull[it % TSTG], (it / TSTG) & 1, &dummy, p.err);
      for (int it = (a_issued > TSTG ? a_issued - TSTG : 0); it < a_issued; ++it)
        mbar_wait(&afull[it % TSTG], (it / TSTG) & 1, &dummy, p.err);
    }
  } else if (warp == Wp::MMA) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f16_f32(BM, BN, TRANS);
      for (int it = 0; it < total; ++it) {
        const int s = it % TSTG, b = it % BSTG;
        if (!mbar_wait(&afull[s], (it / TSTG) & 1, abort_flag, p.err)) break;
        if (!mbar_wait(&bfull[b], (it / BSTG) & 1, abort_flag, p.err)) break;
        tc_fence_after();
        // Descriptors of the stage's first k16 slice; later slices advance the start-address field
        // (bits 0-13, in 16-byte units) by a constant, so the issue loop is adds and MMAs only.
        const uint64_t ad0 = smem_desc_sw128(smem_u32(smem + s * Ly::T_STRIDE + Ly::A_OFF), 16, 1024);
        const uint64_t bd0 = TRANS ? smem_desc_sw128(smem_u32(smem + Ly::B_BASE + b * B_BYTES), 8192, 1024)
                                   : smem_desc_sw128(smem_u32(smem + Ly::B_BASE + b * B_BYTES), 16, 1024);
        constexpr uint64_t A_K16 = 32 >> 4, A_ACC = A_BYTES >> 4, B_K16 = (TRANS ? 2048 : 32) >> 4;
        if (it < num_main) {
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
#pragma unroll
            for (int a = 0; a < NACC; ++a)
              tc_mma_f16(tmem + 256 * a, ad0 + a * A_ACC + kk * A_K16, bd0 + kk * B_K16, idesc,
                         (it > 0 || kk > 0) ? 1u : 0u);
        } else {
          const int nk = min(4, p.kx_steps - 4 * (it - num_main));
          for (int kk = 0; kk < nk; ++kk)
#pragma unroll
            for (int a = 0; a < NACC; ++a)
              tc_mma_f16(tmem + 256 * a, ad0 + a * A_ACC + kk * A_K16, bd0 + kk * B_K16, idesc,
                         (it > 0 || kk > 0) ? 1u : 0u);
        }
        tc_commit(&empty[s]);
        tc_commit(&bempty[b]);
      }
      tc_commit(accf);
    }
  } else {
    // ------------------------------------------------------------ converters, then epilogue
    const int t = threadIdx.x;  // 0 .. Wp::CONV_THREADS-1
    for (int it = 0; it < total; ++it) {
      const int s = it % TSTG, b = it % BSTG;
      if (!mbar_wait(&bempty[b], ((it / BSTG) & 1) ^ 1, abort_flag, p.err)) break;
      uint8_t* bt = smem + Ly::B_BASE + b * B_BYTES;
      if (it < num_main) {
        if (!mbar_wait(&wfull[s], (it / TSTG) & 1, abort_flag, p.err)) break;
        const uint8_t* st = smem + s * Ly::T_STRIDE;
        if (TRANS) convert_trans<Wp::TPR>(st + Ly::P_OFF, st + Ly::S_OFF, bt, t);
        else convert_fwd<Wp::TPR>(st + Ly::P_OFF, st + Ly::S_OFF, bt, t);
      } else {
        griddep_wait();  // the LoRA operand comes from an earlier kernel
        copy_lora_b<TRANS, Wp::TPR>(p, it - num_main, n0, bt, t);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bfull[b]);
    }
    griddep_wait();
    const bool acc_ok = __all_sync(0xffffffffu, mbar_wait(accf, 0, abort_flag, p.err));
    tc_fence_after();
    if (split) stash_partial(tmem, acc_ok && total > 0, warp, lane, smem);
    else if (acc_ok && total > 0) epilogue<TRANS, NACC>(p, tmem, warp, lane, m0, n0, smem + warp * 8192);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == Wp::MMA) {
    if (lane == 0) {  // the accumulator is complete (or every issued MMA has retired) before TMEM is freed
      int dummy = 0;
      mbar_wait(accf, 0, &dummy, p.err);
    }
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, Ly::TMEM_COLS);
  }
  if (split) {  // every thread of every CTA of the cluster passes both barriers
    griddep_wait();
    cluster_sync_all();
    split_reduce(p, smem, m0, n0);
    cluster_sync_all();
  }
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

int make_tmap_3d(CUtensorMap* m, const void* base, CUtensorMapDataType dt, int elem_bytes, uint64_t d0, uint64_t d1,
                 uint64_t d2, uint64_t pitch1_bytes, uint64_t pitch2_bytes, uint32_t b0, uint32_t b1, uint32_t b2,
                 CUtensorMapSwizzle swz) {
  auto enc = get_encode();
  if (!enc) return MEBP_ERR_CUDA;
  if ((reinterpret_cast<uintptr_t>(base) & 15) || (pitch1_bytes & 15) || (pitch2_bytes & 15) ||
      ((b0 * elem_bytes) & 15))
    return MEBP_ERR_INVALID_ARG;
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {pitch1_bytes, pitch2_bytes};
  cuuint32_t box[3] = {b0, b1, b2};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(m, dt, 3, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? MEBP_OK : MEBP_ERR_INVALID_ARG;
}

int gemm_smem_bytes() { return gemm::Layout<1>::SMEM; }

namespace {
template <bool TRANS, int NACC>
bool set_smem_attr() {
  static bool attr = false;
  if (!attr)
    attr = cudaFuncSetAttribute(gemm::dequant_gemm_kernel<TRANS, NACC>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                gemm::Layout<NACC>::SMEM) == cudaSuccess;
  return attr;
}

// Clusters of `s` CTAs (along z) of the one-accumulator kernel that can be resident at once;
// 0 when the cluster shape cannot be scheduled.  Queried once per size.
template <bool TRANS>
int max_active_clusters(int s) {
  static int cache[9] = {-1, -1, -1, -1, -1, -1, -1, -1, -1};
  if (s < 1 || s > 8) return 0;
  if (cache[s] < 0) {
    int n = 0;
    if (set_smem_attr<TRANS, 1>()) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(1, 1, s);
      cfg.blockDim = dim3(gemm::Warps<1>::THREADS);
      cfg.dynamicSmemBytes = gemm::Layout<1>::SMEM;
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = 1;
      at[0].val.clusterDim.y = 1;
      at[0].val.clusterDim.z = s;
      cfg.attrs = at;
      cfg.numAttrs = 1;
      if (cudaOccupancyMaxActiveClusters(&n, gemm::dequant_gemm_kernel<TRANS, 1>, &cfg) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
      }
    }
    cache[s] = n;
  }
  return cache[s];
}

template <bool TRANS, int NACC>
int launch_variant(dim3 grid, const CUtensorMap& tA, const CUtensorMap& tP, const CUtensorMap& tS,
                   const CUtensorMap& tAx, const gemm::Params& p, cudaStream_t st) {
  if (!set_smem_attr<TRANS, NACC>()) return MEBP_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(gemm::Warps<NACC>::THREADS);
  cfg.dynamicSmemBytes = gemm::Layout<NACC>::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute at[2];
  int na = 0;
  if (pdl_take()) {
    at[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  if (grid.z > 1 && p.zstride == 0) {
    at[na].id = cudaLaunchAttributeClusterDimension;
    at[na].val.clusterDim.x = 1;
    at[na].val.clusterDim.y = 1;
    at[na].val.clusterDim.z = grid.z;
    ++na;
  }
  cfg.attrs = at;
  cfg.numAttrs = na;
  count_launch();
  if (cudaLaunchKernelEx(&cfg, gemm::dequant_gemm_kernel<TRANS, NACC>, tA, tP, tS, tAx, p) != cudaSuccess)
    return MEBP_ERR_CUDA;
  return MEBP_OK;
}
}  // namespace

namespace gemm {
// Two 128-row accumulators per CTA (half the decode work per flop) once 256-row tiles alone give
// at least two waves on the 152 SMs (large M, or a large N such as the LM head).
int pick_nacc(int64_t M, int64_t N) {
  const int64_t tiles_n256 = (N + BN - 1) / BN;
  return (M >= 2048 || (M >= 256 && tiles_n256 * ((M + 255) / 256) >= 2 * 152)) ? 2 : 1;
}
}  // namespace gemm

namespace gemm {
// K split through memory for few output tiles over a long K (the LM head's dH pass and long-K
// input gradients at a few hundred tokens).  A cluster split is limited by how many clusters fit
// at once (with one CTA per SM, 16 clusters of 7 or more do not), so 16 tiles got at most 96 of
// the 152 SMs; unbound CTAs fill them.  The accumulator count and the split count minimise a
// per-SM time model: K steps per split x the measured time of a 64-deep step (0.60 us with one
// accumulator, 0.72 with two), plus storing the fp32 partial tile, plus the sum kernel reading
// every partial (at 4 TB/s).  Used from 128 K steps on and with at most 76 one-accumulator tiles
// (below that the cluster split or the narrow kernel serve); never more partials than ws_floats.
struct KSplitPlan {
  int nacc = 0, splits = 0;
};
KSplitPlan plan_ksplit(int64_t M, int64_t N, int64_t K, int64_t ws_floats) {
  KSplitPlan best;
  const int64_t num_k = K / BK, tn = (N + BN - 1) / BN;
  if (M <= 0 || num_k < 128 || tn * ((M + BM - 1) / BM) > 76) return best;
  double best_t = 0.0;
  for (int nacc = 1; nacc <= 2; ++nacc) {
    const int64_t tiles = tn * ((M + BM * nacc - 1) / (BM * nacc));
    const double tk = nacc == 1 ? 0.60 : 0.72;
    for (int64_t s = 2; s * tiles <= 152 && s * M * N <= ws_floats; ++s) {
      const int64_t ks = (num_k + s - 1) / s;
      const double t = ks * tk + 1.0 * nacc + static_cast<double>(s) * M * N * 4.0 / 4.0e6;
      if (best.splits == 0 || t < best_t) {
        best.nacc = nacc;
        best.splits = static_cast<int>(s);
        best_t = t;
      }
    }
  }
  return best;
}
}  // namespace gemm

int64_t gemm_ksplit_floats(int64_t M, int64_t N, int64_t K) {
  const gemm::KSplitPlan k = gemm::plan_ksplit(M, N, K, INT64_MAX);
  return k.splits ? k.splits * M * N : 0;
}

// Whether the [M, N] x K GEMM runs on the wide kernel without a K split (the form that can apply
// the gated activation in its epilogue): two accumulators, or more one-accumulator tiles than
// the narrow kernel and the K split take.
bool gemm_glu_fusable(int64_t M, int64_t N, int64_t K) {
  using namespace gemm;
  if (M <= 0 || N <= 0 || K <= 0) return false;
  return pick_nacc(M, N) == 2 || ((N + BN - 1) / BN) * ((M + BM - 1) / BM) > 76;
}

int launch_dequant_gemm(const GemmArgs& g, cudaStream_t st) {
  using namespace gemm;
  if (g.M <= 0 || g.N <= 0) return MEBP_OK;
  if (g.K % 64 || g.N % 64 || g.K <= 0) return MEBP_ERR_INVALID_ARG;
  const bool glu = g.epi == EPI_GLU;
  if (glu && (g.trans || g.glu_half <= 0 || g.glu_half % 128 || g.N != 2 * g.glu_half)) return MEBP_ERR_UNSUPPORTED;
  const bool plain = g.epi == EPI_F32 || g.epi == EPI_F16;
  const KSplitPlan ks = (plain && g.ksplit_ws) ? plan_ksplit(g.M, g.N, g.K, g.ksplit_floats) : KSplitPlan{};
  const int nacc = ks.splits ? ks.nacc : pick_nacc(g.M, g.N);
  const int bm = BM * nacc;
  // Few tokens and a short K: 128 x 256 tiles would leave most SMs idle; narrow 128 x 64 tiles
  // instead of a K split (a long K keeps the split: its serial chain would dominate).
  if (!ks.splits && nacc == 1 && plain && g.K <= 2560 &&
      ((g.N + BN - 1) / BN) * ((g.M + BM - 1) / BM) <= 76)
    return launch_dequant_gemm_narrow(g, st);

  CUtensorMap tA, tP, tS, tAx;
  int rc;
  // A: fp16 [M, K], row pitch lda elements.
  if ((rc = make_tmap_2d(&tA, g.A, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, g.K, g.M, g.lda * 2, 64, bm,
                         CU_TENSOR_MAP_SWIZZLE_128B)))
    return rc;
  if (!g.trans) {
    // packed [N, K/2] bytes, scales [K/64, N] (pitch = scale_pitch elements)
    // (EPI_GLU: two boxes of 128 rows per tile, the gate rows and the matching up rows)
    const uint32_t wbox = glu ? BN / 2 : BN;
    if ((rc = make_tmap_2d(&tP, g.qpack, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, g.K / 2, g.N, g.K / 2, 32, wbox,
                           CU_TENSOR_MAP_SWIZZLE_NONE)))
      return rc;
    if ((rc = make_tmap_2d(&tS, g.scales, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, g.N, g.K / 64, g.scale_pitch * 2, wbox,
                           1, CU_TENSOR_MAP_SWIZZLE_NONE)))
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
  Params p{};
  int kx_steps = 0;
  if (g.Ax && g.kx > 0) {
    if ((g.kx % 16) || (reinterpret_cast<uintptr_t>(g.Bx) & 15) || (g.ldbx % 8)) return MEBP_ERR_INVALID_ARG;
    kx_steps = static_cast<int>(g.kx / 16);
    if ((rc = make_tmap_2d(&tAx, g.Ax, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, g.kx, g.M, g.ldax * 2, 64, bm,
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
  p.lse_part = g.part;
  p.nparts = g.nparts;
  p.zt = g.zt;
  p.lse = g.lse;
  p.ce_w = g.ce_w;
  p.C2 = g.C2;
  p.ldc2 = g.ldc2;
  p.glu_half = g.glu_half;
  p.act = g.act;
  p.err = g.err;

  const int tiles_n = static_cast<int>((g.N + BN - 1) / BN), tiles_m = static_cast<int>((g.M + bm - 1) / bm);
  const int num_k = static_cast<int>(g.K / BK);
  // Split K when the output tiles leave at least half of the 152 SMs idle: the largest cluster
  // size S <= 8 with >= 2 K tiles per split whose clusters all fit on the GPU at once.
  int splits = 1;
  const int grid_mn = tiles_n * tiles_m;
  if (ks.splits) {  // through memory: partial tiles in the workspace, summed by ksplit_sum_kernel
    splits = ks.splits;
    p.epi = EPI_F32;
    p.C = g.ksplit_ws;
    p.ldc = g.N;
    p.R = nullptr;
    p.alpha = 1.0f;
    p.zstride = g.M * g.N;
  } else if (plain && nacc == 1 && grid_mn <= 76 && num_k >= 4) {
    for (int s = std::min(8, num_k / 2); s >= 2; --s) {
      const int mac = g.trans ? max_active_clusters<true>(s) : max_active_clusters<false>(s);
      if (grid_mn <= mac) {
        splits = s;
        break;
      }
    }
  }
  const int kt_split = (num_k + splits - 1) / splits;
  splits = (num_k + kt_split - 1) / kt_split;  // every split gets >= 1 K tile
  p.kt_split = kt_split;
  dim3 grid(tiles_n, tiles_m, splits);
  // Consecutive CTAs share their row tile of A and walk through the weight tiles, so a weight
  // operand larger than the L2 (the LM head's whole vocabulary) would be streamed once per row
  // tile.  Then run the tiles in groups of 16 row tiles, row-fastest within a group: the weights
  // stream once per group and the group's rows of A stay in L2.
  const double w_bytes = static_cast<double>(g.N) * g.K * (0.5 + 1.0 / 32);
  if (w_bytes > 64.0 * (1 << 20) && tiles_m > 1 && splits == 1) {
    p.m_group = 16;
    p.tiles_m = tiles_m;
    p.tiles_n = tiles_n;
    grid = dim3(static_cast<unsigned>(tiles_m) * static_cast<unsigned>(tiles_n), 1, 1);
  }
  if (g.trans)
    rc = nacc == 2 ? launch_variant<true, 2>(grid, tA, tP, tS, tAx, p, st)
                   : launch_variant<true, 1>(grid, tA, tP, tS, tAx, p, st);
  else
    rc = nacc == 2 ? launch_variant<false, 2>(grid, tA, tP, tS, tAx, p, st)
                   : launch_variant<false, 1>(grid, tA, tP, tS, tAx, p, st);
  if (rc) return rc;
  if (ks.splits) {
    const int64_t n4 = g.M * (g.N / 4);
    launch_k(ksplit_sum_kernel, dim3(static_cast<unsigned>((n4 + 255) / 256)), 256, 0, st,
             static_cast<const float*>(g.ksplit_ws), splits, p.zstride, static_cast<int>(g.M), static_cast<int>(g.N),
             g.alpha, g.R, g.ldr, g.C, g.ldc, g.epi == EPI_F16 ? 1 : 0, g.err);
  }
  return cudaGetLastError() == cudaSuccess ? MEBP_OK : MEBP_ERR_CUDA;
}

}  // namespace mebp
