// Internal kernel launchers (host-callable, stream-ordered).  Not part of the C ABI.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <utility>

namespace mebp {

// Process-wide count of kernel launches issued by the library (reported by mebp_kernel_launches).
extern std::atomic<long long> g_launches;
inline void count_launch(int n = 1) { g_launches.fetch_add(n, std::memory_order_relaxed); }

// Programmatic dependent launch (PDL).  Every kernel of the library starts with griddep_wait()
// (and then griddep_launch()), so a kernel may be launched while its predecessor in the stream
// still runs: its launch latency and prologue overlap the predecessor, and its first access to
// memory still waits for the predecessor to complete.  The first kernel an entry point launches
// is a normal launch (pdl_entry() marks it), so no kernel of one call overlaps an earlier call:
// the fused GEMM may then read the packed weights before its wait (they are written only by
// mebp_compress_weights, a separate call).
// A kernel starts only after every CTA of its predecessor has triggered.  So, at its start,
// everything written before the nearest preceding kernel that waits before it triggers is
// complete.  Every kernel here waits first except the fused GEMMs (whose weight reads need no
// wait) and the attention backward's dK/dV, dQ and split kernels; those issue their q/k/v, lse and
// dO loads before the wait, relying on the dvec kernel (waits first) before them, and read dvec
// after it.  Early reads go through L2 only (cp.async.cg, __ldcg): until the wait, L1 may still
// hold lines of a reused buffer read by an earlier kernel on the same SM.
void pdl_entry();   // the calling thread's next launch is a normal launch
bool pdl_take();    // may this launch use PDL? (consumes the entry mark)

template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                            Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = pdl_take() ? 1 : 0;
  count_launch();
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// launch_k with a thread-block cluster of cluster.x * cluster.y * cluster.z CTAs (1: none).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                                    dim3 cluster, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[2];
  int na = 0;
  if (pdl_take()) {
    at[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  if (cluster.x * cluster.y * cluster.z > 1) {
    at[na].id = cudaLaunchAttributeClusterDimension;
    at[na].val.clusterDim.x = cluster.x;
    at[na].val.clusterDim.y = cluster.y;
    at[na].val.clusterDim.z = cluster.z;
    ++na;
  }
  cfg.attrs = at;
  cfg.numAttrs = na;
  count_launch();
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// EPI_GLU (forward, wide kernel, no K split): the weight is the fused [gate; up] matrix of 2 glu_half rows;
// 256-column tile t holds gate rows 128 t .. 128 t + 127 and the matching up rows, and the epilogue
// writes m = act(gate) * up (fp16, C [M, glu_half]) and, with C2, gate and up (fp16, [M, 2 glu_half]).
enum GemmEpi { EPI_F16 = 0, EPI_F32 = 1, EPI_LSE = 2, EPI_CEGRAD = 3, EPI_GLU = 4 };

struct GemmArgs {
  bool trans = false;            // false: C = A deq(W)^T (W [N,K]);  true: C = A deq(W) (W [K,N])
  const void* A = nullptr;       // fp16 [M, K]
  int64_t lda = 0;
  int64_t M = 0, N = 0, K = 0;
  const uint8_t* qpack = nullptr;
  const uint16_t* scales = nullptr;
  int64_t scale_pitch = 0;       // elements between consecutive scale rows (groups)
  const void* Ax = nullptr;      // fp16 [M, kx] extra (LoRA) operand, or null
  int64_t ldax = 0;
  int64_t kx = 0;
  const void* Bx = nullptr;      // FWD: fp16 [N, kx];  TRANS: fp16 [kx, N]
  int64_t ldbx = 0;
  int epi = EPI_F16;
  void* C = nullptr;
  int64_t ldc = 0;
  const float* R = nullptr;
  int64_t ldr = 0;
  float alpha = 1.0f;            // EPI_F32: C = alpha * acc (+ R)
  const int32_t* targets = nullptr;
  int col_offset = 0;
  int n_valid = 0;
  float* part = nullptr;
  int nparts = 0;
  float* zt = nullptr;
  const float* lse = nullptr;
  const float* ce_w = nullptr;   // EPI_CEGRAD: device scalar weight of a valid row
  void* C2 = nullptr;            // EPI_GLU: gate and up as well (fp16 [M, 2 glu_half]), or null
  int64_t ldc2 = 0;
  int glu_half = 0;              // EPI_GLU: rows of the gate (= of the up) half of the weight
  int act = 0;                   // EPI_GLU: MEBP_ACT_*
  // fp32 scratch for a K split through memory (EPI_F32 / EPI_F16 with few output tiles over a
  // long K); null = cluster splits only.  Not shared between GEMMs that may overlap on the GPU.
  float* ksplit_ws = nullptr;
  int64_t ksplit_floats = 0;
  int* err = nullptr;
};

int launch_dequant_gemm(const GemmArgs& g, cudaStream_t st);
// True when launch_dequant_gemm runs an [M, N] x K GEMM on the wide kernel without a K split:
// then EPI_GLU (the gated activation in the epilogue) costs no parallelism.
bool gemm_glu_fusable(int64_t M, int64_t N, int64_t K);
// fp32 scratch (floats) the K split through memory wants for an [M, N] x K GEMM; 0 when that
// shape does not split through memory.
int64_t gemm_ksplit_floats(int64_t M, int64_t N, int64_t K);
// The 128 x 64-tile variant for few-token GEMMs (EPI_F16 / EPI_F32); launch_dequant_gemm routes
// to it when the 128 x 256 tiles would leave most SMs idle.
int launch_dequant_gemm_narrow(const GemmArgs& g, cudaStream_t st);
// 2-D tiled TMA descriptor: dims {d0 (inner), d1}, row pitch in bytes, box {b0, b1}.
int make_tmap_2d(CUtensorMap* m, const void* base, CUtensorMapDataType dt, int elem_bytes, uint64_t d0, uint64_t d1,
                 uint64_t pitch_bytes, uint32_t b0, uint32_t b1, CUtensorMapSwizzle swz);
// 3-D tiled TMA descriptor: dims {d0 (inner), d1, d2}, pitches of d1 and d2 in bytes, box {b0, b1, b2}.
int make_tmap_3d(CUtensorMap* m, const void* base, CUtensorMapDataType dt, int elem_bytes, uint64_t d0, uint64_t d1,
                 uint64_t d2, uint64_t pitch1_bytes, uint64_t pitch2_bytes, uint32_t b0, uint32_t b1, uint32_t b2,
                 CUtensorMapSwizzle swz);
int gemm_smem_bytes();

void launch_compress(const float* W, int64_t rows, int64_t cols, uint8_t* qpack, uint16_t* scales, cudaStream_t st);
void launch_decode(const uint8_t* qpack, const uint16_t* scales, int64_t rows, int64_t cols, uint16_t* out,
                   cudaStream_t st);
// x0[t] = scale * deq(E)[ids[t]] (scale = sqrt(D) for Gemma3, else 1).
void launch_embed(const uint8_t* qpack, const uint16_t* scales, int64_t V, int64_t D, const int32_t* ids, int64_t T,
                  float* x0, int* err, float scale, cudaStream_t st);

// RMSNorm: y_f16 = x * rstd * g (rstd saved); backward: dx = resid + rstd (g dy) - x rstd^3/D sum(g dy x)
void launch_rmsnorm_fwd(const float* x, const float* g, int64_t T, int D, float eps, uint16_t* y, float* rstd,
                        cudaStream_t st);
// dx = (resid + ...) * (*out_mult) (out_mult may be null = 1); dx_h = fp16(resid + ...) (unmultiplied);
// either output may be null.
void launch_rmsnorm_bwd(const float* dy, const float* x, const float* g, const float* rstd, const float* resid,
                        int64_t T, int D, const float* out_mult, float* dx, uint16_t* dx_h, cudaStream_t st);
// RoPE (half-split) on the q and k heads of a fused [T, (H+2KV)*hd] fp16 buffer, in place.
void launch_rope(uint16_t* qkv, int64_t T, int S, int H, int KV, int hd, const float2* cs, bool inverse,
                 cudaStream_t st);
// Gemma3 QK-norm + RoPE on the q and k heads of the fused qkv buffer, in place; raw fp16 heads
// [T, H+KV, hd] and their 1/rms [T, H+KV] are saved for the backward, which runs in place on dqkv.
void launch_qknorm_rope(uint16_t* qkv, int64_t T, int S, int H, int KV, int hd, const float* qg, const float* kg,
                        float eps, const float2* cs, uint16_t* raw, float* rstd, cudaStream_t st);
void launch_qknorm_rope_bwd(uint16_t* dqkv, int64_t T, int S, int H, int KV, int hd, const float* qg, const float* kg,
                            const float2* cs, const uint16_t* raw, const float* rstd, cudaStream_t st);
// Gemma3 sandwich norms: h1 = x + norm(ao) g_pa and b = fp16(norm(h1) g2) (1/rms of ao and of h1
// saved); y = h1 + norm(dn) g_pf (1/rms of dn saved when rpf != null; y == null computes it only).
void launch_add_norm2(const float* ao, const float* x, const float* gpa, const float* g2, int64_t T, int D, float eps,
                      float* h1, uint16_t* b, float* rpa, float* r2, cudaStream_t st);
void launch_add_norm(const float* dn, const float* h1, const float* gpf, int64_t T, int D, float eps, float* y,
                     float* rpf, cudaStream_t st);
// Gated MLP: m = act(g) * u from gu = [g | u] (fp16 [T, 2I]); backward reads dm fp16 [T, I] and
// writes dgu fp16 [T, 2I].  A result outside the fp16 range sets MEBP_ERR_NONFINITE in *err.
void launch_glu_fwd(const uint16_t* gu, int64_t T, int I, int act, uint16_t* m, int* err, cudaStream_t st);
void launch_glu_bwd(const uint16_t* dm, const uint16_t* gu, int64_t T, int I, int act, uint16_t* dgu, int* err,
                    cudaStream_t st);
// y32 = x * (*scale), y16 = fp16(x * (*scale)); scale may be null (= 1), y32 may be null.
void launch_scale_cast(const float* x, int64_t n, const float* scale, float* y32, uint16_t* y16, cudaStream_t st);
// scal[0] = sigma = 2^-floor(log2(max|x|)) (1 if x == 0), scal[1] = 1/sigma; uses scal[2] as scratch.
void launch_grad_scale(const float* x, int64_t n, float* scal, cudaStream_t st);
void launch_fill_f32(float* x, int64_t n, float v, cudaStream_t st);

// LM head helpers.
void launch_lse_combine(const float* part, int nparts, const float* zt, const int32_t* targets, int64_t T,
                        float* lse, float* tok_loss, cudaStream_t st);
// loss = sum(tok_loss) / n_valid; scal[0] = sigma = 2^ceil(log2(n_valid)), scal[1] = 1/sigma,
// scal[2] = sigma * kCeShift / n_valid (weight of a valid row of the scaled CE gradient).
constexpr float kCeShift = 4096.0f;
void launch_loss_reduce(const float* tok_loss, const int32_t* targets, int64_t T, float* loss, float* scal,
                        cudaStream_t st);

// LoRA helpers.
// out[m, j] = alpha * sum_k X[m, k] W[j, k]  (fp16 in, fp16 out with columns J..ldo-1 zeroed)
// err: device error word for a bounded wait that expires (may be null).
void launch_skinny_gemm(const uint16_t* X, int64_t ldx, int64_t M, int64_t K, const uint16_t* W, int64_t ldw, int J,
                        float alpha, uint16_t* out, int64_t ldo, cudaStream_t st, int* err = nullptr);
// The same on tcgen05 with a TMA ring (large M); ldo in {16, 32, 48, 64, 80, 96}, K % 64 == 0,
// X / W 16-byte aligned with row pitches that are multiples of 8 elements.
int launch_skinny_tc(const uint16_t* X, int64_t ldx, int64_t M, int64_t K, const uint16_t* W, int64_t ldw,
                     float alpha, uint16_t* out, int64_t ldo, int* err, cudaStream_t st);
// C[p, q] (+)= sum_m P[m, p0 + p] Q[m, q0 + q], p < Pw, q < Qw; deterministic split over m.
// The sum is multiplied by *mult (mult may be null = 1) before it is written / added.
int launch_tall_reduce(const uint16_t* P, int64_t ldp, const uint16_t* Q, int64_t ldq, int64_t M, int Pw, int Qw,
                       float* C, int64_t ldc, bool accumulate, const float* mult, float* scratch,
                       int64_t scratch_floats, int* err, cudaStream_t st);
// Several reductions over the same P at once: C[j][p, q] (+)= mult * sum_m P[m, p] Q[m, j r + q],
// j < nq (ldc shared); on tcgen05 (tall_tc.cu) where tall_tc_takes() says so, else nq calls of the
// above.
int launch_tall_reduce_multi(const uint16_t* P, int64_t ldp, const uint16_t* Q, int64_t ldq, int64_t M, int Pw,
                             int nq, int r, float* const* C, int64_t ldc, bool accumulate, const float* mult,
                             float* scratch, int64_t scratch_floats, int* err, cudaStream_t st);
bool tall_tc_takes(int64_t M, int Pw, int nq, int r);
// The tcgen05 reduction; MEBP_ERR_UNSUPPORTED for shapes it does not take.
int launch_tall_tc(const uint16_t* P, int64_t ldp, const uint16_t* Q, int64_t ldq, int64_t M, int Pw, int nq, int r,
                   float* const* C, int64_t ldc, bool accumulate, const float* mult, int* err, cudaStream_t st);
// C[p * sp + q * sq] (+)= mult * sum over splits of part[z][p][q], in split order.
void launch_split_sum(const float* part, int splits, int Pw, int Qw, float* C, int64_t sp, int64_t sq, bool accumulate,
                      const float* mult, cudaStream_t st);
int64_t tall_reduce_scratch_floats(int64_t M, int Pw, int Qw);
// Up to kTallMaxProbs single-pass reductions C (+)= mult * P^T Q over the same M rows in one launch
// (Qw <= 32, Pw and Qw multiples of 8).  tall_batch_add returns false for a problem it cannot take.
constexpr int kTallMaxProbs = 16;
struct TallProb {
  const uint16_t* P;
  const uint16_t* Q;
  float* C;
  int64_t ldp, ldq, sp, sq;
  int Pw, Qw, acc, ctas;
};
struct TallBatch {
  TallProb p[kTallMaxProbs];
  int n = 0;
  int64_t M = 0;
  const float* mult = nullptr;
};
bool tall_batch_add(TallBatch& b, const uint16_t* P, int64_t ldp, const uint16_t* Q, int64_t ldq, int Pw, int Qw,
                    float* C, int64_t ldc, bool accumulate);
void launch_tall_reduce_batched(const TallBatch& b, cudaStream_t st);
// fp16 shadows of the LoRA masters, see lora.cu.
// fp16 LoRA shadows of n_layers layers at once: target t of layer l reads A[3 l + t], B[3 l + t];
// layer l's outputs start at l * stride_a (A_cat) and l * stride_b (B_cat, Bt_cat).
constexpr int kShadowMaxLayers = 64;  // layers per launch
void launch_lora_shadow_layers(int n_layers, const float* const* A, const float* const* B, int nt,
                               const int* ranks_off, const int* n_off, const int* n_len, int r, int K, int N, int kx,
                               uint16_t* A_cat, uint16_t* B_cat, uint16_t* Bt_cat, int64_t stride_a, int64_t stride_b,
                               cudaStream_t st);
void launch_lora_shadow(const float* const* A, const float* const* B, int nt, const int* ranks_off,
                        const int* n_off, const int* n_len, int r, int K, int N, int kx, uint16_t* A_cat,
                        uint16_t* B_cat, uint16_t* Bt_cat, cudaStream_t st);

// Attention (causal GQA).  q/k/v live inside the fused qkv buffer (row pitch ld).
// window > 0: query i sees keys i - window + 1 .. i (sliding-window local layers); 0 = causal.
int launch_attn_fwd(const uint16_t* qkv, int64_t ld, int B, int S, int H, int KV, int hd, uint16_t* o, int64_t ldo,
                    float* lse, int window, int* err, cudaStream_t st);
// The forward on tcgen05 (attention_tc.cu); ld % 64 == 0, ldo % 8 == 0.
int launch_attn_fwd_tc(const uint16_t* qkv, int64_t ld, int B, int S, int H, int KV, int hd, uint16_t* o, int64_t ldo,
                       float* lse, int window, int* err, cudaStream_t st);
void launch_adamw(float* p, const float* g, float* m, float* v, int64_t n, float lr, float b1, float b2, float eps,
                  float wd, float gs, double bc1, double bc2, cudaStream_t st);
// Backward into dqkv.  Small grids run the split mode through the fp32 workspace ws (needs
// 3 * B * ceil(S/64) * H * 2 * 64 * hd floats; a smaller or null ws falls back to the direct mode);
// the split mode also rotates dq, dk back by rope_cs (when not null) and returns true — otherwise
// the caller applies the inverse RoPE.
bool launch_attn_bwd(const uint16_t* qkv, int64_t ld, const uint16_t* o, const uint16_t* dout, int64_t ldo,
                     const float* lse, int B, int S, int H, int KV, int hd, float* dvec, uint16_t* dqkv, int window,
                     const float2* rope_cs, float* ws, int64_t ws_floats, int* err, cudaStream_t st);
// dK/dV and dQ on tcgen05 (attention_tc.cu) from dvec = rowsum(dO o).  parts == 0: writes dqkv
// (no RoPE inverse); parts = P > 0: fp32 partials into wk / wv / wq (see attention.cu) for the
// finish kernel.
int launch_attn_bwd_tc(const uint16_t* qkv, int64_t ld, const uint16_t* dout, int64_t ldo, const float* lse,
                       const float* dvec, int B, int S, int H, int KV, int hd, uint16_t* dqkv, int window, int parts,
                       float* wk, float* wv, float* wq, int* err, cudaStream_t st);

}  // namespace mebp
