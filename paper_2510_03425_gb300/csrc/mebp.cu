// C ABI of the MeBP training step (include/mebp.h): context and workspace, the decoder block's
// recompute-forward and backward, the LM-head cross-entropy and Algorithm 1.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "common.cuh"
#include "kernels.h"

using namespace mebp;

namespace {

enum { LIN_QKV = 0, LIN_O = 1, LIN_GU = 2, LIN_DOWN = 3 };

struct Lin {
  int N = 0, K = 0;
  int nt = 0;        // number of LoRA targets carried by this fused linear
  int tgt[3] = {0, 0, 0};
  int ro[3] = {0, 0, 0};  // rank offset in the concatenated rank axis
  int no[3] = {0, 0, 0};  // first output row of the target
  int nl[3] = {0, 0, 0};  // output rows of the target
  int kx = 0, kxp = 0;    // used / padded width of the rank axis
};

constexpr int kCkptSlots = 3;

// Kinds of kernel the event profiler (mebp_profile_begin / _end / _kernels) tells apart.
enum KKind {
  KK_GEMM_FWD = 0, KK_GEMM_DX, KK_EMBED, KK_RMSNORM_FWD, KK_RMSNORM_BWD, KK_ADD_NORM, KK_ROPE, KK_QKNORM_ROPE,
  KK_GLU_FWD, KK_GLU_BWD, KK_ATTN_FWD, KK_ATTN_BWD, KK_LORA_SKINNY, KK_LORA_REDUCE, KK_LORA_SHADOW, KK_LM_REDUCE,
  KK_SCALE, KK_N
};
const char* const kKindName[KK_N] = {
    "fused_gemm_fwd", "fused_gemm_dx", "embed", "rmsnorm_fwd", "rmsnorm_bwd", "add_norm", "rope", "qknorm_rope",
    "glu_fwd", "glu_bwd", "attention_fwd", "attention_bwd", "lora_skinny", "lora_grad_reduce", "lora_shadow",
    "lmhead_reduce", "grad_scale"};

// One profiled launch: CUDA events on the launching stream around it, and its algorithmic work.
struct ProfRec {
  cudaEvent_t a, b;
  int kind;
  double flops, bytes;
};

// Algorithmic HBM bytes of the memory-bound kernels (each operand read or written once).
double bytes_rms_fwd(int64_t T, int D) { return 6.0 * T * D + 4.0 * T + 4.0 * D; }
double bytes_rms_bwd(int64_t T, int D, bool resid, bool dx, bool dxh) {
  return T * static_cast<double>(D) * (8.0 + (resid ? 4 : 0) + (dx ? 4 : 0) + (dxh ? 2 : 0)) + 4.0 * T + 4.0 * D;
}
double bytes_rope(int64_t T, int S, int H, int KV, int hd) { return 4.0 * T * (H + KV) * hd + 8.0 * S * (hd / 2); }
double bytes_qknorm(int64_t T, int S, int H, int KV, int hd) {
  return 6.0 * T * (H + KV) * hd + 4.0 * T * (H + KV) + 8.0 * S * (hd / 2);
}
// Causal (window W > 0: sliding) attention flops of the forward: QK^T and PV over the visible keys.
double attn_fwd_flops(int B, int S, int H, int hd, int W) {
  double keys = 0.0;
  for (int i = 0; i < S; ++i) keys += (W > 0 && W < i + 1) ? W : i + 1;
  return 4.0 * hd * keys * B * H;
}
double bytes_attn_fwd(int64_t T, int H, int KV, int hd) { return 2.0 * T * (H + 2 * KV) * hd + 2.0 * T * H * hd + 4.0 * T * H; }
double bytes_attn_bwd(int64_t T, int H, int KV, int hd) {
  return 4.0 * T * (H + 2 * KV) * hd + 4.0 * T * H * hd + 12.0 * T * H;
}
double bytes_skinny(int64_t T, int64_t K, int kx, int kxp) { return 2.0 * T * K + 2.0 * kx * K + 2.0 * T * kxp; }
double bytes_tall(int64_t M, int Pw, int Qw, bool acc) { return 2.0 * M * (Pw + Qw) + 4.0 * Pw * Qw * (acc ? 2 : 1); }

}  // namespace

std::atomic<long long> mebp::g_launches{0};
namespace {
thread_local bool t_pdl_entry = false;
}
void mebp::pdl_entry() { t_pdl_entry = true; }
bool mebp::pdl_take() {
  const bool ok = !t_pdl_entry;
  t_pdl_entry = false;
  return ok;
}

// One block's forward intermediates (what the backward consumes) and the fp16 LoRA shadows they
// were computed with.  The step keeps two sets so that the recompute of block i-1 can run on a
// second stream while the backward of block i reads the other set.
// fp16 LoRA shadows of one block's fused linears: A_cat [kxp, K], B_cat [N, kxp], Bt_cat [kxp, N].
struct Shadow {
  uint16_t *A_cat[4] = {}, *B_cat[4] = {}, *Bt_cat[4] = {};
};

struct Acts {
  uint16_t *a = nullptr, *qkv = nullptr, *o = nullptr, *b = nullptr, *gu = nullptr, *m = nullptr;
  float *r1 = nullptr, *r2 = nullptr, *lse_attn = nullptr, *h1 = nullptr;
  uint16_t* us[4] = {nullptr, nullptr, nullptr, nullptr};
  // Gemma3 block only: o-proj and down-proj outputs before their sandwich norms and the norms'
  // 1/rms, the q/k heads before QK-norm ([T, H+KV, hd]) and their 1/rms
  float *ao = nullptr, *dn = nullptr, *rpa = nullptr, *rpf = nullptr, *rqk = nullptr;
  uint16_t* qk_raw = nullptr;
  Shadow own;                  // shadows built by the forward itself
  const Shadow* sh = nullptr;  // the shadows the set was computed with
  // which block / input / token count the set currently holds (-1: none)
  int layer = -1;
  const float* x = nullptr;
  int64_t T = -1;
};

// Backward intermediates that the LoRA-gradient reductions read besides the forward set.
struct Grads2 {
  uint16_t *dqkv = nullptr, *dgu = nullptr, *dh1_h = nullptr;
  uint16_t* ddn_h = nullptr;  // Gemma3: gradient of the down projection's output (fp16)
  uint16_t* du[4] = {nullptr, nullptr, nullptr, nullptr};
};

struct mebp_ctx {
  mebp_model_cfg cfg{};
  int device = 0;
  std::string err_msg = "ok";
  int* d_err = nullptr;
  // device scalars: [0] sigma of the backward working scale, [1] 1/sigma, [2] CE row weight
  // (all written by the loss reduction); [4] / [5] sigma / 1/sigma of a standalone block
  // backward, [6] scratch.
  float* scal = nullptr;
  int D = 0, H = 0, KV = 0, hd = 0, I = 0, V = 0, L = 0, Nqkv = 0, Na = 0, r = 0;
  float s = 1.0f;
  int64_t Tmax = 0;
  Lin lin[4];
  std::vector<void*> dev_allocs;
  int64_t ws_bytes = 0;
  int64_t ws_cat[MEBP_WS_N] = {};  // bytes per purpose (mebp_workspace_breakdown)
  int cur_cat = MEBP_WS_OTHER;     // purpose of the allocations being made

  float2* rope_cs = nullptr;
  float2* rope_cs_local = nullptr;  // RoPE table of the sliding-window layers (their own base)
  bool gemma = false;               // Gemma3 block (QK-norm, sandwich norms, sqrt(D) embedding)
  // forward intermediates: set 0 always, set 1 when the step overlaps recompute and backward
  Acts act[2];
  int nsets = 1;
  std::vector<Shadow> layer_sh;  // the step's shadows, built for every block at once
  cudaStream_t fstream = nullptr;  // recompute stream of the overlapped backward
  cudaEvent_t ev_main = nullptr;   // main-stream progress, waited on by the recompute stream
  cudaEvent_t ev_fwd[2] = {};      // recompute into set k finished
  // backward
  // backward operands of the LoRA-gradient reductions, one copy per layer parity (the reductions
  // of block i run on the gradient stream while the backward of block i-1 runs)
  Grads2 bw[2];
  cudaStream_t gstream = nullptr;  // LoRA-gradient reductions of the overlapped backward
  cudaEvent_t ev_bwd = nullptr;    // backward of the current block issued (main stream)
  cudaEvent_t ev_grad[2] = {};     // reductions of a block of parity k finished
  uint16_t *dout = nullptr, *dy_h[3] = {nullptr, nullptr, nullptr};
  uint16_t* dm = nullptr;  // dE/dm of the gated MLP, fp16 (in the backward's working scale)
  float *dtmp = nullptr, *dh1 = nullptr, *dvec = nullptr, *gbuf[2] = {nullptr, nullptr};
  float* attn_ws = nullptr;  // fp32 partials of the split attention backward (small grids)
  int64_t attn_ws_floats = 0;
  float* red = nullptr;
  int64_t red_floats = 0;
  // fp32 partials of fused GEMMs split over K through memory: [0] for GEMMs on the caller's
  // stream, [1] for the recompute stream (the two overlap on the GPU)
  float* ksplit[2] = {nullptr, nullptr};
  int64_t ksplit_floats = 0;
  // LM head
  uint16_t *hf = nullptr, *dz = nullptr;
  float *rf = nullptr, *part = nullptr, *zt = nullptr, *lse_tok = nullptr, *tok_loss = nullptr,
        *dhf = nullptr;
  int32_t* targets = nullptr;
  int nparts = 0, vchunk = 0;
  // checkpoints
  float* ckpt = nullptr;       // device: (L+1) x Tmax x D, or kCkptSlots slots when spilling
  float* h_ckpt = nullptr;     // pinned host (spill)
  cudaStream_t copy_stream = nullptr;
  cudaEvent_t slot_free[kCkptSlots] = {};
  cudaEvent_t slot_ready[kCkptSlots] = {};
  // CUDA-graph replay of mebp_lora_step (key = every pointer and size the step depends on)
  bool graphs = true;
  std::vector<uintptr_t> graph_key;
  cudaGraphExec_t graph_exec = nullptr;
  long long graph_launches = 0;
  int graph_eager_runs = 0;
  cudaEvent_t copy_join = nullptr;
  // event profiling of every launch (mebp_profile_begin / _end / _kernels)
  bool prof = false;
  std::vector<ProfRec> recs;
  std::vector<mebp_kernel_stat> kstats;
  std::vector<cudaEvent_t> evpool;
  size_t evnext = 0;
};

namespace {

int fail(mebp_ctx* c, int code, const std::string& msg) {
  if (c) c->err_msg = msg;
  return code;
}

int cuda_check(mebp_ctx* c, const char* where) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(c, MEBP_ERR_CUDA, std::string(where) + ": " + cudaGetErrorString(e));
  return MEBP_OK;
}

template <typename T>
int dalloc(mebp_ctx* c, T** p, int64_t count) {
  *p = nullptr;
  if (count <= 0) return MEBP_OK;
  const size_t bytes = static_cast<size_t>(count) * sizeof(T);
  void* q = nullptr;
  if (cudaMalloc(&q, bytes) != cudaSuccess) {
    cudaGetLastError();
    return fail(c, MEBP_ERR_OOM, "device allocation of " + std::to_string(bytes) + " bytes failed");
  }
  c->dev_allocs.push_back(q);
  c->ws_bytes += static_cast<int64_t>(bytes);
  c->ws_cat[c->cur_cat] += static_cast<int64_t>(bytes);
  *p = static_cast<T*>(q);
  return MEBP_OK;
}

cudaStream_t S(void* st) { return static_cast<cudaStream_t>(st); }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

int check_packed(mebp_ctx* c, const mebp_packed* w, int64_t rows, int64_t cols, const char* what) {
  if (!w || !w->qpack || !w->scales) return fail(c, MEBP_ERR_INVALID_ARG, std::string(what) + ": NULL weight");
  if (w->rows != rows || w->cols != cols)
    return fail(c, MEBP_ERR_INVALID_ARG,
                std::string(what) + ": expected [" + std::to_string(rows) + ", " + std::to_string(cols) + "]");
  if (!aligned16(w->qpack) || !aligned16(w->scales))
    return fail(c, MEBP_ERR_INVALID_ARG, std::string(what) + ": weight pointers must be 16-byte aligned");
  return MEBP_OK;
}

void setup_lin(mebp_ctx* c) {
  const int H = c->H, KV = c->KV, hd = c->hd, D = c->D, I = c->I, r = c->r;
  const uint32_t m = c->cfg.lora_targets;
  Lin* L = c->lin;
  L[LIN_QKV].N = (H + 2 * KV) * hd;
  L[LIN_QKV].K = D;
  L[LIN_O].N = D;
  L[LIN_O].K = H * hd;
  L[LIN_GU].N = 2 * I;
  L[LIN_GU].K = D;
  L[LIN_DOWN].N = D;
  L[LIN_DOWN].K = I;
  struct Part { int lin, tgt, no, nl; };
  const Part parts[7] = {{LIN_QKV, MEBP_T_Q, 0, H * hd},           {LIN_QKV, MEBP_T_K, H * hd, KV * hd},
                         {LIN_QKV, MEBP_T_V, (H + KV) * hd, KV * hd}, {LIN_O, MEBP_T_O, 0, D},
                         {LIN_GU, MEBP_T_GATE, 0, I},               {LIN_GU, MEBP_T_UP, I, I},
                         {LIN_DOWN, MEBP_T_DOWN, 0, D}};
  for (const Part& p : parts) {
    if (!(m & (1u << p.tgt)) || r <= 0) continue;
    Lin& l = L[p.lin];
    l.tgt[l.nt] = p.tgt;
    l.ro[l.nt] = l.kx;
    l.no[l.nt] = p.no;
    l.nl[l.nt] = p.nl;
    l.kx += r;
    l.nt++;
  }
  for (int i = 0; i < 4; ++i) L[i].kxp = L[i].kx ? (L[i].kx + 15) / 16 * 16 : 0;
}

// ------------------------------------------------------------------------------------ GEMM glue
GemmArgs gemm_fwd(const uint16_t* X, int64_t ldx, int64_t M, const mebp_packed& W, int N, int K) {
  GemmArgs g;
  g.trans = false;
  g.A = X;
  g.lda = ldx;
  g.M = M;
  g.N = N;
  g.K = K;
  g.qpack = W.qpack;
  g.scales = W.scales;
  g.scale_pitch = W.rows;
  return g;
}
// dX = dY deq(W) for W [N_w, K_w] stored packed: GEMM K = N_w (reduction), N = K_w (output).
GemmArgs gemm_dx(const uint16_t* dY, int64_t ldy, int64_t M, const mebp_packed& W) {
  GemmArgs g;
  g.trans = true;
  g.A = dY;
  g.lda = ldy;
  g.M = M;
  g.N = W.cols;
  g.K = W.rows;
  g.qpack = W.qpack;
  g.scales = W.scales;
  g.scale_pitch = W.rows;
  return g;
}

cudaEvent_t pool_event(mebp_ctx* c) {
  if (c->evnext == c->evpool.size()) {
    cudaEvent_t e;
    cudaEventCreate(&e);
    c->evpool.push_back(e);
  }
  return c->evpool[c->evnext++];
}

// Runs f() (one or more launches on st); when profiling, brackets it with an event pair on st and
// records its kind and algorithmic work.
template <class F>
void KP(mebp_ctx* c, int kind, double bytes, double flops, cudaStream_t st, F&& f) {
  if (!c->prof) {
    f();
    return;
  }
  ProfRec r{};
  r.a = pool_event(c);
  r.b = pool_event(c);
  r.kind = kind;
  r.bytes = bytes;
  r.flops = flops;
  cudaEventRecord(r.a, st);
  f();
  cudaEventRecord(r.b, st);
  c->recs.push_back(r);
}

// Algorithmic bytes of a fused GEMM: the activation operand, the packed weight with its scales,
// the output (and residual), the LoRA operands.
double gemm_bytes(const GemmArgs& g) {
  const double M = static_cast<double>(g.M), N = static_cast<double>(g.N), K = static_cast<double>(g.K);
  double b = 2.0 * M * K + N * K / 2.0 + 2.0 * N * (K / 64.0);
  if (g.epi == EPI_F32) b += 4.0 * M * N;
  else if (g.epi == EPI_F16 || g.epi == EPI_CEGRAD) b += 2.0 * M * N;
  else if (g.epi == EPI_GLU) b += M * N + (g.C2 ? 2.0 * M * N : 0.0);  // m (N / 2 columns), gate and up
  else b += 8.0 * M * g.nparts / 2.0;  // LSE partials
  if (g.R) b += 4.0 * M * N;
  if (g.Ax) b += 2.0 * M * g.kx + 2.0 * N * g.kx;
  return b;
}

int run_gemm(mebp_ctx* c, GemmArgs& g, cudaStream_t st, const char* what) {
  g.err = c->d_err;
  g.ksplit_ws = (st == c->fstream && c->fstream) ? c->ksplit[1] : c->ksplit[0];
  g.ksplit_floats = g.ksplit_ws ? c->ksplit_floats : 0;
  int rc = MEBP_OK;
  KP(c, g.trans ? KK_GEMM_DX : KK_GEMM_FWD, gemm_bytes(g),
     2.0 * g.M * g.N * g.K + (g.Ax ? 2.0 * g.M * g.N * g.kx : 0.0), st, [&] { rc = launch_dequant_gemm(g, st); });
  if (rc) return fail(c, rc, std::string(what) + ": fused GEMM launch failed (" + std::to_string(rc) + ")");
  return MEBP_OK;
}

// fp16 shadows of one fused linear's LoRA masters.
void build_shadow(mebp_ctx* c, Shadow& A, int li, const mebp_lora* lora, cudaStream_t st) {
  const Lin& l = c->lin[li];
  if (!l.kx) return;
  const float* As[3];
  const float* Bs[3];
  for (int t = 0; t < l.nt; ++t) {
    As[t] = lora->A[l.tgt[t]];
    Bs[t] = lora->B[l.tgt[t]];
  }
  launch_lora_shadow(As, Bs, l.nt, l.ro, l.no, l.nl, c->r, l.K, l.N, l.kxp, A.A_cat[li], A.B_cat[li], A.Bt_cat[li],
                     st);
}

int check_lora(mebp_ctx* c, const mebp_lora* lora) {
  for (int li = 0; li < 4; ++li)
    for (int t = 0; t < c->lin[li].nt; ++t) {
      const int tg = c->lin[li].tgt[t];
      if (!lora || !lora->A[tg] || !lora->B[tg])
        return fail(c, MEBP_ERR_INVALID_ARG, "LoRA weights missing for target " + std::to_string(tg));
    }
  return MEBP_OK;
}

// Sliding window of layer `layer` (0 = global: causal over the whole sequence).
int layer_window(const mebp_ctx* c, int layer) {
  const int W = c->cfg.sliding_window;
  return (W > 0 && (layer + 1) % c->cfg.global_every != 0) ? W : 0;
}
const float2* layer_rope(const mebp_ctx* c, int layer) {
  return layer_window(c, layer) ? c->rope_cs_local : c->rope_cs;
}

// y = F(x) for one block.  with_down == false stops after the MLP activation (what the
// backward consumes), so y is not produced; the Gemma3 block still runs the down projection,
// whose output the backward of its sandwich norm reads.
// keep_gu: the gate and up pre-activations are stored in the set (a backward reads them from it); a
// forward whose intermediates are recomputed before any backward can skip them.
int block_forward(mebp_ctx* c, int set, int layer, const mebp_block_weights* w, const mebp_lora* lora, const float* x,
                  float* y, int B, int Sq, bool with_down, cudaStream_t st, const Shadow* sh = nullptr,
                  bool keep_gu = true) {
  Acts& A = c->act[set];
  const int64_t T = static_cast<int64_t>(B) * Sq;
  const int D = c->D, I = c->I;
  int rc;
  if (!sh) {
    for (int li = 0; li < 4; ++li) build_shadow(c, A.own, li, lora, st);
    sh = &A.own;
  }
  A.sh = sh;
  // attention sub-block
  KP(c, KK_RMSNORM_FWD, bytes_rms_fwd(T, D), 0, st,
     [&] { launch_rmsnorm_fwd(x, w->norm1, T, D, c->cfg.rms_eps, A.a, A.r1, st); });
  const Lin& lq = c->lin[LIN_QKV];
  GemmArgs g = gemm_fwd(A.a, D, T, w->qkv, lq.N, lq.K);
  if (lq.kx) {
    KP(c, KK_LORA_SKINNY, bytes_skinny(T, D, lq.kx, lq.kxp), 2.0 * T * D * lq.kx, st, [&] {
      launch_skinny_gemm(A.a, D, T, D, A.sh->A_cat[LIN_QKV], D, lq.kx, c->s, A.us[LIN_QKV], lq.kxp, st, c->d_err);
    });
    g.Ax = A.us[LIN_QKV]; g.ldax = lq.kxp; g.kx = lq.kxp; g.Bx = A.sh->B_cat[LIN_QKV]; g.ldbx = lq.kxp;
  }
  g.epi = EPI_F16; g.C = A.qkv; g.ldc = lq.N;
  if ((rc = run_gemm(c, g, st, "qkv"))) return rc;
  if (c->gemma)
    KP(c, KK_QKNORM_ROPE, bytes_qknorm(T, Sq, c->H, c->KV, c->hd), 0, st, [&] {
      launch_qknorm_rope(A.qkv, T, Sq, c->H, c->KV, c->hd, w->q_norm, w->k_norm, c->cfg.rms_eps,
                         layer_rope(c, layer), A.qk_raw, A.rqk, st);
    });
  else
    KP(c, KK_ROPE, bytes_rope(T, Sq, c->H, c->KV, c->hd), 0, st,
       [&] { launch_rope(A.qkv, T, Sq, c->H, c->KV, c->hd, layer_rope(c, layer), false, st); });
  {
    const int win = layer_window(c, layer) >= Sq ? 0 : layer_window(c, layer);
    KP(c, KK_ATTN_FWD, bytes_attn_fwd(T, c->H, c->KV, c->hd),
       c->prof ? attn_fwd_flops(B, Sq, c->H, c->hd, win) : 0.0, st, [&] {
         rc = launch_attn_fwd(A.qkv, lq.N, B, Sq, c->H, c->KV, c->hd, A.o, c->Na, A.lse_attn, layer_window(c, layer),
                              c->d_err, st);
       });
    if (rc) return fail(c, rc, "attention forward launch failed");
  }
  const Lin& lo = c->lin[LIN_O];
  g = gemm_fwd(A.o, c->Na, T, w->o, lo.N, lo.K);
  if (lo.kx) {
    KP(c, KK_LORA_SKINNY, bytes_skinny(T, c->Na, lo.kx, lo.kxp), 2.0 * T * c->Na * lo.kx, st, [&] {
      launch_skinny_gemm(A.o, c->Na, T, c->Na, A.sh->A_cat[LIN_O], c->Na, lo.kx, c->s, A.us[LIN_O],
          lo.kxp, st, c->d_err);
    });
    g.Ax = A.us[LIN_O]; g.ldax = lo.kxp; g.kx = lo.kxp; g.Bx = A.sh->B_cat[LIN_O]; g.ldbx = lo.kxp;
  }
  if (c->gemma) {  // h1 = x + norm(ao) g_pa, b = norm(h1) g2
    g.epi = EPI_F32; g.C = A.ao; g.ldc = D;
    if ((rc = run_gemm(c, g, st, "o_proj"))) return rc;
    KP(c, KK_ADD_NORM, 14.0 * T * D + 8.0 * T + 8.0 * D, 0, st, [&] {
      launch_add_norm2(A.ao, x, w->post_attn_norm, w->norm2, T, D, c->cfg.rms_eps, A.h1, A.b, A.rpa, A.r2, st);
    });
  } else {
    g.epi = EPI_F32; g.C = A.h1; g.ldc = D; g.R = x; g.ldr = D;
    if ((rc = run_gemm(c, g, st, "o_proj"))) return rc;
    KP(c, KK_RMSNORM_FWD, bytes_rms_fwd(T, D), 0, st,
       [&] { launch_rmsnorm_fwd(A.h1, w->norm2, T, D, c->cfg.rms_eps, A.b, A.r2, st); });
  }
  // MLP sub-block
  const Lin& lg = c->lin[LIN_GU];
  g = gemm_fwd(A.b, D, T, w->gate_up, lg.N, lg.K);
  if (lg.kx) {
    KP(c, KK_LORA_SKINNY, bytes_skinny(T, D, lg.kx, lg.kxp), 2.0 * T * D * lg.kx, st, [&] {
      launch_skinny_gemm(A.b, D, T, D, A.sh->A_cat[LIN_GU], D, lg.kx, c->s, A.us[LIN_GU], lg.kxp, st, c->d_err);
    });
    g.Ax = A.us[LIN_GU]; g.ldax = lg.kxp; g.kx = lg.kxp; g.Bx = A.sh->B_cat[LIN_GU]; g.ldbx = lg.kxp;
  }
  // When the gate|up GEMM runs on the wide kernel without a K split, its epilogue applies the
  // activation itself (EPI_GLU): it writes m and, when a backward will read them, gate and up.
  // Below 2048 tokens (one-accumulator tiles) only when gate and up need not be kept: storing
  // all three from the epilogue lengthened each tile more than the separate GLU launch cost
  // (Gemma3-1B shape, 1024 tokens: 13.59 vs 13.49 ms per step).
  const bool fuse_glu =
      I % 128 == 0 && lg.N == 2 * I && gemm_glu_fusable(T, lg.N, lg.K) && (T >= 2048 || !keep_gu);
  if (fuse_glu) {
    g.epi = EPI_GLU; g.C = A.m; g.ldc = I; g.C2 = keep_gu ? A.gu : nullptr; g.ldc2 = lg.N; g.glu_half = I;
    g.act = c->cfg.act;
    if ((rc = run_gemm(c, g, st, "gate_up"))) return rc;
  } else {
    g.epi = EPI_F16; g.C = A.gu; g.ldc = lg.N;
    if ((rc = run_gemm(c, g, st, "gate_up"))) return rc;
    KP(c, KK_GLU_FWD, 6.0 * T * I, 0, st, [&] { launch_glu_fwd(A.gu, T, I, c->cfg.act, A.m, c->d_err, st); });
  }
  const Lin& ld = c->lin[LIN_DOWN];
  if (ld.kx)
    KP(c, KK_LORA_SKINNY, bytes_skinny(T, I, ld.kx, ld.kxp), 2.0 * T * I * ld.kx, st, [&] {
      launch_skinny_gemm(A.m, I, T, I, A.sh->A_cat[LIN_DOWN], I, ld.kx, c->s, A.us[LIN_DOWN], ld.kxp, st, c->d_err);
    });
  if (with_down || c->gemma) {
    g = gemm_fwd(A.m, I, T, w->down, ld.N, ld.K);
    if (ld.kx) {
      g.Ax = A.us[LIN_DOWN]; g.ldax = ld.kxp; g.kx = ld.kxp; g.Bx = A.sh->B_cat[LIN_DOWN]; g.ldbx = ld.kxp;
    }
    if (c->gemma) {  // y = h1 + norm(dn) g_pf
      g.epi = EPI_F32; g.C = A.dn; g.ldc = D;
      if ((rc = run_gemm(c, g, st, "down"))) return rc;
      KP(c, KK_ADD_NORM, (with_down ? 12.0 : 8.0) * T * D + 4.0 * T + 4.0 * D, 0, st, [&] {
        launch_add_norm(A.dn, A.h1, w->post_ffn_norm, T, D, c->cfg.rms_eps, with_down ? y : nullptr, A.rpf, st);
      });
    } else {
      g.epi = EPI_F32; g.C = y; g.ldc = D; g.R = A.h1; g.ldr = D;
      if ((rc = run_gemm(c, g, st, "down"))) return rc;
    }
  }
  A.layer = (fuse_glu && !keep_gu) ? -1 : layer;  // without gate and up the set cannot serve a backward
  A.x = x;
  A.T = T;
  return cuda_check(c, "block forward");
}

// The batched LoRA-gradient reductions of one block (one launch).
void run_tall_batch(mebp_ctx* c, const TallBatch& b, cudaStream_t st) {
  double bytes = 0.0, flops = 0.0;
  for (int i = 0; i < b.n; ++i) {
    bytes += bytes_tall(b.M, b.p[i].Pw, b.p[i].Qw, b.p[i].acc != 0);
    flops += 2.0 * b.M * b.p[i].Pw * b.p[i].Qw;
  }
  KP(c, KK_LORA_REDUCE, bytes, flops, st, [&] { launch_tall_reduce_batched(b, st); });
}

// Token counts below this run a block's LoRA-gradient reductions as one batched launch (each is a
// single pass over the tokens there); larger ones launch each reduction with its token split.
constexpr int64_t kTallBatchMaxT = 2048;

// LoRA gradients of one fused linear: dB_t = dY[:, rows_t]^T U_s[:, ranks_t], dA_t = dU[:, ranks_t]^T X.
// With tb the reductions are queued in the batch (launched by the caller) where it can take them.
int lin_grads(mebp_ctx* c, const Acts& A, const uint16_t* du, int li, const uint16_t* dY, int64_t ldy,
              const uint16_t* X, int64_t ldx, int64_t T, const mebp_lora_grads* grads, bool acc,
              const float* grad_mult, cudaStream_t st, TallBatch* tb = nullptr) {
  const Lin& l = c->lin[li];
  // dA of all the linear's targets in one pass over X when they sit side by side in dU (their rank
  // blocks consecutive) and the tensor-core reduction takes the shape
  bool dA_fused = false;
  if (grads && !tb && l.nt > 1) {
    bool ok = true;
    float* Cs[3] = {nullptr, nullptr, nullptr};
    for (int t = 0; t < l.nt; ++t) {
      ok = ok && grads->dA[l.tgt[t]] && l.ro[t] == l.ro[0] + t * c->r;
      Cs[t] = grads->dA[l.tgt[t]];
    }
    if (ok && tall_tc_takes(T, l.K, l.nt, c->r)) {
      int rc = MEBP_OK;
      KP(c, KK_LORA_REDUCE, bytes_tall(T, l.K, l.nt * c->r, acc), 2.0 * T * l.K * l.nt * c->r, st, [&] {
        rc = launch_tall_reduce_multi(X, ldx, du + l.ro[0], l.kxp, T, l.K, l.nt, c->r, Cs, -l.K, acc, grad_mult,
                                      c->red, c->red_floats, c->d_err, st);
      });
      if (rc) return fail(c, rc, "LoRA dA reduction");
      dA_fused = true;
    }
  }
  for (int t = 0; t < l.nt; ++t) {
    const int tg = l.tgt[t];
    if (!grads) break;
    if (grads->dB[tg] &&
        !(tb && tall_batch_add(*tb, dY + l.no[t], ldy, A.us[li] + l.ro[t], l.kxp, l.nl[t], c->r, grads->dB[tg], c->r,
                               acc))) {
      int rc = MEBP_OK;
      KP(c, KK_LORA_REDUCE, bytes_tall(T, l.nl[t], c->r, acc), 2.0 * T * l.nl[t] * c->r, st, [&] {
        float* C1[1] = {grads->dB[tg]};
        rc = launch_tall_reduce_multi(dY + l.no[t], ldy, A.us[li] + l.ro[t], l.kxp, T, l.nl[t], 1, c->r, C1, c->r,
                                      acc, grad_mult, c->red, c->red_floats, c->d_err, st);
      });
      if (rc) return fail(c, rc, "LoRA dB reduction");
    }
    if (grads->dA[tg] && !dA_fused &&
        !(tb && tall_batch_add(*tb, X, ldx, du + l.ro[t], l.kxp, l.K, c->r, grads->dA[tg], -l.K, acc))) {
      int rc = MEBP_OK;
      KP(c, KK_LORA_REDUCE, bytes_tall(T, l.K, c->r, acc), 2.0 * T * l.K * c->r, st, [&] {
        float* C1[1] = {grads->dA[tg]};
        rc = launch_tall_reduce_multi(X, ldx, du + l.ro[t], l.kxp, T, l.K, 1, c->r, C1, -l.K, acc, grad_mult, c->red,
                                      c->red_floats, c->d_err, st);
      });
      if (rc) return fail(c, rc, "LoRA dA reduction");
    }
  }
  return MEBP_OK;
}

// dE/dx and LoRA grads of one block from its input checkpoint x and dE/dy.  dy (fp32) and its
// fp16 copy dy_h are in the backward's working scale sigma (a power of two that keeps the fp16
// operands in range); the LoRA gradients are written times *grad_mult and dx times *dx_mult
// (null = 1), so grad_mult = dx_mult = 1/sigma gives true gradients.  dx_h = fp16(sigma dE/dx).
// dx / dx_h may be null.
int block_backward(mebp_ctx* c, int set, int bset, int layer, const mebp_block_weights* w, const mebp_lora* lora,
                   const float* x, const float* dy, const uint16_t* dy_h, float* dx, uint16_t* dx_h,
                   const mebp_lora_grads* grads, int B, int Sq, bool acc, const float* grad_mult,
                   const float* dx_mult, cudaStream_t st, const Shadow* sh = nullptr) {
  Acts& A = c->act[set];
  Grads2& G = c->bw[bset];
  uint16_t* const* du = G.du;
  const int64_t T = static_cast<int64_t>(B) * Sq;
  const int D = c->D, I = c->I;
  int rc;
  TallBatch batch;
  batch.M = T;
  batch.mult = grad_mult;
  TallBatch* tb = T < kTallBatchMaxT ? &batch : nullptr;
  if (!(A.layer == layer && A.x == x && A.T == T)) {
    if ((rc = block_forward(c, set, layer, w, lora, x, nullptr, B, Sq, false, st, sh))) return rc;
  }
  A.layer = -1;  // the set is consumed below
  // ---- down projection: y = h1 + m Wd^T (+ s (m Ad^T) Bd^T); Gemma3: y = h1 + norm(dn) g_pf
  const uint16_t* ddn_h = dy_h;
  if (c->gemma) {
    KP(c, KK_RMSNORM_BWD, bytes_rms_bwd(T, D, false, false, true), 0, st, [&] {
      launch_rmsnorm_bwd(dy, A.dn, w->post_ffn_norm, A.rpf, nullptr, T, D, nullptr, nullptr, G.ddn_h, st);
    });
    ddn_h = G.ddn_h;
  }
  const Lin& ld = c->lin[LIN_DOWN];
  GemmArgs g = gemm_dx(ddn_h, D, T, w->down);
  if (ld.kx) {
    KP(c, KK_LORA_SKINNY, bytes_skinny(T, D, ld.kx, ld.kxp), 2.0 * T * D * ld.kx, st, [&] {
      launch_skinny_gemm(ddn_h, D, T, D, A.sh->Bt_cat[LIN_DOWN], D, ld.kx, c->s, du[LIN_DOWN], ld.kxp, st, c->d_err);
    });
    g.Ax = du[LIN_DOWN]; g.ldax = ld.kxp; g.kx = ld.kxp; g.Bx = A.sh->A_cat[LIN_DOWN]; g.ldbx = I;
  }
  g.epi = EPI_F16; g.C = c->dm; g.ldc = I;
  if ((rc = run_gemm(c, g, st, "down dX"))) return rc;
  if ((rc = lin_grads(c, A, du[LIN_DOWN], LIN_DOWN, ddn_h, D, A.m, I, T, grads, acc, grad_mult, st, tb))) return rc;
  // ---- gated MLP
  KP(c, KK_GLU_BWD, 10.0 * T * I, 0, st,
     [&] { launch_glu_bwd(c->dm, A.gu, T, I, c->cfg.act, G.dgu, c->d_err, st); });
  const Lin& lg = c->lin[LIN_GU];
  g = gemm_dx(G.dgu, 2 * I, T, w->gate_up);
  if (lg.kx) {
    KP(c, KK_LORA_SKINNY, bytes_skinny(T, 2 * I, lg.kx, lg.kxp), 4.0 * T * I * lg.kx, st, [&] {
      launch_skinny_gemm(G.dgu, 2 * I, T, 2 * I, A.sh->Bt_cat[LIN_GU], 2 * I, lg.kx, c->s, du[LIN_GU],
          lg.kxp, st, c->d_err);
    });
    g.Ax = du[LIN_GU]; g.ldax = lg.kxp; g.kx = lg.kxp; g.Bx = A.sh->A_cat[LIN_GU]; g.ldbx = D;
  }
  g.epi = EPI_F32; g.C = c->dtmp; g.ldc = D;
  if ((rc = run_gemm(c, g, st, "gate_up dX"))) return rc;
  if ((rc = lin_grads(c, A, du[LIN_GU], LIN_GU, G.dgu, 2 * I, A.b, D, T, grads, acc, grad_mult, st, tb))) return rc;
  // dh1 = dy + RMSNorm2^T(db); the o projection's output gradient is dh1 (fp16 copy in dh1_h), for
  // Gemma3 the post-attention norm's VJP of it
  if (c->gemma) {
    KP(c, KK_RMSNORM_BWD, bytes_rms_bwd(T, D, true, true, false), 0, st,
       [&] { launch_rmsnorm_bwd(c->dtmp, A.h1, w->norm2, A.r2, dy, T, D, nullptr, c->dh1, nullptr, st); });
    KP(c, KK_RMSNORM_BWD, bytes_rms_bwd(T, D, false, false, true), 0, st, [&] {
      launch_rmsnorm_bwd(c->dh1, A.ao, w->post_attn_norm, A.rpa, nullptr, T, D, nullptr, nullptr, G.dh1_h, st);
    });
  } else {
    KP(c, KK_RMSNORM_BWD, bytes_rms_bwd(T, D, true, true, true), 0, st,
       [&] { launch_rmsnorm_bwd(c->dtmp, A.h1, w->norm2, A.r2, dy, T, D, nullptr, c->dh1, G.dh1_h, st); });
  }
  // ---- o projection
  const Lin& lo = c->lin[LIN_O];
  g = gemm_dx(G.dh1_h, D, T, w->o);
  if (lo.kx) {
    KP(c, KK_LORA_SKINNY, bytes_skinny(T, D, lo.kx, lo.kxp), 2.0 * T * D * lo.kx, st, [&] {
      launch_skinny_gemm(G.dh1_h, D, T, D, A.sh->Bt_cat[LIN_O], D, lo.kx, c->s, du[LIN_O], lo.kxp, st, c->d_err);
    });
    g.Ax = du[LIN_O]; g.ldax = lo.kxp; g.kx = lo.kxp; g.Bx = A.sh->A_cat[LIN_O]; g.ldbx = c->Na;
  }
  g.epi = EPI_F16; g.C = c->dout; g.ldc = c->Na;
  if ((rc = run_gemm(c, g, st, "o dX"))) return rc;
  if ((rc = lin_grads(c, A, du[LIN_O], LIN_O, G.dh1_h, D, A.o, c->Na, T, grads, acc, grad_mult, st, tb))) return rc;
  // ---- attention, RoPE
  const Lin& lq = c->lin[LIN_QKV];
  bool rope_done = false;
  {
    const int win = layer_window(c, layer) >= Sq ? 0 : layer_window(c, layer);
    KP(c, KK_ATTN_BWD, bytes_attn_bwd(T, c->H, c->KV, c->hd),
       c->prof ? 2.5 * attn_fwd_flops(B, Sq, c->H, c->hd, win) : 0.0, st, [&] {
         rope_done = launch_attn_bwd(A.qkv, lq.N, A.o, c->dout, c->Na, A.lse_attn, B, Sq, c->H, c->KV, c->hd, c->dvec,
                                     G.dqkv, layer_window(c, layer), c->gemma ? nullptr : layer_rope(c, layer),
                                     c->attn_ws, c->attn_ws_floats, c->d_err, st);
       });
  }
  if (c->gemma)
    KP(c, KK_QKNORM_ROPE, bytes_qknorm(T, Sq, c->H, c->KV, c->hd), 0, st, [&] {
      launch_qknorm_rope_bwd(G.dqkv, T, Sq, c->H, c->KV, c->hd, w->q_norm, w->k_norm, layer_rope(c, layer), A.qk_raw,
                             A.rqk, st);
    });
  else if (!rope_done)
    KP(c, KK_ROPE, bytes_rope(T, Sq, c->H, c->KV, c->hd), 0, st,
       [&] { launch_rope(G.dqkv, T, Sq, c->H, c->KV, c->hd, layer_rope(c, layer), true, st); });
  // ---- q, k, v projections
  if (lq.kx)
    KP(c, KK_LORA_SKINNY, bytes_skinny(T, lq.N, lq.kx, lq.kxp), 2.0 * T * lq.N * lq.kx, st, [&] {
      launch_skinny_gemm(G.dqkv, lq.N, T, lq.N, A.sh->Bt_cat[LIN_QKV], lq.N, lq.kx, c->s, du[LIN_QKV],
          lq.kxp, st, c->d_err);
    });
  if ((rc = lin_grads(c, A, du[LIN_QKV], LIN_QKV, G.dqkv, lq.N, A.a, D, T, grads, acc, grad_mult, st, tb))) return rc;
  if (dx) {
    g = gemm_dx(G.dqkv, lq.N, T, w->qkv);
    if (lq.kx) {
      g.Ax = du[LIN_QKV]; g.ldax = lq.kxp; g.kx = lq.kxp; g.Bx = A.sh->A_cat[LIN_QKV]; g.ldbx = D;
    }
    g.epi = EPI_F32; g.C = c->dtmp; g.ldc = D;
    if ((rc = run_gemm(c, g, st, "qkv dX"))) return rc;
    KP(c, KK_RMSNORM_BWD, bytes_rms_bwd(T, D, true, dx != nullptr, dx_h != nullptr), 0, st,
       [&] { launch_rmsnorm_bwd(c->dtmp, x, w->norm1, A.r1, c->dh1, T, D, dx_mult, dx, dx_h, st); });
  }
  if (batch.n) run_tall_batch(c, batch, st);
  return cuda_check(c, "block backward");
}

// The LoRA-gradient reductions of one block whose backward (block_backward with grads = null)
// has been issued: the same operands the inline reductions read.
int block_lora_grads(mebp_ctx* c, int set, int bset, const uint16_t* dy_h, int64_t T, const mebp_lora_grads* grads,
                     bool acc, const float* grad_mult, cudaStream_t st) {
  const Acts& A = c->act[set];
  const Grads2& G = c->bw[bset];
  const int D = c->D, I = c->I;
  int rc;
  TallBatch batch;
  batch.M = T;
  batch.mult = grad_mult;
  TallBatch* tb = T < kTallBatchMaxT ? &batch : nullptr;
  const uint16_t* ddn_h = c->gemma ? G.ddn_h : dy_h;
  if ((rc = lin_grads(c, A, G.du[LIN_DOWN], LIN_DOWN, ddn_h, D, A.m, I, T, grads, acc, grad_mult, st, tb))) return rc;
  if ((rc = lin_grads(c, A, G.du[LIN_GU], LIN_GU, G.dgu, 2 * I, A.b, D, T, grads, acc, grad_mult, st, tb))) return rc;
  if ((rc = lin_grads(c, A, G.du[LIN_O], LIN_O, G.dh1_h, D, A.o, c->Na, T, grads, acc, grad_mult, st, tb))) return rc;
  if ((rc = lin_grads(c, A, G.du[LIN_QKV], LIN_QKV, G.dqkv, c->lin[LIN_QKV].N, A.a, D, T, grads, acc, grad_mult, st,
                      tb)))
    return rc;
  if (batch.n) run_tall_batch(c, batch, st);
  return MEBP_OK;
}

// Final RMSNorm + LM head + CE.  dh (fp32) is the true gradient when unscale_dh, else it is
// sigma * dloss/dh (the backward working scale, see loss_reduce_kernel); dh_h = fp16(sigma dloss/dh).
int lmhead(mebp_ctx* c, const mebp_packed* E, const float* gf, const float* h, const int32_t* targets, int64_t T,
           float* loss, float* dh, uint16_t* dh_h, float* tok_loss, bool unscale_dh, cudaStream_t st) {
  const int D = c->D, V = c->V;
  int rc;
  KP(c, KK_RMSNORM_FWD, bytes_rms_fwd(T, D), 0, st,
     [&] { launch_rmsnorm_fwd(h, gf, T, D, c->cfg.rms_eps, c->hf, c->rf, st); });
  GemmArgs g = gemm_fwd(c->hf, D, T, *E, V, D);
  g.epi = EPI_LSE; g.targets = targets; g.col_offset = 0; g.n_valid = V; g.part = c->part; g.nparts = c->nparts;
  g.zt = c->zt;
  if ((rc = run_gemm(c, g, st, "LM head (log-sum-exp pass)"))) return rc;
  float* tl = tok_loss ? tok_loss : c->tok_loss;
  KP(c, KK_LM_REDUCE, 8.0 * T * c->nparts + 20.0 * T, 0, st, [&] {
    launch_lse_combine(c->part, c->nparts, c->zt, targets, T, c->lse_tok, tl, st);
    launch_loss_reduce(tl, targets, T, loss, c->scal, st);
  });
  for (int c0 = 0; c0 < V; c0 += c->vchunk) {
    const int n = std::min(c->vchunk, V - c0);
    mebp_packed Ec = *E;
    Ec.qpack = E->qpack + static_cast<int64_t>(c0) * (D / 2);
    Ec.scales = E->scales + c0;
    Ec.rows = n;
    g = gemm_fwd(c->hf, D, T, Ec, n, D);
    g.scale_pitch = V;
    g.epi = EPI_CEGRAD; g.C = c->dz; g.ldc = c->vchunk; g.targets = targets; g.col_offset = c0; g.n_valid = n;
    g.lse = c->lse_tok; g.ce_w = c->scal + 2;
    if ((rc = run_gemm(c, g, st, "LM head (gradient pass)"))) return rc;
    GemmArgs t;
    t.trans = true;
    t.A = c->dz; t.lda = c->vchunk; t.M = T; t.N = D; t.K = n;
    t.qpack = Ec.qpack; t.scales = Ec.scales; t.scale_pitch = V;
    t.epi = EPI_F32; t.C = c->dhf; t.ldc = D; t.R = c0 ? c->dhf : nullptr; t.ldr = D; t.alpha = 1.0f / kCeShift;
    if ((rc = run_gemm(c, t, st, "LM head (dH pass)"))) return rc;
  }
  KP(c, KK_RMSNORM_BWD, bytes_rms_bwd(T, D, false, dh != nullptr, dh_h != nullptr), 0, st, [&] {
    launch_rmsnorm_bwd(c->dhf, h, gf, c->rf, nullptr, T, D, unscale_dh ? c->scal + 1 : nullptr, dh, dh_h, st);
  });
  return cuda_check(c, "LM head");
}

__global__ void targets_kernel(const int32_t* ids, int B, int Sq, int32_t* tg) {
  griddep_wait();
  griddep_launch();
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= static_cast<int64_t>(B) * Sq) return;
  const int s = static_cast<int>(i % Sq);
  tg[i] = (s < Sq - 1) ? ids[i + 1] : -1;
}

int check_block_ptrs(mebp_ctx* c, const mebp_block_weights* w) {
  int rc;
  if (!w) return fail(c, MEBP_ERR_INVALID_ARG, "NULL block weights");
  if ((rc = check_packed(c, &w->qkv, c->lin[LIN_QKV].N, c->D, "qkv"))) return rc;
  if ((rc = check_packed(c, &w->o, c->D, c->Na, "o"))) return rc;
  if ((rc = check_packed(c, &w->gate_up, 2 * c->I, c->D, "gate_up"))) return rc;
  if ((rc = check_packed(c, &w->down, c->D, c->I, "down"))) return rc;
  if (!w->norm1 || !w->norm2) return fail(c, MEBP_ERR_INVALID_ARG, "NULL norm gain");
  if (c->gemma) {
    const float* gs[4] = {w->q_norm, w->k_norm, w->post_attn_norm, w->post_ffn_norm};
    for (const float* p : gs)
      if (!p || !aligned16(p)) return fail(c, MEBP_ERR_INVALID_ARG, "Gemma3 norm gain NULL or not 16-byte aligned");
  }
  if (!aligned16(w->norm1) || !aligned16(w->norm2))
    return fail(c, MEBP_ERR_INVALID_ARG, "norm gains must be 16-byte aligned");
  return MEBP_OK;
}

// Gemma3 scales the input embeddings by sqrt(D) (rounded to fp32 once).
float embed_scale(const mebp_ctx* c) { return c->gemma ? static_cast<float>(std::sqrt(static_cast<double>(c->D))) : 1.0f; }

int check_tokens(mebp_ctx* c, int B, int Sq) {
  if (B <= 0 || Sq <= 0) return fail(c, MEBP_ERR_INVALID_ARG, "batch and seq must be positive");
  if (static_cast<int64_t>(B) * Sq > c->Tmax) return fail(c, MEBP_ERR_INVALID_ARG, "batch*seq exceeds max_tokens");
  if (Sq > c->cfg.max_seq) return fail(c, MEBP_ERR_INVALID_ARG, "seq exceeds max_seq");
  return MEBP_OK;
}

}  // namespace

// ===================================================================================== C ABI
extern "C" {

int mebp_ctx_create(const mebp_model_cfg* cfg, int device, mebp_ctx** out) {
  if (!cfg || !out) return MEBP_ERR_INVALID_ARG;
  *out = nullptr;
  const mebp_model_cfg& f = *cfg;
  if (f.hidden <= 0 || f.hidden % 64 || f.n_heads <= 0 || f.n_kv_heads <= 0 || f.n_heads % f.n_kv_heads ||
      f.intermediate <= 0 || f.intermediate % 64 || f.n_layers <= 0 || f.max_tokens <= 0 || f.max_seq <= 0 ||
      f.vocab < 0 || f.vocab % 64 || f.lora_rank < 0 || f.lora_rank > 32)
    return MEBP_ERR_INVALID_ARG;
  if (!(f.head_dim == 64 || f.head_dim == 128 || f.head_dim == 256)) return MEBP_ERR_UNSUPPORTED;
  // query heads per kv head <= 8: the split attention backward sums at most 8 heads x 2 parts
  if (f.n_heads / f.n_kv_heads > 8) return MEBP_ERR_UNSUPPORTED;
  if (f.lora_targets && (f.lora_rank % 8)) return MEBP_ERR_UNSUPPORTED;
  if (f.act != MEBP_ACT_SILU && f.act != MEBP_ACT_GELU_TANH) return MEBP_ERR_INVALID_ARG;
  if (f.vocab_chunk < 0 || f.vocab_chunk % 256) return MEBP_ERR_INVALID_ARG;
  if (f.sliding_window < 0 || (f.sliding_window > 0 && (f.global_every < 1 || !(f.rope_theta_local > 0.0f))))
    return MEBP_ERR_INVALID_ARG;
  if (cudaSetDevice(device) != cudaSuccess) {
    cudaGetLastError();
    return MEBP_ERR_CUDA;
  }
  mebp_ctx* c = new mebp_ctx();
  c->cfg = f;
  c->device = device;
  c->D = f.hidden; c->H = f.n_heads; c->KV = f.n_kv_heads; c->hd = f.head_dim; c->I = f.intermediate;
  c->V = f.vocab; c->L = f.n_layers; c->r = f.lora_targets ? f.lora_rank : 0; c->s = f.lora_scale;
  c->Tmax = f.max_tokens;
  c->Na = c->H * c->hd;
  c->gemma = f.gemma_norms != 0;
  setup_lin(c);
  c->Nqkv = c->lin[LIN_QKV].N;
  if (c->Na % 64) {
    delete c;
    return MEBP_ERR_UNSUPPORTED;
  }
  const int64_t T = c->Tmax, D = c->D, I = c->I;
  int rc = MEBP_OK;
  auto A = [&](auto** p, int64_t n) {
    if (rc == MEBP_OK) rc = dalloc(c, p, n);
  };
  c->cur_cat = MEBP_WS_OTHER;
  A(&c->d_err, 4);
  A(&c->scal, 8);
  A(&c->rope_cs, static_cast<int64_t>(f.max_seq) * (c->hd / 2));
  if (f.sliding_window > 0) A(&c->rope_cs_local, static_cast<int64_t>(f.max_seq) * (c->hd / 2));
  // a second intermediate set lets the step overlap recompute and backward (not when spilling:
  // then device memory is the constraint)
  c->nsets = (!f.spill_ckpts && !f.min_memory && c->L > 1) ? 2 : 1;
  for (int k = 0; k < c->nsets; ++k) {
    Acts& s = c->act[k];
    c->cur_cat = MEBP_WS_FWD_SETS;
    A(&s.a, T * D); A(&s.b, T * D); A(&s.qkv, T * c->Nqkv); A(&s.o, T * c->Na); A(&s.gu, T * 2 * I);
    A(&s.m, T * I); A(&s.r1, T); A(&s.r2, T); A(&s.lse_attn, T * c->H); A(&s.h1, T * D);
    if (c->gemma) {
      A(&s.ao, T * D); A(&s.dn, T * D); A(&s.rpa, T); A(&s.rpf, T);
      A(&s.qk_raw, T * (c->H + c->KV) * c->hd); A(&s.rqk, T * (c->H + c->KV));
    }
    for (int li = 0; li < 4; ++li) {
      const Lin& l = c->lin[li];
      if (!l.kx) continue;
      c->cur_cat = MEBP_WS_FWD_SETS;
      A(&s.us[li], T * l.kxp);
      c->cur_cat = MEBP_WS_LORA_SHADOW;
      A(&s.own.A_cat[li], static_cast<int64_t>(l.kxp) * l.K);
      A(&s.own.B_cat[li], static_cast<int64_t>(l.N) * l.kxp);
      A(&s.own.Bt_cat[li], static_cast<int64_t>(l.N) * l.kxp);
    }
  }
  // the step's per-block shadows (one allocation per linear, blocks back to back)
  c->cur_cat = MEBP_WS_LORA_SHADOW;
  c->layer_sh.assign(c->L, Shadow{});
  for (int li = 0; li < 4; ++li) {
    const Lin& l = c->lin[li];
    if (!l.kx) continue;
    uint16_t *pa = nullptr, *pb = nullptr, *pbt = nullptr;
    const int64_t na = static_cast<int64_t>(l.kxp) * l.K, nb = static_cast<int64_t>(l.N) * l.kxp;
    A(&pa, na * c->L); A(&pb, nb * c->L); A(&pbt, nb * c->L);
    if (rc != MEBP_OK) break;
    for (int i = 0; i < c->L; ++i) {
      c->layer_sh[i].A_cat[li] = pa + i * na;
      c->layer_sh[i].B_cat[li] = pb + i * nb;
      c->layer_sh[i].Bt_cat[li] = pbt + i * nb;
    }
  }
  c->cur_cat = MEBP_WS_BWD;
  for (int k = 0; k < c->nsets; ++k) {
    Grads2& g = c->bw[k];
    A(&g.dqkv, T * c->Nqkv); A(&g.dgu, T * 2 * I); A(&g.dh1_h, T * D);
    if (c->gemma) A(&g.ddn_h, T * D);
    for (int li = 0; li < 4; ++li)
      if (c->lin[li].kx) A(&g.du[li], T * c->lin[li].kxp);
  }
  if (rc == MEBP_OK && c->nsets == 2) {
    if (cudaStreamCreateWithFlags(&c->fstream, cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->ev_main, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->ev_fwd[0], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->ev_fwd[1], cudaEventDisableTiming) != cudaSuccess ||
        cudaStreamCreateWithFlags(&c->gstream, cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->ev_bwd, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->ev_grad[0], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->ev_grad[1], cudaEventDisableTiming) != cudaSuccess) {
      cudaGetLastError();
      rc = MEBP_ERR_CUDA;
    }
  }
  c->cur_cat = MEBP_WS_BWD;
  A(&c->dout, T * c->Na);
  for (int k = 0; k < (c->nsets == 2 ? 3 : 2); ++k) A(&c->dy_h[k], T * D);
  A(&c->dm, T * I); A(&c->dtmp, T * D); A(&c->dh1, T * D); A(&c->dvec, T * c->H);
  // split attention backward: 3 arrays of B * ceil(S/64) * H * 2 parts * 64 * hd floats (<= 2 T rows
  // per head and part when S >= 64), at most 192 MB; larger shapes take the direct mode
  c->attn_ws_floats = std::min<int64_t>(3LL * 2 * c->H * c->hd * 2 * T, 48LL << 20);
  c->cur_cat = MEBP_WS_ATTN_SPLIT;
  A(&c->attn_ws, c->attn_ws_floats);
  c->cur_cat = MEBP_WS_BWD;
  A(&c->gbuf[0], T * D); A(&c->gbuf[1], T * D);
  c->red_floats = std::max<int64_t>(tall_reduce_scratch_floats(T, std::max<int64_t>(2 * I, c->Nqkv), 32),
                                    tall_reduce_scratch_floats(T, std::max<int64_t>(I, D), 32));
  c->cur_cat = MEBP_WS_OTHER;
  A(&c->red, c->red_floats);
  c->cur_cat = MEBP_WS_LMHEAD;
  if (c->V > 0) {
    c->nparts = 4 * ((c->V + 255) / 256);  // four (max, sum) parts per 256-column tile
    int64_t vc = f.vocab_chunk;
    if (vc == 0) {
      vc = (int64_t(1) << 30) / (2 * T);
      vc = std::max<int64_t>(4096, vc / 256 * 256);
    }
    c->vchunk = static_cast<int>(std::min<int64_t>(vc, (c->V + 255) / 256 * 256));
    A(&c->hf, T * D); A(&c->rf, T); A(&c->part, T * c->nparts * 2); A(&c->zt, T); A(&c->lse_tok, T);
    A(&c->tok_loss, T); A(&c->dz, T * c->vchunk); A(&c->dhf, T * D); A(&c->targets, T);
  }
  // K-split partials: the largest any of the step's fused GEMMs wants at T tokens (forward and
  // input-gradient shapes of the four linears, the LM head's dH pass over one vocabulary chunk)
  {
    int64_t kf = c->V > 0 ? gemm_ksplit_floats(T, D, c->vchunk) : 0;
    for (int li = 0; li < 4; ++li) {
      kf = std::max(kf, gemm_ksplit_floats(T, c->lin[li].N, c->lin[li].K));
      kf = std::max(kf, gemm_ksplit_floats(T, c->lin[li].K, c->lin[li].N));
    }
    c->ksplit_floats = kf;
    c->cur_cat = MEBP_WS_OTHER;
    if (kf > 0) {
      A(&c->ksplit[0], kf);
      if (c->nsets == 2) A(&c->ksplit[1], kf);
    }
  }
  const int64_t nslots = f.spill_ckpts ? kCkptSlots : (c->L + 1);
  c->cur_cat = MEBP_WS_CKPT;
  A(&c->ckpt, nslots * T * D);
  if (rc == MEBP_OK && f.spill_ckpts) {
    const size_t hb = static_cast<size_t>(c->L + 1) * T * D * sizeof(float);
    c->ws_cat[MEBP_WS_HOST_CKPT] = static_cast<int64_t>(hb);
    if (cudaHostAlloc(reinterpret_cast<void**>(&c->h_ckpt), hb, cudaHostAllocDefault) != cudaSuccess) {
      cudaGetLastError();
      c->h_ckpt = nullptr;
      rc = MEBP_ERR_OOM;
    }
    if (rc == MEBP_OK && cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking) != cudaSuccess) rc = MEBP_ERR_CUDA;
    for (int i = 0; rc == MEBP_OK && i < kCkptSlots; ++i)
      if (cudaEventCreateWithFlags(&c->slot_free[i], cudaEventDisableTiming) != cudaSuccess ||
          cudaEventCreateWithFlags(&c->slot_ready[i], cudaEventDisableTiming) != cudaSuccess)
        rc = MEBP_ERR_CUDA;
    if (rc == MEBP_OK && cudaEventCreateWithFlags(&c->copy_join, cudaEventDisableTiming) != cudaSuccess)
      rc = MEBP_ERR_CUDA;
  }
  if (rc != MEBP_OK) {
    mebp_ctx_destroy(c);
    return rc;
  }
  // RoPE tables: angle(p, j) = p * theta^(-2j/hd), evaluated in double precision on the host.
  auto rope_table = [&](float2* dst, float theta) {
    const int half = c->hd / 2;
    std::vector<float2> cs(static_cast<size_t>(f.max_seq) * half);
    for (int p = 0; p < f.max_seq; ++p)
      for (int j = 0; j < half; ++j) {
        const double ang = p * std::pow(static_cast<double>(theta), -2.0 * j / c->hd);
        cs[static_cast<size_t>(p) * half + j] = make_float2(static_cast<float>(std::cos(ang)),
                                                            static_cast<float>(std::sin(ang)));
      }
    cudaMemcpy(dst, cs.data(), cs.size() * sizeof(float2), cudaMemcpyHostToDevice);
  };
  rope_table(c->rope_cs, f.rope_theta);
  if (c->rope_cs_local) rope_table(c->rope_cs_local, f.rope_theta_local);
  cudaMemset(c->d_err, 0, 16);
  cudaMemset(c->scal, 0, 8 * sizeof(float));
  for (int li = 0; li < 4; ++li) {
    const Lin& l = c->lin[li];
    if (!l.kx) continue;
    for (int k = 0; k < c->nsets; ++k) cudaMemset(c->act[k].us[li], 0, T * l.kxp * 2);
    for (int k = 0; k < c->nsets; ++k) cudaMemset(c->bw[k].du[li], 0, T * l.kxp * 2);
  }
  if (cudaDeviceSynchronize() != cudaSuccess || cudaGetLastError() != cudaSuccess) {
    mebp_ctx_destroy(c);
    return MEBP_ERR_CUDA;
  }
  *out = c;
  return MEBP_OK;
}

void mebp_ctx_destroy(mebp_ctx* c) {
  if (!c) return;
  cudaSetDevice(c->device);
  cudaDeviceSynchronize();
  for (void* p : c->dev_allocs) cudaFree(p);
  for (cudaEvent_t e : c->evpool) cudaEventDestroy(e);
  if (c->graph_exec) cudaGraphExecDestroy(c->graph_exec);
  if (c->copy_join) cudaEventDestroy(c->copy_join);
  if (c->h_ckpt) cudaFreeHost(c->h_ckpt);
  for (int i = 0; i < kCkptSlots; ++i) {
    if (c->slot_free[i]) cudaEventDestroy(c->slot_free[i]);
    if (c->slot_ready[i]) cudaEventDestroy(c->slot_ready[i]);
  }
  if (c->copy_stream) cudaStreamDestroy(c->copy_stream);
  if (c->ev_main) cudaEventDestroy(c->ev_main);
  for (cudaEvent_t e : c->ev_fwd)
    if (e) cudaEventDestroy(e);
  if (c->fstream) cudaStreamDestroy(c->fstream);
  if (c->ev_bwd) cudaEventDestroy(c->ev_bwd);
  for (cudaEvent_t e : c->ev_grad)
    if (e) cudaEventDestroy(e);
  if (c->gstream) cudaStreamDestroy(c->gstream);
  cudaGetLastError();
  delete c;
}

const char* mebp_last_error(const mebp_ctx* c) { return c ? c->err_msg.c_str() : "NULL context"; }

int64_t mebp_workspace_bytes(const mebp_ctx* c) { return c ? c->ws_bytes : 0; }

int mebp_workspace_breakdown(const mebp_ctx* c, int64_t* bytes, int* n_sets) {
  if (!c || !bytes) return MEBP_ERR_INVALID_ARG;
  for (int i = 0; i < MEBP_WS_N; ++i) bytes[i] = c->ws_cat[i];
  if (n_sets) *n_sets = c->nsets;
  return MEBP_OK;
}

int mebp_sync(mebp_ctx* c, void* stream) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  if (cudaStreamSynchronize(S(stream)) != cudaSuccess) return fail(c, MEBP_ERR_CUDA, cudaGetErrorString(cudaGetLastError()));
  int h = 0;
  if (cudaMemcpy(&h, c->d_err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return fail(c, MEBP_ERR_CUDA, cudaGetErrorString(cudaGetLastError()));
  if (h) {
    cudaMemset(c->d_err, 0, sizeof(int));
    return fail(c, h, h == MEBP_ERR_TIMEOUT     ? "a device-side bounded wait expired"
                      : h == MEBP_ERR_NONFINITE ? "an fp16 intermediate overflowed the fp16 range or is NaN"
                                                : "a kernel flagged invalid input (e.g. token id out of range)");
  }
  return MEBP_OK;
}

int64_t mebp_kernel_launches(void) { return g_launches.load(); }

int mebp_enable_graphs(mebp_ctx* c, int on) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  c->graphs = on != 0;
  if (c->graph_exec) cudaGraphExecDestroy(c->graph_exec);
  c->graph_exec = nullptr;
  c->graph_key.clear();
  c->graph_eager_runs = 0;
  return MEBP_OK;
}

int mebp_profile_begin(mebp_ctx* c) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  c->recs.clear();
  c->evnext = 0;
  c->prof = true;
  return MEBP_OK;
}

int mebp_profile_end(mebp_ctx* c, mebp_profile* out) {
  if (!c || !out) return MEBP_ERR_INVALID_ARG;
  c->prof = false;
  mebp_profile p{};
  c->kstats.assign(KK_N, mebp_kernel_stat{});
  for (int k = 0; k < KK_N; ++k) c->kstats[k].name = kKindName[k];
  // [start, end] of every fused-GEMM launch relative to the first record's start event; their union
  // is the time during which some fused GEMM ran (launches on concurrent streams overlap)
  std::vector<std::pair<double, double>> iv;
  iv.reserve(c->recs.size());
  for (const ProfRec& r : c->recs) {
    if (cudaEventSynchronize(r.b) != cudaSuccess) return fail(c, MEBP_ERR_CUDA, cudaGetErrorString(cudaGetLastError()));
    float ms = 0.0f, t0 = 0.0f;
    cudaEventElapsedTime(&ms, r.a, r.b);
    mebp_kernel_stat& ks = c->kstats[r.kind];
    ks.launches++;
    ks.ms += ms;
    ks.bytes += r.bytes;
    ks.flops += r.flops;
    if (r.kind != KK_GEMM_FWD && r.kind != KK_GEMM_DX) continue;
    cudaEventElapsedTime(&t0, c->recs.front().a, r.a);
    iv.emplace_back(t0, static_cast<double>(t0) + ms);
    p.gemm_launches++;
    p.gemm_ms += ms;
    p.gemm_flops += r.flops;
    p.gemm_bytes += r.bytes;
    if (r.kind == KK_GEMM_DX) {
      p.dx_ms += ms;
      p.dx_flops += r.flops;
    } else {
      p.fwd_ms += ms;
      p.fwd_flops += r.flops;
    }
  }
  std::sort(iv.begin(), iv.end());
  double busy = 0.0, cs = 0.0, ce = -1e300;
  for (const auto& v : iv) {
    if (v.first > ce) {
      if (ce > cs) busy += ce - cs;
      cs = v.first;
      ce = v.second;
    } else {
      ce = std::max(ce, v.second);
    }
  }
  if (!iv.empty() && ce > cs) busy += ce - cs;
  p.gemm_busy_ms = busy;
  c->recs.clear();
  c->evnext = 0;
  *out = p;
  return cuda_check(c, "profile");
}

int mebp_profile_kernels(const mebp_ctx* c, mebp_kernel_stat* out, int max, int* n) {
  if (!c || (!out && max > 0) || !n) return MEBP_ERR_INVALID_ARG;
  const int k = static_cast<int>(c->kstats.size());
  for (int i = 0; i < k && i < max; ++i) out[i] = c->kstats[i];
  *n = k;
  return MEBP_OK;
}

int mebp_compress_weights(mebp_ctx* c, const float* W, int64_t rows, int64_t cols, int group, uint8_t* qpack,
                          uint16_t* scales, void* stream) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  if (!W || !qpack || !scales) return fail(c, MEBP_ERR_INVALID_ARG, "NULL pointer");
  if (group != 64) return fail(c, MEBP_ERR_UNSUPPORTED, "group must be 64");
  if (rows <= 0 || cols <= 0 || cols % 64) return fail(c, MEBP_ERR_INVALID_ARG, "cols must be a positive multiple of 64");
  if (reinterpret_cast<uintptr_t>(W) & 7) return fail(c, MEBP_ERR_INVALID_ARG, "W must be 8-byte aligned");
  pdl_entry();
  launch_compress(W, rows, cols, qpack, scales, S(stream));
  return cuda_check(c, "compress");
}

int mebp_decode_weights(mebp_ctx* c, const mebp_packed* w, uint16_t* out, void* stream) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  if (!w || !w->qpack || !w->scales || !out) return fail(c, MEBP_ERR_INVALID_ARG, "NULL pointer");
  if (w->rows <= 0 || w->cols <= 0 || w->cols % 64) return fail(c, MEBP_ERR_INVALID_ARG, "bad shape");
  if (!aligned16(w->qpack) || !aligned16(out)) return fail(c, MEBP_ERR_INVALID_ARG, "pointers must be 16-byte aligned");
  pdl_entry();
  launch_decode(w->qpack, w->scales, w->rows, w->cols, out, S(stream));
  return cuda_check(c, "decode");
}

int mebp_embed(mebp_ctx* c, const mebp_packed* E, const int32_t* ids, int64_t n, float* x0, void* stream) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  if (!E || !E->qpack || !E->scales || !ids || !x0) return fail(c, MEBP_ERR_INVALID_ARG, "NULL pointer");
  if (E->cols % 64 || E->rows <= 0) return fail(c, MEBP_ERR_INVALID_ARG, "bad embedding shape");
  if (!aligned16(x0) || (reinterpret_cast<uintptr_t>(E->qpack) & 3))
    return fail(c, MEBP_ERR_INVALID_ARG, "misaligned pointer");
  if (n <= 0) return MEBP_OK;
  pdl_entry();
  launch_embed(E->qpack, E->scales, E->rows, E->cols, ids, n, x0, c->d_err, embed_scale(c), S(stream));
  return cuda_check(c, "embed");
}

// One standalone LoRA linear (uses stream-ordered temporaries for the fp16 shadows).
static int linear_common(mebp_ctx* c, bool dx_mode, const uint16_t* X, int64_t M, const mebp_packed* W,
                         const float* A, const float* Bm, int r, float s, const float* R, float* y32, uint16_t* y16,
                         cudaStream_t st) {
  if (!W || !W->qpack || !W->scales || !X) return fail(c, MEBP_ERR_INVALID_ARG, "NULL pointer");
  const int64_t N = W->rows, K = W->cols;
  if (N % 64 || K % 64 || N <= 0 || K <= 0) return fail(c, MEBP_ERR_INVALID_ARG, "W dims must be multiples of 64");
  // TMA reads X and the weights; the epilogue stores y and reads R as 16-byte vectors
  if (!aligned16(X) || !aligned16(W->qpack) || !aligned16(W->scales) || !aligned16(y32) || !aligned16(y16) ||
      !aligned16(R))
    return fail(c, MEBP_ERR_INVALID_ARG, "pointers must be 16-byte aligned");
  if ((A == nullptr) != (Bm == nullptr)) return fail(c, MEBP_ERR_INVALID_ARG, "A and B must both be set or both NULL");
  if (A && (r <= 0 || r > 32 || r % 8)) return fail(c, MEBP_ERR_UNSUPPORTED, "rank must be 8, 16, 24 or 32");
  if (M <= 0) return MEBP_OK;
  const int kxp = A ? (r + 15) / 16 * 16 : 0;
  pdl_entry();
  uint16_t *Ac = nullptr, *Bc = nullptr, *Btc = nullptr, *u = nullptr;
  if (A) {
    const size_t bytes = (static_cast<size_t>(kxp) * K + 2 * static_cast<size_t>(N) * kxp + M * kxp) * 2;
    void* base = nullptr;
    if (cudaMallocAsync(&base, bytes, st) != cudaSuccess) {
      cudaGetLastError();
      return fail(c, MEBP_ERR_OOM, "temporary allocation failed");
    }
    Ac = static_cast<uint16_t*>(base);
    Bc = Ac + static_cast<size_t>(kxp) * K;
    Btc = Bc + static_cast<size_t>(N) * kxp;
    u = Btc + static_cast<size_t>(N) * kxp;
    const float* As[1] = {A};
    const float* Bs[1] = {Bm};
    const int ro[1] = {0}, no[1] = {0};
    const int nl[1] = {static_cast<int>(N)};
    launch_lora_shadow(As, Bs, 1, ro, no, nl, r, static_cast<int>(K), static_cast<int>(N), kxp, Ac, Bc, Btc, st);
  }
  GemmArgs g;
  if (!dx_mode) {
    g = gemm_fwd(X, K, M, *W, static_cast<int>(N), static_cast<int>(K));
    if (A) {
      launch_skinny_gemm(X, K, M, K, Ac, K, r, s, u, kxp, st, c->d_err);
      g.Ax = u; g.ldax = kxp; g.kx = kxp; g.Bx = Bc; g.ldbx = kxp;
    }
    if (y32) {
      g.epi = EPI_F32; g.C = y32; g.ldc = N; g.R = R; g.ldr = N;
    } else {
      g.epi = EPI_F16; g.C = y16; g.ldc = N;
    }
  } else {
    g = gemm_dx(X, N, M, *W);
    if (A) {
      launch_skinny_gemm(X, N, M, N, Btc, N, r, s, u, kxp, st, c->d_err);
      g.Ax = u; g.ldax = kxp; g.kx = kxp; g.Bx = Ac; g.ldbx = K;
    }
    g.epi = EPI_F32; g.C = y32; g.ldc = K; g.R = R; g.ldr = K;
  }
  int rc = run_gemm(c, g, st, dx_mode ? "linear dX" : "linear forward");
  if (A) cudaFreeAsync(Ac, st);
  if (rc) return rc;
  return cuda_check(c, "linear");
}

int mebp_linear_fwd(mebp_ctx* c, const uint16_t* X, int64_t M, const mebp_packed* W, const float* A, const float* B,
                    int r, float s, const float* R, float* y_f32, uint16_t* y_f16, void* stream) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  if (!y_f32 && !y_f16) return fail(c, MEBP_ERR_INVALID_ARG, "no output");
  return linear_common(c, false, X, M, W, A, B, r, s, R, y_f32, y_f16, S(stream));
}

int mebp_linear_dx(mebp_ctx* c, const uint16_t* dY, int64_t M, const mebp_packed* W, const float* A, const float* B,
                   int r, float s, const float* R, float* dx, void* stream) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  if (!dx) return fail(c, MEBP_ERR_INVALID_ARG, "no output");
  return linear_common(c, true, dY, M, W, A, B, r, s, R, dx, nullptr, S(stream));
}

int mebp_block_recompute_fwd(mebp_ctx* c, int layer, const mebp_block_weights* w, const mebp_lora* lora,
                             const float* x, float* y, int B, int Sq, int save_for_bwd, void* stream) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  int rc;
  if ((rc = check_tokens(c, B, Sq)) || (rc = check_block_ptrs(c, w)) || (rc = check_lora(c, lora))) return rc;
  if (!x || !y || !aligned16(x) || !aligned16(y)) return fail(c, MEBP_ERR_INVALID_ARG, "x / y must be 16-byte aligned");
  if (x == y) return fail(c, MEBP_ERR_INVALID_ARG, "x and y must not alias");
  pdl_entry();
  // without save_for_bwd gate and up need not be kept (the gate|up GEMM may store m alone)
  rc = block_forward(c, 0, layer, w, lora, x, y, B, Sq, true, S(stream), nullptr, save_for_bwd != 0);
  if (!save_for_bwd) c->act[0].layer = -1;
  return rc;
}

int mebp_block_bwd(mebp_ctx* c, int layer, const mebp_block_weights* w, const mebp_lora* lora, const float* x,
                   const float* dy, float* dx, const mebp_lora_grads* grads, int B, int Sq, int accumulate,
                   void* stream) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  int rc;
  if ((rc = check_tokens(c, B, Sq)) || (rc = check_block_ptrs(c, w)) || (rc = check_lora(c, lora))) return rc;
  if (!x || !dy || !aligned16(x) || !aligned16(dy) || (dx && !aligned16(dx)))
    return fail(c, MEBP_ERR_INVALID_ARG, "x / dy / dx must be 16-byte aligned");
  cudaStream_t st = S(stream);
  const int64_t n = static_cast<int64_t>(B) * Sq * c->D;
  // working scale for this call: sigma = 2^-floor(log2(max|dy|)); the outputs are scaled back
  pdl_entry();
  launch_grad_scale(dy, n, c->scal + 4, st);
  launch_scale_cast(dy, n, c->scal + 4, c->gbuf[0], c->dy_h[1], st);
  return block_backward(c, 0, 0, layer, w, lora, x, c->gbuf[0], c->dy_h[1], dx, nullptr, grads, B, Sq, accumulate != 0,
                        c->scal + 5, c->scal + 5, st);
}

int mebp_lmhead_ce_fwd_bwd(mebp_ctx* c, const mebp_packed* E, const float* gf, const float* h, const int32_t* targets,
                           int64_t T, float* loss, float* dh, float* token_loss, void* stream) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  if (c->V <= 0) return fail(c, MEBP_ERR_INVALID_ARG, "context has no vocabulary");
  int rc;
  if ((rc = check_packed(c, E, c->V, c->D, "embedding"))) return rc;
  if (!gf || !h || !targets || !loss || !dh) return fail(c, MEBP_ERR_INVALID_ARG, "NULL pointer");
  if (T <= 0 || T > c->Tmax) return fail(c, MEBP_ERR_INVALID_ARG, "n_tokens out of range");
  if (!aligned16(h) || !aligned16(dh)) return fail(c, MEBP_ERR_INVALID_ARG, "h / dh must be 16-byte aligned");
  pdl_entry();
  return lmhead(c, E, gf, h, targets, T, loss, dh, nullptr, token_loss, true, S(stream));
}

static int lora_step_body(mebp_ctx* c, const mebp_model_weights* model, const mebp_lora* lora, const int32_t* ids,
                          int B, int Sq, float* loss, const mebp_lora_grads* grads, int accumulate, void* stream) {
  int rc;
  cudaStream_t st = S(stream);
  const int64_t T = static_cast<int64_t>(B) * Sq, D = c->D;
  const int L = c->L;
  const bool spill = c->cfg.spill_ckpts != 0;
  pdl_entry();
  launch_k(targets_kernel, static_cast<unsigned>((T + 255) / 256), 256, 0, st, ids, B, Sq, c->targets);
  // fp16 shadows of every block's LoRA masters, one launch per fused linear
  for (int li = 0; li < 4; ++li) {
    const Lin& l = c->lin[li];
    if (!l.kx) continue;
    std::vector<const float*> As(3 * static_cast<size_t>(L), nullptr), Bs(3 * static_cast<size_t>(L), nullptr);
    for (int i = 0; i < L; ++i)
      for (int t = 0; t < l.nt; ++t) {
        As[3 * i + t] = lora[i].A[l.tgt[t]];
        Bs[3 * i + t] = lora[i].B[l.tgt[t]];
      }
    const Shadow& s0 = c->layer_sh[0];
    launch_lora_shadow_layers(L, As.data(), Bs.data(), l.nt, l.ro, l.no, l.nl, c->r, l.K, l.N, l.kxp, s0.A_cat[li],
                              s0.B_cat[li], s0.Bt_cat[li], static_cast<int64_t>(l.kxp) * l.K,
                              static_cast<int64_t>(l.N) * l.kxp, st);
  }
  // Checkpoint placement (Algorithm 1's ckpts_storage): HBM slot i, or, when spilling, a ring
  // of kCkptSlots device slots whose contents are copied to / from pinned host memory on a
  // side stream (the stand-in for memory-mapped checkpoints).
  if (L + 1 > 4096) return fail(c, MEBP_ERR_UNSUPPORTED, "too many layers");
  std::vector<int> slot_of(L + 1, -1);
  int holds[kCkptSlots];
  for (int k = 0; k < kCkptSlots; ++k) holds[k] = -1;
  auto dev_ckpt = [&](int slot) { return c->ckpt + static_cast<int64_t>(slot) * c->Tmax * D; };
  auto host_ckpt = [&](int i) { return c->h_ckpt + static_cast<int64_t>(i) * c->Tmax * D; };
  // Events recorded during THIS step only (a captured step must not wait on earlier events;
  // work of earlier steps is already ordered before this one on the stream).
  bool freed_rec[kCkptSlots] = {false, false, false};
  // A free slot, else the one holding the lowest-index checkpoint other than `avoid` (every
  // checkpoint below L also lives on the host, so evicting it loses nothing).
  auto take_slot = [&](int i, int avoid) {
    int sl = -1;
    for (int k = 0; k < kCkptSlots && sl < 0; ++k)
      if (holds[k] < 0) sl = k;
    if (sl < 0)
      for (int k = 0; k < kCkptSlots; ++k)
        if (holds[k] != avoid && (sl < 0 || holds[k] < holds[sl])) sl = k;
    if (holds[sl] >= 0) slot_of[holds[sl]] = -1;
    holds[sl] = i;
    slot_of[i] = sl;
    return sl;
  };
  auto release = [&](int i) {
    if (slot_of[i] >= 0) holds[slot_of[i]] = -1;
    slot_of[i] = -1;
  };
  // device -> host copy of checkpoint i once the main stream has produced it
  auto spill_out = [&](int i) {
    const int sl = slot_of[i];
    cudaEventRecord(c->slot_ready[sl], st);
    cudaStreamWaitEvent(c->copy_stream, c->slot_ready[sl], 0);
    cudaMemcpyAsync(host_ckpt(i), dev_ckpt(sl), T * D * sizeof(float), cudaMemcpyDeviceToHost, c->copy_stream);
    cudaEventRecord(c->slot_free[sl], c->copy_stream);
    freed_rec[sl] = true;
  };
  auto wait_free = [&](int sl) {
    if (freed_rec[sl]) cudaStreamWaitEvent(st, c->slot_free[sl], 0);
  };
  // host -> device copy of checkpoint i into a slot the main stream no longer reads
  auto fetch_in = [&](int i, int avoid) {
    const int sl = take_slot(i, avoid);
    cudaEventRecord(c->slot_ready[sl], st);
    cudaStreamWaitEvent(c->copy_stream, c->slot_ready[sl], 0);
    cudaMemcpyAsync(dev_ckpt(sl), host_ckpt(i), T * D * sizeof(float), cudaMemcpyHostToDevice, c->copy_stream);
    cudaEventRecord(c->slot_free[sl], c->copy_stream);
    freed_rec[sl] = true;
  };

  float* x0 = dev_ckpt(0);
  if (spill) {
    const int sl = take_slot(0, -1);
    wait_free(sl);
    x0 = dev_ckpt(sl);
  }
  char rname[32];
  nvtxRangePushA("emb");
  KP(c, KK_EMBED, T * D * (0.5 + 1.0 / 16.0 + 4.0) + 4.0 * T, 0, st, [&] {
    launch_embed(model->embed.qpack, model->embed.scales, c->V, D, ids, T, x0, c->d_err, embed_scale(c), st);
  });
  nvtxRangePop();
  if (spill) spill_out(0);
  // ---- forward loop: store only block-boundary checkpoints
  for (int i = 0; i < L; ++i) {
    const float* xin = spill ? dev_ckpt(slot_of[i]) : dev_ckpt(i);
    float* yout = dev_ckpt(i + 1);
    if (spill) {
      const int sl = take_slot(i + 1, i);
      wait_free(sl);  // its previous contents reached the host
      yout = dev_ckpt(sl);
    }
    std::snprintf(rname, sizeof(rname), "f_%d", i);
    nvtxRangePushA(rname);
    // only the last nsets blocks' intermediates survive to their backward; the others are recomputed
    rc = block_forward(c, i % c->nsets, i, &model->blocks[i], &lora[i], xin, yout, B, Sq, true, st, &c->layer_sh[i],
                       i >= L - c->nsets);
    nvtxRangePop();
    if (rc) return rc;
    if (spill && i + 1 < L) spill_out(i + 1);
  }
  // ---- loss subgraph: final norm + LM head + CE
  const float* hL = spill ? dev_ckpt(slot_of[L]) : dev_ckpt(L);
  int cur = 0;
  nvtxRangePushA("lm");
  rc = lmhead(c, &model->embed, model->final_norm, hL, c->targets, T, loss, c->gbuf[cur], c->dy_h[cur], nullptr, false,
              st);
  nvtxRangePop();
  if (rc) return rc;
  if (spill) release(L);
  // ---- backward loop in reverse order: recompute block i from ckpt_i, apply its VJP.  With two
  // intermediate sets (no spilling) three streams share the work: the recompute of block i-1
  // (recompute stream) and the LoRA-gradient reductions of block i+1 (gradient stream) run while
  // the main stream computes the input gradients of block i.  Buffers alternate by block parity
  // (fp16 upstream gradients over three blocks), so a set is rewritten only after the stream
  // that reads it has finished with it.  Block L-1's intermediates are still in place from the
  // forward loop, and so are block L-2's.
  const bool overlap = c->nsets == 2 && !spill && L > 1;
  auto dyh = [&](int i) { return c->dy_h[(L - 1 - i) % 3]; };  // fp16 dE/dy of block i (overlap)
  for (int i = L - 1; i >= 0; --i) {
    if (spill) {
      if (slot_of[i] < 0) {
        fetch_in(i, i + 1);
        wait_free(slot_of[i]);
      }
      if (i > 0 && slot_of[i - 1] < 0) fetch_in(i - 1, i);  // prefetch while block i runs
    }
    const float* xin = spill ? dev_ckpt(slot_of[i]) : dev_ckpt(i);
    const int set = i % c->nsets;
    const int nxt = cur ^ 1;
    std::snprintf(rname, sizeof(rname), "b_%d", i);
    nvtxRangePushA(rname);
    struct PopOnExit {
      ~PopOnExit() { nvtxRangePop(); }
    } pop_on_exit;
    if (!overlap) {
      if ((rc = block_backward(c, set, 0, i, &model->blocks[i], &lora[i], xin, c->gbuf[cur], c->dy_h[cur],
                               i > 0 ? c->gbuf[nxt] : nullptr, i > 0 ? c->dy_h[nxt] : nullptr, &grads[i], B, Sq,
                               accumulate != 0, c->scal + 1, nullptr, st, &c->layer_sh[i])))
        return rc;
    } else {
      if (i > 0) {  // recompute block i-1 into the other set once its readers are done with it
        const int ps = (i - 1) % 2;
        cudaEventRecord(c->ev_main, st);  // the backward of block i+1 has been issued
        cudaStreamWaitEvent(c->fstream, c->ev_main, 0);
        if (i + 1 < L) cudaStreamWaitEvent(c->fstream, c->ev_grad[ps], 0);  // reductions of block i+1
        const Acts& P = c->act[ps];
        if (!(P.layer == i - 1 && P.x == dev_ckpt(i - 1) && P.T == T) &&
            (rc = block_forward(c, ps, i - 1, &model->blocks[i - 1], &lora[i - 1], dev_ckpt(i - 1), nullptr, B, Sq,
                                false, c->fstream, &c->layer_sh[i - 1])))
          return rc;
        cudaEventRecord(c->ev_fwd[ps], c->fstream);
      }
      if (i < L - 1) cudaStreamWaitEvent(st, c->ev_fwd[set], 0);
      if (i + 2 < L) cudaStreamWaitEvent(st, c->ev_grad[set], 0);  // reductions of block i+2
      if ((rc = block_backward(c, set, set, i, &model->blocks[i], &lora[i], xin, c->gbuf[cur], dyh(i),
                               i > 0 ? c->gbuf[nxt] : nullptr, i > 0 ? dyh(i - 1) : nullptr, nullptr, B, Sq,
                               accumulate != 0, c->scal + 1, nullptr, st)))
        return rc;
      cudaEventRecord(c->ev_bwd, st);
      cudaStreamWaitEvent(c->gstream, c->ev_bwd, 0);
      if ((rc = block_lora_grads(c, set, set, dyh(i), T, &grads[i], accumulate != 0, c->scal + 1, c->gstream)))
        return rc;
      cudaEventRecord(c->ev_grad[set], c->gstream);
    }
    if (spill) {
      release(i);  // the checkpoint is removed once its backward has consumed it
      if (i > 0) wait_free(slot_of[i - 1]);
    }
    cur = nxt;
  }
  if (overlap) {  // join the gradient stream
    cudaStreamWaitEvent(st, c->ev_grad[0], 0);
    cudaStreamWaitEvent(st, c->ev_grad[1], 0);
  }
  if (spill) {  // every copy of this step is complete when the stream reaches this point
    cudaEventRecord(c->copy_join, c->copy_stream);
    cudaStreamWaitEvent(st, c->copy_join, 0);
  }
  for (int k = 0; k < c->nsets; ++k) c->act[k].layer = -1;
  return cuda_check(c, "lora step");
}

int mebp_adamw_step(mebp_ctx* c, float* params, const float* grads, float* m, float* v, int64_t n,
                    const mebp_adamw_cfg* cfg, int64_t step, void* stream) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  if (!cfg || n < 0 || step < 1) return fail(c, MEBP_ERR_INVALID_ARG, "bad AdamW arguments");
  if (n == 0) return MEBP_OK;
  if (!params || !grads || !m || !v) return fail(c, MEBP_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(params) || !aligned16(grads) || !aligned16(m) || !aligned16(v))
    return fail(c, MEBP_ERR_INVALID_ARG, "AdamW buffers must be 16-byte aligned");
  if (!(cfg->lr >= 0.0f) || !(cfg->beta1 >= 0.0f && cfg->beta1 < 1.0f) || !(cfg->beta2 >= 0.0f && cfg->beta2 < 1.0f) ||
      !(cfg->eps > 0.0f) || !(cfg->weight_decay >= 0.0f))
    return fail(c, MEBP_ERR_INVALID_ARG, "bad AdamW hyper-parameters");
  const double bc1 = 1.0 / (1.0 - std::pow(static_cast<double>(cfg->beta1), static_cast<double>(step)));
  const double bc2 = 1.0 / (1.0 - std::pow(static_cast<double>(cfg->beta2), static_cast<double>(step)));
  pdl_entry();
  launch_adamw(params, grads, m, v, n, cfg->lr, cfg->beta1, cfg->beta2, cfg->eps, cfg->weight_decay, cfg->grad_scale,
               bc1, bc2, S(stream));
  return cuda_check(c, "AdamW");
}

int mebp_lora_step(mebp_ctx* c, const mebp_model_weights* model, const mebp_lora* lora, const int32_t* ids, int B,
                   int Sq, float* loss, const mebp_lora_grads* grads, int accumulate, void* stream) {
  if (!c) return MEBP_ERR_INVALID_ARG;
  int rc;
  if (!model || !model->blocks || !lora || !ids || !loss) return fail(c, MEBP_ERR_INVALID_ARG, "NULL pointer");
  if (c->V <= 0) return fail(c, MEBP_ERR_INVALID_ARG, "context has no vocabulary");
  if ((rc = check_tokens(c, B, Sq))) return rc;
  if ((rc = check_packed(c, &model->embed, c->V, c->D, "embedding"))) return rc;
  if (!model->final_norm) return fail(c, MEBP_ERR_INVALID_ARG, "NULL final norm");
  for (int i = 0; i < c->L; ++i)
    if ((rc = check_block_ptrs(c, &model->blocks[i])) || (rc = check_lora(c, &lora[i]))) return rc;
  cudaStream_t st = S(stream);
  // CUDA-graph replay: the first call with a given set of pointers runs eagerly, the second
  // captures the identical launch sequence, later calls replay it (values behind the
  // pointers may change freely between calls).
  std::vector<uintptr_t> key;
  key.reserve(16 + static_cast<size_t>(c->L) * 40);
  auto K = [&](const void* p) { key.push_back(reinterpret_cast<uintptr_t>(p)); };
  K(stream); K(ids); K(loss); K(model->final_norm); K(model->embed.qpack); K(model->embed.scales);
  key.push_back(static_cast<uintptr_t>(B)); key.push_back(static_cast<uintptr_t>(Sq));
  key.push_back(static_cast<uintptr_t>(accumulate != 0));
  for (int i = 0; i < c->L; ++i) {
    const mebp_block_weights& w = model->blocks[i];
    K(w.qkv.qpack); K(w.qkv.scales); K(w.o.qpack); K(w.o.scales); K(w.gate_up.qpack); K(w.gate_up.scales);
    K(w.down.qpack); K(w.down.scales); K(w.norm1); K(w.norm2);
    K(w.q_norm); K(w.k_norm); K(w.post_attn_norm); K(w.post_ffn_norm);
    for (int t = 0; t < MEBP_N_TARGETS; ++t) {
      K(lora[i].A[t]); K(lora[i].B[t]);
      K(grads ? grads[i].dA[t] : nullptr); K(grads ? grads[i].dB[t] : nullptr);
    }
  }
  const bool can_graph = c->graphs && stream != nullptr && !c->prof;
  if (key != c->graph_key) {
    if (c->graph_exec) cudaGraphExecDestroy(c->graph_exec);
    c->graph_exec = nullptr;
    c->graph_key = key;
    c->graph_eager_runs = 0;
  }
  if (can_graph && c->graph_exec) {
    if (cudaGraphLaunch(c->graph_exec, st) != cudaSuccess) return cuda_check(c, "graph launch");
    g_launches.fetch_add(c->graph_launches);
    return MEBP_OK;
  }
  if (can_graph && c->graph_eager_runs >= 1) {
    const long long n0 = g_launches.load();
    if (cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal) != cudaSuccess)
      return cuda_check(c, "begin capture");
    rc = lora_step_body(c, model, lora, ids, B, Sq, loss, grads, accumulate, stream);
    cudaGraph_t graph = nullptr;
    const cudaError_t ce = cudaStreamEndCapture(st, &graph);
    if (rc != MEBP_OK || ce != cudaSuccess) {
      if (graph) cudaGraphDestroy(graph);
      cudaGetLastError();
      return rc != MEBP_OK ? rc : fail(c, MEBP_ERR_CUDA, "stream capture of the step failed");
    }
    const cudaError_t ie = cudaGraphInstantiate(&c->graph_exec, graph, 0);
    cudaGraphDestroy(graph);
    if (ie != cudaSuccess) {
      c->graph_exec = nullptr;
      return cuda_check(c, "graph instantiate");
    }
    c->graph_launches = g_launches.load() - n0;  // kernels in the graph (counted once per replay)
    if (cudaGraphLaunch(c->graph_exec, st) != cudaSuccess) return cuda_check(c, "graph launch");
    return MEBP_OK;
  }
  rc = lora_step_body(c, model, lora, ids, B, Sq, loss, grads, accumulate, stream);
  if (rc == MEBP_OK) c->graph_eager_runs++;
  return rc;
}


}  // extern "C"
