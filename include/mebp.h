/*
 * mebp.h — C ABI of the GB300 (sm_103a) implementation of MeBP's training step
 * (memory-efficient backpropagation for LoRA fine-tuning over 4-bit-compressed
 * base weights; arxiv 2510.03425).
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Pointers are DEVICE pointers owned by the caller unless the name says
 *    "host".  The library never frees caller memory.
 *  - Calls are asynchronous and ordered on `stream` (a cudaStream_t passed as
 *    void*; NULL = the legacy default stream).  Device-side failures (a
 *    bounded wait that expired, a bad token id) are recorded in the context's
 *    device error word and reported by mebp_sync().
 *  - A context's workspace (intermediates, split partials, LM-head buffers) is
 *    shared by its calls: issue the calls of one context on one stream, or
 *    order the streams they use; calls that overlap on the GPU race on it.
 *  - Every call returns an int status (MEBP_OK on success).  No exception or
 *    abort crosses the ABI; mebp_last_error() gives a message.
 *  - Dense activations are row-major [tokens, features]; token t = b*S + s.
 *  - Base weights are frozen and stored compressed (mebp_packed).  LoRA
 *    weights and gradients are fp32 masters in PyTorch Linear layout:
 *    A [r, K_in], B [N_out, r]; the layer computes
 *        Y = X deq(W)^T + s (X A^T) B^T,  s = lora_scale (alpha / r).
 *  - The LoRA targets of a block are indexed MEBP_T_Q .. MEBP_T_DOWN.
 */
#ifndef MEBP_H_
#define MEBP_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes --------------------------------------------------------------------------- */
enum {
  MEBP_OK = 0,
  MEBP_ERR_INVALID_ARG = 1,  /* bad shape, NULL pointer, misalignment, K not a multiple of 64   */
  MEBP_ERR_CUDA = 2,         /* a CUDA runtime call failed                                       */
  MEBP_ERR_OOM = 3,          /* device or pinned-host allocation failed                          */
  MEBP_ERR_TIMEOUT = 4,      /* a device-side bounded wait expired (kernel returned early)       */
  MEBP_ERR_UNSUPPORTED = 5,  /* configuration outside what the kernels implement                 */
  MEBP_ERR_DEVICE = 6,       /* a kernel flagged bad input (e.g. token id out of range)          */
  MEBP_ERR_SCRATCH = 7,      /* mebp_linear_fwd_noalloc: the request needs more than the fixed
                                scratch array (MEBP_NOALLOC_SCRATCH_BYTES) holds                  */
  MEBP_ERR_NONFINITE = 8     /* an fp16 intermediate (a GEMM output stored as fp16, the gated-MLP
                                product or its gradient) overflowed the fp16 range (|x| > 65504)
                                or was NaN; reported by mebp_sync()                                */
};

/* LoRA target index (bit i of mebp_model_cfg.lora_targets). */
enum { MEBP_T_Q = 0, MEBP_T_K, MEBP_T_V, MEBP_T_O, MEBP_T_GATE, MEBP_T_UP, MEBP_T_DOWN, MEBP_N_TARGETS };

enum { MEBP_ACT_SILU = 0, MEBP_ACT_GELU_TANH = 1 };

/* ---- model configuration -------------------------------------------------------------------- */
typedef struct {
  int32_t hidden;        /* D                                                                   */
  int32_t n_heads;       /* H   (query heads)                                                   */
  int32_t n_kv_heads;    /* KV  (key/value heads; H % KV == 0, H / KV <= 8)                     */
  int32_t head_dim;      /* hd  in {64, 128, 256}                                               */
  int32_t intermediate;  /* I   (gated-MLP width)                                               */
  int32_t vocab;         /* V   (tied embedding / LM head rows; 0 = no LM head)                 */
  int32_t n_layers;      /* L                                                                   */
  int32_t act;           /* MEBP_ACT_*                                                          */
  float rope_theta;      /* RoPE base (half-split rotation)                                     */
  float rms_eps;         /* RMSNorm epsilon                                                     */
  int32_t lora_rank;     /* r (1..32)                                                           */
  float lora_scale;      /* s = alpha / r                                                       */
  uint32_t lora_targets; /* bit MEBP_T_* set => that linear carries LoRA                        */
  int32_t max_tokens;    /* workspace sizing: every call has batch*seq <= max_tokens            */
  int32_t max_seq;       /* longest sequence (RoPE table size)                                  */
  int32_t spill_ckpts;   /* 1: mebp_lora_step keeps block checkpoints in pinned host memory     */
  int32_t vocab_chunk;   /* LM-head vocabulary chunk (multiple of 256); 0 = library default     */
  /* Gemma3 block options (Section 4 fine-tunes Gemma3 models; all zero = the plain pre-norm block):
   *  gemma_norms != 0: per-head RMSNorm of q and k (gains q_norm / k_norm, over head_dim) before
   *    RoPE; RMSNorm of the attention output (post_attn_norm) and of the MLP output
   *    (post_ffn_norm) before each residual add; input embeddings multiplied by sqrt(hidden).
   *  sliding_window = W > 0: layer l is local iff (l + 1) % global_every != 0; a local layer's
   *    query at position i attends to keys i - W + 1 .. i and rotates with base rope_theta_local
   *    (global layers: causal, rope_theta).  global_every >= 1 when W > 0. */
  int32_t gemma_norms;
  int32_t sliding_window;
  int32_t global_every;
  float rope_theta_local;
  /* min_memory != 0: one set of block intermediates (Section 3, "Runtime implementation": only
   * one subgraph's intermediates are held at a time).  0: a second set lets mebp_lora_step run the
   * recompute of block i-1 beside the backward of block i (same results, more memory). */
  int32_t min_memory;
} mebp_model_cfg;

/* ---- compressed base weight (Section 3, "Base model weights compression") -------------------
 * A dense W [rows, cols] (cols % 64 == 0) quantised per group of 64 consecutive
 * columns of a row: s = fp16(min(amax/7, 65504)), q = clamp(rint(w/s), -7, 7),
 * stored as offset-binary nibbles u = q + 8:
 *   qpack  uint8 [rows, cols/2]: every run of 8 columns is one little-endian 32-bit word with
 *          column 8w+2j in bits 4j..4j+3 and column 8w+2j+1 in bits 16+4j..16+4j+3 (even
 *          columns in the low half-word, odd ones in the high half-word);
 *   scales fp16 bits [cols/64, rows] (group-major: the scales of one column group are
 *          contiguous over rows).
 * deq(W)[n, k] = (u - 8) * scales[k/64, n]; the tensor cores consume fp16_rne(deq) (IEEE half).
 * Both pointers must be 16-byte aligned. */
typedef struct {
  const uint8_t* qpack;
  const uint16_t* scales;
  int64_t rows;
  int64_t cols;
} mebp_packed;

/* Base weights of one pre-norm decoder block.  Fused matrices stack their parts by rows:
 *   qkv     rows = (H + 2 KV) * hd (q rows, then k rows, then v rows), cols = D
 *   o       rows = D,  cols = H * hd
 *   gate_up rows = 2 I (gate rows, then up rows),                      cols = D
 *   down    rows = D,  cols = I
 * norm1 / norm2: fp32 [D] RMSNorm gains (before attention / before the MLP).
 * With cfg.gemma_norms also (else ignored, may be NULL): q_norm / k_norm fp32 [hd], post_attn_norm
 * / post_ffn_norm fp32 [D].  Every gain pointer 16-byte aligned. */
typedef struct {
  mebp_packed qkv, o, gate_up, down;
  const float* norm1;
  const float* norm2;
  const float* q_norm;
  const float* k_norm;
  const float* post_attn_norm;
  const float* post_ffn_norm;
} mebp_block_weights;

/* LoRA masters of one block (fp32, device).  A[t] = [r, K_in], B[t] = [N_out, r];
 * NULL for a target whose bit is clear in lora_targets. */
typedef struct {
  const float* A[MEBP_N_TARGETS];
  const float* B[MEBP_N_TARGETS];
} mebp_lora;

/* LoRA gradients of one block, same shapes as mebp_lora (NULL for untargeted linears). */
typedef struct {
  float* dA[MEBP_N_TARGETS];
  float* dB[MEBP_N_TARGETS];
} mebp_lora_grads;

/* Whole model: tied embedding/LM head E [V, D], final RMSNorm gain [D], and a HOST array of
 * n_layers block descriptors (the descriptors hold device pointers). */
typedef struct {
  mebp_packed embed;
  const float* final_norm;
  const mebp_block_weights* blocks;
} mebp_model_weights;

typedef struct mebp_ctx mebp_ctx;

/* ---- context ---------------------------------------------------------------------------------
 * Allocates the device workspace (one block's intermediates, LM-head chunk buffers,
 * checkpoint storage in HBM or pinned host) sized from cfg.  `device` is the CUDA
 * ordinal the context and every later call use.  Returns MEBP_ERR_OOM if an
 * allocation fails, MEBP_ERR_UNSUPPORTED for shapes the kernels do not implement. */
int mebp_ctx_create(const mebp_model_cfg* cfg, int device, mebp_ctx** out);
void mebp_ctx_destroy(mebp_ctx* ctx);
/* Message for the last failing call on this context (never NULL; owned by ctx). */
const char* mebp_last_error(const mebp_ctx* ctx);
/* Synchronises `stream`, then reads and clears the device error word: returns
 * MEBP_ERR_TIMEOUT / MEBP_ERR_DEVICE if a kernel flagged one since the last sync. */
int mebp_sync(mebp_ctx* ctx, void* stream);
/* Workspace bytes the context holds on the device (allocated at creation; no call allocates
 * more, so this is also the library's peak). */
int64_t mebp_workspace_bytes(const mebp_ctx* ctx);

/* The workspace by purpose (device bytes, except MEBP_WS_HOST_CKPT: pinned host bytes):
 *   MEBP_WS_CKPT        block-boundary checkpoints (L+1 slots, or a 3-slot ring when spilling)
 *   MEBP_WS_FWD_SETS    forward intermediates of one block, times the number of sets (*n_sets)
 *   MEBP_WS_BWD         backward working buffers of one block (gradients of the intermediates)
 *   MEBP_WS_ATTN_SPLIT  fp32 partials of the split attention backward (small grids)
 *   MEBP_WS_LMHEAD      LM-head + CE buffers (one vocabulary chunk of the CE gradient)
 *   MEBP_WS_LORA_SHADOW fp16 operand copies of the LoRA masters (every block)
 *   MEBP_WS_OTHER       RoPE tables, device scalars, error word, reduction scratch, the fp32
 *                       partials of fused GEMMs split over K through memory
 *   MEBP_WS_HOST_CKPT   pinned host checkpoints (spilling)
 * bytes has MEBP_WS_N entries; n_sets may be NULL. */
enum {
  MEBP_WS_CKPT = 0, MEBP_WS_FWD_SETS, MEBP_WS_BWD, MEBP_WS_ATTN_SPLIT, MEBP_WS_LMHEAD, MEBP_WS_LORA_SHADOW,
  MEBP_WS_OTHER, MEBP_WS_HOST_CKPT, MEBP_WS_N
};
int mebp_workspace_breakdown(const mebp_ctx* ctx, int64_t* bytes, int* n_sets);

/* ---- Section 3 "Base model weights compression": quantise W fp32 [rows, cols] (device)
 * into qpack / scales (layout above).  group must be 64.  Ties round to even. */
int mebp_compress_weights(mebp_ctx* ctx, const float* W, int64_t rows, int64_t cols, int group,
                          uint8_t* qpack, uint16_t* scales, void* stream);

/* Debug decode: out fp16 bits [rows, cols] = fp16_rne(q * s), produced by the same device
 * function that feeds the fused GEMM's shared-memory operand. */
int mebp_decode_weights(mebp_ctx* ctx, const mebp_packed* w, uint16_t* out_f16, void* stream);

/* Embedding gather + dequant: x0[t, :] = deq(E)[ids[t], :] (fp32 [n_tokens, D], exact), times
 * sqrt(D) with cfg.gemma_norms.
 * An id outside [0, V) writes zeros and sets MEBP_ERR_DEVICE. */
int mebp_embed(mebp_ctx* ctx, const mebp_packed* embed, const int32_t* ids, int64_t n_tokens,
               float* x0, void* stream);

/* ---- one LoRA linear with just-in-time dequantised base weight (Algorithm 1,
 * LazyLoadAndDecompressWeights, with the decompression fused into the GEMM mainloop).
 * mebp_linear_fwd:  Y [M, N] = X [M, K] deq(W)^T + s (X A^T) B^T  (+ R if R != NULL)
 *   X fp16 [M, K] (bits), W packed [N, K], A fp32 [r, K] / B fp32 [N, r] or both NULL,
 *   Y fp32 [M, N] when y_f32 != NULL else fp16 bits into y_f16.  R fp32 [M, N] may alias y_f32.
 *   X, the weight pointers, the outputs and R must be 16-byte aligned (MEBP_ERR_INVALID_ARG).
 * mebp_linear_dx:   dX [M, K] = dY [M, N] deq(W) + s (dY B) A  (+ R if R != NULL)
 *   dY fp16 [M, N] (bits), same W / A / B, dX fp32 [M, K].
 * Both use the tcgen05 fused dequant-GEMM kernels; r <= 32. */
int mebp_linear_fwd(mebp_ctx* ctx, const uint16_t* X, int64_t M, const mebp_packed* W,
                    const float* A, const float* B, int r, float s, const float* R,
                    float* y_f32, uint16_t* y_f16, void* stream);
int mebp_linear_dx(mebp_ctx* ctx, const uint16_t* dY, int64_t M, const mebp_packed* W,
                   const float* A, const float* B, int r, float s, const float* R,
                   float* dx, void* stream);

/* ---- mebp_linear_fwd without any device allocation (the paper has no counterpart; this is a
 * deployment convenience).  For callers that may not call cudaMalloc/cudaFree at the point where
 * the layer runs — e.g. a host program whose device memory belongs to an external pool, or code
 * that must keep the process's allocations fixed — and so cannot create a mebp_ctx either.
 * Same arguments and result as mebp_linear_fwd minus the context; the work runs on the device
 * that is current when called.  Its scratch (the fp16 LoRA shadows, the rank-r product and an
 * error word) lives in one static device array of MEBP_NOALLOC_SCRATCH_BYTES per GPU that loads
 * the library, kept until the process exits:
 *   - the first call in each CUDA context (the device's primary context, or one the caller made
 *     current) looks up that array's address (cudaGetSymbolAddress) and must happen before any
 *     stream capture in that context; after a device reset the next call looks it up again;
 *   - every call shares the array and leaves its contents behind: calls that can overlap on the
 *     GPU (different streams without ordering) race on it;
 *   - a request whose scratch (about 2 * (kx*K + 2*N*kx + M*kx) bytes, kx = r rounded up to 16;
 *     none without LoRA) exceeds the array returns MEBP_ERR_SCRATCH before doing anything;
 *   - device-side wait timeouts are not reported (there is no context to read them from): the
 *     output of a call whose bounded wait expired cannot be told apart from a good one;
 *   - X, W's pointers, y_f32 / y_f16 and R must be 16-byte aligned (MEBP_ERR_INVALID_ARG).
 * Allocates nothing: no cudaMalloc, cudaFree or allocating library call. */
#define MEBP_NOALLOC_SCRATCH_BYTES (8u << 20)
int mebp_linear_fwd_noalloc(const uint16_t* X, int64_t M, const mebp_packed* W, const float* A,
                            const float* B, int r, float s, const float* R, float* y_f32,
                            uint16_t* y_f16, void* stream);

/* ---- forward_i of Algorithm 1: y [T, D] = F(x [T, D]) for block `layer`, T = batch*seq.
 * save_for_bwd != 0 keeps the block's intermediates in the context workspace so that a
 * following mebp_block_bwd with the same layer and x skips the recompute.  x, y fp32. */
int mebp_block_recompute_fwd(mebp_ctx* ctx, int layer, const mebp_block_weights* w,
                             const mebp_lora* lora, const float* x, float* y, int batch, int seq,
                             int save_for_bwd, void* stream);

/* ---- backward_i of Algorithm 1 / B_i(x, dE/dy, w) of Section 3: recomputes block `layer`
 * from its input checkpoint x (unless intermediates were saved for exactly this layer and x),
 * then writes dx = dE/dx (fp32 [T, D]; may be NULL when not needed) and the LoRA gradients.
 * accumulate == 0 overwrites the gradients, 1 adds to them (gradient accumulation over
 * micro-batches).  dy fp32 [T, D]. */
int mebp_block_bwd(mebp_ctx* ctx, int layer, const mebp_block_weights* w, const mebp_lora* lora,
                   const float* x, const float* dy, float* dx, const mebp_lora_grads* grads,
                   int batch, int seq, int accumulate, void* stream);

/* ---- final RMSNorm + tied LM head + mean next-token cross-entropy, forward and backward,
 * over vocabulary chunks (full [T, V] logits are never stored).
 *   h fp32 [T, D]; targets int32 [T] with -1 = ignored; loss: device fp32 scalar (mean over
 *   valid targets); dh fp32 [T, D] = dloss/dh; token_loss fp32 [T] (lse - z_target, 0 when
 *   ignored) or NULL. */
int mebp_lmhead_ce_fwd_bwd(mebp_ctx* ctx, const mebp_packed* embed, const float* final_norm,
                           const float* h, const int32_t* targets, int64_t n_tokens, float* loss,
                           float* dh, float* token_loss, void* stream);

/* ---- Algorithm 1, Backpropagation(x): embed ids [batch, seq], forward loop storing only
 * block-boundary checkpoints (HBM, or pinned host when cfg.spill_ckpts), LM head + CE with
 * targets ids[b, s+1] (last position ignored), then the reverse loop of recompute + VJP.
 * lora / grads are HOST arrays of n_layers descriptors.  loss: device fp32 scalar.
 * On a non-NULL stream (and unless disabled with mebp_enable_graphs) the step is replayed as
 * a CUDA graph: the first call with a given set of pointers, sizes, stream and accumulate
 * flag runs eagerly, the second captures the launch sequence, later ones replay it.  Data
 * behind the pointers may change between calls; any pointer change re-captures. */
int mebp_lora_step(mebp_ctx* ctx, const mebp_model_weights* model, const mebp_lora* lora,
                   const int32_t* ids, int batch, int seq, float* loss,
                   const mebp_lora_grads* grads, int accumulate, void* stream);

/* ---- optimizer step (Section 4: every model is trained with AdamW; Section 3 keeps only the LoRA
 * weights, their gradients and the optimizer states, and accumulates gradients over the samples
 * of a batch).  AdamW = Adam with decoupled weight decay; at step t >= 1, per element:
 *   g = grad_scale * grad;  m = b1 m + (1-b1) g;  v = b2 v + (1-b2) g^2;
 *   p = p - lr * ( (m / (1 - b1^t)) / (sqrt(v / (1 - b2^t)) + eps) + weight_decay * p ).
 * grad_scale = 1/n turns a gradient summed over n micro-batches (mebp_lora_step with
 * accumulate = 1) into their mean. */
typedef struct {
  float lr, beta1, beta2, eps, weight_decay;
  float grad_scale;
} mebp_adamw_cfg;

/* One AdamW update, in place, of n fp32 parameters held in one flat device buffer (the LoRA
 * masters of every layer back to back), with their gradients and moment buffers m, v (same
 * length; zero before step 1).  All four pointers 16-byte aligned; params, m, v are read and
 * written, grads only read; none may overlap another.  step >= 1 is the (host) step count t.
 * MEBP_ERR_INVALID_ARG for NULL or misaligned pointers, n < 0, step < 1 or bad hyper-parameters;
 * n = 0 is a no-op. */
int mebp_adamw_step(mebp_ctx* ctx, float* params, const float* grads, float* m, float* v, int64_t n,
                    const mebp_adamw_cfg* cfg, int64_t step, void* stream);

/* ---- instrumentation (Section 4 reports per-layer time and memory; here: device time of every
 * kernel, by kind, measured with CUDA events).
 * mebp_kernel_launches: process-wide number of kernel launches the library has issued.
 * mebp_profile_begin: from now on record a CUDA-event pair on the launching stream around every
 *   kernel launch of this context (mebp_lora_step then runs eagerly, not as a graph replay; the
 *   events serialise each launch against its neighbours on that stream).
 * mebp_profile_end: synchronise those events, stop recording and report the fused dequant-GEMM
 *   launches: summed device time, algorithmic flops (2 M N K, plus 2 M N kx for the LoRA extra
 *   block) and bytes (activation operand, packed weight and scales, output, residual and LoRA
 *   operands, each once), split into forward-mode (Y = X deq(W)^T, LM-head passes) and transposed
 *   (dX) launches.
 * mebp_profile_kernels: after mebp_profile_end, one entry per kind of kernel (fused GEMM forward /
 *   transposed, embedding, RMSNorm forward / backward, RoPE, gated-MLP forward / backward,
 *   attention forward / backward, LoRA kernels, LM-head reductions, ...): launches, summed event
 *   time, algorithmic HBM bytes and flops.  *n = the number of kinds; at most max are written.
 *   name points to a static string. */
typedef struct {
  int64_t gemm_launches;
  double gemm_ms, gemm_flops;  /* summed per-launch device time (launches on concurrent streams
                                  overlap, so this may exceed the wall time) and flops */
  double fwd_ms, fwd_flops;
  double dx_ms, dx_flops;
  double gemm_busy_ms;         /* length of the union of the launches' [start, end] intervals:
                                  wall time during which at least one fused GEMM ran */
  double gemm_bytes;           /* algorithmic bytes of the launches */
} mebp_profile;
typedef struct {
  const char* name;
  int64_t launches;
  double ms, bytes, flops;
} mebp_kernel_stat;
int64_t mebp_kernel_launches(void);
/* Turn CUDA-graph replay of mebp_lora_step on (default) or off; drops any captured graph. */
int mebp_enable_graphs(mebp_ctx* ctx, int on);
int mebp_profile_begin(mebp_ctx* ctx);
int mebp_profile_end(mebp_ctx* ctx, mebp_profile* out);
int mebp_profile_kernels(const mebp_ctx* ctx, mebp_kernel_stat* out, int max, int* n);

#ifdef __cplusplus
}
#endif
#endif /* MEBP_H_ */
