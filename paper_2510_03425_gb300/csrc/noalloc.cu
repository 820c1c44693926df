// mebp_linear_fwd_noalloc: the fused LoRA linear without any device allocation.
//
// Who needs it: code that must not call cudaMalloc / cudaFree (or anything that allocates
// device memory) at the point where it runs the layer — for example a host program whose
// memory is handed out by an external pool it does not own, or a caller running in a
// context where allocation is forbidden or would break its memory accounting.  The regular
// entry points need a mebp_ctx, whose creation allocates the workspace; mebp_linear_fwd also
// takes stream-ordered temporaries for the fp16 LoRA shadows and the rank-r product.
//
// Here that scratch is one file-scope device array of fixed size, present on every GPU that
// loads the library for the life of the process.  Its device address is looked up once per CUDA
// context (on the first call made while that context is current) and reused afterwards; keying
// by context rather than by device ordinal means a context created after a device reset, or a
// non-primary context made current by the caller, gets its own lookup instead of a stale address.
#include <cudaTypedefs.h>

#include <mutex>

#include "../../include/mebp.h"
#include "kernels.h"

#define MEBP_NOALLOC_MAX_CONTEXTS 64

static __device__ __align__(256) unsigned char g_noalloc_scratch[MEBP_NOALLOC_SCRATCH_BYTES];

namespace {

std::mutex g_noalloc_mu;
struct ScratchEntry {
  CUcontext ctx;
  void* addr;
};
ScratchEntry g_noalloc_cache[MEBP_NOALLOC_MAX_CONTEXTS] = {};
int g_noalloc_n = 0;

PFN_cuCtxGetCurrent_v4000 ctx_get_current() {
  static PFN_cuCtxGetCurrent_v4000 fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(f);
    else
      cudaGetLastError();
  }
  return fn;
}

// Device address of g_noalloc_scratch in the current context (looked up on first use).
int noalloc_scratch(unsigned char** out) {
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  PFN_cuCtxGetCurrent_v4000 get = ctx_get_current();
  if (!get) return MEBP_ERR_CUDA;
  CUcontext cur = nullptr;
  if (get(&cur) != CUDA_SUCCESS) return MEBP_ERR_CUDA;
  if (cur)
    for (int i = 0; i < g_noalloc_n; ++i)
      if (g_noalloc_cache[i].ctx == cur) {
        *out = static_cast<unsigned char*>(g_noalloc_cache[i].addr);
        return MEBP_OK;
      }
  // Not cached (or no context current yet: the runtime makes the device's primary context
  // current here).
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) {
    cudaGetLastError();
    return MEBP_ERR_CUDA;
  }
  if (!cur && get(&cur) != CUDA_SUCCESS) return MEBP_ERR_CUDA;
  if (cur && g_noalloc_n < MEBP_NOALLOC_MAX_CONTEXTS) g_noalloc_cache[g_noalloc_n++] = {cur, p};
  *out = static_cast<unsigned char*>(p);
  return MEBP_OK;
}

int64_t align256(int64_t b) { return (b + 255) / 256 * 256; }

}  // namespace

extern "C" int mebp_linear_fwd_noalloc(const uint16_t* X, int64_t M, const mebp_packed* W, const float* A,
                                       const float* B, int r, float s, const float* R, float* y_f32,
                                       uint16_t* y_f16, void* stream) {
  using namespace mebp;
  if (!X || !W || !W->qpack || !W->scales || (!y_f32 && !y_f16)) return MEBP_ERR_INVALID_ARG;
  const int64_t N = W->rows, K = W->cols;
  if (N <= 0 || K <= 0 || N % 64 || K % 64) return MEBP_ERR_INVALID_ARG;
  // 16-byte alignment: TMA reads X and the weights; the epilogue stores y and reads R as 16-byte
  // vectors.
  if ((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(W->qpack) |
       reinterpret_cast<uintptr_t>(W->scales) | reinterpret_cast<uintptr_t>(y_f32) |
       reinterpret_cast<uintptr_t>(y_f16) | reinterpret_cast<uintptr_t>(R)) & 15)
    return MEBP_ERR_INVALID_ARG;
  if ((A == nullptr) != (B == nullptr)) return MEBP_ERR_INVALID_ARG;
  if (A && (r <= 0 || r > 32 || r % 8)) return MEBP_ERR_UNSUPPORTED;
  if (M < 0) return MEBP_ERR_INVALID_ARG;

  // Scratch layout: [error word | A shadow kx x K | B shadow N x kx | B^T shadow kx x N | U M x kx]
  const int kxp = A ? (r + 15) / 16 * 16 : 0;
  const int64_t off_a = 256;
  const int64_t off_b = off_a + align256(2 * static_cast<int64_t>(kxp) * K);
  const int64_t off_bt = off_b + align256(2 * N * kxp);
  const int64_t off_u = off_bt + align256(2 * N * kxp);
  const int64_t need = off_u + align256(2 * M * kxp);
  if (need > MEBP_NOALLOC_SCRATCH_BYTES) return MEBP_ERR_SCRATCH;
  if (M == 0) return MEBP_OK;

  unsigned char* scratch = nullptr;
  int rc = noalloc_scratch(&scratch);
  if (rc) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int* err = reinterpret_cast<int*>(scratch);
  cudaMemsetAsync(err, 0, sizeof(int), st);  // the only scratch that must start at zero
  pdl_entry();  // no kernel of this call overlaps work issued before it

  GemmArgs g;
  g.trans = false;
  g.A = X;
  g.lda = K;
  g.M = M;
  g.N = N;
  g.K = K;
  g.qpack = W->qpack;
  g.scales = W->scales;
  g.scale_pitch = N;
  g.err = err;
  if (A) {
    uint16_t* Ac = reinterpret_cast<uint16_t*>(scratch + off_a);
    uint16_t* Bc = reinterpret_cast<uint16_t*>(scratch + off_b);
    uint16_t* Btc = reinterpret_cast<uint16_t*>(scratch + off_bt);
    uint16_t* U = reinterpret_cast<uint16_t*>(scratch + off_u);
    const float* As[1] = {A};
    const float* Bs[1] = {B};
    const int ro[1] = {0}, no[1] = {0};
    const int nl[1] = {static_cast<int>(N)};
    launch_lora_shadow(As, Bs, 1, ro, no, nl, r, static_cast<int>(K), static_cast<int>(N), kxp, Ac, Bc, Btc, st);
    launch_skinny_gemm(X, K, M, K, Ac, K, r, s, U, kxp, st, err);
    g.Ax = U;
    g.ldax = kxp;
    g.kx = kxp;
    g.Bx = Bc;
    g.ldbx = kxp;
  }
  if (y_f32) {
    g.epi = EPI_F32;
    g.C = y_f32;
    g.ldc = N;
    g.R = R;
    g.ldr = N;
  } else {
    g.epi = EPI_F16;
    g.C = y_f16;
    g.ldc = N;
  }
  rc = launch_dequant_gemm(g, st);
  if (rc) return rc;
  return cudaGetLastError() == cudaSuccess ? MEBP_OK : MEBP_ERR_CUDA;
}
