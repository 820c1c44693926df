// AdamW update of the flat LoRA parameter buffer (Section 4 trains with AdamW; Section 3 keeps
// the LoRA weights, gradients and optimizer states in memory).  One pass over HBM: reads p, g,
// m, v and writes p, m, v (28 bytes per parameter), 16-byte vector accesses, grid-stride.
#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace mebp {

struct AdamWArgs {
  float lr, b1, b2, eps, wd, gs;
  float bc1, bc2;  // 1 / (1 - beta^t), from the host in double precision
};

__device__ __forceinline__ void adamw_elem(float& p, float g, float& m, float& v, const AdamWArgs& a) {
  g *= a.gs;
  m = a.b1 * m + (1.0f - a.b1) * g;
  v = a.b2 * v + (1.0f - a.b2) * g * g;
  const float upd = (m * a.bc1) / (sqrtf(v * a.bc2) + a.eps);
  p = p - a.lr * (upd + a.wd * p);
}

__global__ void adamw_kernel(float* __restrict__ p, const float* __restrict__ g, float* __restrict__ m,
                             float* __restrict__ v, int64_t n, const AdamWArgs a) {
  griddep_wait();
  griddep_launch();
  const int64_t n4 = n / 4;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4; i += stride) {
    float4 pp = reinterpret_cast<const float4*>(p)[i];
    const float4 gg = reinterpret_cast<const float4*>(g)[i];
    float4 mm = reinterpret_cast<const float4*>(m)[i];
    float4 vv = reinterpret_cast<const float4*>(v)[i];
    adamw_elem(pp.x, gg.x, mm.x, vv.x, a);
    adamw_elem(pp.y, gg.y, mm.y, vv.y, a);
    adamw_elem(pp.z, gg.z, mm.z, vv.z, a);
    adamw_elem(pp.w, gg.w, mm.w, vv.w, a);
    reinterpret_cast<float4*>(p)[i] = pp;
    reinterpret_cast<float4*>(m)[i] = mm;
    reinterpret_cast<float4*>(v)[i] = vv;
  }
  // tail (n % 4 elements)
  const int64_t t = 4 * n4 + static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (t < n) adamw_elem(p[t], g[t], m[t], v[t], a);
}

void launch_adamw(float* p, const float* g, float* m, float* v, int64_t n, float lr, float b1, float b2, float eps,
                  float wd, float gs, double bc1, double bc2, cudaStream_t st) {
  if (n <= 0) return;
  const AdamWArgs a{lr, b1, b2, eps, wd, gs, static_cast<float>(bc1), static_cast<float>(bc2)};
  // enough 256-thread blocks for ~8 float4 per thread at most, at least one wave of 152 x 8 CTAs
  const int64_t n4 = (n + 3) / 4;
  const int64_t blocks = std::max<int64_t>(1, std::min<int64_t>((n4 + 255) / 256, 152 * 8));
  launch_k(adamw_kernel, static_cast<unsigned>(blocks), 256, 0, st, p, g, m, v, n, a);
}

}  // namespace mebp
