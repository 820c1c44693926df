// Bandwidth-bound kernels of the block: RMSNorm forward/backward, RoPE, gated-MLP activation
// forward/backward, casts, and the LM-head's log-sum-exp combine and loss reduction.
// Every kernel streams rows with 16-byte vector accesses, one warp per row where a row
// reduction is needed.
#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace mebp {

// ------------------------------------------------------------------------------------ RMSNorm
// y = x / sqrt(mean(x^2) + eps) * g  ->  fp16 (the GEMM operand); rstd saved for the backward.
__global__ void rmsnorm_fwd_kernel(const float* __restrict__ x, const float* __restrict__ g, int64_t T, int D,
                                   float eps, uint16_t* __restrict__ y, float* __restrict__ rstd) {
  griddep_wait();
  griddep_launch();
  const int64_t row = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= T) return;
  const float4* xr = reinterpret_cast<const float4*>(x + row * D);
  const int n4 = D >> 2;
  float ss = 0.0f;
  for (int i = lane; i < n4; i += 32) {
    const float4 v = xr[i];
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = warp_sum(ss);
  const float r = rsqrtf(ss / static_cast<float>(D) + eps);
  if (lane == 0 && rstd) rstd[row] = r;
  const float4* gr = reinterpret_cast<const float4*>(g);
  uint2* yr = reinterpret_cast<uint2*>(y + row * D);
  for (int i = lane; i < n4; i += 32) {
    const float4 v = xr[i], w = gr[i];
    yr[i] = make_uint2(pack_half2(v.x * r * w.x, v.y * r * w.y), pack_half2(v.z * r * w.z, v.w * r * w.w));
  }
}

// v = resid + r (g*dy) - x r^3 / D * sum(g*dy*x);  dx = v * mult,  dxb = fp16(v)
__global__ void rmsnorm_bwd_kernel(const float* __restrict__ dy, const float* __restrict__ x,
                                   const float* __restrict__ g, const float* __restrict__ rstd,
                                   const float* __restrict__ resid, int64_t T, int D, const float* __restrict__ mult,
                                   float* __restrict__ dx, uint16_t* __restrict__ dxb) {
  griddep_wait();
  griddep_launch();
  const int64_t row = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= T) return;
  const int n4 = D >> 2;
  const float4* dr = reinterpret_cast<const float4*>(dy + row * D);
  const float4* xr = reinterpret_cast<const float4*>(x + row * D);
  const float4* gr = reinterpret_cast<const float4*>(g);
  float dot = 0.0f;
  for (int i = lane; i < n4; i += 32) {
    const float4 a = dr[i], b = xr[i], w = gr[i];
    dot += a.x * w.x * b.x + a.y * w.y * b.y + a.z * w.z * b.z + a.w * w.w * b.w;
  }
  dot = warp_sum(dot);
  const float r = rstd[row];
  const float c = r * r * r * dot / static_cast<float>(D);
  const float mu = mult ? *mult : 1.0f;
  const float4* rr = resid ? reinterpret_cast<const float4*>(resid + row * D) : nullptr;
  float4* outr = reinterpret_cast<float4*>(dx + row * D);
  uint2* outb = dxb ? reinterpret_cast<uint2*>(dxb + row * D) : nullptr;
  for (int i = lane; i < n4; i += 32) {
    const float4 a = dr[i], b = xr[i], w = gr[i];
    float4 o = make_float4(r * w.x * a.x - b.x * c, r * w.y * a.y - b.y * c, r * w.z * a.z - b.z * c,
                           r * w.w * a.w - b.w * c);
    if (rr) {
      const float4 q = rr[i];
      o.x += q.x; o.y += q.y; o.z += q.z; o.w += q.w;
    }
    if (outb) outb[i] = make_uint2(pack_half2(o.x, o.y), pack_half2(o.z, o.w));
    if (dx) outr[i] = make_float4(o.x * mu, o.y * mu, o.z * mu, o.w * mu);
  }
}

void launch_rmsnorm_fwd(const float* x, const float* g, int64_t T, int D, float eps, uint16_t* y, float* rstd,
                        cudaStream_t st) {
  if (T <= 0) return;
  launch_k(rmsnorm_fwd_kernel, static_cast<unsigned>((T * 32 + 255) / 256), 256, 0, st, x, g, T, D, eps, y, rstd);
}
void launch_rmsnorm_bwd(const float* dy, const float* x, const float* g, const float* rstd, const float* resid,
                        int64_t T, int D, const float* out_mult, float* dx, uint16_t* dxb, cudaStream_t st) {
  if (T <= 0) return;
  launch_k(rmsnorm_bwd_kernel, static_cast<unsigned>((T * 32 + 255) / 256), 256, 0, st, dy, x, g, rstd, resid, T, D,
           out_mult, dx, dxb);
}

// ------------------------------------------------------------------------------------ RoPE
// Half-split rotation: (x1, x2) -> (x1 c - x2 s, x2 c + x1 s) with (c, s) = table[pos][j];
// inverse rotates by -angle (the VJP).  One thread per (token, group of 8 pairs j .. j+7, up to
// four heads): the eight (c, s) pairs are read once and applied to every head of the thread, and
// the eight x1 and eight x2 values of a head move as one 16-byte load / store each.
constexpr int kRopeHeadsPerThread = 4;
__global__ void rope_kernel(uint16_t* __restrict__ qkv, int64_t T, int S, int nheads, int ld, int hd,
                            const float2* __restrict__ cs, int inverse) {
  griddep_wait();
  griddep_launch();
  const int half = hd >> 1, ng = half >> 3, nhc = (nheads + kRopeHeadsPerThread - 1) / kRopeHeadsPerThread;
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= T * ng * nhc) return;
  const int g = static_cast<int>(i % ng);
  const int64_t th = i / ng;
  const int hc = static_cast<int>(th % nhc);
  const int64_t t = th / nhc;
  const int pos = static_cast<int>(t % S);
  const float4* tab = reinterpret_cast<const float4*>(cs + static_cast<int64_t>(pos) * half + 8 * g);
  const float sg = inverse ? -1.0f : 1.0f;
  float c[8], sn[8];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float4 v = tab[k];
    c[2 * k] = v.x;
    sn[2 * k] = sg * v.y;
    c[2 * k + 1] = v.z;
    sn[2 * k + 1] = sg * v.w;
  }
  const int h0 = hc * kRopeHeadsPerThread, h1 = min(nheads, h0 + kRopeHeadsPerThread);
  uint4 a[kRopeHeadsPerThread], b[kRopeHeadsPerThread];
#pragma unroll
  for (int k = 0; k < kRopeHeadsPerThread; ++k)
    if (h0 + k < h1) {
      const uint16_t* base = qkv + t * ld + static_cast<int64_t>(h0 + k) * hd + 8 * g;
      a[k] = *reinterpret_cast<const uint4*>(base);
      b[k] = *reinterpret_cast<const uint4*>(base + half);
    }
#pragma unroll
  for (int k = 0; k < kRopeHeadsPerThread; ++k)
    if (h0 + k < h1) {
      const uint32_t x1[4] = {a[k].x, a[k].y, a[k].z, a[k].w}, x2[4] = {b[k].x, b[k].y, b[k].z, b[k].w};
      uint32_t y1[4], y2[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float p0 = h2_lo(x1[q]), p1 = h2_hi(x1[q]), q0 = h2_lo(x2[q]), q1 = h2_hi(x2[q]);
        const int j0 = 2 * q, j1 = 2 * q + 1;
        y1[q] = pack_half2(p0 * c[j0] - q0 * sn[j0], p1 * c[j1] - q1 * sn[j1]);
        y2[q] = pack_half2(q0 * c[j0] + p0 * sn[j0], q1 * c[j1] + p1 * sn[j1]);
      }
      uint16_t* base = qkv + t * ld + static_cast<int64_t>(h0 + k) * hd + 8 * g;
      *reinterpret_cast<uint4*>(base) = make_uint4(y1[0], y1[1], y1[2], y1[3]);
      *reinterpret_cast<uint4*>(base + half) = make_uint4(y2[0], y2[1], y2[2], y2[3]);
    }
}

void launch_rope(uint16_t* qkv, int64_t T, int S, int H, int KV, int hd, const float2* cs, bool inverse,
                 cudaStream_t st) {
  const int nheads = H + KV;  // q heads then k heads
  const int64_t n = T * (hd / 16) * ((nheads + kRopeHeadsPerThread - 1) / kRopeHeadsPerThread);
  if (n <= 0) return;
  launch_k(rope_kernel, static_cast<unsigned>((n + 255) / 256), 256, 0, st, qkv, T, S, nheads, (H + 2 * KV) * hd, hd,
           cs, inverse ? 1 : 0);
}

// ------------------------------------------------------------------------------------ Gemma3 block
// QK-norm then RoPE: each q or k head (token t, head h < H + KV) is RMS-normalised over its hd
// elements with the head gain (q_norm for q heads, k_norm for k heads) and rotated in place; the
// raw head and its 1/rms are kept for the backward.  One warp per (token, head); lane handles
// the rotation pairs (j, j + hd/2) for j = lane + 32 i.
template <int HD>
__global__ void qknorm_rope_kernel(uint16_t* __restrict__ qkv, int64_t T, int S, int H, int KV, int64_t ld,
                                   const float* __restrict__ qg, const float* __restrict__ kg, float eps,
                                   const float2* __restrict__ cs, uint16_t* __restrict__ raw,
                                   float* __restrict__ rstd) {
  griddep_wait();
  griddep_launch();
  constexpr int HALF = HD / 2, NP = HALF / 32;
  const int nh = H + KV;
  const int64_t wid = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (wid >= T * nh) return;
  const int head = static_cast<int>(wid % nh);
  const int64_t t = wid / nh;
  const int pos = static_cast<int>(t % S);
  uint16_t* base = qkv + t * ld + static_cast<int64_t>(head) * HD;
  uint16_t* rb = raw + wid * HD;
  const float* g = head < H ? qg : kg;
  float x1[NP], x2[NP];
  float ss = 0.0f;
#pragma unroll
  for (int i = 0; i < NP; ++i) {
    const int j = lane + 32 * i;
    const uint16_t a = base[j], b = base[j + HALF];
    rb[j] = a;
    rb[j + HALF] = b;
    x1[i] = h_to_f(a);
    x2[i] = h_to_f(b);
    ss += x1[i] * x1[i] + x2[i] * x2[i];
  }
  ss = warp_sum(ss);
  const float r = rsqrtf(ss / static_cast<float>(HD) + eps);
  if (lane == 0) rstd[wid] = r;
#pragma unroll
  for (int i = 0; i < NP; ++i) {
    const int j = lane + 32 * i;
    const float y1 = x1[i] * r * g[j], y2 = x2[i] * r * g[j + HALF];
    const float2 c = cs[static_cast<int64_t>(pos) * HALF + j];
    base[j] = f_to_h(y1 * c.x - y2 * c.y);
    base[j + HALF] = f_to_h(y2 * c.x + y1 * c.y);
  }
}

// Backward of qknorm_rope on dqkv in place: rotate the head gradient back (by -angle), then
// the RMSNorm VJP dx = r (g dy) - x r^3 / hd * sum(g dy x) with the saved raw head x and r.
template <int HD>
__global__ void qknorm_rope_bwd_kernel(uint16_t* __restrict__ dqkv, int64_t T, int S, int H, int KV, int64_t ld,
                                       const float* __restrict__ qg, const float* __restrict__ kg,
                                       const float2* __restrict__ cs, const uint16_t* __restrict__ raw,
                                       const float* __restrict__ rstd) {
  griddep_wait();
  griddep_launch();
  constexpr int HALF = HD / 2, NP = HALF / 32;
  const int nh = H + KV;
  const int64_t wid = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (wid >= T * nh) return;
  const int head = static_cast<int>(wid % nh);
  const int64_t t = wid / nh;
  const int pos = static_cast<int>(t % S);
  uint16_t* base = dqkv + t * ld + static_cast<int64_t>(head) * HD;
  const uint16_t* rb = raw + wid * HD;
  const float* g = head < H ? qg : kg;
  float gd1[NP], gd2[NP], x1[NP], x2[NP];
  float dot = 0.0f;
#pragma unroll
  for (int i = 0; i < NP; ++i) {
    const int j = lane + 32 * i;
    const float d1 = h_to_f(base[j]), d2 = h_to_f(base[j + HALF]);
    const float2 c = cs[static_cast<int64_t>(pos) * HALF + j];
    gd1[i] = g[j] * (d1 * c.x + d2 * c.y);
    gd2[i] = g[j + HALF] * (d2 * c.x - d1 * c.y);
    x1[i] = h_to_f(rb[j]);
    x2[i] = h_to_f(rb[j + HALF]);
    dot += gd1[i] * x1[i] + gd2[i] * x2[i];
  }
  dot = warp_sum(dot);
  const float r = rstd[wid];
  const float cc = r * r * r * dot / static_cast<float>(HD);
#pragma unroll
  for (int i = 0; i < NP; ++i) {
    const int j = lane + 32 * i;
    base[j] = f_to_h(r * gd1[i] - x1[i] * cc);
    base[j + HALF] = f_to_h(r * gd2[i] - x2[i] * cc);
  }
}

void launch_qknorm_rope(uint16_t* qkv, int64_t T, int S, int H, int KV, int hd, const float* qg, const float* kg,
                        float eps, const float2* cs, uint16_t* raw, float* rstd, cudaStream_t st) {
  const int64_t n = T * (H + KV) * 32;
  if (n <= 0) return;
  const int64_t ld = static_cast<int64_t>(H + 2 * KV) * hd;
  const unsigned grid = static_cast<unsigned>((n + 255) / 256);
  if (hd == 64) launch_k(qknorm_rope_kernel<64>, grid, 256, 0, st, qkv, T, S, H, KV, ld, qg, kg, eps, cs, raw, rstd);
  else if (hd == 128) launch_k(qknorm_rope_kernel<128>, grid, 256, 0, st, qkv, T, S, H, KV, ld, qg, kg, eps, cs, raw, rstd);
  else launch_k(qknorm_rope_kernel<256>, grid, 256, 0, st, qkv, T, S, H, KV, ld, qg, kg, eps, cs, raw, rstd);
}
void launch_qknorm_rope_bwd(uint16_t* dqkv, int64_t T, int S, int H, int KV, int hd, const float* qg, const float* kg,
                            const float2* cs, const uint16_t* raw, const float* rstd, cudaStream_t st) {
  const int64_t n = T * (H + KV) * 32;
  if (n <= 0) return;
  const int64_t ld = static_cast<int64_t>(H + 2 * KV) * hd;
  const unsigned grid = static_cast<unsigned>((n + 255) / 256);
  if (hd == 64) launch_k(qknorm_rope_bwd_kernel<64>, grid, 256, 0, st, dqkv, T, S, H, KV, ld, qg, kg, cs, raw, rstd);
  else if (hd == 128)
    launch_k(qknorm_rope_bwd_kernel<128>, grid, 256, 0, st, dqkv, T, S, H, KV, ld, qg, kg, cs, raw, rstd);
  else launch_k(qknorm_rope_bwd_kernel<256>, grid, 256, 0, st, dqkv, T, S, H, KV, ld, qg, kg, cs, raw, rstd);
}

// Sandwich norm after attention, residual add and the MLP pre-norm in one pass per row:
// h1 = x + ao * r_pa * g_pa (r_pa = 1/rms(ao)), b = fp16(h1 * r2 * g2) (r2 = 1/rms(h1)).
__global__ void add_norm2_kernel(const float* __restrict__ ao, const float* __restrict__ x,
                                 const float* __restrict__ gpa, const float* __restrict__ g2, int64_t T, int D,
                                 float eps, float* __restrict__ h1, uint16_t* __restrict__ b, float* __restrict__ rpa,
                                 float* __restrict__ r2) {
  griddep_wait();
  griddep_launch();
  const int64_t row = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= T) return;
  const int n4 = D >> 2;
  const float4* ar = reinterpret_cast<const float4*>(ao + row * D);
  const float4* xr = reinterpret_cast<const float4*>(x + row * D);
  const float4* gp = reinterpret_cast<const float4*>(gpa);
  const float4* gq = reinterpret_cast<const float4*>(g2);
  float4* hr = reinterpret_cast<float4*>(h1 + row * D);
  float ss = 0.0f;
  for (int i = lane; i < n4; i += 32) {
    const float4 v = ar[i];
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  const float ra = rsqrtf(warp_sum(ss) / static_cast<float>(D) + eps);
  float sh = 0.0f;
  for (int i = lane; i < n4; i += 32) {
    const float4 v = ar[i], w = gp[i], xx = xr[i];
    const float4 h = make_float4(xx.x + v.x * ra * w.x, xx.y + v.y * ra * w.y, xx.z + v.z * ra * w.z,
                                 xx.w + v.w * ra * w.w);
    hr[i] = h;
    sh += h.x * h.x + h.y * h.y + h.z * h.z + h.w * h.w;
  }
  const float rb = rsqrtf(warp_sum(sh) / static_cast<float>(D) + eps);
  if (lane == 0) {
    rpa[row] = ra;
    r2[row] = rb;
  }
  uint2* br = reinterpret_cast<uint2*>(b + row * D);
  for (int i = lane; i < n4; i += 32) {  // the row this thread just wrote
    const float4 h = hr[i], w = gq[i];
    br[i] = make_uint2(pack_half2(h.x * rb * w.x, h.y * rb * w.y), pack_half2(h.z * rb * w.z, h.w * rb * w.w));
  }
}

// Sandwich norm after the MLP and the residual add: y = h1 + dn * r_pf * g_pf.
__global__ void add_norm_kernel(const float* __restrict__ dn, const float* __restrict__ h1,
                                const float* __restrict__ gpf, int64_t T, int D, float eps, float* __restrict__ y,
                                float* __restrict__ rpf) {
  griddep_wait();
  griddep_launch();
  const int64_t row = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= T) return;
  const int n4 = D >> 2;
  const float4* dr = reinterpret_cast<const float4*>(dn + row * D);
  const float4* hr = reinterpret_cast<const float4*>(h1 + row * D);
  const float4* gp = reinterpret_cast<const float4*>(gpf);
  float4* yr = reinterpret_cast<float4*>(y ? y + row * D : nullptr);
  float ss = 0.0f;
  for (int i = lane; i < n4; i += 32) {
    const float4 v = dr[i];
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  const float r = rsqrtf(warp_sum(ss) / static_cast<float>(D) + eps);
  if (lane == 0 && rpf) rpf[row] = r;
  if (!y) return;  // the backward's recompute wants the 1/rms only
  for (int i = lane; i < n4; i += 32) {
    const float4 v = dr[i], w = gp[i], h = hr[i];
    yr[i] = make_float4(h.x + v.x * r * w.x, h.y + v.y * r * w.y, h.z + v.z * r * w.z, h.w + v.w * r * w.w);
  }
}

void launch_add_norm2(const float* ao, const float* x, const float* gpa, const float* g2, int64_t T, int D, float eps,
                      float* h1, uint16_t* b, float* rpa, float* r2, cudaStream_t st) {
  if (T <= 0) return;
  launch_k(add_norm2_kernel, static_cast<unsigned>((T * 32 + 255) / 256), 256, 0, st, ao, x, gpa, g2, T, D, eps, h1,
           b, rpa, r2);
}
void launch_add_norm(const float* dn, const float* h1, const float* gpf, int64_t T, int D, float eps, float* y,
                     float* rpf, cudaStream_t st) {
  if (T <= 0) return;
  launch_k(add_norm_kernel, static_cast<unsigned>((T * 32 + 255) / 256), 256, 0, st, dn, h1, gpf, T, D, eps, y, rpf);
}

// ------------------------------------------------------------------------------------ gated MLP

// m = act(g) * u; gu row = [g (I) | u (I)].  8 elements per thread.
// A product outside the fp16 range (or NaN) sets MEBP_ERR_NONFINITE in *err.
__global__ void glu_fwd_kernel(const uint16_t* __restrict__ gu, int64_t T, int I, int act, uint16_t* __restrict__ m,
                               int* err) {
  griddep_wait();
  griddep_launch();
  const int per = I / 8;
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= T * per) return;
  const int64_t t = i / per;
  const int c = static_cast<int>(i % per) * 8;
  const uint4 gv = *reinterpret_cast<const uint4*>(gu + t * 2 * I + c);
  const uint4 uv = *reinterpret_cast<const uint4*>(gu + t * 2 * I + I + c);
  const uint32_t ga[4] = {gv.x, gv.y, gv.z, gv.w}, ua[4] = {uv.x, uv.y, uv.z, uv.w};
  uint32_t o[4];
#pragma unroll
  for (int k = 0; k < 4; ++k)
    o[k] = pack_half2(act_f(h2_lo(ga[k]), act) * h2_lo(ua[k]), act_f(h2_hi(ga[k]), act) * h2_hi(ua[k]));
  if (h2_nonfinite(o[0]) | h2_nonfinite(o[1]) | h2_nonfinite(o[2]) | h2_nonfinite(o[3])) flag_error(err, kErrNonFinite);
  *reinterpret_cast<uint4*>(m + t * I + c) = make_uint4(o[0], o[1], o[2], o[3]);
}

// dg = dm * u * act'(g), du = dm * act(g)
__global__ void glu_bwd_kernel(const uint16_t* __restrict__ dm, const uint16_t* __restrict__ gu, int64_t T, int I, int act,
                               uint16_t* __restrict__ dgu, int* err) {
  griddep_wait();
  griddep_launch();
  const int per = I / 8;
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= T * per) return;
  const int64_t t = i / per;
  const int c = static_cast<int>(i % per) * 8;
  const uint4 gv = *reinterpret_cast<const uint4*>(gu + t * 2 * I + c);
  const uint4 uv = *reinterpret_cast<const uint4*>(gu + t * 2 * I + I + c);
  const uint4 dv = *reinterpret_cast<const uint4*>(dm + t * I + c);
  const float dd[8] = {h2_lo(dv.x), h2_hi(dv.x), h2_lo(dv.y), h2_hi(dv.y),
                       h2_lo(dv.z), h2_hi(dv.z), h2_lo(dv.w), h2_hi(dv.w)};
  const uint32_t ga[4] = {gv.x, gv.y, gv.z, gv.w}, ua[4] = {uv.x, uv.y, uv.z, uv.w};
  uint32_t og[4], ou[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float g0 = h2_lo(ga[k]), g1 = h2_hi(ga[k]), u0 = h2_lo(ua[k]), u1 = h2_hi(ua[k]);
    og[k] = pack_half2(dd[2 * k] * u0 * act_grad(g0, act), dd[2 * k + 1] * u1 * act_grad(g1, act));
    ou[k] = pack_half2(dd[2 * k] * act_f(g0, act), dd[2 * k + 1] * act_f(g1, act));
  }
  uint32_t bad = 0;
#pragma unroll
  for (int k = 0; k < 4; ++k) bad |= h2_nonfinite(og[k]) | h2_nonfinite(ou[k]);
  if (bad) flag_error(err, kErrNonFinite);
  *reinterpret_cast<uint4*>(dgu + t * 2 * I + c) = make_uint4(og[0], og[1], og[2], og[3]);
  *reinterpret_cast<uint4*>(dgu + t * 2 * I + I + c) = make_uint4(ou[0], ou[1], ou[2], ou[3]);
}

void launch_glu_fwd(const uint16_t* gu, int64_t T, int I, int act, uint16_t* m, int* err, cudaStream_t st) {
  const int64_t n = T * (I / 8);
  if (n <= 0) return;
  launch_k(glu_fwd_kernel, static_cast<unsigned>((n + 255) / 256), 256, 0, st, gu, T, I, act, m, err);
}
void launch_glu_bwd(const uint16_t* dm, const uint16_t* gu, int64_t T, int I, int act, uint16_t* dgu, int* err,
                    cudaStream_t st) {
  const int64_t n = T * (I / 8);
  if (n <= 0) return;
  launch_k(glu_bwd_kernel, static_cast<unsigned>((n + 255) / 256), 256, 0, st, dm, gu, T, I, act, dgu, err);
}

// ------------------------------------------------------------------------------------ casts
__global__ void scale_cast_kernel(const float* __restrict__ x, int64_t n4, const float* __restrict__ scale,
                                  float* __restrict__ y32, uint16_t* __restrict__ y16) {
  griddep_wait();
  griddep_launch();
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= n4) return;
  const float sc = scale ? *scale : 1.0f;
  float4 v = reinterpret_cast<const float4*>(x)[i];
  v.x *= sc; v.y *= sc; v.z *= sc; v.w *= sc;
  if (y32) reinterpret_cast<float4*>(y32)[i] = v;
  reinterpret_cast<uint2*>(y16)[i] = make_uint2(pack_half2(v.x, v.y), pack_half2(v.z, v.w));
}
// max |x| into *amax_bits (as the bit pattern of a non-negative float; atomicMax on the
// integer view is order independent, so the result is deterministic).
__global__ void amax_kernel(const float* __restrict__ x, int64_t n, unsigned int* __restrict__ amax_bits) {
  griddep_wait();
  griddep_launch();
  float m = 0.0f;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    m = fmaxf(m, fabsf(x[i]));
  m = warp_max(m);
  if ((threadIdx.x & 31) == 0) atomicMax(amax_bits, __float_as_uint(m));
}
// sigma = 2^-floor(log2(amax)) so that max|x * sigma| lies in [1, 2); 1 when amax is 0 or not finite.
__global__ void sigma_kernel(float* scal) {
  griddep_wait();
  griddep_launch();
  const float amax = __uint_as_float(reinterpret_cast<unsigned int*>(scal)[2]);
  float sg = 1.0f;
  if (amax > 0.0f && amax < INFINITY) sg = exp2f(-floorf(log2f(amax)));
  scal[0] = sg;
  scal[1] = 1.0f / sg;
}
void launch_scale_cast(const float* x, int64_t n, const float* scale, float* y32, uint16_t* y16, cudaStream_t st) {
  const int64_t n4 = n / 4;
  if (n4 <= 0) return;
  launch_k(scale_cast_kernel, static_cast<unsigned>((n4 + 255) / 256), 256, 0, st, x, n4, scale, y32, y16);
}
void launch_grad_scale(const float* x, int64_t n, float* scal, cudaStream_t st) {
  cudaMemsetAsync(scal + 2, 0, sizeof(float), st);
  const int64_t blocks = std::min<int64_t>(1184, (n + 255) / 256);
  launch_k(amax_kernel, static_cast<unsigned>(std::max<int64_t>(1, blocks)), 256, 0, st, x, n,
           reinterpret_cast<unsigned int*>(scal + 2));
  launch_k(sigma_kernel, 1, 1, 0, st, scal);
}
__global__ void fill_kernel(float* __restrict__ x, int64_t n, float v) {
  griddep_wait();
  griddep_launch();
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i < n) x[i] = v;
}
void launch_fill_f32(float* x, int64_t n, float v, cudaStream_t st) {
  if (n <= 0) return;
  launch_k(fill_kernel, static_cast<unsigned>((n + 255) / 256), 256, 0, st, x, n, v);
}

// ------------------------------------------------------------------------------------ LM head
// lse[t] = M + log(sum_i l_i exp(m_i - M)) over the per-tile partials (m_i, l_i);
// tok_loss[t] = lse[t] - z_target[t] for valid targets, else 0.
__global__ void lse_combine_kernel(const float2* __restrict__ part, int nparts, const float* __restrict__ zt,
                                   const int32_t* __restrict__ targets, int64_t T, float* __restrict__ lse,
                                   float* __restrict__ tok_loss) {
  griddep_wait();
  griddep_launch();
  const int64_t row = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= T) return;
  const float2* pr = part + row * nparts;
  float mx = -INFINITY;
  for (int i = lane; i < nparts; i += 32) mx = fmaxf(mx, pr[i].x);
  mx = warp_max(mx);
  float s = 0.0f;
  for (int i = lane; i < nparts; i += 32) {
    const float2 v = pr[i];
    if (v.x > -INFINITY) s += v.y * expf(v.x - mx);
  }
  s = warp_sum(s);
  if (lane == 0) {
    const float l = mx + logf(s);
    lse[row] = l;
    tok_loss[row] = targets[row] >= 0 ? l - zt[row] : 0.0f;
  }
}

// loss = sum(tok_loss) / n_valid: one block, fixed reduction order.  Also the backward's
// power-of-two working scale sigma = 2^ceil(log2(n_valid)) (the gradient of the mean loss times
// sigma keeps fp16 operands in range), 1/sigma, and the CE-gradient row weight sigma*shift/n.
__global__ void loss_reduce_kernel(const float* __restrict__ tok_loss, const int32_t* __restrict__ targets, int64_t T,
                                   float* __restrict__ loss, float* __restrict__ scal) {
  griddep_wait();
  griddep_launch();
  __shared__ double ssum[1024];
  __shared__ int scnt[1024];
  double s = 0.0;
  int c = 0;
  for (int64_t i = threadIdx.x; i < T; i += blockDim.x) {
    s += static_cast<double>(tok_loss[i]);
    c += targets[i] >= 0 ? 1 : 0;
  }
  ssum[threadIdx.x] = s;
  scnt[threadIdx.x] = c;
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) {
      ssum[threadIdx.x] += ssum[threadIdx.x + w];
      scnt[threadIdx.x] += scnt[threadIdx.x + w];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const int n = scnt[0];
    *loss = n > 0 ? static_cast<float>(ssum[0] / n) : 0.0f;
    float sg = 1.0f;
    while (sg < static_cast<float>(n)) sg *= 2.0f;
    scal[0] = sg;
    scal[1] = 1.0f / sg;
    scal[2] = n > 0 ? static_cast<float>(static_cast<double>(sg) * kCeShift / n) : 0.0f;
  }
}

void launch_lse_combine(const float* part, int nparts, const float* zt, const int32_t* targets, int64_t T, float* lse,
                        float* tok_loss, cudaStream_t st) {
  if (T <= 0) return;
  launch_k(lse_combine_kernel, static_cast<unsigned>((T * 32 + 255) / 256), 256, 0, st,
           reinterpret_cast<const float2*>(part), nparts, zt, targets, T, lse, tok_loss);
}
void launch_loss_reduce(const float* tok_loss, const int32_t* targets, int64_t T, float* loss, float* scal,
                        cudaStream_t st) {
  launch_k(loss_reduce_kernel, 1, 1024, 0, st, tok_loss, targets, T, loss, scal);
}

}  // namespace mebp
