// Small fused row ops of the drafter forward.
//
// combine_kernel (Sec. 2.3, input slots): c_t is the sum of the boundary-fusion
// GEMM's split-K partials; x_i = E[u_i] + P_i + c_t with u_0 = a (the committed
// token) and the mask embedding for slots holding -1, written to the fp32
// residual stream and fused with the first layer's input RMSNorm.  The same
// launch fills the rotary cos/sin table of every (request, slot) at absolute
// position t + i: the angle is formed and reduced modulo 2*pi in fp64, so
// positions near 1.3e5 keep full fp32 accuracy, and sin/cos run in fp32.
//
// resid_norm_kernel: x += sum of a projection's split-K partials (the
// residual add of the o and down projections, in split order), then
// x / sqrt(mean(x^2) + eps) * w (Qwen3 RMSNorm) into the storage dtype that
// the next projection's TMA reads; one CTA of up to 1024 threads per row.

#include <algorithm>

#include "common.cuh"
#include "lsp_internal.h"

namespace lsp {

constexpr int kRowThreads = 256;
constexpr int kMaxPerThread = 32;   // H <= 8192

__device__ __forceinline__ float block_sum(float v, float* red) {
  v = warp_sum(v);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float s = 0.f;
  if (threadIdx.x < 32) {
    s = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
    s = warp_sum(s);
    if (threadIdx.x == 0) red[0] = s;
  }
  __syncthreads();
  s = red[0];
  __syncthreads();
  return s;
}

// four consecutive elements as fp32 (16-byte fp32 or 8-byte bf16 accesses)
__device__ __forceinline__ float4 ld4(const float* p, int i4) { return reinterpret_cast<const float4*>(p)[i4]; }
__device__ __forceinline__ float4 ld4(const bf16* p, int i4) {
  const uint2 r = reinterpret_cast<const uint2*>(p)[i4];
  const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r.x));
  const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r.y));
  return make_float4(a.x, a.y, b.x, b.y);
}
// A split-K partial is read once: streaming load (evict first in L1 and L2).
__device__ __forceinline__ float4 ld4_last(const float* p, int i4) { return __ldcs(reinterpret_cast<const float4*>(p) + i4); }
__device__ __forceinline__ void st4(float* p, int i4, float4 v) { reinterpret_cast<float4*>(p)[i4] = v; }
__device__ __forceinline__ void st4(bf16* p, int i4, float4 v) {
  const __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
  uint2 r;
  r.x = *reinterpret_cast<const uint32_t*>(&a);
  r.y = *reinterpret_cast<const uint32_t*>(&b);
  reinterpret_cast<uint2*>(p)[i4] = r;
}
__device__ __forceinline__ float4 add4(float4 a, float4 b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float dot4(float4 a) { return a.x * a.x + a.y * a.y + a.z * a.z + a.w * a.w; }

constexpr int kMaxVec = kMaxPerThread / 4;   // float4 per thread (H <= 8192)

template <typename T>
__global__ void __launch_bounds__(kRowThreads) combine_kernel(const CombineParams p) {
  __shared__ float red[32];
  __shared__ double inv_freq[128];
  griddep_launch();
  const int M = p.C * p.B;
  if ((int)blockIdx.x >= M) {
    // rotary table of request b: rope[b][i][f] = (cos, sin)(pos * theta^(-2f/d))
    const int b = blockIdx.x - M;
    const int half = p.d / 2;
    for (int f = threadIdx.x; f < half; f += blockDim.x)
      inv_freq[f] = pow(p.theta, -2.0 * (double)f / (double)p.d);
    __syncthreads();
    griddep_wait();
    const long long t0 = p.t[b];
    const double two_pi = 6.283185307179586476925286766559;
    for (int idx = threadIdx.x; idx < p.B * half; idx += blockDim.x) {
      const int i = idx / half, f = idx % half;
      const double ang = (double)(t0 + i) * inv_freq[f];
      const double red_ang = ang - rint(ang * (1.0 / two_pi)) * two_pi;
      float sn, cs;
      sincosf((float)red_ang, &sn, &cs);
      float* dst = p.rope + ((size_t)(b * p.B + i) * half + f) * 2;
      dst[0] = cs;
      dst[1] = sn;
    }
    return;
  }
  griddep_wait();
  const int m = blockIdx.x, b = m / p.B, i = m % p.B;
  int u = p.tokens[(size_t)b * p.B + i];
  const bool ok = (i == 0) ? (u >= 0 && u < p.V) : (u >= -1 && u < p.V);
  if (!ok) {
    if (threadIdx.x == 0) set_err(p.err, LSP_DEV_BAD_TOKEN);
    u = -1;
  }
  const T* src = u >= 0 ? static_cast<const T*>(p.embed) + (size_t)u * p.H
                        : static_cast<const T*>(p.mask_emb);
  const T* pos = static_cast<const T*>(p.pos) + (size_t)i * p.H;
  const size_t cstride = (size_t)p.C * p.H;
  // c_t split partials (absent with LSP_NO_BOUNDARY: c == nullptr, c_splits == 0)
  const float* c = p.c ? p.c + (size_t)b * p.H : nullptr;
  const int h4 = p.H / 4;
  float4 xv[kMaxVec];
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < kMaxVec; ++k) {
    const int j = threadIdx.x + k * kRowThreads;
    if (j < h4) {
      float4 cv = c ? ld4_last(c, j) : make_float4(0.f, 0.f, 0.f, 0.f);
      for (int s0 = 1; s0 < p.c_splits; s0 += 4) {
        float4 t[4];
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (s0 + u < p.c_splits) t[u] = ld4_last(c + (s0 + u) * cstride, j);
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (s0 + u < p.c_splits) cv = add4(cv, t[u]);
      }
      xv[k] = add4(add4(ld4(src, j), ld4(pos, j)), cv);
      st4(p.x + (size_t)m * p.H, j, xv[k]);
      ss += dot4(xv[k]);
    }
  }
  const float rstd = rsqrtf(block_sum(ss, red) / (float)p.H + p.eps);
  const T* w = static_cast<const T*>(p.norm_w);
  T* out = static_cast<T*>(p.xn) + (size_t)m * p.H;
#pragma unroll
  for (int k = 0; k < kMaxVec; ++k) {
    const int j = threadIdx.x + k * kRowThreads;
    if (j < h4) {
      const float4 wv = ld4(w, j);
      st4(out, j, make_float4(xv[k].x * rstd * wv.x, xv[k].y * rstd * wv.y, xv[k].z * rstd * wv.z,
                              xv[k].w * rstd * wv.w));
    }
  }
}

// One CTA of up to 512 threads per token row (two 16-byte vectors a thread
// at H = 4096): every partial load of a thread is in flight at once, and an SM
// keeps room (threads and registers) for a CTA of the projection launched
// after this kernel, which then starts its weight stream while the norm runs.
constexpr int kNormThreads = 512;

template <typename T, int VPT>
__global__ void __launch_bounds__(kNormThreads, 2)
    resid_norm_kernel(float* __restrict__ x, const float* __restrict__ part, int splits,
                      const T* __restrict__ w, T* __restrict__ out, int M, int H, float eps) {
  __shared__ float red[32];
  griddep_launch();
  const int m = blockIdx.x;
  const int h4 = H / 4;
  // the norm weight is a constant: load it before waiting for the producer
  float4 wv[VPT];
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int j = threadIdx.x + k * blockDim.x;
    if (j < h4) wv[k] = ld4(w, j);
  }
  griddep_wait();
  float* row = x + (size_t)m * H;
  const float* prow = part + (size_t)m * H;
  const size_t pstride = (size_t)M * H;
  float4 xv[VPT];
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int j = threadIdx.x + k * blockDim.x;
    if (j < h4) xv[k] = ld4(row, j);
  }
  // splits in groups with all loads of a group issued before the adds (in split order)
  constexpr int kGrp = VPT <= 1 ? 8 : VPT == 2 ? 4 : 2;
  for (int s0 = 0; s0 < splits; s0 += kGrp) {
    float4 t[VPT][kGrp];
#pragma unroll
    for (int k = 0; k < VPT; ++k) {
      const int j = threadIdx.x + k * blockDim.x;
#pragma unroll
      for (int u = 0; u < kGrp; ++u)
        if (j < h4 && s0 + u < splits) t[k][u] = ld4_last(prow + (s0 + u) * pstride, j);
    }
#pragma unroll
    for (int k = 0; k < VPT; ++k) {
      const int j = threadIdx.x + k * blockDim.x;
#pragma unroll
      for (int u = 0; u < kGrp; ++u)
        if (j < h4 && s0 + u < splits) xv[k] = add4(xv[k], t[k][u]);
    }
  }
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int j = threadIdx.x + k * blockDim.x;
    if (j < h4) {
      if (splits > 0) st4(row, j, xv[k]);
      ss += dot4(xv[k]);
    }
  }
  const float rstd = rsqrtf(block_sum(ss, red) / (float)H + eps);
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int j = threadIdx.x + k * blockDim.x;
    if (j < h4)
      st4(out + (size_t)m * H, j, make_float4(xv[k].x * rstd * wv[k].x, xv[k].y * rstd * wv[k].y,
                                              xv[k].z * rstd * wv[k].z, xv[k].w * rstd * wv[k].w));
  }
}

int launch_combine(const CombineParams& p, int dtype, cudaStream_t s) {
  if (p.H > kRowThreads * kMaxPerThread || p.d / 2 > 128) return LSP_ERR_SHAPE;
  const dim3 grid(p.C * p.B + p.C);
  cudaError_t e = dtype == LSP_DTYPE_BF16
                      ? launch_pdl(combine_kernel<bf16>, grid, dim3(kRowThreads), 0, s, p)
                      : launch_pdl(combine_kernel<float>, grid, dim3(kRowThreads), 0, s, p);
  return e == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

template <typename T>
static cudaError_t launch_norm_t(float* x, const float* part, int splits, const void* w, void* out, int M,
                                 int H, float eps, cudaStream_t s) {
  const int h4 = H / 4;
  const int threads = std::min(kNormThreads, (h4 + 31) / 32 * 32);
  const int vpt = (h4 + threads - 1) / threads;
  const T* wt = static_cast<const T*>(w);
  T* ot = static_cast<T*>(out);
  switch (vpt) {
    case 1: return launch_pdl(resid_norm_kernel<T, 1>, dim3(M), dim3(threads), 0, s, x, part, splits, wt, ot, M, H, eps);
    case 2: return launch_pdl(resid_norm_kernel<T, 2>, dim3(M), dim3(threads), 0, s, x, part, splits, wt, ot, M, H, eps);
    case 3: return launch_pdl(resid_norm_kernel<T, 3>, dim3(M), dim3(threads), 0, s, x, part, splits, wt, ot, M, H, eps);
    case 4: return launch_pdl(resid_norm_kernel<T, 4>, dim3(M), dim3(threads), 0, s, x, part, splits, wt, ot, M, H, eps);
    default: return cudaErrorInvalidValue;
  }
}

int launch_resid_norm(float* x, const float* part, int splits, const void* w, void* out, int M,
                      int H, float eps, int dtype, cudaStream_t s) {
  if (H > 4 * 4 * kNormThreads || H % 4) return LSP_ERR_SHAPE;
  const cudaError_t e = dtype == LSP_DTYPE_BF16
                            ? launch_norm_t<bf16>(x, part, splits, w, out, M, H, eps, s)
                            : launch_norm_t<float>(x, part, splits, w, out, M, H, eps, s);
  return e == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

}  // namespace lsp
