// Small fused row ops of the drafter forward.
//
// combine_kernel (Sec. 2.3, input slots): x_i = E[u_i] + P_i + c_t with u_0 = a
// (the committed token) and the mask embedding for slots holding -1, written
// to the fp32 residual stream, fused with the first layer's input RMSNorm; the
// same launch fills the rotary cos/sin table of every (request, slot) at
// absolute position t + i, with the angle formed and reduced in fp64 so that
// positions near 1.3e5 keep full fp32 accuracy.
//
// rmsnorm_kernel: x / sqrt(mean(x^2) + eps) * w (Qwen3 RMSNorm) of fp32 rows
// into the storage dtype that the next projection's TMA reads.
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

template <typename T>
__global__ void __launch_bounds__(kRowThreads) combine_kernel(const CombineParams p) {
  __shared__ float red[32];
  const int M = p.C * p.B;
  if ((int)blockIdx.x >= M) {
    // rotary table of request b: rope[b][i][f] = (cos, sin)(pos * theta^(-2f/d))
    const int b = blockIdx.x - M;
    const int half = p.d / 2;
    const long long t0 = p.t[b];
    for (int idx = threadIdx.x; idx < p.B * half; idx += blockDim.x) {
      const int i = idx / half, f = idx % half;
      const double inv = pow(p.theta, -2.0 * (double)f / (double)p.d);
      const double ang = (double)(t0 + i) * inv;
      double sn, cs;
      sincos(ang, &sn, &cs);
      float* dst = p.rope + ((size_t)(b * p.B + i) * half + f) * 2;
      dst[0] = (float)cs;
      dst[1] = (float)sn;
    }
    return;
  }
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
  const float* c = p.c + (size_t)b * p.H;
  float xv[kMaxPerThread];
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < kMaxPerThread; ++k) {
    const int h = threadIdx.x + k * kRowThreads;
    xv[k] = 0.f;
    if (h < p.H) {
      xv[k] = to_f(src[h]) + to_f(pos[h]) + c[h];
      p.x[(size_t)m * p.H + h] = xv[k];
      ss += xv[k] * xv[k];
    }
  }
  const float rstd = rsqrtf(block_sum(ss, red) / (float)p.H + p.eps);
  const T* w = static_cast<const T*>(p.norm_w);
  T* out = static_cast<T*>(p.xn) + (size_t)m * p.H;
#pragma unroll
  for (int k = 0; k < kMaxPerThread; ++k) {
    const int h = threadIdx.x + k * kRowThreads;
    if (h < p.H) out[h] = from_f<T>(xv[k] * rstd * to_f(w[h]));
  }
}

template <typename T>
__global__ void __launch_bounds__(kRowThreads)
    rmsnorm_kernel(const float* __restrict__ x, const T* __restrict__ w, T* __restrict__ out, int H,
                   float eps) {
  __shared__ float red[32];
  const int m = blockIdx.x;
  const float* row = x + (size_t)m * H;
  float xv[kMaxPerThread];
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < kMaxPerThread; ++k) {
    const int h = threadIdx.x + k * kRowThreads;
    xv[k] = h < H ? row[h] : 0.f;
    ss += xv[k] * xv[k];
  }
  const float rstd = rsqrtf(block_sum(ss, red) / (float)H + eps);
#pragma unroll
  for (int k = 0; k < kMaxPerThread; ++k) {
    const int h = threadIdx.x + k * kRowThreads;
    if (h < H) out[(size_t)m * H + h] = from_f<T>(xv[k] * rstd * to_f(w[h]));
  }
}

int launch_combine(const CombineParams& p, int dtype, cudaStream_t s) {
  if (p.H > kRowThreads * kMaxPerThread) return LSP_ERR_SHAPE;
  const dim3 grid(p.C * p.B + p.C);
  if (dtype == LSP_DTYPE_BF16)
    combine_kernel<bf16><<<grid, kRowThreads, 0, s>>>(p);
  else
    combine_kernel<float><<<grid, kRowThreads, 0, s>>>(p);
  return cudaGetLastError() == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

int launch_rmsnorm(const float* x, const void* w, void* out, int M, int H, float eps, int dtype,
                   cudaStream_t s) {
  if (H > kRowThreads * kMaxPerThread) return LSP_ERR_SHAPE;
  if (dtype == LSP_DTYPE_BF16)
    rmsnorm_kernel<bf16><<<M, kRowThreads, 0, s>>>(x, static_cast<const bf16*>(w),
                                                   static_cast<bf16*>(out), H, eps);
  else
    rmsnorm_kernel<float><<<M, kRowThreads, 0, s>>>(x, static_cast<const float*>(w),
                                                    static_cast<float*>(out), H, eps);
  return cudaGetLastError() == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

}  // namespace lsp
