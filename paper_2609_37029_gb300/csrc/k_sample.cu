// Markov correction + sequential proposal sampling (Eq. markov,
// Eq. proposal-factorization):  for i = 1..B in order,
//     z_i = z_i^(0) + W_c E_c(y_{i-1}),   y_0 = a,
//     y_i = argmax_v z_i[v]                      (temperature 0, greedy)
//     y_i = argmax_v (z_i[v] / T + g_{b,i,v})    (T > 0, Gumbel-max == sampling softmax(z_i / T))
// with g = -log(-log u) from Philox4x32-10 (Salmon et al., SC'11).
//
// One launch per step i: every CTA first finishes step i-1's argmax from the
// per-CTA partials (so y_{i-1} is known everywhere), gathers E_c(y_{i-1}) of
// all C requests into shared memory, then sweeps its share of 16-row vocabulary
// tiles: the correction W_c[v0:v0+16] E_c^T is one mma.sync tile per warp
// (bf16 in, fp32 accumulate; fp32 storage uses FMA), the corrected logits are
// read/written as float4, one Philox call feeds four vocabulary entries, and
// a per-lane running argmax (ties to the lowest index) is reduced to one
// partial per CTA and request.  A last tiny launch resolves y_B.
#include <algorithm>

#include "common.cuh"
#include "lsp_internal.h"

namespace lsp {

constexpr int kSampThreads = 256;
constexpr int kSampWarps = kSampThreads / 32;
constexpr int kMaxC = 64;
constexpr int kMaxPartialsPerLane = 16;    // sampler grids of up to 512 CTAs

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
  const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;
  const uint32_t W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t hi0 = __umulhi(M0, c.x), lo0 = M0 * c.x;
    const uint32_t hi1 = __umulhi(M1, c.z), lo1 = M1 * c.z;
    c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
    k.x += W0;
    k.y += W1;
  }
  return c;
}

// g = -log(-log u): the inner log keeps full relative accuracy (u can be within
// 2^-24 of 1, where -log u is tiny); the outer log only needs absolute accuracy.
__device__ __forceinline__ float gumbel_of(uint32_t x) {
  const float u = ((float)(x >> 9) + 0.5f) * 1.1920928955078125e-07f;   // 2^-23
  return -__logf(-logf(u));
}

__device__ __forceinline__ bool better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}

__device__ __forceinline__ void mma_bf16_s(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9},"
      " {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// argmax over the previous step's per-CTA partials of request b (one warp);
// partials are laid out [buf][b][block] so the lanes read consecutive blocks.
__device__ __forceinline__ int resolve_prev(const SampleParams& p, int buf, int b, int lane) {
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  const float* pv = p.part_val + ((size_t)buf * p.C + b) * p.nblk;
  const int* pi = p.part_idx + ((size_t)buf * p.C + b) * p.nblk;
  // every load in flight before the first compare (nblk <= 32 * kMaxPartialsPerLane)
  float v[kMaxPartialsPerLane];
  int ix[kMaxPartialsPerLane];
#pragma unroll
  for (int k = 0; k < kMaxPartialsPerLane; ++k) {
    const int g = lane + 32 * k;
    v[k] = g < p.nblk ? pv[g] : -INFINITY;
    ix[k] = g < p.nblk ? pi[g] : 0x7fffffff;
  }
#pragma unroll
  for (int k = 0; k < kMaxPartialsPerLane; ++k)
    if (better(v[k], ix[k], bv, bi)) { bv = v[k]; bi = ix[k]; }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (better(ov, oi, bv, bi)) { bv = ov; bi = oi; }
  }
  return bi;
}

// KG = ceil(4 * C / 32): groups of four vocabulary entries each lane handles per tile.
template <typename T, int KG>
__global__ void __launch_bounds__(kSampThreads, 2) sample_step_kernel(const SampleParams p, const int step) {
  extern __shared__ __align__(16) uint8_t ssm_raw[];
  const int C = p.C, rc = p.rc;
  const int C8 = (C + 7) / 8 * 8;
  const int lde = rc + 8;                                   // padded row (elements)
  int* yprev = reinterpret_cast<int*>(ssm_raw);             // [kMaxC]
  float* red_v = reinterpret_cast<float*>(yprev + kMaxC);   // [warps][C]
  int* red_i = reinterpret_cast<int*>(red_v + kSampWarps * kMaxC);
  float* corr_s = reinterpret_cast<float*>(red_i + kSampWarps * kMaxC);   // [warps][C][17]
  T* e_s = reinterpret_cast<T*>(corr_s + kSampWarps * kMaxC * 17);        // [C8][lde]
  // per-warp double buffer of the 16 W_c rows of the current / next tile (bf16 path)
  bf16* wbuf = reinterpret_cast<bf16*>(e_s + (size_t)kMaxC * lde) + (size_t)(threadIdx.x >> 5) * 2 * 16 * lde;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  griddep_launch();
  griddep_wait();

  // ---- y_{i-1} for every request
  if (step == 0) {
    for (int b = tid; b < C; b += kSampThreads) {
      int y = p.prev[(size_t)b * p.prev_stride];
      if (y < 0 || y >= p.V) {
        if (blockIdx.x == 0) set_err(p.err, LSP_DEV_BAD_TOKEN);
        y = 0;
      }
      yprev[b] = y;
    }
  } else {
    for (int b = warp; b < C; b += kSampWarps) {
      const int y = resolve_prev(p, (step - 1) & 1, b, lane);
      if (lane == 0) {
        yprev[b] = y;
        if (blockIdx.x == 0) p.out_tokens[(size_t)b * p.B + step - 1] = y;
      }
    }
  }
  __syncthreads();
  // ---- E_c(y_{i-1}) rows
  const T* Ec = static_cast<const T*>(p.Ec);
  for (int idx = tid; idx < C8 * rc; idx += kSampThreads) {
    const int b = idx / rc, r = idx % rc;
    e_s[b * lde + r] = b < C ? Ec[(size_t)yprev[b] * rc + r] : from_f<T>(0.f);
  }
  __syncthreads();

  const T* Wc = static_cast<const T*>(p.Wc);
  const uint2 key = make_uint2((uint32_t)p.seed, (uint32_t)(p.seed >> 32));
  const bool sample = p.temperature > 0.f;
  const float inv_temp = sample ? 1.0f / p.temperature : 1.0f;   // exact for T = 1
  float* cw = corr_s + (size_t)warp * kMaxC * 17;
  float bv[KG];
  int bi[KG];
#pragma unroll
  for (int k = 0; k < KG; ++k) { bv[k] = -INFINITY; bi[k] = 0x7fffffff; }

  const int ntiles = p.V / 16;
  const int stride = gridDim.x * kSampWarps;
  auto zoff = [&](int tile, int k) {
    const int gi = lane + 32 * k;
    return ((size_t)(gi >> 2) * p.B + step) * p.V + tile * 16 + 4 * (gi & 3);
  };
  float4 zc[KG], zn[KG];
  int tile = blockIdx.x * kSampWarps + warp;
  // the 16 W_c rows of a tile -> this warp's buffer `buf` (16-byte cp.async chunks)
  auto stage_wc = [&](int t, int buf) {
    if constexpr (sizeof(T) == 2) {
      if (t < ntiles) {
        const int chunks = 16 * rc / 8;
        for (int c = lane; c < chunks; c += 32) {
          const int r = c / (rc / 8), e = (c % (rc / 8)) * 8;
          const bf16* src = reinterpret_cast<const bf16*>(Wc) + (size_t)(t * 16 + r) * rc + e;
          bf16* dst = wbuf + (size_t)buf * 16 * lde + (size_t)r * lde + e;
          asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
        }
      }
      asm volatile("cp.async.commit_group;" ::: "memory");
    }
  };
  stage_wc(tile, 0);
#pragma unroll
  for (int k = 0; k < KG; ++k)
    if (tile < ntiles && lane + 32 * k < 4 * C) zc[k] = *reinterpret_cast<const float4*>(p.src + zoff(tile, k));
  int cur = 0;
  for (; tile < ntiles; tile += stride, cur ^= 1) {
    const int next = tile + stride;
    stage_wc(next, cur ^ 1);
#pragma unroll
    for (int k = 0; k < KG; ++k)
      if (next < ntiles && lane + 32 * k < 4 * C) zn[k] = *reinterpret_cast<const float4*>(p.src + zoff(next, k));
    const int v0 = tile * 16;
    // correction W_c[v0:v0+16] . E_c(y)^T for all requests -> cw[b][v]
    if constexpr (sizeof(T) == 2) {
      asm volatile("cp.async.wait_group 1;" ::: "memory");   // this tile's rows have landed
      __syncwarp();
      const bf16* es = reinterpret_cast<const bf16*>(e_s);
      const bf16* wr = wbuf + (size_t)cur * 16 * lde + (size_t)(lane >> 2) * lde + (lane & 3) * 2;
      float acc[KG][4];                                     // KG = ceil(C / 8) n-tiles of 8 requests
#pragma unroll
      for (int nt = 0; nt < KG; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.f;
      for (int kk = 0; kk < rc / 16; ++kk) {
        uint32_t a[4];
        a[0] = *reinterpret_cast<const uint32_t*>(wr + kk * 16);
        a[1] = *reinterpret_cast<const uint32_t*>(wr + 8 * lde + kk * 16);
        a[2] = *reinterpret_cast<const uint32_t*>(wr + kk * 16 + 8);
        a[3] = *reinterpret_cast<const uint32_t*>(wr + 8 * lde + kk * 16 + 8);
#pragma unroll
        for (int nt = 0; nt < KG; ++nt) {
          const bf16* er = es + (size_t)(nt * 8 + (lane >> 2)) * lde + (lane & 3) * 2 + kk * 16;
          mma_bf16_s(acc[nt], a, *reinterpret_cast<const uint32_t*>(er),
                     *reinterpret_cast<const uint32_t*>(er + 8));
        }
      }
#pragma unroll
      for (int nt = 0; nt < KG; ++nt) {
        const int bcol = nt * 8 + (lane & 3) * 2, vr = lane >> 2;
        if (bcol < C) { cw[bcol * 17 + vr] = acc[nt][0]; cw[bcol * 17 + vr + 8] = acc[nt][2]; }
        if (bcol + 1 < C) { cw[(bcol + 1) * 17 + vr] = acc[nt][1]; cw[(bcol + 1) * 17 + vr + 8] = acc[nt][3]; }
      }
    } else {
      for (int idx = lane; idx < 16 * C; idx += 32) {
        const int v = idx & 15, b = idx >> 4;
        const T* wrow = Wc + (size_t)(v0 + v) * rc;
        const T* er = e_s + (size_t)b * lde;
        float acc = 0.f;
        for (int r = 0; r < rc; ++r) acc = fmaf(to_f(wrow[r]), to_f(er[r]), acc);
        cw[b * 17 + v] = acc;
      }
    }
    __syncwarp();
    // corrected logits, noise and running argmax: lane handles groups of 4 entries
#pragma unroll
    for (int k = 0; k < KG; ++k) {
      const int gi = lane + 32 * k;
      if (gi < 4 * C) {
        const int b = gi >> 2, vq = gi & 3;
        const int v = v0 + 4 * vq;
        float4 z = zc[k];
        z.x += cw[b * 17 + 4 * vq + 0];
        z.y += cw[b * 17 + 4 * vq + 1];
        z.z += cw[b * 17 + 4 * vq + 2];
        z.w += cw[b * 17 + 4 * vq + 3];
        if (p.dst) *reinterpret_cast<float4*>(p.dst + zoff(tile, k)) = z;
        float sc[4] = {z.x, z.y, z.z, z.w};
        if (sample) {
          const uint4 x = philox4x32_10(make_uint4((uint32_t)(v >> 2), (uint32_t)step, (uint32_t)b, p.round), key);
          sc[0] = sc[0] * inv_temp + gumbel_of(x.x);
          sc[1] = sc[1] * inv_temp + gumbel_of(x.y);
          sc[2] = sc[2] * inv_temp + gumbel_of(x.z);
          sc[3] = sc[3] * inv_temp + gumbel_of(x.w);
        }
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (better(sc[e], v + e, bv[k], bi[k])) { bv[k] = sc[e]; bi[k] = v + e; }
      }
    }
    __syncwarp();                                           // wbuf[cur] is refilled next iteration
#pragma unroll
    for (int k = 0; k < KG; ++k) zc[k] = zn[k];
  }
  if constexpr (sizeof(T) == 2) asm volatile("cp.async.wait_all;" ::: "memory");

  // ---- per-CTA partial argmax of every request
#pragma unroll
  for (int k = 0; k < KG; ++k) {
#pragma unroll
    for (int o = 1; o <= 2; o <<= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv[k], o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi[k], o);
      if (better(ov, oi, bv[k], bi[k])) { bv[k] = ov; bi[k] = oi; }
    }
    const int b = (lane >> 2) + 8 * k;
    if ((lane & 3) == 0 && b < C) {
      red_v[warp * kMaxC + b] = bv[k];
      red_i[warp * kMaxC + b] = bi[k];
    }
  }
  __syncthreads();
  for (int b = tid; b < C; b += kSampThreads) {
    float v = red_v[b];
    int i = red_i[b];
    for (int w = 1; w < kSampWarps; ++w)
      if (better(red_v[w * kMaxC + b], red_i[w * kMaxC + b], v, i)) {
        v = red_v[w * kMaxC + b];
        i = red_i[w * kMaxC + b];
      }
    const size_t o = ((size_t)(step & 1) * C + b) * p.nblk + blockIdx.x;
    p.part_val[o] = v;
    p.part_idx[o] = i;
  }
}

__global__ void __launch_bounds__(kSampThreads) sample_final_kernel(const SampleParams p) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  griddep_launch();
  griddep_wait();
  for (int b = warp; b < p.C; b += kSampWarps) {
    const int y = resolve_prev(p, (p.B - 1) & 1, b, lane);
    if (lane == 0) p.out_tokens[(size_t)b * p.B + p.B - 1] = y;
  }
}

__global__ void philox_words_kernel(uint64_t seed, uint32_t round, uint32_t b, uint32_t i,
                                    uint32_t* out, int count) {
  const int n = blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= count) return;
  const uint4 x = philox4x32_10(make_uint4((uint32_t)(n >> 2), i, b, round),
                                make_uint2((uint32_t)seed, (uint32_t)(seed >> 32)));
  const int w = n & 3;
  out[n] = w == 0 ? x.x : w == 1 ? x.y : w == 2 ? x.z : x.w;
}

int sample_blocks(int num_sms) { return std::min(2 * num_sms, 32 * kMaxPartialsPerLane); }

static size_t sample_smem(int rc, int es) {
  return kMaxC * sizeof(int) + 2 * kSampWarps * kMaxC * sizeof(float) +
         (size_t)kSampWarps * kMaxC * 17 * sizeof(float) + (size_t)kMaxC * (rc + 8) * es +
         (size_t)kSampWarps * 2 * 16 * (rc + 8) * 2;
}

template <typename T, int KG>
static cudaError_t launch_step(const SampleParams& p, int step, size_t smem, cudaStream_t s) {
  static size_t attr = 0;                 // largest dynamic shared memory granted so far
  if (smem > attr) {
    const cudaError_t e = cudaFuncSetAttribute(sample_step_kernel<T, KG>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr = smem;
  }
  return launch_pdl(sample_step_kernel<T, KG>, dim3(p.nblk), dim3(kSampThreads), smem, s, p, step);
}

int launch_sample(const SampleParams& p, int dtype, cudaStream_t s) {
  if (p.C > kMaxC || p.V % 16 || p.rc % 16 || p.rc > 256) return LSP_ERR_SHAPE;
  if (p.nblk > 32 * kMaxPartialsPerLane) return LSP_ERR_SHAPE;
  const int es = dtype == LSP_DTYPE_BF16 ? 2 : 4;
  const size_t smem = sample_smem(p.rc, es);
  if (smem > 227 * 1024) return LSP_ERR_SHAPE;

  const int kg = (4 * p.C + 31) / 32;
  for (int step = 0; step < p.B; ++step) {
    cudaError_t e;
    if (dtype == LSP_DTYPE_BF16)
      e = kg <= 1 ? launch_step<bf16, 1>(p, step, smem, s)
        : kg <= 2 ? launch_step<bf16, 2>(p, step, smem, s)
        : kg <= 4 ? launch_step<bf16, 4>(p, step, smem, s)
                  : launch_step<bf16, 8>(p, step, smem, s);
    else
      e = kg <= 1 ? launch_step<float, 1>(p, step, smem, s)
        : kg <= 2 ? launch_step<float, 2>(p, step, smem, s)
        : kg <= 4 ? launch_step<float, 4>(p, step, smem, s)
                  : launch_step<float, 8>(p, step, smem, s);
    if (e != cudaSuccess) return LSP_ERR_CUDA;
  }
  if (launch_pdl(sample_final_kernel, dim3(1), dim3(kSampThreads), 0, s, p) != cudaSuccess)
    return LSP_ERR_CUDA;
  return LSP_OK;
}

int launch_philox_words(uint64_t seed, uint32_t round, uint32_t b, uint32_t i, uint32_t* out,
                        int count, cudaStream_t s) {
  if (count <= 0) return LSP_OK;
  philox_words_kernel<<<(count + 255) / 256, 256, 0, s>>>(seed, round, b, i, out, count);
  return cudaGetLastError() == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

}  // namespace lsp
