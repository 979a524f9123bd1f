// Markov correction + sequential proposal sampling (Eq. markov,
// Eq. proposal-factorization):  for i = 1..B in order,
//     z_i = z_i^(0) + W_c E_c(y_{i-1}),   y_0 = a,
//     y_i = argmax_v z_i[v]                      (temperature 0, greedy)
//     y_i = argmax_v (z_i[v] / T + g_{b,i,v})    (T > 0, Gumbel-max == sampling softmax(z_i / T))
// with g = -log(-log u) from Philox4x32-10 (Salmon et al., SC'11).
//
// Two kernels compute the same thing.
//
// sample_persistent_kernel (bf16, C <= 16, rc in {32, 64}, vocabulary slice
// fits shared memory): one cooperative launch for all B steps, one CTA per SM.
// Each CTA owns a contiguous slice of 16-row vocabulary tiles and keeps its
// W_c rows resident in shared memory for the whole launch.  Sixteen compute
// warps form the correction as mma.sync tiles with the requests on M (16) and
// the vocabulary on N, add the base logits (staged one step ahead by
// cp.async), add the noise and keep a running argmax.  A control warp
// publishes the CTA's best (value, index) of every request as one 64-bit
// atomicMax key, arrives on the step's counter, waits (bounded) for every CTA,
// reads y_i and gathers E_c(y_i) for the next step, while the compute warps
// draw the next step's noise.  The k index of the contraction is permuted
// identically in both operands so that each lane's operand words are
// contiguous in shared memory, and the vocabulary columns are permuted so that
// each lane's accumulators are four consecutive vocabulary entries (one
// Philox call, one float4 of logits).
//
// sample_step_kernel (every other shape): one launch per step i: every CTA
// first finishes step i-1's argmax from the per-CTA partials (so y_{i-1} is
// known everywhere), gathers E_c(y_{i-1}) of all C requests into shared
// memory, then sweeps its share of 16-row vocabulary tiles: the correction
// W_c[v0:v0+16] E_c^T is one mma.sync tile per warp (bf16 in, fp32
// accumulate; fp32 storage uses FMA), the corrected logits are read/written
// as float4, one Philox call feeds four vocabulary entries, and a per-lane
// running argmax (ties to the lowest index) is reduced to one partial per CTA
// and request.  A last tiny launch resolves y_B.
#include <algorithm>

#include "common.cuh"
#include "lsp_internal.h"

namespace lsp {

constexpr int kSampThreads = 256;
constexpr int kSampWarps = kSampThreads / 32;
constexpr int kMaxC = 64;
constexpr int kMaxPartialsPerLane = 16;    // sampler grids of up to 512 CTAs


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
          const uint4 x = philox4x32_10(make_uint4((uint32_t)(v >> 2), (uint32_t)step, (uint32_t)(p.b0 + b), p.round), key);
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

// ------------------------------------------------------------------ persistent kernel
constexpr int kPWarps = 16;                          // compute warps
constexpr int kPThreads = (kPWarps + 1) * 32;        // + the control warp
constexpr int kPTilesPerWarp = 4;
constexpr int kPMaxTiles = kPWarps * kPTilesPerWarp; // 64 tiles = 1024 vocabulary rows per CTA
constexpr int kPMaxC = 16;
constexpr int kSlotStride = 16;                      // u64 words between step keys: one 128-byte line
                                                     // per (step, request) spreads the atomics over L2
constexpr int kBarKeys = 1;                          // compute warps -> control warp: keys ready
constexpr int kBarNext = 2;                          // control warp -> compute warps: E_c(y_i) ready
constexpr int kBarPub = 3;                           // control warp -> compute warps: keys published (T = 0)

// Order-preserving 64-bit key of (value, index): a larger value wins, equal
// values go to the lower index; -0 ranks as +0.
__device__ __forceinline__ unsigned long long arg_key(float v, int i) {
  uint32_t u = __float_as_uint(v);
  if (u == 0x80000000u) u = 0u;
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ((unsigned long long)u << 32) | (uint32_t)~(uint32_t)i;
}

__device__ __forceinline__ unsigned long long max_u64(unsigned long long a, unsigned long long b) {
  return a > b ? a : b;
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src),
               "r"(src_bytes)
               : "memory");
}

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void red_release_add(unsigned* p, unsigned v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ void named_arrive(int id, int count) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Wait (every lane of a warp, same address) until *c >= target; false after kWaitLimitNs.
__device__ __forceinline__ bool wait_count(const unsigned* c, unsigned target) {
  if (ld_acquire_u32(c) >= target) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t i = 1;; ++i) {
    if (ld_acquire_u32(c) >= target) return true;
    if ((i & 63u) == 0 && global_ns() - t0 > kWaitLimitNs) return false;
  }
}

// Control warp: E_c rows of the current tokens (lane r < C holds y_r) into Es,
// 16-byte chunk c of row r stored at chunk c ^ (r & 1).
template <int CH>
__device__ __forceinline__ void gather_e(const bf16* Ec, int y, int C, int rc, uint8_t* Es, int lane) {
#pragma unroll
  for (int i0 = 0; i0 < kPMaxC * CH; i0 += 32) {
    const int i = i0 + lane, r = i / CH, c = i % CH;
    const int yr = __shfl_sync(0xffffffffu, y, r);
    if (r < C) {
      const uint4 v = *reinterpret_cast<const uint4*>(Ec + (size_t)yr * rc + c * 8);
      *reinterpret_cast<uint4*>(Es + r * (CH * 16) + ((c ^ (r & 1)) * 16)) = v;
    }
  }
}

// KS = rc / 16 k-steps of the m16n8k16 contraction.
// (17 warps of 32 threads: at 120 registers a thread the occupancy query
// reports no resident CTA, so the bound stays at 96 registers)
template <int KS>
__global__ void __launch_bounds__(kPThreads, 1)
    sample_persistent_kernel(const SampleParams p, const int ntiles) {
  constexpr int RB = KS * 32;        // bytes of one W_c / E_c row
  constexpr int CH = RB / 16;        // 16-byte chunks per row
  constexpr int TCH = KS / 2;        // chunks of one lane's k range
  extern __shared__ __align__(128) uint8_t psm[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nblk = gridDim.x;
  const int t_begin = (int)(((long long)blockIdx.x * ntiles) / nblk);
  const int cnt = (int)(((long long)(blockIdx.x + 1) * ntiles) / nblk) - t_begin;
  const int tpc = (ntiles + nblk - 1) / nblk;
  uint8_t* Ws = psm;                                                    // [tpc*16][RB]
  float4* Zs = reinterpret_cast<float4*>(psm + (size_t)tpc * 16 * RB);  // [tpc][2][32]
  uint8_t* Es = reinterpret_cast<uint8_t*>(Zs + (size_t)tpc * 64);      // [16][RB]
  unsigned long long* red = reinterpret_cast<unsigned long long*>(Es + kPMaxC * RB);   // [warps][16]
  volatile int* abort_flag = reinterpret_cast<volatile int*>(red + kPWarps * kPMaxC);
  unsigned long long* slots = p.sync;                                   // [B][16][kSlotStride]
  unsigned* counts = reinterpret_cast<unsigned*>(p.sync + (size_t)p.B * kPMaxC * kSlotStride);   // [B]
  const bf16* Wc = static_cast<const bf16*>(p.Wc);
  const bf16* Ec = static_cast<const bf16*>(p.Ec);
  const int C = p.C, B = p.B, V = p.V, rc = p.rc;
  const bool sample = p.temperature > 0.f;
  const float inv_temp = sample ? 1.0f / p.temperature : 1.0f;
  const uint2 key = make_uint2((uint32_t)p.seed, (uint32_t)(p.seed >> 32));
  const int g = lane >> 2, q = lane & 3;                               // mma group / thread in group

  // ---- prologue: W_c slice, zero E rows, step-0 logits, y_0, E_c(y_0)
  for (int i = tid; i < cnt * 16 * CH; i += kPThreads) {
    const int r = i / CH, c = i % CH;
    cp_async16(Ws + r * RB + ((c ^ (r & 1)) * 16), Wc + (size_t)(t_begin * 16 + r) * rc + c * 8, 16);
  }
  for (int i = tid; i < kPMaxC * RB / 16; i += kPThreads)
    reinterpret_cast<uint4*>(Es)[i] = make_uint4(0u, 0u, 0u, 0u);
  if (tid == 0) *abort_flag = 0;
  // E_c rows are gathered at random every step: keep the table in L2 (this CTA's share)
  if (tid == kPWarps * 32) {
    const size_t bytes = (size_t)V * rc * 2;
    const size_t share = (bytes / nblk + 4095) / 4096 * 4096;
    const size_t lo = share * blockIdx.x, hi = lo + share < bytes ? lo + share : bytes;
    const uint64_t pol = policy_evict_last();
    for (size_t o = lo; o < hi; o += 4096) {
      const uint32_t n = (uint32_t)(hi - o < 4096 ? hi - o : 4096);
      asm volatile("cp.async.bulk.prefetch.L2.global.L2::cache_hint [%0], %1, %2;" ::"l"(
                       reinterpret_cast<const char*>(Ec) + o),
                   "r"(n), "l"(pol)
                   : "memory");
    }
  }

  // this lane's own logits of step s for local tile lt (the same lane reads them)
  auto issue_z_tile = [&](int s, int lt) {
    const int v = (t_begin + lt) * 16 + 4 * q;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int r = g + 8 * h;
      const bool ok = r < C;
      cp_async16(&Zs[(lt * 2 + h) * 32 + lane], p.src + (ok ? ((size_t)r * B + s) * V + v : 0), ok ? 16u : 0u);
    }
  };
  float gn[kPTilesPerWarp][2][4];      // noise of the step about to be scored
  auto draw_noise_tile = [&](int s, int j, int lt) {
    const int v = (t_begin + lt) * 16 + 4 * q;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const uint4 x = philox4x32_10(make_uint4((uint32_t)(v >> 2), (uint32_t)s, (uint32_t)(p.b0 + g + 8 * h), p.round), key);
      gn[j][h][0] = gumbel_of(x.x);
      gn[j][h][1] = gumbel_of(x.y);
      gn[j][h][2] = gumbel_of(x.z);
      gn[j][h][3] = gumbel_of(x.w);
    }
  };

  int y = 0;                                                            // control warp: y of lane < C
  if (warp < kPWarps) {
#pragma unroll
    for (int j = 0; j < kPTilesPerWarp; ++j)
      if (warp + kPWarps * j < cnt) issue_z_tile(0, warp + kPWarps * j);
  } else {
    __syncwarp();
    if (lane < C) {
      y = p.prev[(size_t)lane * p.prev_stride];
      if (y < 0 || y >= V) {
        if (blockIdx.x == 0) set_err(p.err, LSP_DEV_BAD_TOKEN);
        y = 0;
      }
    }
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
  __syncthreads();                                                      // E rows zeroed
  if (warp == kPWarps) gather_e<CH>(Ec, y, C, rc, Es, lane);
  if (warp < kPWarps && sample) {
#pragma unroll
    for (int j = 0; j < kPTilesPerWarp; ++j)
      if (warp + kPWarps * j < cnt) draw_noise_tile(0, j, warp + kPWarps * j);
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  __syncthreads();                                                      // W_c slice and E_c(y_0) visible

  if (warp < kPWarps) {
    // ================= compute warps
    for (int s = 0; s < B; ++s) {
      // A operand: E_c(y) rows g and g + 8 over this lane's k range
      uint32_t a[KS][4];
      {
        uint32_t e0[2 * KS], e1[2 * KS];
#pragma unroll
        for (int c = 0; c < TCH; ++c) {
          const int pc = (TCH * q + c) ^ (g & 1);
          const uint4 u0 = *reinterpret_cast<const uint4*>(Es + g * RB + pc * 16);
          const uint4 u1 = *reinterpret_cast<const uint4*>(Es + (g + 8) * RB + pc * 16);
          e0[4 * c] = u0.x; e0[4 * c + 1] = u0.y; e0[4 * c + 2] = u0.z; e0[4 * c + 3] = u0.w;
          e1[4 * c] = u1.x; e1[4 * c + 1] = u1.y; e1[4 * c + 2] = u1.z; e1[4 * c + 3] = u1.w;
        }
#pragma unroll
        for (int ks = 0; ks < KS; ++ks) {
          a[ks][0] = e0[2 * ks];
          a[ks][1] = e1[2 * ks];
          a[ks][2] = e0[2 * ks + 1];
          a[ks][3] = e1[2 * ks + 1];
        }
      }
      asm volatile("cp.async.wait_all;" ::: "memory");                  // this lane's z_s landed
      const int v_first = (t_begin + warp) * 16 + 4 * q;
      float bv[2] = {-INFINITY, -INFINITY};
      int bi[2] = {v_first, v_first};
#pragma unroll
      for (int j = 0; j < kPTilesPerWarp; ++j) {
        const int lt = warp + kPWarps * j;
        if (lt >= cnt) break;                                           // warp-uniform
        const int v = (t_begin + lt) * 16 + 4 * q;
        float acc[2][4];
#pragma unroll
        for (int t = 0; t < 2; ++t) {
          // column n = g of n-tile t is vocabulary row 4 (g >> 1) + 2 t + (g & 1) of the tile
          const int row = lt * 16 + 4 * (g >> 1) + 2 * t + (g & 1);
          uint32_t bw[2 * KS];
#pragma unroll
          for (int c = 0; c < TCH; ++c) {
            const uint4 u = *reinterpret_cast<const uint4*>(Ws + row * RB + (((TCH * q + c) ^ (g & 1)) * 16));
            bw[4 * c] = u.x; bw[4 * c + 1] = u.y; bw[4 * c + 2] = u.z; bw[4 * c + 3] = u.w;
          }
          acc[t][0] = acc[t][1] = acc[t][2] = acc[t][3] = 0.f;
#pragma unroll
          for (int ks = 0; ks < KS; ++ks) mma_bf16_s(acc[t], a[ks], bw[2 * ks], bw[2 * ks + 1]);
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const float4 z = Zs[(lt * 2 + h) * 32 + lane];
          float zc[4] = {z.x + acc[0][2 * h], z.y + acc[0][2 * h + 1], z.z + acc[1][2 * h],
                         z.w + acc[1][2 * h + 1]};
          // corrected logits go out after the keys are published (below)
          if (p.dst) Zs[(lt * 2 + h) * 32 + lane] = make_float4(zc[0], zc[1], zc[2], zc[3]);
          if (sample) {
#pragma unroll
            for (int e = 0; e < 4; ++e) zc[e] = zc[e] * inv_temp + gn[j][h][e];
          }
#pragma unroll
          for (int e = 0; e < 4; ++e)
            if (zc[e] > bv[h]) { bv[h] = zc[e]; bi[h] = v + e; }
        }
      }
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        unsigned long long k = warp < cnt ? arg_key(bv[h], bi[h]) : 0ull;
        k = max_u64(k, __shfl_xor_sync(0xffffffffu, k, 1));
        k = max_u64(k, __shfl_xor_sync(0xffffffffu, k, 2));
        if (q == 0) red[warp * kPMaxC + g + 8 * h] = k;
      }
      named_arrive(kBarKeys, kPThreads);
      // HBM traffic of this lane (corrected logits out, next logits in) and the
      // next step's noise overlap the grid-wide wait; tile by tile, so that the
      // noise arithmetic of a tile runs while its memory operations drain
      // instead of the warp stalling on a full store queue.  Greedy (no noise):
      // the traffic waits until the control warp has published the step's keys,
      // so that the key atomics and their release do not queue behind it
      // (measured at the Qwen3-8B shape: 6.0 -> 5.3 us per step at T = 0; at
      // T = 1 the same wait, filled with noise, made the round 8 us slower).
      if (!sample) named_bar(kBarPub, kPThreads);
      const bool more = s + 1 < B;
#pragma unroll
      for (int j = 0; j < kPTilesPerWarp; ++j) {
        const int lt = warp + kPWarps * j;
        if (lt < cnt) {
          if (p.dst) {
            const int v = (t_begin + lt) * 16 + 4 * q;
#pragma unroll
            for (int h = 0; h < 2; ++h)
              if (g + 8 * h < C)
                *reinterpret_cast<float4*>(p.dst + ((size_t)(g + 8 * h) * B + s) * V + v) =
                    Zs[(lt * 2 + h) * 32 + lane];
          }
          if (more) {
            issue_z_tile(s + 1, lt);                                    // slot already consumed
            if (sample) draw_noise_tile(s + 1, j, lt);
          }
        }
      }
      if (!more) break;
      asm volatile("cp.async.commit_group;" ::: "memory");
      named_bar(kBarNext, kPThreads);
      if (*abort_flag) break;
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
    return;
  }

  // ================= control warp
  const size_t zrow = (size_t)cnt * 16 * sizeof(float);                  // this CTA's slice of one logits row
  for (int s = 0; s < B; ++s) {
    // pull the next step's logits slice into L2 while the compute warps score this one
    if (s + 1 < B && lane < C && zrow > 0)
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(
                       p.src + ((size_t)lane * B + s + 1) * V + (size_t)t_begin * 16),
                   "r"((uint32_t)zrow)
                   : "memory");
    named_bar(kBarKeys, kPThreads);
    if (lane < C) {
      unsigned long long k = 0ull;
#pragma unroll
      for (int w = 0; w < kPWarps; ++w) k = max_u64(k, red[w * kPMaxC + lane]);
      atomicMax(&slots[(s * kPMaxC + lane) * kSlotStride], k);
    }
    __syncwarp();
    if (lane == 0) red_release_add(&counts[s], 1u);                     // orders the warp's key atomics
    if (!sample) {
      __syncwarp();
      named_arrive(kBarPub, kPThreads);                                 // compute warps may store now
    }
    const bool last = s + 1 == B;
    if (last && blockIdx.x != 0) return;                                // only CTA 0 needs y_B
    const bool ok = __all_sync(0xffffffffu, wait_count(&counts[s], (unsigned)nblk));
    if (!ok) {
      if (lane == 0) set_err(p.err, LSP_DEV_TIMEOUT);
      if (!last) {
        if (lane == 0) *abort_flag = 1;
        __syncwarp();
        named_arrive(kBarNext, kPThreads);
      }
      return;
    }
    if (lane < C) {
      y = (int)~(uint32_t)ld_relaxed_u64(&slots[(s * kPMaxC + lane) * kSlotStride]);
      if (y < 0 || y >= V) {                                            // no key arrived: corrupt sync words
        set_err(p.err, LSP_DEV_TIMEOUT);
        y = 0;
      }
      if (blockIdx.x == 0) p.out_tokens[(size_t)lane * B + s] = y;
    }
    if (last) {
      // every CTA has arrived on every counter, so no one reads the sync words
      // again: leave them zero for the next launch
      __syncwarp();
      for (int i = lane; i < B * kPMaxC; i += 32) slots[i * kSlotStride] = 0ull;
      for (int i = lane; i < B; i += 32) counts[i] = 0u;
      return;
    }
    gather_e<CH>(Ec, y, C, rc, Es, lane);
    __syncwarp();
    named_arrive(kBarNext, kPThreads);
  }
}

// ------------------------------------------------------------------ persistent kernel, fp32 storage
// One cooperative launch for all B steps with fp32 W_c / E_c (the fp32
// reference shape): CTA k owns 16-row vocabulary tiles [t_begin, t_begin +
// cnt) and keeps their W_c rows resident in shared memory.  Per step, a warp
// takes one request at a time: its lanes form z = z^(0) + W_c[v] . E_c(y)
// (fp32 FMA) over the slice, write the corrected logits, add the noise and
// keep a running argmax, which the warp publishes as one 64-bit atomicMax key.
// Thread 0 then arrives on the step's counter (release) and waits, bounded,
// for every CTA; y_i is read back from the keys and E_c(y_i) gathered for the
// next step.  The synchronisation words are those of the bf16 kernel and are
// left zero at exit.
constexpr int kPfThreads = 256;

__global__ void __launch_bounds__(kPfThreads, 1)
    sample_persistent_f32_kernel(const SampleParams p, const int ntiles) {
  extern __shared__ __align__(16) float pfs[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, nw = kPfThreads / 32;
  const int nblk = gridDim.x;
  const int t_begin = (int)(((long long)blockIdx.x * ntiles) / nblk);
  const int cnt = (int)(((long long)(blockIdx.x + 1) * ntiles) / nblk) - t_begin;
  const int C = p.C, B = p.B, V = p.V, rc = p.rc;
  const int v0 = t_begin * 16, nv = cnt * 16;
  float* Ws = pfs;                                  // [nv][rc]
  float* Es = Ws + (size_t)nv * rc;                 // [C][rc]
  __shared__ int s_y[kPMaxC];
  __shared__ int s_ok;
  unsigned long long* slots = p.sync;
  unsigned* counts = reinterpret_cast<unsigned*>(p.sync + (size_t)B * kPMaxC * kSlotStride);
  const float* Wc = static_cast<const float*>(p.Wc);
  const float* Ec = static_cast<const float*>(p.Ec);
  const bool sample = p.temperature > 0.f;
  const float inv_temp = sample ? 1.0f / p.temperature : 1.0f;
  const uint2 key = make_uint2((uint32_t)p.seed, (uint32_t)(p.seed >> 32));

  for (int i = tid; i < nv * rc / 4; i += kPfThreads)
    reinterpret_cast<float4*>(Ws)[i] = reinterpret_cast<const float4*>(Wc + (size_t)v0 * rc)[i];
  if (tid < C) {
    int y = p.prev[(size_t)tid * p.prev_stride];
    if (y < 0 || y >= V) {
      if (blockIdx.x == 0) set_err(p.err, LSP_DEV_BAD_TOKEN);
      y = 0;
    }
    s_y[tid] = y;
  }
  __syncthreads();
  for (int s = 0; s < B; ++s) {
    for (int i = tid; i < C * rc; i += kPfThreads) Es[i] = Ec[(size_t)s_y[i / rc] * rc + i % rc];
    __syncthreads();
    for (int c = warp; c < C; c += nw) {
      const float* zr = p.src + ((size_t)c * B + s) * V;
      float bv = -INFINITY;
      int bi = 0x7fffffff;
      for (int v = v0 + lane; v < v0 + nv; v += 32) {
        const float* w = Ws + (size_t)(v - v0) * rc;
        const float* e = Es + (size_t)c * rc;
        float corr = 0.f;
        for (int r = 0; r < rc; r += 4) {
          const float4 a = *reinterpret_cast<const float4*>(w + r), b = *reinterpret_cast<const float4*>(e + r);
          corr = fmaf(a.x, b.x, corr);
          corr = fmaf(a.y, b.y, corr);
          corr = fmaf(a.z, b.z, corr);
          corr = fmaf(a.w, b.w, corr);
        }
        const float z = zr[v] + corr;
        if (p.dst) p.dst[((size_t)c * B + s) * V + v] = z;
        float sc = z;
        if (sample) {
          const uint4 x = philox4x32_10(make_uint4((uint32_t)(v >> 2), (uint32_t)s, (uint32_t)(p.b0 + c), p.round), key);
          const uint32_t wd = (v & 3) == 0 ? x.x : (v & 3) == 1 ? x.y : (v & 3) == 2 ? x.z : x.w;
          sc = z * inv_temp + gumbel_of(wd);
        }
        if (better(sc, v, bv, bi)) { bv = sc; bi = v; }
      }
      unsigned long long k = nv > 0 && bi != 0x7fffffff ? arg_key(bv, bi) : 0ull;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) k = max_u64(k, __shfl_xor_sync(0xffffffffu, k, o));
      if (lane == 0 && k) atomicMax(&slots[(s * kPMaxC + c) * kSlotStride], k);
    }
    __syncthreads();                                // this CTA's keys of step s are published
    const bool last = s + 1 == B;
    if (tid == 0) {
      red_release_add(&counts[s], 1u);
      s_ok = (last && blockIdx.x != 0) ? 1 : (wait_count(&counts[s], (unsigned)nblk) ? 1 : 0);
      if (!s_ok) set_err(p.err, LSP_DEV_TIMEOUT);
    }
    __syncthreads();
    if (!s_ok || (last && blockIdx.x != 0)) return;   // only CTA 0 needs y_B
    if (tid < C) {
      int y = (int)~(uint32_t)ld_relaxed_u64(&slots[(s * kPMaxC + tid) * kSlotStride]);
      if (y < 0 || y >= V) {                          // no key arrived: corrupt sync words
        set_err(p.err, LSP_DEV_TIMEOUT);
        y = 0;
      }
      s_y[tid] = y;
      if (blockIdx.x == 0) p.out_tokens[(size_t)tid * B + s] = y;
    }
    __syncthreads();
  }
  // CTA 0 after the last step: every CTA has arrived on every counter, so no
  // one reads the sync words again -- leave them zero for the next launch
  for (int i = tid; i < B * kPMaxC; i += kPfThreads) slots[i * kSlotStride] = 0ull;
  for (int i = tid; i < B; i += kPfThreads) counts[i] = 0u;
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

size_t sample_sync_bytes(int B) {
  return ((size_t)B * kPMaxC * kSlotStride * sizeof(unsigned long long) + (size_t)B * sizeof(unsigned) +
          255) / 256 * 256;
}

static size_t persistent_smem(int tpc, int rc) {
  const size_t rb = (size_t)rc * 2;
  return (size_t)tpc * 16 * rb + (size_t)tpc * 64 * 16 + kPMaxC * rb +
         (size_t)kPWarps * kPMaxC * sizeof(unsigned long long) + 16;
}

template <int KS>
static int launch_persistent(const SampleParams& p, cudaStream_t s) {
  const int ntiles = p.V / 16;
  const int nblk = std::min(p.num_sms, ntiles);
  const int tpc = (ntiles + nblk - 1) / nblk;
  if (tpc > kPMaxTiles) return LSP_ERR_SHAPE;
  const size_t smem = persistent_smem(tpc, p.rc);
  if (smem > 227 * 1024) return LSP_ERR_SHAPE;
  static size_t attr = 0;
  if (smem > attr) {
    if (cudaFuncSetAttribute(sample_persistent_kernel<KS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem) != cudaSuccess)
      return LSP_ERR_CUDA;
    attr = smem;
  }
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, sample_persistent_kernel<KS>, kPThreads,
                                                    smem) != cudaSuccess)
    return LSP_ERR_CUDA;
  if (per_sm < 1) return LSP_ERR_SHAPE;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(nblk);
  cfg.blockDim = dim3(kPThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr_c[1];
  attr_c[0].id = cudaLaunchAttributeCooperative;       // every CTA resident: the step waits are safe
  attr_c[0].val.cooperative = 1;
  cfg.attrs = attr_c;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, sample_persistent_kernel<KS>, p, ntiles) == cudaSuccess ? LSP_OK
                                                                                          : LSP_ERR_CUDA;
}

// The persistent kernel's shape limits (anything else takes the per-step kernel).
static size_t persistent_f32_smem(int tpc, int rc) { return ((size_t)tpc * 16 + kPMaxC) * rc * sizeof(float); }

static bool coop_ok() {
  int dev = 0, coop = 0;
  return cudaGetDevice(&dev) == cudaSuccess &&
         cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev) == cudaSuccess && coop != 0;
}

// fp32 storage: the whole B-step loop in one cooperative launch when the W_c
// slice of a CTA fits shared memory.
static bool persistent_f32_ok(const SampleParams& p, int dtype) {
  if (dtype != LSP_DTYPE_F32 || p.C > kPMaxC || !p.sync || p.num_sms < 1 || p.rc % 4) return false;
  const int ntiles = p.V / 16;
  const int nblk = std::min(p.num_sms, ntiles);
  const int tpc = (ntiles + nblk - 1) / nblk;
  return persistent_f32_smem(tpc, p.rc) <= 200 * 1024 && coop_ok();
}

static int launch_persistent_f32(const SampleParams& p, cudaStream_t s) {
  const int ntiles = p.V / 16;
  const int nblk = std::min(p.num_sms, ntiles);
  const int tpc = (ntiles + nblk - 1) / nblk;
  const size_t smem = persistent_f32_smem(tpc, p.rc);
  static size_t attr = 0;
  if (smem > attr) {
    if (cudaFuncSetAttribute(sample_persistent_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem) != cudaSuccess)
      return LSP_ERR_CUDA;
    attr = smem;
  }
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, sample_persistent_f32_kernel, kPfThreads,
                                                    smem) != cudaSuccess)
    return LSP_ERR_CUDA;
  if (per_sm < 1) return LSP_ERR_SHAPE;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(nblk);
  cfg.blockDim = dim3(kPfThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr_c[1];
  attr_c[0].id = cudaLaunchAttributeCooperative;       // every CTA resident: the step waits are safe
  attr_c[0].val.cooperative = 1;
  cfg.attrs = attr_c;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, sample_persistent_f32_kernel, p, ntiles) == cudaSuccess ? LSP_OK
                                                                                         : LSP_ERR_CUDA;
}

static bool persistent_ok(const SampleParams& p, int dtype) {
  if (dtype != LSP_DTYPE_BF16 || p.C > kPMaxC || (p.rc != 32 && p.rc != 64) || !p.sync || p.num_sms < 1)
    return false;
  const int ntiles = p.V / 16;
  const int nblk = std::min(p.num_sms, ntiles);
  const int tpc = (ntiles + nblk - 1) / nblk;
  if (tpc > kPMaxTiles || persistent_smem(tpc, p.rc) > 227 * 1024) return false;
  return coop_ok();
}

// More than kPMaxC requests: the requests' proposal chains are independent,
// so the one-launch loop runs once per group of up to kPMaxC requests
// whenever every group fits it (the Philox counter keeps the global request
// index, so the draws are those of one launch over all requests); the
// per-step kernel covers all C otherwise.
static SampleParams request_group(const SampleParams& p, int g0) {
  SampleParams q = p;
  q.C = std::min(kPMaxC, p.C - g0);
  q.src = p.src + (size_t)g0 * p.B * p.V;
  if (p.dst) q.dst = p.dst + (size_t)g0 * p.B * p.V;
  q.prev = p.prev + (size_t)g0 * p.prev_stride;
  q.out_tokens = p.out_tokens + (size_t)g0 * p.B;
  q.b0 = p.b0 + g0;
  return q;
}

static int persistent_groups(const SampleParams& p, int dtype) {
  if (p.C <= kPMaxC) return persistent_ok(p, dtype) || persistent_f32_ok(p, dtype) ? 1 : 0;
  for (int g0 = 0; g0 < p.C; g0 += kPMaxC) {
    const SampleParams q = request_group(p, g0);
    if (!persistent_ok(q, dtype) && !persistent_f32_ok(q, dtype)) return 0;
  }
  return (p.C + kPMaxC - 1) / kPMaxC;
}

int sample_launches(const SampleParams& p, int dtype) {
  const int groups = persistent_groups(p, dtype);
  return groups > 0 ? groups : p.B + 1;
}

int launch_sample(const SampleParams& p, int dtype, cudaStream_t s) {
  if (p.C > kMaxC || p.V % 16 || p.rc % 16 || p.rc > 256) return LSP_ERR_SHAPE;
  // float4 / 16-byte accesses to the logits and the correction tables
  if ((reinterpret_cast<uintptr_t>(p.src) | reinterpret_cast<uintptr_t>(p.dst) |
       reinterpret_cast<uintptr_t>(p.Ec) | reinterpret_cast<uintptr_t>(p.Wc)) & 15)
    return LSP_ERR_ARG;
  if (persistent_groups(p, dtype) > 0) {
    for (int g0 = 0; g0 < p.C; g0 += kPMaxC) {
      const SampleParams q = request_group(p, g0);
      const int rc = persistent_ok(q, dtype) ? (q.rc == 32 ? launch_persistent<2>(q, s) : launch_persistent<4>(q, s))
                                             : launch_persistent_f32(q, s);
      if (rc != LSP_OK) return rc;
    }
    return LSP_OK;
  }

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
