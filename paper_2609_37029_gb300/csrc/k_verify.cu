// Target-side verification of the drafted blocks (Sec. 2.1): candidates y_i
// drawn from q_i are tested in order and y_i is accepted with probability
// alpha_i = min(1, p_i(y_i) / q_i(y_i)) (Eq. acceptance); at the first
// rejected position i a correction token is drawn from [p_i - q_i]_+ (Eq.
// residual); if all B are accepted, a bonus token is drawn from p_{B+1}.
// p_i = softmax(target logits_i / T), q_i = softmax(draft logits_i / T); T = 0
// is the greedy limit (accept y_i iff y_i = argmax p_i, emit argmax p_{r+1}).
//
// verify_stats_kernel: CTA (request, row, chunk) streams every logit row the
// decision needs and writes the chunk's partial: (max, sum of 2^x) of
// x = z log2(e) / T over the target and draft rows (T > 0), or the
// lowest-index argmax of the target rows (T = 0).  verify_greedy_kernel
// (T = 0): CTA per request -- merges the argmax partials and accepts the prefix
// of candidates equal to the target argmax.  verify_draw_kernel (T > 0): CTA
// (vocabulary chunk, request) -- merges the request's row partials, tests the
// B candidates one lane each (the acceptance uniforms are Philox words, so
// every CTA finds the same first rejected position j), takes the Gumbel-max
// of the correction or bonus draw over its chunk, and the CTA that finishes
// the request's last chunk merges the chunk winners (its counter resets
// itself).  One wave of draw CTAs pays the merge latency once.
//
// Randomness (Philox4x32-10, key = seed): the acceptance uniform of position i
// is word 0 of counter (0, 2^30 + i, b, round), u = ((x >> 9) + 1/2) 2^-23,
// accepted iff u q_i(y_i) < p_i(y_i); the draw at position i uses the words of
// counters (v >> 2, 2^31 + i, b, round), g_v = -log(-log u_v).  The drafter's
// counters have a second word < 2^30, so the streams never meet.
#include <algorithm>
#include <climits>


#include "common.cuh"
#include "lsp_internal.h"

namespace lsp {

constexpr int kVerThreads = 256;
constexpr uint32_t kAcceptStream = 1u << 30;
constexpr uint32_t kDrawStream = 1u << 31;
constexpr unsigned kFull = 0xffffffffu;
constexpr int kDrawBatch = 2;
constexpr int kDrawCtasPerSm = 5;     // float4 groups of both rows in flight per thread in the draw

__device__ __forceinline__ float ver_uniform(uint32_t x) {
  return ((float)(x >> 9) + 0.5f) * 1.1920928955078125e-07f;   // 2^-23
}

__device__ __forceinline__ bool ver_better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}

template <int W>
__device__ __forceinline__ void group_argmax(float& v, int& i) {
#pragma unroll
  for (int o = W / 2; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(kFull, v, o);
    const int oi = __shfl_xor_sync(kFull, i, o);
    if (ver_better(ov, oi, v, i)) { v = ov; i = oi; }
  }
}

// Rows of request b, r in [0, rpr): r <= B is target row (b, r); r > B is draft
// row (b, r - B - 1) (T > 0 only).  Chunk partials are [b][r][nst].
__device__ __forceinline__ const float* ver_row(const VerifyParams& p, int b, int r) {
  return r <= p.B ? p.zt + ((size_t)b * (p.B + 1) + r) * p.V
                  : p.zq + ((size_t)b * p.B + (r - p.B - 1)) * p.V;
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// base-2 log-sum-exp pair combine: (m, s) represents m + log2(s)
__device__ __forceinline__ void lse2_combine(float& m, float& s, float om, float os) {
  const float nm = fmaxf(m, om);
  s = (nm > -INFINITY) ? s * ex2(m - nm) + os * ex2(om - nm) : 0.f;
  m = nm;
}

template <int W>
__device__ __forceinline__ void group_lse2(float& m, float& s) {
#pragma unroll
  for (int o = W / 2; o > 0; o >>= 1)
    lse2_combine(m, s, __shfl_xor_sync(kFull, m, o), __shfl_xor_sync(kFull, s, o));
}

template <bool kGreedy, int kBatch>
__global__ void __launch_bounds__(kVerThreads) verify_stats_kernel(const VerifyParams p, const int rpr) {
  __shared__ float sv[32];
  __shared__ int si[32];
  // dependents launch only after this grid's inputs are complete: the draw
  // kernel reads the call's inputs before its own wait
  griddep_wait();
  griddep_launch();
  const int u = blockIdx.x;
  const int ch = u % p.nst, rr = u / p.nst;
  const int b = rr / rpr, r = rr - b * rpr;
  const int ng = p.V / 4;
  const int g0 = (int)((long long)ch * ng / p.nst), g1 = (int)((long long)(ch + 1) * ng / p.nst);
  const float4* z4 = reinterpret_cast<const float4*>(ver_row(p, b, r));
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float4 pad = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
  if (kGreedy) {
    float bv = -INFINITY;
    int bi = INT_MAX;
    for (int base = g0 + threadIdx.x; base < g1; base += kBatch * kVerThreads) {
      float4 x[kBatch];
#pragma unroll
      for (int k = 0; k < kBatch; ++k) {
        const int g = base + k * kVerThreads;
        x[k] = g < g1 ? __ldg(z4 + g) : pad;
      }
#pragma unroll
      for (int k = 0; k < kBatch; ++k) {
        // indices rise with (k, e) within a thread: a strict > keeps the lowest on ties
        const int v0 = 4 * (base + k * kVerThreads);
        if (x[k].x > bv) { bv = x[k].x; bi = v0; }
        if (x[k].y > bv) { bv = x[k].y; bi = v0 + 1; }
        if (x[k].z > bv) { bv = x[k].z; bi = v0 + 2; }
        if (x[k].w > bv) { bv = x[k].w; bi = v0 + 3; }
      }
    }
    group_argmax<32>(bv, bi);
    if (lane == 0) { sv[warp] = bv; si[warp] = bi; }
    __syncthreads();
    if (threadIdx.x == 0) {
      for (int w = 1; w < kVerThreads / 32; ++w)
        if (ver_better(sv[w], si[w], bv, bi)) { bv = sv[w]; bi = si[w]; }
      p.st_a[u] = bv;
      p.st_i[u] = bi;
    }
  } else {
    const float it2 = 1.4426950408889634f / p.temperature;   // log2(e) / T
    float m = -INFINITY, s = 0.f;
    for (int base = g0 + threadIdx.x; base < g1; base += kBatch * kVerThreads) {
      float4 x[kBatch];
#pragma unroll
      for (int k = 0; k < kBatch; ++k) {
        const int g = base + k * kVerThreads;
        x[k] = g < g1 ? __ldg(z4 + g) : pad;
      }
      float bm = -INFINITY;
#pragma unroll
      for (int k = 0; k < kBatch; ++k)
        bm = fmaxf(bm, fmaxf(fmaxf(x[k].x, x[k].y), fmaxf(x[k].z, x[k].w)));
      const float nm = fmaxf(m, bm * it2);
      if (nm > -INFINITY) {
        float acc = 0.f;
#pragma unroll
        for (int k = 0; k < kBatch; ++k)
          acc += ex2(fmaf(x[k].x, it2, -nm)) + ex2(fmaf(x[k].y, it2, -nm)) + ex2(fmaf(x[k].z, it2, -nm)) +
                 ex2(fmaf(x[k].w, it2, -nm));
        s = s * ex2(m - nm) + acc;
        m = nm;
      }
    }
    group_lse2<32>(m, s);
    if (lane == 0) { sv[warp] = m; reinterpret_cast<float*>(si)[warp] = s; }
    __syncthreads();
    if (threadIdx.x == 0) {
      for (int w = 1; w < kVerThreads / 32; ++w) lse2_combine(m, s, sv[w], reinterpret_cast<float*>(si)[w]);
      p.st_a[u] = m;
      p.st_b[u] = s;
    }
  }
}

// T = 0, CTA per request: argmax of each position (8 lanes per row), then the
// greedy prefix and the emitted token.
__global__ void __launch_bounds__(kVerThreads) verify_greedy_kernel(const VerifyParams p) {
  __shared__ int s_arg[kVerMaxB + 1];
  griddep_launch();
  griddep_wait();
  const int b = blockIdx.x, B = p.B, nst = p.nst, rpr = B + 1;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int grp = threadIdx.x >> 3, sub = threadIdx.x & 7;
  const size_t base = (size_t)b * rpr * nst;
  for (int r0 = 0; r0 < rpr; r0 += kVerThreads / 8) {
    const int r = r0 + grp;
    float v = -INFINITY;
    int i = INT_MAX;
    if (r < rpr)
      for (int k = sub; k < nst; k += 8)
        if (ver_better(p.st_a[base + (size_t)r * nst + k], p.st_i[base + (size_t)r * nst + k], v, i)) {
          v = p.st_a[base + (size_t)r * nst + k];
          i = p.st_i[base + (size_t)r * nst + k];
        }
    group_argmax<8>(v, i);
    if (r < rpr && sub == 0) s_arg[r] = i;
  }
  __syncthreads();
  if (warp != 0) return;
  for (int i0 = 0; i0 <= B; i0 += 32) {
    const int i = i0 + lane;
    bool stop = false;
    if (i < B) {
      const int y = p.y[(size_t)b * B + i];
      if (y < 0 || y >= p.V) set_err(p.err, LSP_DEV_BAD_TOKEN);
      stop = y != s_arg[i];
    } else if (i == B) {
      stop = true;
    }
    const unsigned m = __ballot_sync(kFull, stop);
    if (m) {
      const int j = i0 + __ffs(m) - 1;
      if (lane == 0) {
        p.accepted[b] = j;
        p.next_token[b] = s_arg[j] < p.V ? s_arg[j] : 0;
      }
      return;
    }
  }
}

// CTA (chunk, b), T > 0: decide j, then the Gumbel-max of the correction /
// bonus draw over the chunk's vocabulary; the last chunk merges the winners.
__global__ void __launch_bounds__(kVerThreads, kDrawCtasPerSm) verify_draw_kernel(const VerifyParams p) {
  __shared__ float s_lse[2 * kVerMaxB + 1];    // base-2 log-normalisers of the request's rows
  __shared__ float sv[32];
  __shared__ int si[32];
  __shared__ int s_j;
  __shared__ unsigned s_last;
  const int b = blockIdx.y, ch = blockIdx.x, nch = gridDim.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float it2 = 1.4426950408889634f / p.temperature;
  const uint2 key = make_uint2((uint32_t)p.seed, (uint32_t)(p.seed >> 32));
  const int B = p.B, nst = p.nst, rpr = 2 * B + 1;
  // candidate logits: inputs of the call, complete before the row pass began,
  // so they load while the row pass finishes
  float zy_t = 0.f, zy_q = 0.f;
  if (warp == 0 && lane < B) {
    int y = p.y[(size_t)b * B + lane];
    if (y < 0 || y >= p.V) {
      set_err(p.err, LSP_DEV_BAD_TOKEN);
      y = 0;
    }
    zy_t = p.zt[((size_t)b * (B + 1) + lane) * p.V + y];
    zy_q = p.zq[((size_t)b * B + lane) * p.V + y];
  }
  griddep_launch();
  griddep_wait();
  {
    const int grp = threadIdx.x >> 3, sub = threadIdx.x & 7;
    const size_t base = (size_t)b * rpr * nst;
    for (int r0 = 0; r0 < rpr; r0 += kVerThreads / 8) {
      const int r = r0 + grp;
      float m = -INFINITY, s = 0.f;
      if (r < rpr)
        for (int k = sub; k < nst; k += 8)
          lse2_combine(m, s, p.st_a[base + (size_t)r * nst + k], p.st_b[base + (size_t)r * nst + k]);
      group_lse2<8>(m, s);
      if (r < rpr && sub == 0) s_lse[r] = m + __log2f(s);
    }
  }
  __syncthreads();
  if (warp == 0) {
    int j = B;
    for (int i0 = 0; i0 < B; i0 += 32) {
      const int i = i0 + lane;
      bool rej = false;
      if (i < B) {
        float zt_i = zy_t, zq_i = zy_q;
        if (i0 > 0) {   // candidates past the first 32 (f32 configurations with B > 32)
          int y = p.y[(size_t)b * B + i];
          if (y < 0 || y >= p.V) {
            set_err(p.err, LSP_DEV_BAD_TOKEN);
            y = 0;
          }
          zt_i = p.zt[((size_t)b * (B + 1) + i) * p.V + y];
          zq_i = p.zq[((size_t)b * B + i) * p.V + y];
        }
        // p_i(y) = 2^(z_t it2 - lse2_t), q_i(y) = 2^(z_q it2 - lse2_q)
        const float lp = zt_i * it2 - s_lse[i];
        const float lq = zq_i * it2 - s_lse[B + 1 + i];
        const uint4 x = philox4x32_10(make_uint4(0u, kAcceptStream + (uint32_t)i, (uint32_t)b, p.round), key);
        rej = !(ver_uniform(x.x) * exp2f(lq) < exp2f(lp));
      }
      const unsigned rm = __ballot_sync(kFull, rej);
      if (rm) { j = i0 + __ffs(rm) - 1; break; }
    }
    if (lane == 0) s_j = j;
  }
  __syncthreads();
  const int j = s_j;
  const bool corr = j < B;
  const float lse_t = s_lse[j], lse_q = corr ? s_lse[B + 1 + j] : 0.f;
  const float* zt = p.zt + ((size_t)b * (B + 1) + j) * p.V;
  const float* zq = corr ? p.zq + ((size_t)b * B + j) * p.V : zt;
  const int ng = p.V / 4;
  const int g0 = (int)((long long)ch * ng / nch), g1 = (int)((long long)(ch + 1) * ng / nch);
  constexpr float kLn2 = 0.69314718055994531f;
  float bv = -INFINITY;
  int bi = INT_MAX;
  for (int base = g0 + threadIdx.x; base < g1; base += kDrawBatch * kVerThreads) {
    float4 a[kDrawBatch], c[kDrawBatch];
#pragma unroll
    for (int k = 0; k < kDrawBatch; ++k) {
      const int gi = base + k * kVerThreads;
      const bool in = gi < g1;
      a[k] = in ? __ldg(reinterpret_cast<const float4*>(zt) + gi) : make_float4(0.f, 0.f, 0.f, 0.f);
      c[k] = in && corr ? __ldg(reinterpret_cast<const float4*>(zq) + gi) : a[k];
    }
#pragma unroll
    for (int k = 0; k < kDrawBatch; ++k) {
      const int gi = base + k * kVerThreads;
      if (gi >= g1) break;
      const float at[4] = {a[k].x, a[k].y, a[k].z, a[k].w}, aq[4] = {c[k].x, c[k].y, c[k].z, c[k].w};
      // log-weight of each entry: log[p - q]_+ (correction) or log p (bonus), natural log
      float lw[4];
      bool any = false;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        if (corr) {
          const float w = ex2(fmaf(at[e], it2, -lse_t)) - ex2(fmaf(aq[e], it2, -lse_q));
          lw[e] = w > 0.f ? __logf(w) : -INFINITY;
        } else {
          lw[e] = fmaf(at[e], it2, -lse_t) * kLn2;
        }
        any |= lw[e] > -INFINITY;
      }
      if (!any) continue;    // no weight in this group: no entry can win
      const uint4 x = philox4x32_10(make_uint4((uint32_t)gi, kDrawStream + (uint32_t)j, (uint32_t)b, p.round), key);
      const uint32_t xs[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float sc = lw[e] + gumbel_of(xs[e]);
        if (ver_better(sc, 4 * gi + e, bv, bi)) { bv = sc; bi = 4 * gi + e; }
      }
    }
  }
  group_argmax<32>(bv, bi);
  if (lane == 0) { sv[warp] = bv; si[warp] = bi; }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < kVerThreads / 32; ++w)
      if (ver_better(sv[w], si[w], bv, bi)) { bv = sv[w]; bi = si[w]; }
    p.part_val[(size_t)b * nch + ch] = bv;
    p.part_idx[(size_t)b * nch + ch] = bi;
    __threadfence();
    s_last = atomicAdd(&p.ctr[b], 1u) == (unsigned)nch - 1u;
  }
  __syncthreads();
  if (s_last && warp == 0) {
    __threadfence();
    float v = -INFINITY;
    int i = INT_MAX;
    for (int k = lane; k < nch; k += 32) {
      const float kv = __ldcg(p.part_val + (size_t)b * nch + k);
      const int ki = __ldcg(p.part_idx + (size_t)b * nch + k);
      if (ver_better(kv, ki, v, i)) { v = kv; i = ki; }
    }
    group_argmax<32>(v, i);
    if (lane == 0) {
      p.accepted[b] = j;
      p.next_token[b] = i < p.V ? i : 0;
      atomicExch(&p.ctr[b], 0u);
    }
  }
}

int verify_max_stat_chunks(int V) { return std::max(1, std::min(kVerMaxStatChunks, V / 8192)); }

int launch_verify(const VerifyParams& p, int num_sms, cudaStream_t s) {
  if (p.V % 4 || p.C < 1 || p.B < 1 || p.B > kVerMaxB) return LSP_ERR_SHAPE;
  const bool greedy = !(p.temperature > 0.f);
  const int rpr = greedy ? p.B + 1 : 2 * p.B + 1;
  VerifyParams q = p;
  // about eight chunk CTAs per SM in all (the row pass streams; many chunks keep SMs fed)
  q.nst = std::max(1, std::min(verify_max_stat_chunks(p.V), (8 * num_sms + p.C * rpr - 1) / (p.C * rpr)));
  const dim3 grid(p.C * rpr * q.nst);
  cudaError_t e;
  if (greedy) {
    e = launch_pdl(verify_stats_kernel<true, 8>, grid, dim3(kVerThreads), 0, s, q, rpr);
    if (e == cudaSuccess) e = launch_pdl(verify_greedy_kernel, dim3(p.C), dim3(kVerThreads), 0, s, q);
  } else {
    e = launch_pdl(verify_stats_kernel<false, 4>, grid, dim3(kVerThreads), 0, s, q, rpr);
    // one wave of draw CTAs, at least one float4 group per thread
    const int nch = std::max(1, std::min({kDrawCtasPerSm * num_sms / p.C, kVerMaxDrawChunks, std::max(1, p.V / 4 / kVerThreads)}));
    // (the draw kernel's pre-wait loads need the row pass to trigger after its own wait)
    if (e == cudaSuccess) e = launch_pdl(verify_draw_kernel, dim3(nch, p.C), dim3(kVerThreads), 0, s, q);
  }
  return e == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

}  // namespace lsp
