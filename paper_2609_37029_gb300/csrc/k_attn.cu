// Fixed-context block attention of a draft layer (Sec. 2.3, Eq. draft-context).
//
// Each block query of request b and query head h attends, with one softmax
// (scale 1/sqrt(d)) and no mask inside the block, over
//     K = [K^b ; K^w ; G_h],   V = [V^b ; V^w ; M_h]
// -- the B block keys/values of its KV head g = h / (nq/nkv), the valid rows
// of the recent window of the paired tapped layer, and the R summary entries
// of head h.  At most B + W + R entries per head, independent of t (Sec. 2.4).
// The block q and k get the per-head RMSNorm and the rotary embedding here,
// fused into the load of the q/k/v projection output.
//
// The bf16 shapes the tcgen05 kernel serves (k_attn_tc.cu) run there, with the
// q/k/v finalisation folded in; the kernels below cover the rest.
// attn_mma_kernel (bf16, d = 128): one CTA per (request, KV head) stages the
// window once in shared memory for all nq/nkv query heads (HBM traffic = one
// read of the window and summary); each head gets 8 / (nq/nkv) warps (key
// splits over contiguous ranges of 16-key groups), each running an online
// softmax over 64-key chunks with mma.sync m16n8k16 (bf16 in, fp32
// accumulate; the row max and rescale once per 64 keys), and the split-0
// warp of a head merges the others' records in its registers and writes the
// head's rows.  Measured per CTA at the Qwen3-8B shape (clock stamps): with
// 16 warps and 16-key chunks, 14.2 us (staging 4.5, softmax 5.7, merge 2.4);
// with this layout 12.7 us (staging 4.8, bounded by the window's HBM read,
// softmax 4.0, merge 0.9 plus the wait for the slower split).
// attn_simple_kernel (fp32 storage): FMA version, one CTA per (request, query
// head), for the fp32 reference shape: window and summary rows are staged in
// shared memory 64 at a time (float4 loads, several in flight per thread), a
// warp scores each staged key against all block queries (lanes split over
// queries and head dims), one softmax, then P V over the re-staged values.
#include <algorithm>
#include <type_traits>

#include "common.cuh"
#include "lsp_internal.h"

namespace lsp {

constexpr int kHD = 128;         // head dim of the tensor-core path
constexpr int kLd = kHD + 8;     // smem row stride (bf16): 272 B, conflict-free ldmatrix

struct AttnLayout {
  int rep, ksplit, nwarps, rows_bw;
  size_t off_q, off_kbw, off_vbw, off_ks, off_vs, bytes;
};

static AttnLayout attn_layout(int B, int W, int nq, int nkv, int ksplit) {
  AttnLayout a;
  a.rep = nq / nkv;
  a.ksplit = ksplit;
  a.nwarps = a.rep * ksplit;
  a.rows_bw = (B + W + 15) / 16 * 16;
  const size_t row = kLd * sizeof(bf16);
  a.off_q = 0;
  a.off_kbw = a.off_q + (size_t)a.rep * 16 * row;
  a.off_vbw = a.off_kbw + (size_t)a.rows_bw * row;
  a.off_ks = a.off_vbw + (size_t)a.rows_bw * row;
  a.off_vs = a.off_ks + (size_t)a.rep * 16 * row;
  a.bytes = a.off_vs + (size_t)a.rep * 16 * row;
  return a;
}
// Key-split merge record of one warp: o[16][kOs] (padded: conflict-free
// float2 stores of the mma accumulator layout) then max[16] and sum[16].
constexpr int kOs = kHD + 8;
constexpr int kMergeRec = 16 * kOs + 32;

// 2^x with the MUFU approximation (relative error ~2^-22; -inf gives +0):
// softmax weights that are rounded to bf16 for the P V product anyway.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Up to 64 keys (ng <= 4 groups of 16 rows at Kc / Vc, `nvalid` of them
// valid) of one online-softmax step for the warp's 16 query rows: S = Q K^T
// by mma.sync m16n8k16, one row max / rescale per 64 keys, then O += P V.
__device__ __forceinline__ void attn_chunk(const bf16* qbase, const bf16* Kc, const bf16* Vc, int ng,
                                           int nvalid, float sl2, int lane, float (&rmax)[2],
                                           float (&rsum)[2], float (&o)[16][4]) {
  const size_t row = kLd;
  float s[8][4];
#pragma unroll
  for (int n = 0; n < 8; ++n) s[n][0] = s[n][1] = s[n][2] = s[n][3] = 0.f;
  const bf16* kb = Kc + (size_t)((lane & 7) + (lane >> 4) * 8) * row + ((lane >> 3) & 1) * 8;
#pragma unroll
  for (int kk = 0; kk < kHD / 16; ++kk) {
    uint32_t a[4];
    ldsm_x4(a, qbase + kk * 16);
#pragma unroll
    for (int gi = 0; gi < 4; ++gi)
      if (gi < ng) {
        uint32_t bk[4];
        ldsm_x4(bk, kb + (size_t)gi * 16 * row + kk * 16);
        mma_bf16(s[2 * gi], a, bk[0], bk[1]);
        mma_bf16(s[2 * gi + 1], a, bk[2], bk[3]);
      }
  }
  float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
  for (int n = 0; n < 8; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      if (n * 8 + (lane & 3) * 2 + (e & 1) >= nvalid) s[n][e] = -INFINITY;   // invalid or empty group
      if (e < 2) mx0 = fmaxf(mx0, s[n][e]);
      else mx1 = fmaxf(mx1, s[n][e]);
    }
  mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
  mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
  mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
  mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
  const float n0 = fmaxf(rmax[0], mx0), n1 = fmaxf(rmax[1], mx1);
  const float b0 = (n0 == -INFINITY) ? 0.f : n0, b1 = (n1 == -INFINITY) ? 0.f : n1;
  const float sc0 = ex2_approx((rmax[0] - b0) * sl2), sc1 = ex2_approx((rmax[1] - b1) * sl2);
  rmax[0] = n0;
  rmax[1] = n1;
  float t0 = 0.f, t1 = 0.f;
#pragma unroll
  for (int n = 0; n < 8; ++n) {
    s[n][0] = ex2_approx((s[n][0] - b0) * sl2);
    s[n][1] = ex2_approx((s[n][1] - b0) * sl2);
    s[n][2] = ex2_approx((s[n][2] - b1) * sl2);
    s[n][3] = ex2_approx((s[n][3] - b1) * sl2);
    t0 += s[n][0] + s[n][1];
    t1 += s[n][2] + s[n][3];
  }
  rsum[0] = rsum[0] * sc0 + t0;
  rsum[1] = rsum[1] * sc1 + t1;
#pragma unroll
  for (int n = 0; n < 16; ++n) {
    o[n][0] *= sc0; o[n][1] *= sc0;
    o[n][2] *= sc1; o[n][3] *= sc1;
  }
  const bf16* vb = Vc + (size_t)((lane & 7) + ((lane >> 3) & 1) * 8) * row + (lane >> 4) * 8;
#pragma unroll
  for (int gi = 0; gi < 4; ++gi)
    if (gi < ng) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * gi][0], s[2 * gi][1]);
      pa[1] = pack_bf16(s[2 * gi][2], s[2 * gi][3]);
      pa[2] = pack_bf16(s[2 * gi + 1][0], s[2 * gi + 1][1]);
      pa[3] = pack_bf16(s[2 * gi + 1][2], s[2 * gi + 1][3]);
#pragma unroll
      for (int np = 0; np < kHD / 16; ++np) {
        uint32_t bv[4];
        ldsm_x4_t(bv, vb + (size_t)gi * 16 * row + np * 16);
        mma_bf16(o[2 * np], pa, bv[0], bv[1]);
        mma_bf16(o[2 * np + 1], pa, bv[2], bv[3]);
      }
    }
}

__global__ void __launch_bounds__(512)
    attn_mma_kernel(const AttnParams p, const int rep, const int ksplit, const int rows_bw) {
  extern __shared__ __align__(16) uint8_t asmem[];
  const size_t row = kLd;
  bf16* sQ = reinterpret_cast<bf16*>(asmem);
  bf16* sKbw = sQ + (size_t)rep * 16 * row;
  bf16* sVbw = sKbw + (size_t)rows_bw * row;
  bf16* sKs = sVbw + (size_t)rows_bw * row;
  bf16* sVs = sKs + (size_t)rep * 16 * row;

  const int nwarps = rep * ksplit;
  const int nthr = nwarps * 32;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int b = blockIdx.x / p.nkv, g = blockIdx.x % p.nkv;
  griddep_launch();
  // The window, summary and t come from the view update at the start of the
  // round: the q/k/v finalize before this kernel triggers its dependents only
  // after its own wait, so every kernel before the q/k/v projection has
  // completed and these loads may start before this kernel's own wait,
  // overlapping the finalize.  Only the block q/k/v waits for it.
  const int B = p.B, L = p.L, l = p.layer;
  const long long t = p.t[b];
  const int count = (int)(t < p.W ? t : p.W);
  const int nbw = B + count;                       // valid block + window keys
  const int nbw16 = (nbw + 15) / 16 * 16;

  // ---- window rows (valid slots are 0..count-1) straight into smem
  const bf16* wk = static_cast<const bf16*>(p.win_k) + ((size_t)(b * L + l) * p.nkv + g) * p.W * kHD;
  const bf16* wv = static_cast<const bf16*>(p.win_v) + ((size_t)(b * L + l) * p.nkv + g) * p.W * kHD;
  for (int idx = tid; idx < count * 16; idx += nthr) {
    const int r = idx >> 4, c = (idx & 15) * 8;
    cp_async16(sKbw + (size_t)(B + r) * row + c, wk + (size_t)r * kHD + c);
    cp_async16(sVbw + (size_t)(B + r) * row + c, wv + (size_t)r * kHD + c);
  }
  // ---- summary keys G_h (bf16) and values M_h (fp32 -> bf16): every value
  //      load of this thread is issued before the first conversion
  const bf16* Gp = static_cast<const bf16*>(p.G) + ((size_t)l * p.nq + (size_t)g * rep) * p.R * kHD;
  const float* Mp = p.m + (((size_t)(b * L + l) * p.nq + (size_t)g * rep) * p.R) * kHD;
  {
    constexpr int kMaxItems = 8;                   // rep * 16 * 16 / (rep * ksplit * 32) <= 8
    float4 mv[kMaxItems][2];
#pragma unroll
    for (int u = 0; u < kMaxItems; ++u) {
      const int idx = tid + u * nthr;
      const int hr = idx >> 4, c = (idx & 15) * 8, hh = hr >> 4, r = hr & 15;
      if (idx < rep * 256 && r < p.R) {
        cp_async16(sKs + (size_t)hr * row + c, Gp + ((size_t)hh * p.R + r) * kHD + c);
        const float4* src = reinterpret_cast<const float4*>(Mp + ((size_t)hh * p.R + r) * kHD + c);
        mv[u][0] = src[0];
        mv[u][1] = src[1];
      }
    }
#pragma unroll
    for (int u = 0; u < kMaxItems; ++u) {
      const int idx = tid + u * nthr;
      const int hr = idx >> 4, c = (idx & 15) * 8, r = hr & 15;
      if (idx < rep * 256) {
        bf16* dk = sKs + (size_t)hr * row + c;
        bf16* dv = sVs + (size_t)hr * row + c;
        if (r < p.R) {
          uint4 o;
          o.x = pack_bf16(mv[u][0].x, mv[u][0].y);
          o.y = pack_bf16(mv[u][0].z, mv[u][0].w);
          o.z = pack_bf16(mv[u][1].x, mv[u][1].y);
          o.w = pack_bf16(mv[u][1].z, mv[u][1].w);
          *reinterpret_cast<uint4*>(dv) = o;
        } else {
          *reinterpret_cast<uint4*>(dk) = make_uint4(0, 0, 0, 0);
          *reinterpret_cast<uint4*>(dv) = make_uint4(0, 0, 0, 0);
        }
      }
    }
  }
  // ---- zero the tail of the last block/window group, and the padded query rows
  for (int idx = tid; idx < (nbw16 - nbw) * 16; idx += nthr) {
    const int r = nbw + (idx >> 4), c = (idx & 15) * 8;
    *reinterpret_cast<uint4*>(sKbw + (size_t)r * row + c) = make_uint4(0, 0, 0, 0);
    *reinterpret_cast<uint4*>(sVbw + (size_t)r * row + c) = make_uint4(0, 0, 0, 0);
  }
  for (int idx = tid; idx < rep * (16 - B) * 16; idx += nthr) {
    const int hr = idx >> 4, c = (idx & 15) * 8;
    const int hh = hr / (16 - B), i = B + hr % (16 - B);
    *reinterpret_cast<uint4*>(sQ + (size_t)(hh * 16 + i) * row + c) = make_uint4(0, 0, 0, 0);
  }
  // ---- block q (rep heads), k, v of KV head g, already normalised and rotated
  {
    const bf16* qkv = static_cast<const bf16*>(p.qkv);
    const int ldq = (p.nq + 2 * p.nkv) * kHD;
    const int kinds = rep + 2;
    griddep_wait();                                 // the q/k/v finalize has completed
    for (int idx = tid; idx < B * kinds * 16; idx += nthr) {
      const int c = (idx & 15) * 8, item = idx >> 4;
      const int i = item / kinds, kind = item % kinds;
      const size_t mrow = (size_t)(b * B + i) * ldq;
      const bf16* src;
      bf16* dst;
      if (kind < rep) {
        src = qkv + mrow + (size_t)(g * rep + kind) * kHD;
        dst = sQ + (size_t)(kind * 16 + i) * row;
      } else if (kind == rep) {
        src = qkv + mrow + (size_t)(p.nq + g) * kHD;
        dst = sKbw + (size_t)i * row;
      } else {
        src = qkv + mrow + (size_t)(p.nq + p.nkv + g) * kHD;
        dst = sVbw + (size_t)i * row;
      }
      cp_async16(dst + c, src + c);
    }
  }
  cp_async_wait_all();
  __syncthreads();

  // ---- online softmax of head hh over this warp's contiguous range of
  //      16-key groups, 64 keys at a time.  The summary is one more 16-key
  //      unit after the last group, so the ranges balance the splits' work.
  const int hh = warp / ksplit, ks = warp % ksplit;
  const int ngrp = nbw16 / 16;
  const int nunits = ngrp + (p.R > 0 ? 1 : 0);
  const int u0 = ks * nunits / ksplit, u1 = (ks + 1) * nunits / ksplit;
  const int g0 = min(u0, ngrp), g1 = min(u1, ngrp);
  const bool take_summary = p.R > 0 && u1 == nunits && u0 < nunits;
  const float sl2 = 1.4426950408889634f * rsqrtf((float)kHD);
  float rmax[2] = {-INFINITY, -INFINITY}, rsum[2] = {0.f, 0.f};
  float o[16][4];
#pragma unroll
  for (int n = 0; n < 16; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  const bf16* qbase = sQ + (size_t)(hh * 16 + (lane & 15)) * row + (lane >> 4) * 8;
  for (int cg = g0; cg < g1; cg += 4) {
    const int ng = min(4, g1 - cg);
    attn_chunk(qbase, sKbw + (size_t)cg * 16 * row, sVbw + (size_t)cg * 16 * row, ng,
               min(ng * 16, nbw - cg * 16), sl2, lane, rmax, rsum, o);
  }
  if (take_summary)
    attn_chunk(qbase, sKs + (size_t)hh * 16 * row, sVs + (size_t)hh * 16 * row, 1, p.R, sl2, lane, rmax,
               rsum, o);
  rsum[0] += __shfl_xor_sync(0xffffffffu, rsum[0], 1);
  rsum[0] += __shfl_xor_sync(0xffffffffu, rsum[0], 2);
  rsum[1] += __shfl_xor_sync(0xffffffffu, rsum[1], 1);
  rsum[1] += __shfl_xor_sync(0xffffffffu, rsum[1], 2);

  // ---- the split-0 warp of each head merges the other splits' records in
  //      its registers (scratch reuses the K/V staging area) and writes out
  const int r0 = lane >> 2;
  if (ksplit > 1) {
    __syncthreads();                                // every warp is done with the K/V tiles
    float* scratch = reinterpret_cast<float*>(sKbw);
    if (ks > 0) {
      float* so = scratch + (size_t)(hh * (ksplit - 1) + ks - 1) * kMergeRec;
      float* sml = so + 16 * kOs;
#pragma unroll
      for (int n = 0; n < 16; ++n) {
        const int col = n * 8 + (lane & 3) * 2;
        *reinterpret_cast<float2*>(so + r0 * kOs + col) = make_float2(o[n][0], o[n][1]);
        *reinterpret_cast<float2*>(so + (r0 + 8) * kOs + col) = make_float2(o[n][2], o[n][3]);
      }
      if ((lane & 3) == 0) {
        sml[r0] = rmax[0];
        sml[r0 + 8] = rmax[1];
        sml[16 + r0] = rsum[0];
        sml[16 + r0 + 8] = rsum[1];
      }
    }
    __syncthreads();
    if (ks > 0) return;
    for (int k = 1; k < ksplit; ++k) {
      const float* so = scratch + (size_t)(hh * (ksplit - 1) + k - 1) * kMergeRec;
      const float* sml = so + 16 * kOs;
      const float m0 = sml[r0], m1 = sml[r0 + 8];
      const float n0 = fmaxf(rmax[0], m0), n1 = fmaxf(rmax[1], m1);
      const float b0 = (n0 == -INFINITY) ? 0.f : n0, b1 = (n1 == -INFINITY) ? 0.f : n1;
      const float a0 = ex2_approx((rmax[0] - b0) * sl2), a1 = ex2_approx((rmax[1] - b1) * sl2);
      const float c0 = ex2_approx((m0 - b0) * sl2), c1 = ex2_approx((m1 - b1) * sl2);
      rsum[0] = rsum[0] * a0 + sml[16 + r0] * c0;
      rsum[1] = rsum[1] * a1 + sml[16 + r0 + 8] * c1;
      rmax[0] = n0;
      rmax[1] = n1;
#pragma unroll
      for (int n = 0; n < 16; ++n) {
        const int col = n * 8 + (lane & 3) * 2;
        const float2 x0 = *reinterpret_cast<const float2*>(so + r0 * kOs + col);
        const float2 x1 = *reinterpret_cast<const float2*>(so + (r0 + 8) * kOs + col);
        o[n][0] = o[n][0] * a0 + x0.x * c0;
        o[n][1] = o[n][1] * a0 + x0.y * c0;
        o[n][2] = o[n][2] * a1 + x1.x * c1;
        o[n][3] = o[n][3] * a1 + x1.y * c1;
      }
    }
  }
  // ---- normalise and store this head's rows (query rows r0 and r0 + 8 of the block)
  bf16* out = static_cast<bf16*>(p.out);
  const int ldo = p.nq * kHD;
  const float inv0 = 1.0f / rsum[0], inv1 = 1.0f / rsum[1];
  bf16* o0 = out + (size_t)(b * B + r0) * ldo + (size_t)(g * rep + hh) * kHD + (lane & 3) * 2;
  bf16* o1 = o0 + (size_t)8 * ldo;
#pragma unroll
  for (int n = 0; n < 16; ++n) {
    if (r0 < B) *reinterpret_cast<uint32_t*>(o0 + n * 8) = pack_bf16(o[n][0] * inv0, o[n][1] * inv0);
    if (r0 + 8 < B) *reinterpret_cast<uint32_t*>(o1 + n * 8) = pack_bf16(o[n][2] * inv1, o[n][3] * inv1);
  }
}

// ------------------------------------------------------------ fp32 reference shape
constexpr int kSimpleChunk = 64;    // window / summary rows staged per round trip

// Lanes per block query in the score loop: the largest power of two with
// lpq * B <= 32 (1 when B > 16).
__host__ __device__ inline int simple_lpq(int B) {
  int lpq = 1;
  while (lpq * 2 * B <= 32) lpq *= 2;
  return lpq;
}

// Rows [j0, j0 + nr) of the context list "count window rows, then summary rows"
// into shared memory as [nr][d] floats: float4 loads (d % 4 == 0), four in
// flight per thread before their stores.
__device__ __forceinline__ void stage_rows(float* dst, const float* win, const float* summ, int count,
                                           int j0, int nr, int d) {
  const int d4 = d / 4, n4 = nr * d4;
  for (int base = threadIdx.x; base < n4; base += 4 * blockDim.x) {
    float4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int idx = base + u * blockDim.x;
      v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (idx < n4) {
        const int r = j0 + idx / d4, c4 = idx % d4;
        const float* src = r < count ? win + (size_t)r * d : summ + (size_t)(r - count) * d;
        v[u] = reinterpret_cast<const float4*>(src)[c4];
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int idx = base + u * blockDim.x;
      if (idx < n4) reinterpret_cast<float4*>(dst)[idx] = v[u];
    }
  }
}

template <typename T>
__global__ void __launch_bounds__(256) attn_simple_kernel(const AttnParams p, const int whole) {
  extern __shared__ float ssm[];
  const int d = p.d, B = p.B;
  const int rep = p.nq / p.nkv;
  const int b = blockIdx.x / p.nq, h = blockIdx.x % p.nq, g = h / rep;
  const long long t = p.t[b];
  const int count = (int)(t < p.W ? t : p.W);
  const int ctx = B + count + p.R;
  // Query rows padded to d + lpq floats: with d a multiple of 32 the lanes of a
  // score pass (query qi, dims c + lpq k) then fall in distinct banks.
  const int lpq = simple_lpq(B), dq = d + lpq;
  float* sq = ssm;
  float* sk = sq + (B * dq + 3) / 4 * 4;
  float* sv = sk + B * d;
  float* ss = sv + B * d;                 // [B][ctx]
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, nw = blockDim.x >> 5;
  griddep_launch();
  griddep_wait();
  const T* qkv = static_cast<const T*>(p.qkv);
  const int ldq = (p.nq + 2 * p.nkv) * d;
  for (int idx = tid; idx < 3 * B * d; idx += blockDim.x) {
    const int kind = idx / (B * d), i = (idx / d) % B, e = idx % d;
    const size_t mrow = (size_t)(b * B + i) * ldq;
    const size_t col = kind == 0 ? (size_t)h * d : kind == 1 ? (size_t)(p.nq + g) * d
                                                                : (size_t)(p.nq + p.nkv + g) * d;
    (kind == 0 ? sq + i * dq : (kind == 1 ? sk : sv) + i * d)[e] = to_f(qkv[mrow + col + e]);
  }
  __syncthreads();
  const size_t wbase = ((size_t)(b * p.L + p.layer) * p.nkv + g) * p.W * d;
  const T* wk = static_cast<const T*>(p.win_k) + wbase;
  const T* wv = static_cast<const T*>(p.win_v) + wbase;
  const T* Gh = static_cast<const T*>(p.G) + ((size_t)p.layer * p.nq + h) * p.R * d;
  const float* Mh = p.m + (((size_t)(b * p.L + p.layer) * p.nq + h) * p.R) * d;
  const float scale = rsqrtf((float)d);
  float* sc = ss + ((size_t)B * ctx + 3) / 4 * 4;   // [kSimpleChunk][d] staged rows (16-B aligned)
  const int nctx = count + p.R;           // window rows, then summary rows
  // Lanes split into groups of `lpq` per block query (queries in passes of
  // 32 / lpq); lane c of a group covers dims c, c + lpq, ... so a score needs
  // log2(lpq) shuffles.
  const int qpp = 32 / lpq, qi = lane / lpq, c = lane % lpq;
  auto score = [&](const float* krow, int j) {   // j: context index of the key
    for (int i0 = 0; i0 < B; i0 += qpp) {
      const int i = i0 + qi;
      float part = 0.f;
      if (i < B)
        for (int e = c; e < d; e += lpq) part = fmaf(sq[i * dq + e], krow[e], part);
      for (int o = lpq / 2; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
      if (i < B && c == 0) ss[i * ctx + j] = part * scale;
    }
  };
  if (whole) {
    // every window and summary key and value row at once (cp.async, one round
    // trip for all of them; fp32 rows of d floats, 16-byte chunks)
    float* sK = sc;
    float* sV = sc + (size_t)nctx * d;
    const int d4 = d / 4;
    for (int idx = tid; idx < nctx * d4; idx += blockDim.x) {
      const int r = idx / d4, c4 = (idx % d4) * 4;
      const float* srck = r < count ? reinterpret_cast<const float*>(wk) + (size_t)r * d
                                    : reinterpret_cast<const float*>(Gh) + (size_t)(r - count) * d;
      const float* srcv = r < count ? reinterpret_cast<const float*>(wv) + (size_t)r * d : Mh + (size_t)(r - count) * d;
      cp_async16(sK + (size_t)r * d + c4, srck + c4);
      cp_async16(sV + (size_t)r * d + c4, srcv + c4);
    }
    for (int j = warp; j < B; j += nw) score(sk + j * d, j);
    cp_async_wait_all();
    __syncthreads();
    for (int r = warp; r < nctx; r += nw) score(sK + (size_t)r * d, B + r);
    __syncthreads();
    for (int i = warp; i < B; i += nw) {
      float mx = -INFINITY;
      for (int j = lane; j < ctx; j += 32) mx = fmaxf(mx, ss[i * ctx + j]);
      mx = warp_max(mx);
      float sum = 0.f;
      for (int j = lane; j < ctx; j += 32) {
        const float e = expf(ss[i * ctx + j] - mx);
        ss[i * ctx + j] = e;
        sum += e;
      }
      sum = warp_sum(sum);
      for (int j = lane; j < ctx; j += 32) ss[i * ctx + j] /= sum;
    }
    __syncthreads();
    T* out = static_cast<T*>(p.out);
    for (int idx = tid; idx < B * d; idx += blockDim.x) {
      const int i = idx / d, e = idx % d;
      const float* pr = ss + (size_t)i * ctx;
      float a = 0.f, a4[4] = {0.f, 0.f, 0.f, 0.f};   // four independent FMA chains
      for (int j = 0; j < B; ++j) a = fmaf(pr[j], sv[j * d + e], a);
      int r = 0;
      for (; r + 4 <= nctx; r += 4) {
#pragma unroll
        for (int u = 0; u < 4; ++u) a4[u] = fmaf(pr[B + r + u], sV[(size_t)(r + u) * d + e], a4[u]);
      }
      for (; r < nctx; ++r) a = fmaf(pr[B + r], sV[(size_t)r * d + e], a);
      a += (a4[0] + a4[1]) + (a4[2] + a4[3]);
      out[(size_t)(b * B + i) * p.nq * d + (size_t)h * d + e] = from_f<T>(a);
    }
    return;
  }
  // ---- scores: block keys from shared memory, then the window and summary
  // keys staged kSimpleChunk rows at a time (one coalesced round trip each)
  for (int j = warp; j < B; j += nw) score(sk + j * d, j);
  for (int j0 = 0; j0 < nctx; j0 += kSimpleChunk) {
    const int nr = min(kSimpleChunk, nctx - j0);
    __syncthreads();
    stage_rows(sc, wk, Gh, count, j0, nr, d);
    __syncthreads();
    for (int r = warp; r < nr; r += nw) score(sc + r * d, B + j0 + r);
  }
  __syncthreads();
  // ---- one softmax per query over the B + count + R scores
  for (int i = warp; i < B; i += nw) {
    float mx = -INFINITY;
    for (int j = lane; j < ctx; j += 32) mx = fmaxf(mx, ss[i * ctx + j]);
    mx = warp_max(mx);
    float sum = 0.f;
    for (int j = lane; j < ctx; j += 32) {
      const float e = expf(ss[i * ctx + j] - mx);
      ss[i * ctx + j] = e;
      sum += e;
    }
    sum = warp_sum(sum);
    for (int j = lane; j < ctx; j += 32) ss[i * ctx + j] /= sum;
  }
  __syncthreads();
  // ---- P V, accumulated in place of the (no longer needed) queries: block
  // values first, then the window and summary values staged like the keys
  float* acc = sq;
  for (int idx = tid; idx < B * d; idx += blockDim.x) {
    const int i = idx / d, e = idx % d;
    float a = 0.f;
    for (int j = 0; j < B; ++j) a = fmaf(ss[i * ctx + j], sv[j * d + e], a);
    acc[idx] = a;
  }
  for (int j0 = 0; j0 < nctx; j0 += kSimpleChunk) {
    const int nr = min(kSimpleChunk, nctx - j0);
    __syncthreads();
    stage_rows(sc, wv, Mh, count, j0, nr, d);
    __syncthreads();
    for (int idx = tid; idx < B * d; idx += blockDim.x) {
      const int i = idx / d, e = idx % d;
      const float* pr = ss + (size_t)i * ctx + B + j0;
      float a = acc[idx];
      for (int r = 0; r < nr; ++r) a = fmaf(pr[r], sc[r * d + e], a);
      acc[idx] = a;
    }
  }
  __syncthreads();
  T* out = static_cast<T*>(p.out);
  for (int idx = tid; idx < B * d; idx += blockDim.x) {
    const int i = idx / d, e = idx % d;
    out[(size_t)(b * B + i) * p.nq * d + (size_t)h * d + e] = from_f<T>(acc[idx]);
  }
}

// ------------------------------------------------------------ q/k/v finalisation
// N (2 or 4) consecutive fp32 / bf16 values <-> fp32 registers, one vector access
template <int N>
__device__ __forceinline__ void load_vec(const float* p, float* v) {
  if constexpr (N == 4) {
    const float4 x = *reinterpret_cast<const float4*>(p);
    v[0] = x.x; v[1] = x.y; v[2] = x.z; v[3] = x.w;
  } else {
    const float2 x = *reinterpret_cast<const float2*>(p);
    v[0] = x.x; v[1] = x.y;
  }
}
template <int N>
__device__ __forceinline__ void load_vec(const bf16* p, float* v) {
  if constexpr (N == 4) {
    const uint2 r = *reinterpret_cast<const uint2*>(p);
    const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r.x));
    const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r.y));
    v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y;
  } else {
    const __nv_bfloat162 r = *reinterpret_cast<const __nv_bfloat162*>(p);
    const float2 a = __bfloat1622float2(r);
    v[0] = a.x; v[1] = a.y;
  }
}
template <int N>
__device__ __forceinline__ void store_vec(float* p, const float* v) {
  if constexpr (N == 4) *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  else *reinterpret_cast<float2*>(p) = make_float2(v[0], v[1]);
}
template <int N>
__device__ __forceinline__ void store_vec(bf16* p, const float* v) {
  if constexpr (N == 4) *reinterpret_cast<uint2*>(p) = make_uint2(pack_bf16(v[0], v[1]), pack_bf16(v[2], v[3]));
  else *reinterpret_cast<uint32_t*>(p) = pack_bf16(v[0], v[1]);
}

// One warp per group of kFinRows (block row, head) rows: the sum of the q/k/v
// projection's split-K partials in split order, then for q and k heads the
// per-head RMSNorm and the rotary embedding (pairs f, f + d/2; lane l holds
// elements EPL*l .. EPL*l+EPL-1, its rotary partner lives in lane l ^ 16).
// The grid is capped at two CTAs per SM (a grid-stride loop covers the rest),
// so every CTA is resident as soon as the projection's CTAs leave: the
// attention kernel, which launches once every CTA here has passed its wait,
// then starts staging its window while these rows are still being formed.
// Measured at the Qwen3-8B round with one row per warp (1536 CTAs, 1.4 waves):
// the attention started ~8.5 us after the projection ended.
constexpr int kFinRows = 6;

template <typename T, int EPL>
__global__ void __launch_bounds__(256, 2) qkv_finalize_kernel(const QkvParams p) {
  // wait first, then let the attention kernel launch: it reads the view
  // state before its own wait, which is safe once the q/k/v projection (and
  // so every kernel before it) has completed
  griddep_wait();
  griddep_launch();
  const int heads = p.nq + 2 * p.nkv;
  const int items = p.M * heads;
  const int lane = threadIdx.x & 31;
  const int d = EPL * 32, half = d / 2;
  const size_t ldq = (size_t)heads * d;
  const size_t pstride = (size_t)p.M * ldq;
  using V = typename std::conditional<EPL == 4, float4, float2>::type;
  const int nw = gridDim.x * 8;
  for (int base = (blockIdx.x * 8 + (threadIdx.x >> 5)) * kFinRows; base < items; base += nw * kFinRows) {
    // kFinRows rows x up to three splits of vector loads in flight before the
    // adds (which run in split order); partials are read once
    float x[kFinRows][EPL];
#pragma unroll
    for (int u = 0; u < kFinRows; ++u)
#pragma unroll
      for (int e = 0; e < EPL; ++e) x[u][e] = 0.f;
    const float* src0 = p.part + (size_t)base * d + EPL * lane;   // rows base.. are contiguous
    for (int s0 = 0; s0 < p.splits; s0 += 3) {
      V y[3][kFinRows];
#pragma unroll
      for (int v = 0; v < 3; ++v) {
        const float* sv = src0 + (size_t)(s0 + v) * pstride;
#pragma unroll
        for (int u = 0; u < kFinRows; ++u)
          if (s0 + v < p.splits && base + u < items) y[v][u] = __ldcs(reinterpret_cast<const V*>(sv + u * d));
      }
#pragma unroll
      for (int v = 0; v < 3; ++v)
#pragma unroll
        for (int u = 0; u < kFinRows; ++u)
          if (s0 + v < p.splits && base + u < items) {
            const float* f = reinterpret_cast<const float*>(&y[v][u]);
#pragma unroll
            for (int e = 0; e < EPL; ++e) x[u][e] += f[e];
          }
    }
#pragma unroll
    for (int u = 0; u < kFinRows; ++u) {
      const int item = base + u;
      if (item >= items) break;                      // warp-uniform
      const int m = item / heads, h = item % heads;
      if (h < p.nq + p.nkv) {
        // the lane's norm weights and (cos, sin) pairs as vector loads, issued before the reduction
        float w[EPL], cs[2 * EPL];
        load_vec<EPL>(static_cast<const T*>(h < p.nq ? p.q_norm : p.k_norm) + EPL * lane, w);
        const int b = m / p.B, i = m % p.B;
        const float* csp = p.rope + ((size_t)(b * p.B + i) * half + EPL * (lane & 15)) * 2;
        load_vec<EPL>(csp, cs);
        load_vec<EPL>(csp + EPL, cs + EPL);
        float ss = 0.f;
#pragma unroll
        for (int e = 0; e < EPL; ++e) ss += x[u][e] * x[u][e];
        const float rstd = rsqrtf(warp_sum(ss) / (float)d + p.eps);
#pragma unroll
        for (int e = 0; e < EPL; ++e) x[u][e] *= rstd * w[e];
        const float sg = lane < 16 ? -1.f : 1.f;
#pragma unroll
        for (int e = 0; e < EPL; ++e) {
          const float partner = __shfl_xor_sync(0xffffffffu, x[u][e], 16);
          x[u][e] = x[u][e] * cs[2 * e] + sg * partner * cs[2 * e + 1];
        }
      }
      store_vec<EPL>(static_cast<T*>(p.out) + (size_t)item * d + EPL * lane, x[u]);
    }
  }
}

int launch_qkv_finalize(const QkvParams& p, int dtype, cudaStream_t s) {
  const int items = p.M * (p.nq + 2 * p.nkv);
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
    return LSP_ERR_CUDA;
  const int need = (items + 8 * kFinRows - 1) / (8 * kFinRows);
  const dim3 grid(std::min(need, 2 * sms));
  cudaError_t e;
  if (p.d == 128)
    e = dtype == LSP_DTYPE_BF16 ? launch_pdl(qkv_finalize_kernel<bf16, 4>, grid, dim3(256), 0, s, p)
                                : launch_pdl(qkv_finalize_kernel<float, 4>, grid, dim3(256), 0, s, p);
  else if (p.d == 64)
    e = dtype == LSP_DTYPE_BF16 ? launch_pdl(qkv_finalize_kernel<bf16, 2>, grid, dim3(256), 0, s, p)
                                : launch_pdl(qkv_finalize_kernel<float, 2>, grid, dim3(256), 0, s, p);
  else
    return LSP_ERR_SHAPE;
  return e == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

// Key splits per query head.  Measured on one GB300 (A/B): Qwen3-8B (4 heads
// per KV head) 8 warps (2 splits) beat 16 warps by 8.7 us per round; the large
// shape (5 heads per KV head) gained 27 us per round with 3 splits (15 warps)
// over 1 split.
int attn_ksplit(int B, int W, int nq, int nkv) {
  const int rep = nq / nkv;
  int ks = rep >= 16 ? 1 : (rep <= 4 ? 8 / rep : 16 / rep);
  while (ks > 1) {
    AttnLayout a = attn_layout(B, W, nq, nkv, ks);
    const size_t scratch = (size_t)rep * (ks - 1) * kMergeRec * sizeof(float);
    if (scratch <= a.bytes - a.off_kbw && a.nwarps <= 16) break;
    --ks;
  }
  return ks;
}

size_t attn_smem_bytes(int B, int W, int nq, int nkv) {
  AttnLayout a = attn_layout(B, W, nq, nkv, attn_ksplit(B, W, nq, nkv));
  return a.bytes;
}

int launch_attention(const AttnParams& p, int dtype, cudaStream_t s, const AttnTcPlan* tc) {
  if (dtype == LSP_DTYPE_BF16) {
    if (tc && tc->ok) return launch_attention_tc(p, *tc, s);
    if (p.d != kHD || p.B > 16 || p.R > 16) return LSP_ERR_SHAPE;
    const int ks = attn_ksplit(p.B, p.W, p.nq, p.nkv);
    AttnLayout a = attn_layout(p.B, p.W, p.nq, p.nkv, ks);
    if (a.bytes > 227 * 1024 || (size_t)a.rep * (ks - 1) * kMergeRec * sizeof(float) > a.bytes - a.off_kbw)
      return LSP_ERR_SHAPE;
    static bool attr_set = false;
    if (!attr_set) {
      cudaFuncSetAttribute(attn_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
      attr_set = true;
    }
    if (launch_pdl(attn_mma_kernel, dim3(p.C * p.nkv), dim3(a.nwarps * 32), a.bytes, s, p, a.rep, ks,
                   a.rows_bw) != cudaSuccess)
      return LSP_ERR_CUDA;
  } else {
    const int ctx = p.B + p.W + p.R;
    const size_t fixed = (size_t)(3 * p.B * p.d + p.B * simple_lpq(p.B) + 4 + p.B * ctx + 4) * sizeof(float);
    // all window and summary rows staged at once when they fit (fp32 and d % 4 == 0
    // for the 16-byte copies), else kSimpleChunk rows at a time
    const size_t whole_bytes = fixed + (size_t)2 * (p.W + p.R) * p.d * sizeof(float);
    const int whole = (dtype == LSP_DTYPE_F32 && p.d % 4 == 0 && whole_bytes <= 227 * 1024) ? 1 : 0;
    const size_t smem = whole ? whole_bytes : fixed + (size_t)kSimpleChunk * p.d * sizeof(float);
    if (smem > 227 * 1024) return LSP_ERR_SHAPE;
    static bool attr32 = false;
    if (!attr32) {
      cudaFuncSetAttribute(attn_simple_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           227 * 1024);
      attr32 = true;
    }
    if (launch_pdl(attn_simple_kernel<float>, dim3(p.C * p.nq), dim3(256), smem, s, p, whole) != cudaSuccess)
      return LSP_ERR_CUDA;
  }
  return cudaGetLastError() == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

}  // namespace lsp
