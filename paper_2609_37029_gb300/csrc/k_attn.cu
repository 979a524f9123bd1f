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
// attn_mma_kernel (bf16, d = 128): one CTA per (request, KV head) stages the
// window once in shared memory for all nq/nkv query heads (HBM traffic = one
// read of the window and summary); warps are (query head x key split); each
// warp runs an online softmax over 16-key chunks with mma.sync m16n8k16
// (bf16 in, fp32 accumulate), and the key splits merge through shared memory.
// attn_simple_kernel (fp32 storage): FMA version, one CTA per (request, query
// head), for the fp32 reference shape: window and summary rows are staged in
// shared memory 64 at a time (float4 loads, several in flight per thread), a
// warp scores each staged key against all block queries (lanes split over
// queries and head dims), one softmax, then P V over the re-staged values.
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
// Key-split merge scratch per warp: o[16][kOs] (padded: conflict-free float2
// stores of the mma accumulator layout) then max[16] and sum[16].
constexpr int kOs = kHD + 8;
constexpr int kMergeRec = 16 * kOs + 32;
static size_t attn_merge_bytes(int nwarps) { return (size_t)nwarps * kMergeRec * sizeof(float); }

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
  // ---- summary keys G_h (bf16) and values M_h (fp32 -> bf16)
  const bf16* Gp = static_cast<const bf16*>(p.G) + ((size_t)l * p.nq + (size_t)g * rep) * p.R * kHD;
  const float* Mp = p.m + (((size_t)(b * L + l) * p.nq + (size_t)g * rep) * p.R) * kHD;
  for (int idx = tid; idx < rep * 16 * 16; idx += nthr) {
    const int hr = idx >> 4, c = (idx & 15) * 8;     // hr = hh * 16 + r
    const int hh = hr >> 4, r = hr & 15;
    bf16* dk = sKs + (size_t)hr * row + c;
    bf16* dv = sVs + (size_t)hr * row + c;
    if (r < p.R) {
      cp_async16(dk, Gp + ((size_t)hh * p.R + r) * kHD + c);
      const float4* src = reinterpret_cast<const float4*>(Mp + ((size_t)hh * p.R + r) * kHD + c);
      const float4 x0 = src[0], x1 = src[1];
      uint4 o;
      o.x = pack_bf16(x0.x, x0.y);
      o.y = pack_bf16(x0.z, x0.w);
      o.z = pack_bf16(x1.x, x1.y);
      o.w = pack_bf16(x1.z, x1.w);
      *reinterpret_cast<uint4*>(dv) = o;
    } else {
      *reinterpret_cast<uint4*>(dk) = make_uint4(0, 0, 0, 0);
      *reinterpret_cast<uint4*>(dv) = make_uint4(0, 0, 0, 0);
    }
  }
  // ---- zero the tail of the last block/window chunk, and the padded query rows
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

  // ---- online softmax over this warp's 16-key chunks
  const int hh = warp / ksplit, ks = warp % ksplit;
  const int nch_bw = nbw16 / 16;
  const int nch = nch_bw + (p.R > 0 ? 1 : 0);
  const float sl2 = 1.4426950408889634f * rsqrtf((float)kHD);
  float rmax[2] = {-INFINITY, -INFINITY}, rsum[2] = {0.f, 0.f};
  float o[16][4];
#pragma unroll
  for (int n = 0; n < 16; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  const bf16* qbase = sQ + (size_t)(hh * 16 + (lane & 15)) * row + (lane >> 4) * 8;

  for (int c = ks; c < nch; c += ksplit) {
    const bool summ = (c == nch_bw);
    const bf16* Kc = summ ? sKs + (size_t)hh * 16 * row : sKbw + (size_t)c * 16 * row;
    const bf16* Vc = summ ? sVs + (size_t)hh * 16 * row : sVbw + (size_t)c * 16 * row;
    const int nvalid = summ ? p.R : min(16, nbw - c * 16);
    float s[2][4];
#pragma unroll
    for (int n = 0; n < 2; ++n) s[n][0] = s[n][1] = s[n][2] = s[n][3] = 0.f;
    const bf16* kb = Kc + (size_t)((lane & 7) + (lane >> 4) * 8) * row + ((lane >> 3) & 1) * 8;
#pragma unroll
    for (int kk = 0; kk < kHD / 16; ++kk) {
      uint32_t a[4], bk[4];
      ldsm_x4(a, qbase + kk * 16);
      ldsm_x4(bk, kb + kk * 16);
      mma_bf16(s[0], a, bk[0], bk[1]);
      mma_bf16(s[1], a, bk[2], bk[3]);
    }
#pragma unroll
    for (int n = 0; n < 2; ++n)
#pragma unroll
      for (int e = 0; e < 4; ++e)
        if (n * 8 + (lane & 3) * 2 + (e & 1) >= nvalid) s[n][e] = -INFINITY;
    float mx0 = fmaxf(fmaxf(s[0][0], s[0][1]), fmaxf(s[1][0], s[1][1]));
    float mx1 = fmaxf(fmaxf(s[0][2], s[0][3]), fmaxf(s[1][2], s[1][3]));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float n0 = fmaxf(rmax[0], mx0), n1 = fmaxf(rmax[1], mx1);
    const float b0 = (n0 == -INFINITY) ? 0.f : n0, b1 = (n1 == -INFINITY) ? 0.f : n1;
    const float sc0 = exp2f((rmax[0] - b0) * sl2), sc1 = exp2f((rmax[1] - b1) * sl2);
    rmax[0] = n0;
    rmax[1] = n1;
    float pr[2][4];
#pragma unroll
    for (int n = 0; n < 2; ++n) {
      pr[n][0] = exp2f((s[n][0] - b0) * sl2);
      pr[n][1] = exp2f((s[n][1] - b0) * sl2);
      pr[n][2] = exp2f((s[n][2] - b1) * sl2);
      pr[n][3] = exp2f((s[n][3] - b1) * sl2);
    }
    rsum[0] = rsum[0] * sc0 + pr[0][0] + pr[0][1] + pr[1][0] + pr[1][1];
    rsum[1] = rsum[1] * sc1 + pr[0][2] + pr[0][3] + pr[1][2] + pr[1][3];
#pragma unroll
    for (int n = 0; n < 16; ++n) {
      o[n][0] *= sc0; o[n][1] *= sc0;
      o[n][2] *= sc1; o[n][3] *= sc1;
    }
    uint32_t pa[4];
    pa[0] = pack_bf16(pr[0][0], pr[0][1]);
    pa[1] = pack_bf16(pr[0][2], pr[0][3]);
    pa[2] = pack_bf16(pr[1][0], pr[1][1]);
    pa[3] = pack_bf16(pr[1][2], pr[1][3]);
    const bf16* vb = Vc + (size_t)((lane & 7) + ((lane >> 3) & 1) * 8) * row + (lane >> 4) * 8;
#pragma unroll
    for (int np = 0; np < kHD / 16; ++np) {
      uint32_t bv[4];
      ldsm_x4_t(bv, vb + np * 16);
      mma_bf16(o[2 * np], pa, bv[0], bv[1]);
      mma_bf16(o[2 * np + 1], pa, bv[2], bv[3]);
    }
  }
  rsum[0] += __shfl_xor_sync(0xffffffffu, rsum[0], 1);
  rsum[0] += __shfl_xor_sync(0xffffffffu, rsum[0], 2);
  rsum[1] += __shfl_xor_sync(0xffffffffu, rsum[1], 1);
  rsum[1] += __shfl_xor_sync(0xffffffffu, rsum[1], 2);

  // ---- merge the key splits of each head (scratch reuses the K/V staging area)
  __syncthreads();
  float* scratch = reinterpret_cast<float*>(sKbw);
  float* so = scratch + (size_t)warp * kMergeRec;
  float* sml = so + 16 * kOs;
  const int r0 = lane >> 2;
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
  __syncthreads();
  bf16* out = static_cast<bf16*>(p.out);
  const int ldo = p.nq * kHD;
  // thread -> (head h2, query i, 4 columns e..e+3)
  for (int idx = tid; idx < rep * B * (kHD / 4); idx += nthr) {
    const int e = (idx % (kHD / 4)) * 4, i = (idx / (kHD / 4)) % B, h2 = idx / ((kHD / 4) * B);
    const float* base = scratch + (size_t)h2 * ksplit * kMergeRec;
    float M = -INFINITY;
    for (int k = 0; k < ksplit; ++k) M = fmaxf(M, base[(size_t)k * kMergeRec + 16 * kOs + i]);
    float4 num = make_float4(0.f, 0.f, 0.f, 0.f);
    float den = 0.f;
    for (int k = 0; k < ksplit; ++k) {
      const float* sw = base + (size_t)k * kMergeRec;
      const float f = exp2f((sw[16 * kOs + i] - M) * sl2);
      den += f * sw[16 * kOs + 16 + i];
      const float4 v = *reinterpret_cast<const float4*>(sw + i * kOs + e);
      num.x += f * v.x;
      num.y += f * v.y;
      num.z += f * v.z;
      num.w += f * v.w;
    }
    const float inv = 1.0f / den;
    uint2 wv;
    wv.x = pack_bf16(num.x * inv, num.y * inv);
    wv.y = pack_bf16(num.z * inv, num.w * inv);
    *reinterpret_cast<uint2*>(out + (size_t)(b * B + i) * ldo + (size_t)(g * rep + h2) * kHD + e) = wv;
  }
}

// ------------------------------------------------------------ fp32 reference shape
constexpr int kSimpleChunk = 64;    // window / summary rows staged per round trip

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
__global__ void __launch_bounds__(256) attn_simple_kernel(const AttnParams p) {
  extern __shared__ float ssm[];
  const int d = p.d, B = p.B;
  const int rep = p.nq / p.nkv;
  const int b = blockIdx.x / p.nq, h = blockIdx.x % p.nq, g = h / rep;
  const long long t = p.t[b];
  const int count = (int)(t < p.W ? t : p.W);
  const int ctx = B + count + p.R;
  float* sq = ssm;
  float* sk = sq + B * d;
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
    (kind == 0 ? sq : kind == 1 ? sk : sv)[i * d + e] = to_f(qkv[mrow + col + e]);
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
  // Lanes split into groups of `lpq` per block query (lpq = the largest power
  // of two with lpq * B <= 32, queries in passes of 32 / lpq); lane c of a
  // group covers dims c, c + lpq, ... so a score needs log2(lpq) shuffles.
  int lpq = 1;
  while (lpq * 2 * B <= 32) lpq *= 2;
  const int qpp = 32 / lpq, qi = lane / lpq, c = lane % lpq;
  auto score = [&](const float* krow, int j) {   // j: context index of the key
    for (int i0 = 0; i0 < B; i0 += qpp) {
      const int i = i0 + qi;
      float part = 0.f;
      if (i < B)
        for (int e = c; e < d; e += lpq) part = fmaf(sq[i * d + e], krow[e], part);
      for (int o = lpq / 2; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
      if (i < B && c == 0) ss[i * ctx + j] = part * scale;
    }
  };
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
// One warp per (block row, head): the sum of the q/k/v projection's split-K
// partials in split order, then for q and k heads the per-head RMSNorm and the
// rotary embedding (pairs f, f + d/2; lane l holds elements EPL*l .. EPL*l+EPL-1,
// its rotary partner lives in lane l ^ 16).
template <typename T, int EPL>
__global__ void __launch_bounds__(256) qkv_finalize_kernel(const QkvParams p) {
  // wait first, then let the attention kernel launch: it reads the view
  // state before its own wait, which is safe once the q/k/v projection (and
  // so every kernel before it) has completed
  griddep_wait();
  griddep_launch();
  const int heads = p.nq + 2 * p.nkv;
  const int item = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (item >= p.M * heads) return;
  const int m = item / heads, h = item % heads;
  const int d = EPL * 32, half = d / 2;
  const size_t ldq = (size_t)heads * d;
  const size_t pstride = (size_t)p.M * ldq;
  const float* src = p.part + (size_t)m * ldq + (size_t)h * d + EPL * lane;
  // the lane's EPL consecutive values of every split as one vector load each,
  // all in flight before the adds (which run in split order)
  using V = typename std::conditional<EPL == 4, float4, float2>::type;
  float x[EPL];
  {
    const V v0 = __ldcs(reinterpret_cast<const V*>(src));     // partials are read once
    const float* f0 = reinterpret_cast<const float*>(&v0);
#pragma unroll
    for (int e = 0; e < EPL; ++e) x[e] = f0[e];
  }
  for (int s0 = 1; s0 < p.splits; s0 += 8) {
    V y[8];
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (s0 + u < p.splits) y[u] = __ldcs(reinterpret_cast<const V*>(src + (size_t)(s0 + u) * pstride));
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (s0 + u < p.splits) {
        const float* f = reinterpret_cast<const float*>(&y[u]);
#pragma unroll
        for (int e = 0; e < EPL; ++e) x[e] += f[e];
      }
  }
  if (h < p.nq + p.nkv) {
    const T* w = static_cast<const T*>(h < p.nq ? p.q_norm : p.k_norm) + EPL * lane;
    float ss = 0.f;
#pragma unroll
    for (int e = 0; e < EPL; ++e) ss += x[e] * x[e];
    const float rstd = rsqrtf(warp_sum(ss) / (float)d + p.eps);
#pragma unroll
    for (int e = 0; e < EPL; ++e) x[e] *= rstd * to_f(w[e]);
    const int b = m / p.B, i = m % p.B;
    const float* cs = p.rope + ((size_t)(b * p.B + i) * half + EPL * (lane & 15)) * 2;
    const float sg = lane < 16 ? -1.f : 1.f;
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
      const float partner = __shfl_xor_sync(0xffffffffu, x[e], 16);
      x[e] = x[e] * cs[2 * e] + sg * partner * cs[2 * e + 1];
    }
  }
  T* out = static_cast<T*>(p.out) + (size_t)m * ldq + (size_t)h * d + EPL * lane;
#pragma unroll
  for (int e = 0; e < EPL; ++e) out[e] = from_f<T>(x[e]);
}

int launch_qkv_finalize(const QkvParams& p, int dtype, cudaStream_t s) {
  const int items = p.M * (p.nq + 2 * p.nkv);
  const dim3 grid((items + 7) / 8);
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

int attn_ksplit(int B, int W, int nq, int nkv) {
  const int rep = nq / nkv;
  int ks = rep >= 16 ? 1 : 16 / rep;
  while (ks > 1) {
    AttnLayout a = attn_layout(B, W, nq, nkv, ks);
    if (attn_merge_bytes(a.nwarps) <= a.bytes - a.off_kbw && a.nwarps <= 16) break;
    --ks;
  }
  return ks;
}

size_t attn_smem_bytes(int B, int W, int nq, int nkv) {
  AttnLayout a = attn_layout(B, W, nq, nkv, attn_ksplit(B, W, nq, nkv));
  return a.bytes;
}

int launch_attention(const AttnParams& p, int dtype, cudaStream_t s) {
  if (dtype == LSP_DTYPE_BF16) {
    if (p.d != kHD || p.B > 16 || p.R > 16) return LSP_ERR_SHAPE;
    const int ks = attn_ksplit(p.B, p.W, p.nq, p.nkv);
    AttnLayout a = attn_layout(p.B, p.W, p.nq, p.nkv, ks);
    if (a.bytes > 227 * 1024 || attn_merge_bytes(a.nwarps) > a.bytes - a.off_kbw) return LSP_ERR_SHAPE;
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
    const size_t smem = (size_t)(3 * p.B * p.d + p.B * ctx + 4 + kSimpleChunk * p.d) * sizeof(float);
    if (smem > 227 * 1024) return LSP_ERR_SHAPE;
    static bool attr32 = false;
    if (!attr32) {
      cudaFuncSetAttribute(attn_simple_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           227 * 1024);
      attr32 = true;
    }
    if (launch_pdl(attn_simple_kernel<float>, dim3(p.C * p.nq), dim3(256), smem, s, p) != cudaSuccess)
      return LSP_ERR_CUDA;
  }
  return cudaGetLastError() == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

}  // namespace lsp
