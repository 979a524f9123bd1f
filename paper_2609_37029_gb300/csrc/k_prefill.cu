// Prefill: build one request's interface from its whole prefix (Sec. 2.2,
// Eq. global-summary, App. A.2; the summary is initialised over the full prefix
// during target prefill, Fig. 3).
//
// For every tapped layer l and query head h the summary is attention of the R
// summary queries over all t prefix rows,
//     s_j = g_r . k_j / sqrt(d),  eta = log sum_j exp(s_j),
//     m   = sum_j exp(s_j - eta) v_j,
// and the interface also keeps the last min(t, W) rows in the window ring
// (prefix row p in slot p mod W), the hidden state of row t-1 as the boundary,
// and t.  This is the drafter's one O(t) step: at 128K rows it reads ~2.7 GB of
// tapped K/V per request at the Qwen3-8B shape, so it is split over the GPU:
//
// prefill_partial_kernel: one CTA per (prefix segment, tapped layer x KV head),
// one warp per query head of that KV head (R <= 16 queries = one m16 tile).
// 64-row K/V chunks are double-buffered through shared memory with cp.async;
// scores G K^T come from mma.sync m16n8k16 (bf16 inputs are exact, fp32
// accumulate) with an online softmax; P V uses P split into a bf16 high part
// and a bf16 remainder (two MMAs), which keeps the probabilities to ~16
// significant bits.  Each CTA writes the segment's (eta_s, m_s).
//
// prefill_merge_kernel: folds the segments in segment order with Eq.
// summary-update (eta = log(e^eta_a + e^eta_s), m = e^(eta_a - eta) m_a +
// e^(eta_s - eta) m_s) -- deterministic -- and writes (eta, m) into the state;
// further CTAs copy the window rows and the boundary hidden state and set t.
#include <algorithm>
#include <cstdlib>

#include "common.cuh"
#include "lsp_internal.h"

namespace lsp {

constexpr int kPfD = 128;                 // head dim of this path
constexpr int kPfLd = kPfD + 8;           // smem row stride (bf16): conflict-free ldmatrix
constexpr int kPfChunk = 64;              // segment granularity (a multiple of every stage size)
constexpr int kPfRec = 16 + 16 * kPfD;    // floats per (segment, layer, query head): eta[16], m[16][d]
constexpr int kPrefillStage = 32;         // default K/V rows per pipeline stage (measured: 745 vs 897 us at 64)

// CH = K/V rows per pipeline stage (32 or 64): smaller stages leave room for
// more CTAs per SM (shared memory and registers) at the same MMA work.
template <int CH>
__global__ void __launch_bounds__(256)
    prefill_partial_kernel(const PrefillParams p, const int rep, const int seg_rows) {
  extern __shared__ __align__(16) uint8_t psm[];
  const size_t row = kPfLd;
  bf16* sG = reinterpret_cast<bf16*>(psm);                   // [rep * 16][kPfLd]
  bf16* sK = sG + (size_t)rep * 16 * row;                    // [2][CH][kPfLd]
  bf16* sV = sK + (size_t)2 * CH * row;                      // [2][CH][kPfLd]

  const int nthr = rep * 32;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int seg = blockIdx.x, lg = blockIdx.y;
  const int l = lg / p.nkv, g = lg % p.nkv;
  const int r_begin = seg * seg_rows;
  const int r_end = min(p.rows, r_begin + seg_rows);
  const int nrows = r_end - r_begin;
  const int nchunks = (nrows + CH - 1) / CH;
  griddep_launch();
  griddep_wait();

  // ---- summary queries of the rep heads of KV head g (rows >= R are zero)
  const bf16* Gp = static_cast<const bf16*>(p.G) + ((size_t)l * p.nq + (size_t)g * rep) * p.R * kPfD;
  for (int idx = tid; idx < rep * 16 * 16; idx += nthr) {
    const int hr = idx >> 4, c8 = (idx & 15) * 8, hh = hr >> 4, r = hr & 15;
    bf16* dq = sG + (size_t)hr * row + c8;
    if (r < p.R) cp_async16(dq, Gp + ((size_t)hh * p.R + r) * kPfD + c8);
    else *reinterpret_cast<uint4*>(dq) = make_uint4(0, 0, 0, 0);
  }
  // ---- one CH-row chunk of this segment's K/V into buffer `buf`; rows past the
  // segment are zero (their scores are masked and their value rows add nothing)
  const bf16* kin = static_cast<const bf16*>(p.k) + (size_t)l * p.rows * p.nkv * kPfD + (size_t)g * kPfD;
  const bf16* vin = static_cast<const bf16*>(p.v) + (size_t)l * p.rows * p.nkv * kPfD + (size_t)g * kPfD;
  const size_t rstride = (size_t)p.nkv * kPfD;
  auto stage = [&](int c, int buf) {
    for (int idx = tid; idx < CH * 16; idx += nthr) {
      const int j = idx >> 4, c8 = (idx & 15) * 8;
      const int rr = r_begin + c * CH + j;
      bf16* dk = sK + ((size_t)buf * CH + j) * row + c8;
      bf16* dv = sV + ((size_t)buf * CH + j) * row + c8;
      if (rr < r_end) {
        cp_async16(dk, kin + (size_t)rr * rstride + c8);
        cp_async16(dv, vin + (size_t)rr * rstride + c8);
      } else {
        *reinterpret_cast<uint4*>(dk) = make_uint4(0, 0, 0, 0);
        *reinterpret_cast<uint4*>(dv) = make_uint4(0, 0, 0, 0);
      }
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  stage(0, 0);
  if (nchunks > 1) stage(1, 1);
  else asm volatile("cp.async.commit_group;" ::: "memory");

  const int hh = warp;
  const float sl2 = 1.4426950408889634f * rsqrtf((float)kPfD);
  float rmax[2] = {-INFINITY, -INFINITY}, rsum[2] = {0.f, 0.f};
  float o[16][4];
#pragma unroll
  for (int n = 0; n < 16; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  const bf16* qbase = sG + (size_t)(hh * 16 + (lane & 15)) * row + (lane >> 4) * 8;

  for (int c = 0; c < nchunks; ++c) {
    const int buf = c & 1;
    asm volatile("cp.async.wait_group 1;" ::: "memory");      // chunk c has landed
    __syncthreads();
    const bf16* Kc = sK + (size_t)buf * CH * row;
    const bf16* Vc = sV + (size_t)buf * CH * row;
    const int nvalid = min(CH, nrows - c * CH);
    // scores of the warp's 16 queries against the CH rows: s[n] covers keys 8n..8n+7
    constexpr int NS = CH / 8;
    float s[NS][4];
#pragma unroll
    for (int n = 0; n < NS; ++n) s[n][0] = s[n][1] = s[n][2] = s[n][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < kPfD / 16; ++kk) {
      uint32_t a[4];
      ldsm_x4(a, qbase + kk * 16);
#pragma unroll
      for (int nt = 0; nt < CH / 16; ++nt) {
        uint32_t bk[4];
        ldsm_x4(bk, Kc + (size_t)(nt * 16 + (lane & 7) + (lane >> 4) * 8) * row + ((lane >> 3) & 1) * 8 + kk * 16);
        mma_bf16(s[2 * nt], a, bk[0], bk[1]);
        mma_bf16(s[2 * nt + 1], a, bk[2], bk[3]);
      }
    }
#pragma unroll
    for (int n = 0; n < NS; ++n)
#pragma unroll
      for (int e = 0; e < 4; ++e)
        if (n * 8 + (lane & 3) * 2 + (e & 1) >= nvalid) s[n][e] = -INFINITY;
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int n = 0; n < NS; ++n) {
      mx0 = fmaxf(mx0, fmaxf(s[n][0], s[n][1]));
      mx1 = fmaxf(mx1, fmaxf(s[n][2], s[n][3]));
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float n0 = fmaxf(rmax[0], mx0), n1 = fmaxf(rmax[1], mx1);
    const float b0 = (n0 == -INFINITY) ? 0.f : n0, b1 = (n1 == -INFINITY) ? 0.f : n1;
    const float sc0 = exp2f((rmax[0] - b0) * sl2), sc1 = exp2f((rmax[1] - b1) * sl2);
    rmax[0] = n0;
    rmax[1] = n1;
    float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
    for (int n = 0; n < NS; ++n) {
      s[n][0] = exp2f((s[n][0] - b0) * sl2);
      s[n][1] = exp2f((s[n][1] - b0) * sl2);
      s[n][2] = exp2f((s[n][2] - b1) * sl2);
      s[n][3] = exp2f((s[n][3] - b1) * sl2);
      ps0 += s[n][0] + s[n][1];
      ps1 += s[n][2] + s[n][3];
    }
    rsum[0] = rsum[0] * sc0 + ps0;
    rsum[1] = rsum[1] * sc1 + ps1;
#pragma unroll
    for (int n = 0; n < 16; ++n) {
      o[n][0] *= sc0; o[n][1] *= sc0;
      o[n][2] *= sc1; o[n][3] *= sc1;
    }
    // P V over the CH rows in 16-row steps; P = hi + lo, both bf16
#pragma unroll
    for (int ks = 0; ks < CH / 16; ++ks) {
      uint32_t ph[4], pl[4];
      const float* q0 = s[2 * ks];
      const float* q1 = s[2 * ks + 1];
      const float pv[8] = {q0[0], q0[1], q0[2], q0[3], q1[0], q1[1], q1[2], q1[3]};
      float hi[8], lo[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        hi[e] = __bfloat162float(__float2bfloat16_rn(pv[e]));
        lo[e] = pv[e] - hi[e];
      }
      // A fragment of m16n8k16: (row r0, keys 2q..2q+1), (row r0+8, ...), (row r0, keys 8+2q..), (row r0+8, ...)
      ph[0] = pack_bf16(hi[0], hi[1]); ph[1] = pack_bf16(hi[2], hi[3]);
      ph[2] = pack_bf16(hi[4], hi[5]); ph[3] = pack_bf16(hi[6], hi[7]);
      pl[0] = pack_bf16(lo[0], lo[1]); pl[1] = pack_bf16(lo[2], lo[3]);
      pl[2] = pack_bf16(lo[4], lo[5]); pl[3] = pack_bf16(lo[6], lo[7]);
      const bf16* vb = Vc + (size_t)(ks * 16 + (lane & 7) + ((lane >> 3) & 1) * 8) * row + (lane >> 4) * 8;
#pragma unroll
      for (int np = 0; np < kPfD / 16; ++np) {
        uint32_t bv[4];
        ldsm_x4_t(bv, vb + np * 16);
        mma_bf16(o[2 * np], ph, bv[0], bv[1]);
        mma_bf16(o[2 * np + 1], ph, bv[2], bv[3]);
        mma_bf16(o[2 * np], pl, bv[0], bv[1]);
        mma_bf16(o[2 * np + 1], pl, bv[2], bv[3]);
      }
    }
    __syncthreads();                                          // buffer `buf` is free again
    if (c + 2 < nchunks) stage(c + 2, buf);
    else asm volatile("cp.async.commit_group;" ::: "memory");
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  rsum[0] += __shfl_xor_sync(0xffffffffu, rsum[0], 1);
  rsum[0] += __shfl_xor_sync(0xffffffffu, rsum[0], 2);
  rsum[1] += __shfl_xor_sync(0xffffffffu, rsum[1], 1);
  rsum[1] += __shfl_xor_sync(0xffffffffu, rsum[1], 2);

  // ---- this segment's (eta_s, m_s) of query head g*rep + hh: eta in natural log
  float* rec = p.ws + (((size_t)seg * gridDim.y + lg) * rep + hh) * kPfRec;
  const int r0 = lane >> 2;
  const float inv0 = 1.0f / rsum[0], inv1 = 1.0f / rsum[1];
  const float isd = rsqrtf((float)kPfD);
  if ((lane & 3) == 0) {
    rec[r0] = rmax[0] * isd + logf(rsum[0]);
    rec[r0 + 8] = rmax[1] * isd + logf(rsum[1]);
  }
  float* mrec = rec + 16;
#pragma unroll
  for (int n = 0; n < 16; ++n) {
    const int col = n * 8 + (lane & 3) * 2;
    *reinterpret_cast<float2*>(mrec + r0 * kPfD + col) = make_float2(o[n][0] * inv0, o[n][1] * inv0);
    *reinterpret_cast<float2*>(mrec + (r0 + 8) * kPfD + col) = make_float2(o[n][2] * inv1, o[n][3] * inv1);
  }
}

// blockIdx.x < L*nq: (l, h) summary merge, 256 threads = 16 rows x 16 eight-column groups.
// blockIdx.x >= L*nq: (l, g) window rows and boundary state (and t).
template <typename T>
__global__ void __launch_bounds__(256) prefill_merge_kernel(const PrefillParams p, const int nseg) {
  griddep_launch();
  griddep_wait();
  const int b = p.b;
  const int nsum = p.L * p.nq;
  if ((int)blockIdx.x < nsum) {
    const int l = blockIdx.x / p.nq, h = blockIdx.x % p.nq;
    const int rep = p.nq / p.nkv, g = h / rep, hh = h % rep;
    const int r = threadIdx.x >> 4, c0 = (threadIdx.x & 15) * 8;
    if (r >= p.R) return;
    const int lg = l * p.nkv + g;
    float eta = -INFINITY, m[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) m[e] = 0.f;
    for (int s = 0; s < nseg; ++s) {
      const float* rec = p.ws + (((size_t)s * p.L * p.nkv + lg) * rep + hh) * kPfRec;
      const float es = __ldcg(rec + r);
      const float4 a = __ldcg(reinterpret_cast<const float4*>(rec + 16 + r * kPfD + c0));
      const float4 bb = __ldcg(reinterpret_cast<const float4*>(rec + 16 + r * kPfD + c0 + 4));
      const float ms[8] = {a.x, a.y, a.z, a.w, bb.x, bb.y, bb.z, bb.w};
      // Eq. summary-update (eta = -inf before the first segment gives (eta_s, m_s))
      const float mx = fmaxf(eta, es);
      const float ne = mx + logf(expf(eta - mx) + expf(es - mx));
      const float ca = expf(eta - ne), cs = expf(es - ne);
#pragma unroll
      for (int e = 0; e < 8; ++e) m[e] = ca * m[e] + cs * ms[e];
      eta = ne;
    }
    const size_t q = (((size_t)b * p.L + l) * p.nq + h) * p.R + r;
    float* mo = p.m + q * p.d + c0;
    *reinterpret_cast<float4*>(mo) = make_float4(m[0], m[1], m[2], m[3]);
    *reinterpret_cast<float4*>(mo + 4) = make_float4(m[4], m[5], m[6], m[7]);
    if ((threadIdx.x & 15) == 0) p.eta[q] = eta;
    return;
  }
  // ---- window ring (prefix row q in slot q mod W) and boundary of layer l
  const int lg = blockIdx.x - nsum, l = lg / p.nkv, g = lg % p.nkv;
  const int vec = 16 / (int)sizeof(T), vpr = p.d / vec;           // 16-byte vectors per row
  const int first = p.rows > p.W ? p.rows - p.W : 0;
  const size_t rstride = (size_t)p.nkv * p.d;
  const T* kin = static_cast<const T*>(p.k) + (size_t)l * p.rows * rstride + (size_t)g * p.d;
  const T* vin = static_cast<const T*>(p.v) + (size_t)l * p.rows * rstride + (size_t)g * p.d;
  T* wk = static_cast<T*>(p.win_k) + (((size_t)b * p.L + l) * p.nkv + g) * p.W * p.d;
  T* wv = static_cast<T*>(p.win_v) + (((size_t)b * p.L + l) * p.nkv + g) * p.W * p.d;
  for (int idx = threadIdx.x; idx < (p.rows - first) * vpr; idx += blockDim.x) {
    const int q = first + idx / vpr, c = (idx % vpr) * vec;
    const size_t slot = (size_t)(q % p.W) * p.d + c;
    *reinterpret_cast<uint4*>(wk + slot) = *reinterpret_cast<const uint4*>(kin + (size_t)q * rstride + c);
    *reinterpret_cast<uint4*>(wv + slot) = *reinterpret_cast<const uint4*>(vin + (size_t)q * rstride + c);
  }
  if (g == 0) {
    if (p.h) {   // no boundary state is kept with LSP_NO_BOUNDARY
      const T* hin = static_cast<const T*>(p.hid) + ((size_t)l * p.h_rows + (p.h_rows - 1)) * p.H;
      T* hout = static_cast<T*>(p.h) + ((size_t)b * p.L + l) * p.H;
      for (int i = threadIdx.x * vec; i < p.H; i += blockDim.x * vec)
        *reinterpret_cast<uint4*>(hout + i) = *reinterpret_cast<const uint4*>(hin + i);
    }
    if (l == 0 && threadIdx.x == 0) p.t[b] = p.rows;
  }
}

size_t prefill_ws_floats(int L, int nq) { return (size_t)kPrefillMaxSeg * L * nq * kPfRec; }

int launch_prefill(const PrefillParams& p, int dtype, cudaStream_t s) {
  const int rep = p.nq / p.nkv;
  if (dtype != LSP_DTYPE_BF16 || p.d != kPfD || p.R > 16 || p.R < 0 || rep > 8 || p.rows < 1 || !p.ws)
    return LSP_ERR_UNSUPPORTED;
  if (p.H % 8) return LSP_ERR_SHAPE;
  // segments of a multiple of 64 rows, at most kPrefillMaxSeg of them
  int seg_rows = (p.rows + kPrefillMaxSeg - 1) / kPrefillMaxSeg;
  seg_rows = std::max(kPfChunk, (seg_rows + kPfChunk - 1) / kPfChunk * kPfChunk);
  const int nseg = (p.rows + seg_rows - 1) / seg_rows;
  // K/V rows per pipeline stage
  constexpr int ch = kPrefillStage;
  const size_t smem = ((size_t)rep * 16 + 4 * ch) * kPfLd * sizeof(bf16);
  if (smem > 227 * 1024) return LSP_ERR_SHAPE;
  auto kern = prefill_partial_kernel<ch>;
  static size_t attr = 0;
  if (smem > attr) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
      return LSP_ERR_CUDA;
    attr = smem;
  }
  // R = 0 (no summary): only the window, boundary and t are written
  if ((p.R > 0 && launch_pdl(kern, dim3(nseg, p.L * p.nkv), dim3(rep * 32), smem, s, p, rep, seg_rows) !=
                      cudaSuccess) ||
      launch_pdl(prefill_merge_kernel<bf16>, dim3(p.L * p.nq + p.L * p.nkv), dim3(256), 0, s, p, nseg) !=
          cudaSuccess)
    return LSP_ERR_CUDA;
  return LSP_OK;
}

}  // namespace lsp
