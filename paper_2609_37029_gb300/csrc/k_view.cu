// View update: fold newly accepted target rows into the fixed-size interface.
//
// Sec. 2.2 / App. A.2: for every tapped layer l, query head h and summary
// query g_r, the statistics of the new rows N are
//     s_j = g_r . k_j / sqrt(d),  eta_N = log sum_j exp(s_j),
//     m_N = sum_j exp(s_j - eta_N) v_j,
// and they merge into the stored (eta_A, m_A) by Eq. summary-update:
//     eta = log(e^eta_A + e^eta_N),  m = e^(eta_A-eta) m_A + e^(eta_N-eta) m_N.
// The same pass writes the new K/V rows into the window ring (prefix row p in
// slot p mod W), copies the boundary hidden state of the last new row, and the
// last CTA of each request advances t.
//
// One CTA per (request b, tapped layer l, KV head g) covers the nq/nkv query
// heads sharing that KV head (rep * R queries); the new K/V rows are read from
// HBM once (16-byte vectors) and only the new rows are touched.
// view_update_mma_kernel (bf16, d = 128, rep * R a multiple of 16 up to
// 128): the statistics are an attention of the summary queries over the new
// rows, run as mma.sync tiles with an online softmax (below).  view_update_kernel (every
// other shape): rows staged in shared memory as fp32; each warp owns whole
// queries, lanes split the head dimension, and the dot products and the row
// max/sum reduce with warp shuffles.
#include <cstdlib>

#include "common.cuh"
#include "lsp_internal.h"

namespace lsp {

constexpr int kViewThreads = 256;
constexpr int kViewWarps = kViewThreads / 32;
constexpr int kViewChunk = 32;       // new rows staged per pass (one per lane)

// N (2 or 4) consecutive fp32 / bf16 values <-> registers with one vector access
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
    const uint32_t r = *reinterpret_cast<const uint32_t*>(p);
    const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&r));
    v[0] = a.x; v[1] = a.y;
  }
}
template <int N>
__device__ __forceinline__ void store_vec(float* p, const float* v) {
  if constexpr (N == 4) *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  else *reinterpret_cast<float2*>(p) = make_float2(v[0], v[1]);
}

template <typename T, int DPL, int QPW>
__global__ void __launch_bounds__(kViewThreads)
    view_update_kernel(const ViewParams p) {
  extern __shared__ float vsm[];
  const int d = DPL * 32;
  float* sK = vsm;                              // [kViewChunk][d]
  float* sV = vsm + kViewChunk * d;             // [kViewChunk][d]

  const int unit = blockIdx.x;
  const int g = unit % p.nkv;
  const int l = (unit / p.nkv) % p.L;
  const int b = unit / (p.nkv * p.L);
  const int rep = p.nq / p.nkv;
  const int Q = rep * p.R;                      // queries handled by this CTA
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  griddep_launch();
  griddep_wait();

  int delta = p.acc[b];
  if (delta < 0 || delta > p.rows) {
    if (threadIdx.x == 0 && g == 0 && l == 0) set_err(p.err, LSP_DEV_BAD_DELTA);
    return;
  }
  if (delta == 0) return;                        // empty new set: state unchanged (App. A.2)
  const long long t0 = p.t[b];
  const size_t es = sizeof(T);

  // ---- this warp's queries: stored state and summary query vectors
  const size_t qbase = ((size_t)(b * p.L + l) * p.nq + (size_t)g * rep) * p.R;   // first query row
  const size_t gbase = ((size_t)l * p.nq + (size_t)g * rep) * p.R;
  const T* Gp = static_cast<const T*>(p.G);
  float ma[QPW][DPL], gq[QPW][DPL], eta_a[QPW];
#pragma unroll
  for (int i = 0; i < QPW; ++i) {
    const int q = warp + i * kViewWarps;
    eta_a[i] = -INFINITY;
#pragma unroll
    for (int e = 0; e < DPL; ++e) { ma[i][e] = 0.f; gq[i][e] = 0.f; }
    if (q < Q) {
      eta_a[i] = p.eta[qbase + q];
      // the lane's DPL consecutive entries as one vector load each
      load_vec<DPL>(p.m + (qbase + q) * d + lane * DPL, ma[i]);
      load_vec<DPL>(Gp + (gbase + q) * d + lane * DPL, gq[i]);
    }
  }
  const float scale = rsqrtf((float)d);

  // ---- stream the new rows in chunks
  const T* kin = static_cast<const T*>(p.k_new);
  const T* vin = static_cast<const T*>(p.v_new);
  T* wk = static_cast<T*>(p.win_k);
  T* wv = static_cast<T*>(p.win_v);
  const size_t row_stride = (size_t)p.nkv * d;                         // elements per new row
  const size_t in_base = (size_t)(b * p.L + l) * p.rows * row_stride + (size_t)g * d;
  const size_t win_base = ((size_t)(b * p.L + l) * p.nkv + g) * (size_t)p.W * d;
  const int vec = 16 / (int)es;                                        // elements per 16-byte vector
  const int vecs_per_row = d / vec;

  for (int j0 = 0; j0 < delta; j0 += kViewChunk) {
    const int nrows = min(kViewChunk, delta - j0);
    __syncthreads();                     // previous chunk fully consumed
    for (int idx = threadIdx.x; idx < 2 * nrows * vecs_per_row; idx += kViewThreads) {
      const int which = idx / (nrows * vecs_per_row);                  // 0 = K, 1 = V
      const int rem = idx % (nrows * vecs_per_row);
      const int j = rem / vecs_per_row, c = rem % vecs_per_row;
      const T* src = (which ? vin : kin) + in_base + (size_t)(j0 + j) * row_stride + c * vec;
      const uint4 raw = *reinterpret_cast<const uint4*>(src);
      const long long pabs = t0 + j0 + j;                              // absolute prefix row
      if (p.W > 0 && j0 + j >= delta - p.W) {
        T* dst = (which ? wv : wk) + win_base + (size_t)(pabs % p.W) * d + c * vec;
        *reinterpret_cast<uint4*>(dst) = raw;
      }
      const T* ev = reinterpret_cast<const T*>(&raw);
      float* sd = (which ? sV : sK) + j * d + c * vec;
#pragma unroll
      for (int e = 0; e < 16 / (int)sizeof(T); ++e) sd[e] = to_f(ev[e]);
    }
    __syncthreads();

#pragma unroll
    for (int i = 0; i < QPW; ++i) {
      const int q = warp + i * kViewWarps;
      if (q >= Q) continue;                                            // warp-uniform
      // scores of this query over the chunk: lane j keeps s_j
      float s_mine = -INFINITY;
#pragma unroll 4
      for (int j = 0; j < nrows; ++j) {
        const float* kr = sK + j * d + lane * DPL;
        float part = 0.f;
#pragma unroll
        for (int e = 0; e < DPL; ++e) part = fmaf(gq[i][e], kr[e], part);
        const float s = warp_sum(part) * scale;
        if (lane == j) s_mine = s;
      }
      // eta_N and m_N of the chunk (max-subtracted log-sum-exp)
      const float mx_n = warp_max(s_mine);
      const float e_mine = (lane < nrows) ? __expf(s_mine - mx_n) : 0.f;
      const float z_n = warp_sum(e_mine);
      const float eta_n = mx_n + logf(z_n);
      float mn[DPL];
#pragma unroll
      for (int e = 0; e < DPL; ++e) mn[e] = 0.f;
#pragma unroll 4
      for (int j = 0; j < nrows; ++j) {
        const float pj = __shfl_sync(0xffffffffu, e_mine, j);
        const float* vr = sV + j * d + lane * DPL;
#pragma unroll
        for (int e = 0; e < DPL; ++e) mn[e] = fmaf(pj, vr[e], mn[e]);
      }
      const float inv_z = 1.0f / z_n;
      // merge (Eq. summary-update); eta_A = -inf gives (eta_N, m_N)
      const float mx = fmaxf(eta_a[i], eta_n);
      const float wa = __expf(eta_a[i] - mx), wn = __expf(eta_n - mx);
      const float eta = mx + logf(wa + wn);
      const float ca = __expf(eta_a[i] - eta), cn = __expf(eta_n - eta) * inv_z;
#pragma unroll
      for (int e = 0; e < DPL; ++e) ma[i][e] = ca * ma[i][e] + cn * mn[e];
      eta_a[i] = eta;
    }
  }

  // ---- write back the merged summary
#pragma unroll
  for (int i = 0; i < QPW; ++i) {
    const int q = warp + i * kViewWarps;
    if (q < Q) {
      store_vec<DPL>(p.m + (qbase + q) * d + lane * DPL, ma[i]);
      if (lane == 0) p.eta[qbase + q] = eta_a[i];
    }
  }

  // ---- boundary: hidden state of the last new row, this CTA's 1/nkv share
  if (p.h) {   // no boundary state is kept with LSP_NO_BOUNDARY
    const T* hin = static_cast<const T*>(p.h_new) +
                   ((size_t)(b * p.L + l) * p.h_rows + (p.h_rows == 1 ? 0 : delta - 1)) * p.H;
    T* hout = static_cast<T*>(p.h) + (size_t)(b * p.L + l) * p.H;
    const int per = p.H / p.nkv;
    for (int i = g * per + threadIdx.x * vec; i < (g + 1) * per; i += kViewThreads * vec)
      *reinterpret_cast<uint4*>(hout + i) = *reinterpret_cast<const uint4*>(hin + i);
  }

  // ---- the last CTA of request b advances t
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const int old = atomicAdd(&p.done[b], 1);
    if (old == p.L * p.nkv - 1) {
      p.t[b] = t0 + delta;
      p.done[b] = 0;
      __threadfence();
    }
  }
}

// ---------------------------------------------------------------- tensor-core variant
// bf16 storage, d = 128, Q = rep * R = 16 * MT queries (MT <= 8): the summary
// update is the attention of the Q summary queries over the new rows, so it
// runs as mma.sync m16n8k16 tiles.  Warp w owns query tile w (16 queries) and
// all 128 dims: per 16-row key chunk S = G K^T (bf16 products are exact, fp32
// accumulate), an online softmax in registers, and P V with P split into a
// bf16 high part and the bf16 remainder (two MMAs: ~16 significant bits of
// every weight).  Few registers a thread (the G fragments come from shared
// memory at each k-step, the stored state is not held), so 5 CTAs share an
// SM: at the Qwen3-8B shape all 640 CTAs run in one wave of 760 slots.
//
// The kernel is a latency chain per CTA (the whole grid moves ~45 MB), so the
// steps overlap where they can: G is staged before the dependency wait; the
// stored m block is prefetched into L2 and the boundary row copied while the
// new K/V rows land; the merge goes through shared memory so that one
// coalesced pass has all 16 loads a thread in flight at once (instead of four
// dependent rounds from the MMA fragment layout); and the t advance takes a
// ticket early instead of a fence after the stores.
constexpr int kVuRows = 32;                // new rows staged per pass
constexpr int kVuLd = 128 + 8;             // smem row (bf16): conflict-free ldmatrix
constexpr int kVuMLd = 128 + 8;            // merge row (fp32): conflict-free float2 stores

// dynamic shared memory: the staging buffers, later reused by the merge
constexpr size_t vu_smem_bytes(int MT) {
  const size_t stage = (size_t)(16 * MT + 2 * kVuRows) * kVuLd * 2;
  const size_t merge = (size_t)16 * MT * (kVuMLd + 1) * 4;
  return stage > merge ? stage : merge;
}

// CTAs per SM the launch bounds ask for, at most 8: 96 registers a thread
// suffice for 4 and 5 query tiles (no spills), the other counts take 112
constexpr int vu_min_blocks(int MT) {
  return (MT == 4 || MT == 5) ? 65536 / (MT * 32 * 96)
                              : (65536 / (MT * 32 * 112) > 8 ? 8 : 65536 / (MT * 32 * 112));
}

template <int MT>
__global__ void __launch_bounds__(MT * 32, vu_min_blocks(MT)) view_update_mma_kernel(const ViewParams p) {
  constexpr int NT = 16;                                   // 8-dim output tiles per warp (all 128 dims)
  constexpr int Q = 16 * MT;
  constexpr int kThreads = MT * 32;
  extern __shared__ __align__(16) uint8_t vsm_raw[];
  bf16* sG = reinterpret_cast<bf16*>(vsm_raw);             // [Q][kVuLd]
  bf16* sK = sG + Q * kVuLd;                               // [kVuRows][kVuLd]
  bf16* sV = sK + kVuRows * kVuLd;
  constexpr int d = 128;
  const int unit = blockIdx.x;
  const int g = unit % p.nkv;
  const int l = (unit / p.nkv) % p.L;
  const int b = unit / (p.nkv * p.L);
  const int rep = p.nq / p.nkv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  griddep_launch();
  // the summary queries are a constant of the state: stage them before the wait
  const size_t gbase = ((size_t)l * p.nq + (size_t)g * rep) * p.R;
  const bf16* Gp = static_cast<const bf16*>(p.G) + gbase * d;
  for (int i = tid; i < Q * 16; i += kThreads) {
    const int q = i >> 4, c = (i & 15) * 8;
    cp_async16(sG + q * kVuLd + c, Gp + (size_t)q * d + c);
  }
  const bf16* kin = static_cast<const bf16*>(p.k_new);
  const bf16* vin = static_cast<const bf16*>(p.v_new);
  const size_t row_stride = (size_t)p.nkv * d;
  const size_t in_base = (size_t)(b * p.L + l) * p.rows * row_stride + (size_t)g * d;
  // rows [j0, j0 + nv) of the new K and V into sK / sV by cp.async, zeros up to n16
  auto stage = [&](int j0, int nv, int n16) {
    for (int idx = tid; idx < 2 * n16 * 16; idx += kThreads) {
      const int which = idx / (n16 * 16), rem = idx % (n16 * 16);
      const int j = rem >> 4, c = (rem & 15) * 8;
      bf16* dst = (which ? sV : sK) + j * kVuLd + c;
      if (j < nv) cp_async16(dst, (which ? vin : kin) + in_base + (size_t)(j0 + j) * row_stride + c);
      else *reinterpret_cast<uint4*>(dst) = make_uint4(0u, 0u, 0u, 0u);
    }
  };
  griddep_wait();
  const int delta = p.acc[b];
  const long long t0 = p.t[b];
  const size_t qbase = ((size_t)(b * p.L + l) * p.nq + (size_t)g * rep) * p.R;
  const int r0 = warp * 16 + (lane >> 2);
  const float etaA[2] = {p.eta[qbase + r0], p.eta[qbase + r0 + 8]};
  if (delta < 0 || delta > p.rows) {
    if (tid == 0 && g == 0 && l == 0) set_err(p.err, LSP_DEV_BAD_DELTA);
    cp_async_wait_all();
    return;
  }
  if (delta == 0) { cp_async_wait_all(); return; }        // empty new set: state unchanged (App. A.2)
  // t[b] may change once every CTA of request b has read it: each CTA takes a
  // ticket now (a release atomic, ordered after the read of t) and the CTA that
  // takes the last one writes t[b] when it is done.  The ticket is consumed
  // only at the end, so nothing waits on it.
  int ticket = 0;
  if (tid == 0)
    asm volatile("atom.add.release.gpu.global.s32 %0, [%1], 1;" : "=r"(ticket) : "l"(p.done + b) : "memory");

  const float sl2 = 1.4426950408889634f * rsqrtf((float)d);   // log2(e) / sqrt(d)
  float rmax[2] = {-INFINITY, -INFINITY}, rsum[2] = {0.f, 0.f};
  float o[NT][4];
#pragma unroll
  for (int n = 0; n < NT; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;

  bf16* wk = static_cast<bf16*>(p.win_k);
  bf16* wv = static_cast<bf16*>(p.win_v);
  const size_t win_base = ((size_t)(b * p.L + l) * p.nkv + g) * (size_t)p.W * d;
  const bf16* qa = sG + (size_t)(warp * 16 + (lane & 15)) * kVuLd + (lane >> 4) * 8;

  for (int j0 = 0; j0 < delta; j0 += kVuRows) {
    const int nrows = min(kVuRows, delta - j0);
    const int nrows16 = (nrows + 15) / 16 * 16;
    if (j0 > 0) __syncthreads();                           // previous rows consumed
    stage(j0, nrows, nrows16);
    if (j0 == 0) {
      if (tid == 0)                                        // the stored m block into L2 for the merge
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p.m + qbase * d), "r"((uint32_t)(Q * d * 4))
                     : "memory");
      // boundary: hidden state of the last new row, this CTA's 1/nkv share
      if (p.h) {
        const bf16* hin = static_cast<const bf16*>(p.h_new) +
                          ((size_t)(b * p.L + l) * p.h_rows + (p.h_rows == 1 ? 0 : delta - 1)) * p.H;
        bf16* hout = static_cast<bf16*>(p.h) + (size_t)(b * p.L + l) * p.H;
        const int per = p.H / p.nkv;
        for (int i = g * per + tid * 8; i < (g + 1) * per; i += kThreads * 8)
          *reinterpret_cast<uint4*>(hout + i) = *reinterpret_cast<const uint4*>(hin + i);
      }
    }
    cp_async_wait_all();                                   // (the first pass also lands sG)
    __syncthreads();
    // the window ring: the last W rows of the new set, from shared memory
    if (p.W > 0) {
      for (int idx = tid; idx < 2 * nrows * 16; idx += kThreads) {
        const int which = idx / (nrows * 16), rem = idx % (nrows * 16);
        const int j = rem >> 4, c = (rem & 15) * 8;
        if (j0 + j >= delta - p.W) {
          const long long pabs = t0 + j0 + j;
          *reinterpret_cast<uint4*>((which ? wv : wk) + win_base + (size_t)(pabs % p.W) * d + c) =
              *reinterpret_cast<const uint4*>((which ? sV : sK) + j * kVuLd + c);
        }
      }
    }
    for (int c16 = 0; c16 < nrows16; c16 += 16) {
      // S = G K^T over 16 keys: two n8 tiles
      float sc[2][4];
#pragma unroll
      for (int n = 0; n < 2; ++n) sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
      const bf16* kb = sK + (size_t)(c16 + (lane & 7) + (lane >> 4) * 8) * kVuLd + ((lane >> 3) & 1) * 8;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        uint32_t ga[4], bk[4];
        ldsm_x4(ga, qa + kk * 16);
        ldsm_x4(bk, kb + kk * 16);
        mma_bf16(sc[0], ga, bk[0], bk[1]);
        mma_bf16(sc[1], ga, bk[2], bk[3]);
      }
      const int nvalid = nrows - c16;
#pragma unroll
      for (int n = 0; n < 2; ++n)
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (n * 8 + (lane & 3) * 2 + (e & 1) >= nvalid) sc[n][e] = -INFINITY;
      float mx0 = fmaxf(fmaxf(sc[0][0], sc[0][1]), fmaxf(sc[1][0], sc[1][1]));
      float mx1 = fmaxf(fmaxf(sc[0][2], sc[0][3]), fmaxf(sc[1][2], sc[1][3]));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
      const float n0 = fmaxf(rmax[0], mx0), n1 = fmaxf(rmax[1], mx1);   // finite: key 0 of a chunk is valid
      const float s0 = exp2f((rmax[0] - n0) * sl2), s1 = exp2f((rmax[1] - n1) * sl2);
      rmax[0] = n0;
      rmax[1] = n1;
      float pr[2][4];
#pragma unroll
      for (int n = 0; n < 2; ++n) {
        pr[n][0] = exp2f((sc[n][0] - n0) * sl2);
        pr[n][1] = exp2f((sc[n][1] - n0) * sl2);
        pr[n][2] = exp2f((sc[n][2] - n1) * sl2);
        pr[n][3] = exp2f((sc[n][3] - n1) * sl2);
      }
      rsum[0] = rsum[0] * s0 + pr[0][0] + pr[0][1] + pr[1][0] + pr[1][1];
      rsum[1] = rsum[1] * s1 + pr[0][2] + pr[0][3] + pr[1][2] + pr[1][3];
#pragma unroll
      for (int n = 0; n < NT; ++n) {
        o[n][0] *= s0; o[n][1] *= s0;
        o[n][2] *= s1; o[n][3] *= s1;
      }
      // P = high + remainder, both bf16
      uint32_t ph[4], pl[4];
      {
        const float q00 = pr[0][0], q01 = pr[0][1], q02 = pr[0][2], q03 = pr[0][3];
        const float q10 = pr[1][0], q11 = pr[1][1], q12 = pr[1][2], q13 = pr[1][3];
        ph[0] = pack_bf16(q00, q01); ph[1] = pack_bf16(q02, q03);
        ph[2] = pack_bf16(q10, q11); ph[3] = pack_bf16(q12, q13);
        auto rem_of = [](float x) { return x - __bfloat162float(__float2bfloat16_rn(x)); };
        pl[0] = pack_bf16(rem_of(q00), rem_of(q01)); pl[1] = pack_bf16(rem_of(q02), rem_of(q03));
        pl[2] = pack_bf16(rem_of(q10), rem_of(q11)); pl[3] = pack_bf16(rem_of(q12), rem_of(q13));
      }
      const bf16* vb = sV + (size_t)(c16 + (lane & 7) + ((lane >> 3) & 1) * 8) * kVuLd + (lane >> 4) * 8;
#pragma unroll
      for (int np = 0; np < NT / 2; ++np) {
        uint32_t bv[4];
        ldsm_x4_t(bv, vb + np * 16);
        mma_bf16(o[2 * np], ph, bv[0], bv[1]);
        mma_bf16(o[2 * np + 1], ph, bv[2], bv[3]);
        mma_bf16(o[2 * np], pl, bv[0], bv[1]);
        mma_bf16(o[2 * np + 1], pl, bv[2], bv[3]);
      }
    }
  }
  rsum[0] += __shfl_xor_sync(0xffffffffu, rsum[0], 1);
  rsum[0] += __shfl_xor_sync(0xffffffffu, rsum[0], 2);
  rsum[1] += __shfl_xor_sync(0xffffffffu, rsum[1], 1);
  rsum[1] += __shfl_xor_sync(0xffffffffu, rsum[1], 2);

  // ---- (eta_N, m_N) of the new rows, merged into (eta_A, m_A) by Eq. summary-update
  const float isd = rsqrtf((float)d);
  const float etaN[2] = {rmax[0] * isd + logf(rsum[0]), rmax[1] * isd + logf(rsum[1])};
  float ca[2], cn[2], eta[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const float mx = fmaxf(etaA[h], etaN[h]);
    eta[h] = mx + logf(__expf(etaA[h] - mx) + __expf(etaN[h] - mx));
    ca[h] = __expf(etaA[h] - eta[h]);
    cn[h] = __expf(etaN[h] - eta[h]) / rsum[h];            // m_N = o / rsum
  }
  // e^(eta_N - eta) m_N and e^(eta_A - eta) into shared memory (over the
  // staging buffers, once every warp is done with them) ...
  float* sM = reinterpret_cast<float*>(vsm_raw);           // [Q][kVuMLd]
  float* sCa = sM + Q * kVuMLd;                            // [Q]
  __syncthreads();
#pragma unroll
  for (int n = 0; n < NT; ++n) {
    *reinterpret_cast<float2*>(sM + r0 * kVuMLd + n * 8 + (lane & 3) * 2) = make_float2(cn[0] * o[n][0], cn[0] * o[n][1]);
    *reinterpret_cast<float2*>(sM + (r0 + 8) * kVuMLd + n * 8 + (lane & 3) * 2) =
        make_float2(cn[1] * o[n][2], cn[1] * o[n][3]);
  }
  if ((lane & 3) == 0) {
    sCa[r0] = ca[0];
    sCa[r0 + 8] = ca[1];
    p.eta[qbase + r0] = eta[0];                            // each eta_A was read above by its own lane
    p.eta[qbase + r0 + 8] = eta[1];
  }
  __syncthreads();
  // ... then one coalesced pass over the CTA's Q x d block of m with every load
  // in flight at once (16 float4 a thread)
  constexpr int kPer = Q * d / 4 / kThreads;
  float4* mrow = reinterpret_cast<float4*>(p.m + qbase * d);
  float4 xa[kPer];
#pragma unroll
  for (int u = 0; u < kPer; ++u) xa[u] = mrow[tid + u * kThreads];
#pragma unroll
  for (int u = 0; u < kPer; ++u) {
    const int i = tid + u * kThreads, q = i >> 5, c = (i & 31) * 4;
    const float a = sCa[q];
    const float4 nv = *reinterpret_cast<const float4*>(sM + q * kVuMLd + c);
    mrow[i] = make_float4(a * xa[u].x + nv.x, a * xa[u].y + nv.y, a * xa[u].z + nv.z, a * xa[u].w + nv.w);
  }

  // ---- the CTA with the last ticket of request b advances t
  if (tid == 0 && ticket == p.L * p.nkv - 1) {
    __threadfence();
    p.t[b] = t0 + delta;
    p.done[b] = 0;
  }
}

template <int MT>
static int launch_mma(const ViewParams& p, cudaStream_t s) {
  const size_t smem = vu_smem_bytes(MT);
  static size_t attr = 0;
  if (smem > attr) {
    if (cudaFuncSetAttribute(view_update_mma_kernel<MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
        cudaSuccess)
      return LSP_ERR_CUDA;
    attr = smem;
  }
  return launch_pdl(view_update_mma_kernel<MT>, dim3(p.C * p.L * p.nkv), dim3(MT * 32), smem, s, p) ==
                 cudaSuccess
             ? LSP_OK
             : LSP_ERR_CUDA;
}

template <typename T, int DPL>
static int launch_dpl(const ViewParams& p, cudaStream_t s) {
  const int Q = (p.nq / p.nkv) * p.R;
  const int qpw = (Q + kViewWarps - 1) / kViewWarps;
  const size_t smem = 2 * kViewChunk * DPL * 32 * sizeof(float);
  const dim3 grid(p.C * p.L * p.nkv);
  cudaError_t e;
  if (qpw <= 4)
    e = launch_pdl(view_update_kernel<T, DPL, 4>, grid, dim3(kViewThreads), smem, s, p);
  else if (qpw <= 8)
    e = launch_pdl(view_update_kernel<T, DPL, 8>, grid, dim3(kViewThreads), smem, s, p);
  else if (qpw <= 16)
    e = launch_pdl(view_update_kernel<T, DPL, 16>, grid, dim3(kViewThreads), smem, s, p);
  else
    return LSP_ERR_SHAPE;
  return e == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

int launch_view_update(const ViewParams& p, int dtype, cudaStream_t s) {
  // tensor-core path: bf16, d = 128, Q = rep * R a multiple of 16 up to 128
  const int Q = (p.nq / p.nkv) * p.R;
  if (dtype == LSP_DTYPE_BF16 && p.d == 128 && Q % 16 == 0) {
    switch (Q / 16) {
      case 1: return launch_mma<1>(p, s);
      case 2: return launch_mma<2>(p, s);
      case 3: return launch_mma<3>(p, s);
      case 4: return launch_mma<4>(p, s);
      case 5: return launch_mma<5>(p, s);
      case 6: return launch_mma<6>(p, s);
      case 7: return launch_mma<7>(p, s);
      case 8: return launch_mma<8>(p, s);
      default: break;
    }
  }
  if (p.d == 128) return dtype == LSP_DTYPE_BF16 ? launch_dpl<bf16, 4>(p, s) : launch_dpl<float, 4>(p, s);
  if (p.d == 64) return dtype == LSP_DTYPE_BF16 ? launch_dpl<bf16, 2>(p, s) : launch_dpl<float, 2>(p, s);
  return LSP_ERR_SHAPE;
}

}  // namespace lsp
