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
// heads sharing that KV head (rep * R queries): the new K/V rows are read from
// HBM once (16-byte vectors) and staged in shared memory as fp32; each warp
// owns whole queries, lanes split the head dimension, and the dot products and
// the row max/sum reduce with warp shuffles.  Only the new rows are touched.
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
                   ((size_t)(b * p.L + l) * p.rows + (delta - 1)) * p.H;
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
  if (p.d == 128) return dtype == LSP_DTYPE_BF16 ? launch_dpl<bf16, 4>(p, s) : launch_dpl<float, 4>(p, s);
  if (p.d == 64) return dtype == LSP_DTYPE_BF16 ? launch_dpl<bf16, 2>(p, s) : launch_dpl<float, 2>(p, s);
  return LSP_ERR_SHAPE;
}

}  // namespace lsp
