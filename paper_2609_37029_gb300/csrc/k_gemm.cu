// Weight-streaming projection GEMM on the 5th-generation tensor cores (sm_103a).
//
// Every dense projection of the drafter -- boundary fusion (Sec. 2.2), the
// q/k/v, output, gate/up and down projections of each draft layer and the
// frozen LM head (Sec. 2.3) -- has a small token count M = C*B (or C) and a
// large weight.  The kernel therefore puts 128 weight rows on the UMMA M axis
// and the tokens on its N axis ("swap AB"): D^T[n][m] = sum_k W[n][k] X[m][k].
//
//   warp 0      TMA producer: one 128 x BK weight tile (16 KB) and the M x BK
//               activation tile per stage into an S-deep mbarrier ring
//   warp 1      TMEM allocation and the single-thread tcgen05.mma issue
//   warps 2-5   epilogue: tcgen05.ld of the fp32 accumulator, fused
//               store / residual add / SwiGLU, or a split-K partial
//
// Split-K partials go to a workspace; the last CTA of a tile (atomic ticket)
// sums them in split order, so results are deterministic.  Every mbarrier wait
// is bounded and records LSP_DEV_TIMEOUT instead of spinning forever.
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "lsp_internal.h"

namespace lsp {

template <typename T> struct GemmType;
template <> struct GemmType<bf16> {
  static constexpr int BK = 64;   // one 128-byte swizzle row of bf16
  static constexpr int UK = 16;   // K of one kind::f16 MMA
  static constexpr uint32_t FMT = 1;
};
template <> struct GemmType<float> {
  static constexpr int BK = 32;   // one 128-byte swizzle row of fp32 (read as tf32)
  static constexpr int UK = 8;    // K of one kind::tf32 MMA
  static constexpr uint32_t FMT = 2;
};

// Instruction descriptor: fp32 accumulate, A/B format `fmt`, both K-major,
// N = n, M = 128.
__device__ __forceinline__ uint32_t make_idesc(int n, uint32_t fmt) {
  return (1u << 4) | (fmt << 7) | (fmt << 10) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(kTileRows >> 4) << 24);
}

template <typename T>
__device__ __forceinline__ void emit_chunk(const GemmParams& p, int tile, int r, int m0,
                                           const float* v, float* xchg) {
  const int M = p.M;
  if (p.mode == EPI_SWIGLU) {
#pragma unroll
    for (int j = 0; j < 16; ++j) xchg[r * 17 + j] = v[j];
    named_bar(1, 128);
    if (r < 64) {
      const int f = tile * 64 + r;
      T* Y = static_cast<T*>(p.Y);
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int m = m0 + j;
        if (m < M && f < p.N) {
          const float g = xchg[r * 17 + j];
          const float u = xchg[(r + 64) * 17 + j];
          Y[(size_t)m * p.ldy + f] = from_f<T>(g / (1.0f + expf(-g)) * u);
        }
      }
    }
    named_bar(1, 128);
    return;
  }
  const int n = tile * kTileRows + r;
  if (n >= p.N) return;
  if (p.mode == EPI_T) {
    T* Y = static_cast<T*>(p.Y);
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (m0 + j < M) Y[(size_t)(m0 + j) * p.ldy + n] = from_f<T>(v[j]);
  } else if (p.mode == EPI_RESID) {
    float* Y = static_cast<float*>(p.Y);
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (m0 + j < M) Y[(size_t)(m0 + j) * p.ldy + n] += v[j];
  } else {
    float* Y = static_cast<float*>(p.Y);
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (m0 + j < M) Y[(size_t)(m0 + j) * p.ldy + n] = v[j];
  }
}

template <typename T>
__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap ta0, const __grid_constant__ CUtensorMap ta1,
                const __grid_constant__ CUtensorMap ta2, const __grid_constant__ CUtensorMap tb,
                const GemmParams p) {
  using G = GemmType<T>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int S = p.stages;
  const uint32_t stage_a = kTileRows * 128;
  const uint32_t stage_bytes = stage_a + (uint32_t)p.m_pad * 128;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)S * stage_bytes);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S + 1);
  volatile int* s_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);  // [0] last CTA, [1] abort

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int tile = blockIdx.x;
  const int split = blockIdx.y;
  const int kb0 = (int)((long long)split * p.kblocks / p.splits);
  const int kb1 = (int)((long long)(split + 1) * p.kblocks / p.splits);
  const int nk = kb1 - kb0;

  const uint32_t bar0 = smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (S + s); };
  const uint32_t acc_bar = bar0 + 8u * (2 * S);

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(acc_bar, 1);
    s_flag[0] = 0;
    s_flag[1] = 0;
    fence_barrier_init();
    tma_prefetch_desc(&ta0);
    tma_prefetch_desc(&tb);
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), (uint32_t)p.tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  int issued = 0;
  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------------ TMA producer
    const uint64_t pol_w = policy_evict_first();
    const uint64_t pol_x = policy_evict_last();
    int seg = 0;
    if (p.mode != EPI_SWIGLU) {
      if (p.nseg > 2 && tile >= p.seg_tile0[2]) seg = 2;
      else if (p.nseg > 1 && tile >= p.seg_tile0[1]) seg = 1;
    }
    const CUtensorMap* ta = seg == 0 ? &ta0 : (seg == 1 ? &ta1 : &ta2);
    const int arow = (tile - p.seg_tile0[seg]) * kTileRows;
    for (int i = 0; i < nk; ++i) {
      const int s = i % S;
      const uint32_t ph = (uint32_t)(i / S) & 1u;
      if (!mbar_wait(empty_bar(s), ph ^ 1u, p.err)) { s_flag[1] = 1; break; }
      mbar_expect_tx(full_bar(s), stage_bytes);
      const uint32_t sa = smem_u32(smem + (size_t)s * stage_bytes);
      const uint32_t sb = sa + stage_a;
      const int kx = (kb0 + i) * G::BK;
      if (p.mode == EPI_SWIGLU) {
        tma_load_2d(sa, &ta0, full_bar(s), kx, tile * 64, pol_w);
        tma_load_2d(sa + 64 * 128, &ta1, full_bar(s), kx, tile * 64, pol_w);
      } else {
        tma_load_2d(sa, ta, full_bar(s), kx, arow, pol_w);
      }
      for (int tt = 0; tt < p.n_tok_tiles; ++tt)
        tma_load_2d(sb + (uint32_t)(tt * p.bn * 128), &tb, full_bar(s), kx, tt * p.bn, pol_x);
      issued = i + 1;
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------------------ MMA issue
    const uint32_t idesc = make_idesc(p.bn, G::FMT);
    for (int i = 0; i < nk; ++i) {
      const int s = i % S;
      const uint32_t ph = (uint32_t)(i / S) & 1u;
      if (!mbar_wait(full_bar(s), ph, p.err)) { s_flag[1] = 1; break; }
      tc_fence_after();
      const uint32_t sa = smem_u32(smem + (size_t)s * stage_bytes);
      const uint32_t sb = sa + stage_a;
#pragma unroll
      for (int kk = 0; kk < G::BK / G::UK; ++kk) {
        const uint64_t ad = sdesc_sw128(sa + kk * 32);
        for (int tt = 0; tt < p.n_tok_tiles; ++tt) {
          const uint64_t bd = sdesc_sw128(sb + (uint32_t)(tt * p.bn * 128) + kk * 32);
          const uint32_t acc = (i > 0 || kk > 0) ? 1u : 0u;
          if constexpr (sizeof(T) == 2)
            umma_f16(tmem_base + (uint32_t)(tt * p.bn), ad, bd, idesc, acc);
          else
            umma_tf32(tmem_base + (uint32_t)(tt * p.bn), ad, bd, idesc, acc);
        }
      }
      umma_commit(empty_bar(s));
    }
    umma_commit(acc_bar);
  } else if (warp >= 2) {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const int etid = threadIdx.x - 64;
    float* xchg = reinterpret_cast<float*>(smem);   // pipeline smem is idle once acc_bar fired
    const bool ok = mbar_wait(acc_bar, 0, p.err);
    if (!ok) s_flag[1] = 1;
    tc_fence_after();
    named_bar(1, 128);
    const bool abort = s_flag[1] != 0;
    const uint32_t tb_addr = tmem_base + ((uint32_t)(q * 32) << 16);
    if (!abort) {
      if (p.splits == 1) {
        for (int tt = 0; tt < p.n_tok_tiles; ++tt)
          for (int c0 = 0; c0 < p.bn; c0 += 16) {
            float v[16];
            tmem_ld16(tb_addr + (uint32_t)(tt * p.bn + c0), v);
            emit_chunk<T>(p, tile, r, tt * p.bn + c0, v, xchg);
          }
      } else {
        float* part = p.ws + (size_t)(tile * p.splits + split) * p.m_pad * kTileRows;
        for (int tt = 0; tt < p.n_tok_tiles; ++tt)
          for (int c0 = 0; c0 < p.bn; c0 += 16) {
            float v[16];
            tmem_ld16(tb_addr + (uint32_t)(tt * p.bn + c0), v);
            const int m0 = tt * p.bn + c0;
#pragma unroll
            for (int j = 0; j < 16; ++j) part[(size_t)(m0 + j) * kTileRows + r] = v[j];
          }
        __threadfence();
        named_bar(1, 128);
        if (etid == 0) {
          const int old = atomicAdd(&p.counters[tile], 1);
          s_flag[0] = (old == p.splits - 1) ? 1 : 0;
        }
        named_bar(1, 128);
        if (s_flag[0]) {
          __threadfence();
          const float* base = p.ws + (size_t)tile * p.splits * p.m_pad * kTileRows;
          for (int m0 = 0; m0 < p.M; m0 += 16) {
            float v[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) v[j] = 0.0f;
            for (int s2 = 0; s2 < p.splits; ++s2) {
              const float* ps = base + (size_t)s2 * p.m_pad * kTileRows;
#pragma unroll
              for (int j = 0; j < 16; ++j) v[j] += __ldcg(ps + (size_t)(m0 + j) * kTileRows + r);
            }
            emit_chunk<T>(p, tile, r, m0, v, xchg);
          }
          if (etid == 0) p.counters[tile] = 0;
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 0 && lane == 0 && s_flag[1]) {
    // A wait gave up: let every TMA copy this CTA issued land before exit.
    for (int i = (issued > S ? issued - S : 0); i < issued; ++i)
      mbar_wait(full_bar(i % S), (uint32_t)(i / S) & 1u, p.err);
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, (uint32_t)p.tmem_cols);
  }
}

// ====================================================================== host

static PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
static std::once_flag g_encode_once;

static PFN_cuTensorMapEncodeTiled_v12000 encoder() {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  return g_encode;
}

// 2-D K-major map: rows x K elements, box (BK, box_rows), 128-byte swizzle.
static int make_map(CUtensorMap* m, int dtype, const void* ptr, int K, int rows, int box_rows) {
  auto enc = encoder();
  if (!enc) return LSP_ERR_UNSUPPORTED;
  const int es = dtype == LSP_DTYPE_BF16 ? 2 : 4;
  const int bk = 128 / es;
  cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)K * es};
  cuuint32_t box[2] = {(cuuint32_t)bk, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(m, dtype == LSP_DTYPE_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16
                                              : CU_TENSOR_MAP_DATA_TYPE_TFLOAT32,
                   2, const_cast<void*>(ptr), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? LSP_OK : LSP_ERR_CUDA;
}

int gemm_tiles(int mode, const int* seg_rows, int nseg) {
  if (mode == EPI_SWIGLU) return (seg_rows[0] + 63) / 64;
  int t = 0;
  for (int i = 0; i < nseg; ++i) t += (seg_rows[i] + kTileRows - 1) / kTileRows;
  return t;
}

static void token_tiling(int M, int* bn, int* ntt) {
  *ntt = (M + 255) / 256;
  int per = (M + *ntt - 1) / *ntt;
  *bn = std::max(16, (per + 15) / 16 * 16);
}

size_t gemm_ws_bytes(int M, int n_tiles, int splits) {
  int bn, ntt;
  token_tiling(M, &bn, &ntt);
  return splits <= 1 ? 0 : (size_t)n_tiles * splits * (size_t)bn * ntt * kTileRows * sizeof(float);
}

static constexpr int kSmemBudget = 227 * 1024;

// split-K factor: minimise waves x (k-blocks per CTA + fixed per-CTA overhead)
int gemm_auto_splits(int n_tiles, int kblocks, int num_sms) {
  double best = 1e30;
  int splits = 1;
  for (int s = 1; s <= std::min(16, kblocks); ++s) {
    const long long ctas = (long long)n_tiles * s;
    const long long waves = (ctas + num_sms - 1) / num_sms;
    const double per = (double)((kblocks + s - 1) / s) + 3.0 + (s > 1 ? 1.5 : 0.0);
    const double cost = (double)waves * per;
    if (cost < best - 1e-9) { best = cost; splits = s; }
  }
  return splits;
}

int gemm_plan(GemmOp* op, int dtype, const void* X, int M, int K, const void* const* W,
              const int* seg_rows, int nseg, int mode, void* Y, int ldy, float* ws,
              size_t ws_bytes, int* counters, int n_counters, unsigned* err, int num_sms,
              int splits) {
  if (M < 1 || M > 512 || K < 1 || nseg < 1 || nseg > 3) return LSP_ERR_SHAPE;
  if (mode == EPI_SWIGLU && nseg != 2) return LSP_ERR_SHAPE;
  const int es = dtype == LSP_DTYPE_BF16 ? 2 : 4;
  if ((K * es) % 16) return LSP_ERR_SHAPE;
  for (int i = 0; i + 1 < nseg && mode != EPI_SWIGLU; ++i)
    if (seg_rows[i] % kTileRows) return LSP_ERR_SHAPE;
  GemmParams& p = op->p;
  p = GemmParams{};
  p.M = M;
  p.K = K;
  p.mode = mode;
  p.nseg = nseg;
  p.n_tiles = gemm_tiles(mode, seg_rows, nseg);
  p.N = 0;
  if (mode == EPI_SWIGLU) {
    p.N = seg_rows[0];
    p.seg_tile0[0] = p.seg_tile0[1] = p.seg_tile0[2] = 0;
  } else {
    int t0 = 0;
    for (int i = 0; i < 3; ++i) {
      p.seg_tile0[i] = i < nseg ? t0 : p.n_tiles;
      if (i < nseg) t0 += (seg_rows[i] + kTileRows - 1) / kTileRows;
    }
    for (int i = 0; i < nseg; ++i) p.N += seg_rows[i];
  }
  const int bk = 128 / es;
  p.kblocks = (K + bk - 1) / bk;
  token_tiling(M, &p.bn, &p.n_tok_tiles);
  p.m_pad = p.bn * p.n_tok_tiles;
  int cols = 32;
  while (cols < p.m_pad) cols *= 2;
  p.tmem_cols = cols;
  const int stage_bytes = kTileRows * 128 + p.m_pad * 128;
  p.stages = std::min(8, (kSmemBudget - 2048) / stage_bytes);
  if (p.stages < 2) return LSP_ERR_SHAPE;
  if (splits <= 0) splits = gemm_auto_splits(p.n_tiles, p.kblocks, num_sms);
  splits = std::max(1, std::min(splits, p.kblocks));
  if (splits > 1) {
    if (!ws || !counters || n_counters < p.n_tiles || gemm_ws_bytes(M, p.n_tiles, splits) > ws_bytes)
      return LSP_ERR_SHAPE;
  }
  p.splits = splits;
  p.Y = Y;
  p.ldy = ldy;
  p.ws = ws;
  p.counters = counters;
  p.err = err;
  op->dtype = dtype;
  const int box_rows = mode == EPI_SWIGLU ? 64 : kTileRows;
  int rc;
  for (int i = 0; i < 3; ++i) {
    const int si = i < nseg ? i : 0;
    if ((rc = make_map(&op->a[i], dtype, W[si], K, seg_rows[si], box_rows)) != LSP_OK) return rc;
  }
  if ((rc = make_map(&op->b, dtype, X, K, M, p.bn)) != LSP_OK) return rc;
  op->grid = dim3((unsigned)p.n_tiles, (unsigned)splits, 1);
  op->smem = (size_t)p.stages * stage_bytes + 1024 + 256;
  return LSP_OK;
}

template <typename T>
static int launch_t(const GemmOp* op, cudaStream_t s) {
  static std::once_flag once;
  std::call_once(once, [] {
    cudaFuncSetAttribute(gemm_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget);
  });
  gemm_kernel<T><<<op->grid, kGemmThreads, op->smem, s>>>(op->a[0], op->a[1], op->a[2], op->b,
                                                           op->p);
  return cudaGetLastError() == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

int gemm_launch(const GemmOp* op, cudaStream_t s) {
  return op->dtype == LSP_DTYPE_BF16 ? launch_t<bf16>(op, s) : launch_t<float>(op, s);
}

}  // namespace lsp
