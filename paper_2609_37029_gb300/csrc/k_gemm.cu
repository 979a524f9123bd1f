// Weight-streaming projection GEMM on the 5th-generation tensor cores (sm_103a).
//
// Every dense projection of the drafter -- boundary fusion (Sec. 2.2), the
// q/k/v, output, gate/up and down projections of each draft layer and the
// frozen LM head (Sec. 2.3) -- has a small token count M = C*B (or C) and a
// large weight.  The kernel therefore puts 128 weight rows on the UMMA M axis
// and the tokens on its N axis ("swap AB"): D^T[n][m] = sum_k W[n][k] X[m][k].
//
//   warp 0      TMA producer: the CTA's 128 x BK weight tile and its
//               m_pad x BK activation tile per stage into an S-deep mbarrier
//               ring, plus an L2 prefetch of the next stage's weight tile
//   warp 1      TMEM allocation and the single-thread tcgen05.mma issue (a
//               lean loop: this one thread's instructions set the issue rate)
//   warps 2-5   epilogue: tcgen05.ld of the fp32 accumulators, the fused
//               output (fp32, storage dtype, SwiGLU, or a split-K partial)
//               staged in shared memory 16-32 tokens at a time and written
//               by TMA tensor stores (double-buffered), so the global writes
//               are full-line bulk copies that overlap the next chunk
//
// Grid: x = weight-tile CTAs x token groups (a group's CTAs share the weight
// tile, each over m_pad consecutive tokens; the SwiGLU gate/up projection
// takes two groups when its tiles fill under one wave of two CTAs per SM),
// y = split-K.
//
// Launched as a programmatic dependent: before the preceding kernel finishes,
// the producer already streams this launch's weights (L2 prefetch and the
// weight halves of the first stages); activation loads wait for it.  Split-K
// partials are summed in split order by the consuming kernel, so results are
// deterministic and no CTA waits on another.  Every mbarrier wait is bounded
// and records LSP_DEV_TIMEOUT instead of spinning forever.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstdlib>
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

constexpr uint32_t kTileBytes = kTileRows * 128;   // one weight tile per stage: 16 KB
// L2 prefetch distance of the weight stream, in k-blocks (one ahead: 318 -> 281 us at the
// LM-head shape; longer distances were slower)
constexpr int kPrefetchDist = 1;

// The epilogue's named barrier (id 1) counts exactly the four epilogue warps
// 2-5: any other warp taking that branch would leave bar.sync waiting forever.
constexpr int kEpilogueThreads = 128;
static_assert(kGemmThreads == 64 + kEpilogueThreads, "warp 0 TMA, warp 1 MMA, warps 2-5 epilogue");

// Instruction descriptor: fp32 accumulate, A/B format `fmt`, both K-major,
// N = n, M = 128.
__device__ __forceinline__ uint32_t make_idesc(int n, uint32_t fmt) {
  return (1u << 4) | (fmt << 7) | (fmt << 10) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(kTileRows >> 4) << 24);
}

template <typename T>
__device__ __forceinline__ void emit_chunk(const GemmParams& p, int tile, int split, int r, int m0,
                                           const float* v, float* xchg) {
  const int M = p.M;
  if (p.mode == EPI_SWIGLU) {
#pragma unroll
    for (int j = 0; j < 16; ++j) xchg[r * 17 + j] = v[j];
    named_bar(1, kEpilogueThreads);
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
    named_bar(1, kEpilogueThreads);
    return;
  }
  const int n = tile * kTileRows + r;
  if (n >= p.N) return;
  if (p.mode == EPI_T) {
    T* Y = static_cast<T*>(p.Y);
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (m0 + j < M) Y[(size_t)(m0 + j) * p.ldy + n] = from_f<T>(v[j]);
  } else {
    float* Y = static_cast<float*>(p.Y);
    if (p.mode == EPI_PARTIAL) Y += (size_t)split * M * p.ldy;
#pragma unroll
    for (int j = 0; j < 16; ++j)
      if (m0 + j < M) Y[(size_t)(m0 + j) * p.ldy + n] = v[j];
  }
}

constexpr uint32_t kXchgStride = 33;                          // SwiGLU exchange row (floats)
constexpr uint32_t kXchgBytes = 17408;                        // 128 x 33 floats, 1 KB aligned

// silu(gate) * up for NT tokens of gate feature f (exchange rows f and f + 64)
// into the staged [token][64] output tile.  Every input is loaded before the
// arithmetic, and the fast exponential and division keep the chain short
// (their relative error is far below the bf16 rounding of the result).  Measured
// at the Qwen3-8B gate/up shape: 1.5 -> 0.2 us per 32-token chunk.
template <typename T, int NT>
__device__ __forceinline__ void swiglu_rows(const float* xchg, T* o, int f, int t0) {
  float g[NT], u[NT];
#pragma unroll
  for (int j = 0; j < NT; ++j) {
    g[j] = xchg[f * kXchgStride + t0 + j];
    u[j] = xchg[(f + 64) * kXchgStride + t0 + j];
  }
#pragma unroll
  for (int j = 0; j < NT; ++j) o[(t0 + j) * 64 + f] = from_f<T>(__fdividef(g[j], 1.0f + __expf(-g[j])) * u[j]);
}

// Epilogue through shared memory and TMA stores (4 warps, r = accumulator
// row = output feature of the tile).  Chunk c of TT tokens: every thread
// loads its row's TT accumulators, writes them (or, for SwiGLU, the
// activation of its share after a gate/up exchange) into staging buffer
// c & 1, and one thread stores the buffer with a TMA tensor store into the
// [split][token][feature] view of Y at the CTA's first token row tok0.
// Token rows past M and feature columns past N fall outside the view and are
// not written; the chunks tile the CTA's m_pad tokens exactly, so no store
// reaches the next token group's rows.
template <typename T>
__device__ __forceinline__ void epilogue_tma(const GemmParams& p, const CUtensorMap* to, uint8_t* smem,
                                             uint32_t lane_base, int tile, int tok0, int split,
                                             int r) {
  const bool swiglu = p.mode == EPI_SWIGLU;
  const bool f32out = p.mode == EPI_F32 || p.mode == EPI_PARTIAL;
  const int es = f32out ? 4 : (int)sizeof(T);
  const int cols = swiglu ? 64 : kTileRows;                   // output features of one weight tile
  const int TT = p.out_tok;
  float* xchg = reinterpret_cast<float*>(smem);              // SwiGLU: [128][kXchgStride]
  uint8_t* stg0 = smem + (swiglu ? kXchgBytes : 0);
  const uint32_t buf_bytes = (uint32_t)(TT * cols * es);     // <= 16 KB
  const bool issuer = r == 0;
  const uint64_t pol_part = policy_evict_last();
  const int m_end = min(p.m_pad, p.M - tok0);                 // > 0: no token group is empty
  int chunk = 0;
  {
    for (int m0 = 0; m0 < m_end; m0 += TT, ++chunk) {       // no store box starts past row M
      float v[32];
      const uint32_t col = (uint32_t)m0;
      if (TT == 32) tmem_ld32(lane_base + col, v);
      else tmem_ld16(lane_base + col, v);
      uint8_t* stg = stg0 + (chunk & 1) * buf_bytes;
      if (issuer && chunk >= 2) bulk_wait_read<1>();         // the store two chunks back has read stg
      named_bar(1, kEpilogueThreads);
      if (swiglu) {
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (j < TT) xchg[r * kXchgStride + j] = v[j];
        named_bar(1, kEpilogueThreads);
        // thread (f = r & 63, half = r >> 6) forms tokens [half * TT/2, (half + 1) * TT/2)
        const int f = r & 63, t0 = (r >> 6) * (TT / 2);
        T* o = reinterpret_cast<T*>(stg);
        if (TT == 32) swiglu_rows<T, 16>(xchg, o, f, t0);
        else swiglu_rows<T, 8>(xchg, o, f, t0);
      } else if (f32out) {
        float* o = reinterpret_cast<float*>(stg);
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (j < TT) o[j * kTileRows + r] = v[j];
      } else {
        T* o = reinterpret_cast<T*>(stg);
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (j < TT) o[j * kTileRows + r] = from_f<T>(v[j]);
      }
      fence_proxy_async_smem();
      named_bar(1, kEpilogueThreads);
      if (issuer) {
        if (p.mode == EPI_PARTIAL)   // read once more, by the consumer: kept in L2 past the weight stream
          tma_store_3d_hint(to, smem_u32(stg), tile * cols, tok0 + m0, split, pol_part);
        else
          tma_store_3d(to, smem_u32(stg), tile * cols, tok0 + m0, split);
        bulk_commit();
      }
    }
  }
  if (issuer) bulk_wait_read<0>();                            // staging smem is released at exit
}

template <typename T, int kOcc>
__global__ void __launch_bounds__(kGemmThreads, kOcc)
    gemm_kernel(const __grid_constant__ CUtensorMap ta0, const __grid_constant__ CUtensorMap ta1,
                const __grid_constant__ CUtensorMap ta2, const __grid_constant__ CUtensorMap tb,
                const __grid_constant__ CUtensorMap to, const __grid_constant__ GemmParams p) {
  using G = GemmType<T>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int S = p.stages;
  const uint32_t stage_a = kTileBytes;
  const uint32_t stage_bytes = stage_a + (uint32_t)p.m_pad * 128;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)S * stage_bytes);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // blockIdx.x = weight tile x token groups + group: the CTAs of one weight
  // tile are adjacent, so they run together and share the tile through L2
  const int group = (int)blockIdx.x % p.tok_groups;
  const int tile = (int)blockIdx.x / p.tok_groups;
  const int tok0 = group * p.m_pad;                            // first token row of this CTA
  const int split = blockIdx.y;
  const int kb0 = (int)((long long)split * p.kblocks / p.splits);
  const int kb1 = (int)((long long)(split + 1) * p.kblocks / p.splits);
  const int nk = kb1 - kb0;
  const uint32_t expect = kTileBytes + (uint32_t)p.m_pad * 128;

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
    *s_abort = 0;
    fence_barrier_init();
    tma_prefetch_desc(&ta0);
    tma_prefetch_desc(&tb);
    if (p.tma_out) tma_prefetch_desc(&to);
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), (uint32_t)p.tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (!p.late_trigger) griddep_launch();
  const uint32_t tmem_base = *tmem_slot;

  int issued = 0;
  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------------ TMA producer
    // a weight tile read by one CTA goes first; shared by token groups, it stays
    const uint64_t pol_w = p.tok_groups > 1 ? policy_evict_normal() : policy_evict_first();
    const uint64_t pol_x = policy_evict_last();
    // the tile's tensor map (segment) and first row within it
    const int seg = (p.nseg > 2 && tile >= p.seg_tile0[2]) ? 2 : (p.nseg > 1 && tile >= p.seg_tile0[1]) ? 1 : 0;
    const CUtensorMap* amap = seg == 0 ? &ta0 : (seg == 1 ? &ta1 : &ta2);
    const int arow = p.mode == EPI_SWIGLU ? tile * 64 : (tile - p.seg_tile0[seg]) * kTileRows;
    auto load_a = [&](int i, uint32_t sa, uint32_t bar) {
      const int kx = (kb0 + i) * G::BK;
      if (p.mode == EPI_SWIGLU) {                  // 64 gate rows, then the 64 matching up rows
        tma_load_2d(sa, &ta0, bar, kx, arow, pol_w);
        tma_load_2d(sa + 64 * 128, &ta1, bar, kx, arow, pol_w);
      } else {
        tma_load_2d(sa, amap, bar, kx, arow, pol_w);
      }
    };
    auto prefetch_a = [&](int i) {
      if (group != 0) return;                // one CTA of the tile prefetches it
      const int kx = (kb0 + i) * G::BK;
      if (p.mode == EPI_SWIGLU) {
        tma_prefetch_l2(&ta0, kx, arow);
        tma_prefetch_l2(&ta1, kx, arow);
      } else {
        tma_prefetch_l2(amap, kx, arow);
      }
    };
    auto load_b = [&](int i, uint32_t sb, uint32_t bar) {
      const int kx = (kb0 + i) * G::BK;
      for (int tt = 0; tt < p.n_tok_tiles; ++tt)
        tma_load_2d(sb + (uint32_t)(tt * p.bn * 128), &tb, bar, kx, tok0 + tt * p.bn, pol_x);
    };
    // Weights do not depend on the preceding kernel: start streaming them now
    // (the first stages, and an L2 prefetch one k-block ahead of the ring).
    int next_pf = 0;
    const int pre = min(S, nk);
    while (next_pf < min(kPrefetchDist, nk)) prefetch_a(next_pf++);
    for (int i = 0; i < pre; ++i) {
      mbar_expect_tx(full_bar(i), expect);
      load_a(i, smem_u32(smem + (size_t)i * stage_bytes), full_bar(i));
    }
    griddep_wait();                       // activations come from the preceding kernel
    // A late trigger lets the next kernel start only once every kernel before
    // this one has completed (it may then read their outputs before its own
    // wait, as the attention does with the view state).
    if (p.late_trigger) griddep_launch();
    for (int i = 0; i < pre; ++i)
      load_b(i, smem_u32(smem + (size_t)i * stage_bytes) + stage_a, full_bar(i));
    issued = pre;
    // stage and phase of k-block i advance by counters (no division per block)
    int s = pre % S;
    uint32_t ph = (uint32_t)(pre / S) & 1u;
    const uint32_t ring0 = smem_u32(smem);
    for (int i = pre; i < nk; ++i) {
      while (next_pf < nk && next_pf < i + kPrefetchDist) prefetch_a(next_pf++);
      if (!mbar_wait(empty_bar(s), ph ^ 1u, p.err)) { *s_abort = 1; break; }
      mbar_expect_tx(full_bar(s), expect);
      const uint32_t sa = ring0 + (uint32_t)s * stage_bytes;
      load_a(i, sa, full_bar(s));
      load_b(i, sa + stage_a, full_bar(s));
      issued = i + 1;
      if (++s == S) { s = 0; ph ^= 1u; }
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------------------ MMA issue
    // One thread issues every MMA, so its own instructions set the issue rate
    // (measured: 0.60 -> 0.24 us per k-block with the loop below): the two
    // descriptors are formed once per stage and stepped by the byte offset
    // >> 4 in their address field (offsets stay inside the stage, so the
    // field never carries), and the stage and phase advance by counters.
    const uint32_t idesc = make_idesc(p.bn, G::FMT);
    const uint32_t ring0 = smem_u32(smem);
    const bool one_tile = p.n_tok_tiles == 1;
    int s = 0;
    uint32_t ph = 0;
    for (int i = 0; i < nk; ++i) {
      if (!mbar_wait(full_bar(s), ph, p.err)) { *s_abort = 1; break; }
      tc_fence_after();
      const uint32_t sa = ring0 + (uint32_t)s * stage_bytes;
      const uint64_t ad0 = sdesc_sw128(sa), bd0 = sdesc_sw128(sa + stage_a);
      if (one_tile) {
#pragma unroll
        for (int kk = 0; kk < G::BK / G::UK; ++kk) {
          const uint32_t acc = (i > 0 || kk > 0) ? 1u : 0u;
          if constexpr (sizeof(T) == 2)
            umma_f16(tmem_base, ad0 + (uint64_t)(2 * kk), bd0 + (uint64_t)(2 * kk), idesc, acc);
          else
            umma_tf32(tmem_base, ad0 + (uint64_t)(2 * kk), bd0 + (uint64_t)(2 * kk), idesc, acc);
        }
      } else {
#pragma unroll
        for (int kk = 0; kk < G::BK / G::UK; ++kk) {
          const uint64_t ad = ad0 + (uint64_t)((kk * 32) >> 4);
          for (int tt = 0; tt < p.n_tok_tiles; ++tt) {
            const uint64_t bd = bd0 + (uint64_t)((tt * p.bn * 128 + kk * 32) >> 4);
            const uint32_t acc = (i > 0 || kk > 0) ? 1u : 0u;
            if constexpr (sizeof(T) == 2)
              umma_f16(tmem_base + (uint32_t)(tt * p.bn), ad, bd, idesc, acc);
            else
              umma_tf32(tmem_base + (uint32_t)(tt * p.bn), ad, bd, idesc, acc);
          }
        }
      }
      umma_commit(empty_bar(s));
      if (++s == S) { s = 0; ph ^= 1u; }
    }
    umma_commit(acc_bar);
  } else if (warp >= 2) {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;
    const int r = q * 32 + lane;
    float* xchg = reinterpret_cast<float*>(smem);   // pipeline smem is idle once acc_bar fired
    griddep_wait();
    const bool ok = mbar_wait(acc_bar, 0, p.err);
    if (!ok) *s_abort = 1;
    tc_fence_after();
    named_bar(1, kEpilogueThreads);
    // one thread's snapshot of s_abort (which another role may set at any
    // time), so that all four warps take the same branch below
    volatile int* s_stop = s_abort + 1;
    if (r == 0) *s_stop = *s_abort;
    named_bar(1, kEpilogueThreads);
    const bool go = *s_stop == 0;
    const uint32_t lane_base = tmem_base + ((uint32_t)(q * 32) << 16);
    if (go && p.tma_out) {
      epilogue_tma<T>(p, &to, smem, lane_base, tile, tok0, split, r);
    } else if (go) {
      for (int tt = 0; tt < p.n_tok_tiles; ++tt)
        for (int c0 = 0; c0 < p.bn; c0 += 16) {
          float v[16];
          tmem_ld16(lane_base + (uint32_t)(tt * p.bn + c0), v);
          emit_chunk<T>(p, tile, split, r, tok0 + tt * p.bn + c0, v, xchg);
        }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 0 && lane == 0 && *s_abort) {
    // A wait gave up: let every TMA copy this CTA issued land before exit.
    for (int i = (issued > S ? issued - S : 0); i < issued; ++i)
      mbar_wait(full_bar(i % S), (uint32_t)(i / S) & 1u, p.err);
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, (uint32_t)p.tmem_cols);
  }
}

__global__ void sum_partials_kernel(const float* __restrict__ part, int splits, size_t n,
                                    float* __restrict__ y) {
  griddep_launch();
  griddep_wait();
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x) {
    float acc = part[i];
    for (int s = 1; s < splits; ++s) acc += part[(size_t)s * n + i];
    y[i] = acc;
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

int tmap_2d_bf16_sw128(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t rows, uint64_t row_bytes,
                       uint32_t box_inner, uint32_t box_rows) {
  auto enc = encoder();
  if (!enc) return LSP_ERR_UNSUPPORTED;
  if (((uintptr_t)ptr & 15) || (row_bytes % 16) || box_inner * 2 > 128 || box_rows < 1 || box_rows > 256)
    return LSP_ERR_SHAPE;
  cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)row_bytes};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? LSP_OK : LSP_ERR_CUDA;
}

// [splits][M][N] view of the output (row stride ldy) for TMA stores of
// box (cols features, tok tokens, 1 split); no swizzle.
static int make_out_map(CUtensorMap* m, bool f32, const void* Y, int N, int M, int splits, int ldy,
                        int cols, int tok) {
  auto enc = encoder();
  if (!enc) return LSP_ERR_UNSUPPORTED;
  const int es = f32 ? 4 : 2;
  if (((uintptr_t)Y & 15) || ((size_t)ldy * es) % 16) return LSP_ERR_SHAPE;
  cuuint64_t dims[3] = {(cuuint64_t)N, (cuuint64_t)M, (cuuint64_t)splits};
  cuuint64_t strides[2] = {(cuuint64_t)ldy * es, (cuuint64_t)M * ldy * es};
  cuuint32_t box[3] = {(cuuint32_t)cols, (cuuint32_t)tok, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(m, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3,
                   const_cast<void*>(Y), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? LSP_OK : LSP_ERR_CUDA;
}

int gemm_tiles(int mode, const int* seg_rows, int nseg) {
  if (mode == EPI_SWIGLU) return (seg_rows[0] + 63) / 64;
  int t = 0;
  for (int i = 0; i < nseg; ++i) t += (seg_rows[i] + kTileRows - 1) / kTileRows;
  return t;
}

int gemm_kblocks(int K, int dtype) {
  const int bk = dtype == LSP_DTYPE_BF16 ? 64 : 32;
  return (K + bk - 1) / bk;
}

static void token_tiling(int M, int* bn, int* ntt) {
  *ntt = (M + 255) / 256;
  int per = (M + *ntt - 1) / *ntt;
  *bn = std::max(16, (per + 15) / 16 * 16);
}

int gemm_group_rows(int M, int G) {
  int bn, ntt;
  token_tiling((M + G - 1) / G, &bn, &ntt);
  return bn * ntt;
}

static constexpr int kSmemBudget = 227 * 1024;

// Two 2-stage CTAs per SM keep the tensor pipe fed from two MMA issuers and
// overlap one CTA's prologue/epilogue with the other's weight stream; the pair
// must fit one SM's shared memory and TMEM.
static bool two_per_sm_fits(int m_pad) {
  const int stage_bytes = (int)kTileBytes + m_pad * 128;
  return 2 * stage_bytes + 2048 <= kSmemBudget / 2 && 2 * m_pad <= 512;
}

static bool use_two_per_sm(long long ctas, int num_sms, int m_pad) {
  return ctas * 4 >= (long long)num_sms * 5 && two_per_sm_fits(m_pad);
}

// Three 2-stage CTAs per SM (shared memory incl. the 1 KB each CTA reserves,
// TMEM columns, and the kernel instance bounded to 3 x 192 threads' registers)
// when token groups give enough CTAs for most SMs to hold a third.
constexpr int kSmemPerSm = 228 * 1024;
static bool three_per_sm_fits(int m_pad, int groups) {
  if (groups < 2) return false;
  int cols = 32;
  while (cols < m_pad) cols *= 2;
  const int stage_bytes = (int)kTileBytes + m_pad * 128;
  return 3 * (2 * stage_bytes + 1280 + 1024) <= kSmemPerSm && 3 * cols <= 512;
}

static bool use_three_per_sm(long long ctas, int num_sms, int m_pad, int groups) {
  return ctas >= 2LL * num_sms && three_per_sm_fits(m_pad, groups);
}

// Token groups: the CTAs of a weight tile split the M tokens G ways (each
// streams the tile; the copies after the first come from L2).  Smaller stages
// let three CTAs share an SM.  Two groups for the SwiGLU gate/up projection
// when its tiles fill at least one wave of one CTA per SM but less than one
// of two and the token count allows it (Qwen3-8B round, M = 256, 192 tiles:
// gate/up 368 -> 359 us per round, round 1.243 -> 1.231 ms).  Two groups for
// every projection above 256 tokens (the large shape, M = 512: round 2600 ->
// 2485 us), where one group would need a 512-column accumulator, one CTA per
// SM and two 80 KB stages.  One otherwise (at M = 256 every other projection
// and the LM head measured slower with two or three: more CTAs re-stream each
// weight tile for the same work).
static int token_groups(int M, int mode, int n_tiles, int num_sms) {
  const int g = (M > 256 || (mode == EPI_SWIGLU && M >= 128 && n_tiles <= 2 * num_sms && n_tiles >= num_sms)) ? 2 : 1;
  if (g == 1) return 1;
  int bn, ntt;
  token_tiling((M + g - 1) / g, &bn, &ntt);
  return (g - 1) * bn * ntt < M ? g : 1;     // every group holds at least one token row
}

// Split-K factor from a cost model in units of one k-block of one of two
// co-resident CTAs (~0.8 us measured at M = 256): waves x (k-blocks per CTA +
// fixed per-CTA cost) + the cost of combining the splits (per_split_cost per
// split: the consumer's re-read of fp32 partials from L2).  A lone CTA on an
// SM, with its deeper ring, moves a k-block in 0.53 of that time (0.42 vs
// 0.80 us measured at M = 256 with the MMA issue loop at 0.24 us per k-block).
constexpr double kLoneCtaCost = 0.53;

int gemm_auto_splits(int n_ctas, int kblocks, int num_sms, double per_split_cost, int max_splits,
                     int occ_max) {
  double best = 1e30;
  int splits = 1;
  for (int s = 1; s <= std::min(max_splits, kblocks); ++s) {
    const long long ctas = (long long)n_ctas * s;
    const int occ = (occ_max >= 3 && ctas >= 2LL * num_sms) ? 3
                    : (occ_max >= 2 && ctas * 4 >= (long long)num_sms * 5) ? 2 : 1;
    const long long slots = (long long)occ * num_sms;
    const long long waves = (ctas + slots - 1) / slots;
    const double per = (double)((kblocks + s - 1) / s) * (occ > 1 ? 1.0 : kLoneCtaCost) + 2.0;
    const double cost = (double)waves * per + (s > 1 ? per_split_cost * s : 0.0);
    if (cost < best - 1e-9) { best = cost; splits = s; }
  }
  return splits;
}

// Consumer cost of one M x N fp32 partial read back from L2 (~5 TB/s), in the
// model's k-block units (~1.56 us).
double gemm_partial_cost(int M, int N) { return (double)M * N * 4.0 / 5e12 / 1.56e-6; }

void gemm_choose(int dtype, int M, int K, int n_tiles, int mode, int num_sms, int* splits, int* groups) {
  const int G = token_groups(M, mode, n_tiles, num_sms);
  if (groups) *groups = G;
  int bn, ntt;
  token_tiling((M + G - 1) / G, &bn, &ntt);
  const int m_pad = bn * ntt;
  const int kblocks = gemm_kblocks(K, dtype);
  const int n_ctas = n_tiles * G;
  const int occ_max = three_per_sm_fits(m_pad, G) ? 3 : two_per_sm_fits(m_pad) ? 2 : 1;
  if (*splits <= 0)
    *splits = mode == EPI_PARTIAL
                  ? gemm_auto_splits(n_ctas, kblocks, num_sms, gemm_partial_cost(M, n_tiles * kTileRows), 16, occ_max)
                  : 1;
  *splits = std::max(1, std::min(*splits, kblocks));
}

int gemm_plan(GemmOp* op, int dtype, const void* X, int M, int K, const void* const* W,
              const int* seg_rows, int nseg, int mode, void* Y, int ldy, unsigned* err,
              int num_sms, int splits) {
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
  } else {
    int t0 = 0;
    for (int i = 0; i < 3; ++i) {
      p.seg_tile0[i] = i < nseg ? t0 : p.n_tiles;
      if (i < nseg) t0 += (seg_rows[i] + kTileRows - 1) / kTileRows;
    }
    for (int i = 0; i < nseg; ++i) p.N += seg_rows[i];
  }
  p.kblocks = gemm_kblocks(K, dtype);
  int G = 1;
  gemm_choose(dtype, M, K, p.n_tiles, mode, num_sms, &splits, &G);
  p.tok_groups = G;
  token_tiling((M + G - 1) / G, &p.bn, &p.n_tok_tiles);      // per token group
  p.m_pad = p.bn * p.n_tok_tiles;
  if (p.m_pad > 512) return LSP_ERR_SHAPE;
  int cols = 32;
  while (cols < p.m_pad) cols *= 2;
  p.tmem_cols = cols;
  const int stage_bytes = (int)kTileBytes + p.m_pad * 128;
  p.stages = std::min(8, (kSmemBudget - 2048) / stage_bytes);
  const int n_ctas = p.n_tiles * G;
  op->occ = 1;
  if (use_three_per_sm((long long)n_ctas * splits, num_sms, p.m_pad, G)) {
    p.stages = 2;
    op->occ = 3;
  } else if (use_two_per_sm((long long)n_ctas * splits, num_sms, p.m_pad)) {
    p.stages = 2;
  }
  if (p.stages < 2) return LSP_ERR_SHAPE;
  p.splits = splits;
  if (splits > 1 && mode != EPI_PARTIAL) return LSP_ERR_SHAPE;
  p.Y = Y;
  p.ldy = ldy;
  p.err = err;
  op->dtype = dtype;
  const int box_rows = mode == EPI_SWIGLU ? 64 : kTileRows;
  int rc;
  for (int i = 0; i < 3; ++i) {
    const int si = i < nseg ? i : 0;
    if ((rc = make_map(&op->a[i], dtype, W[si], K, seg_rows[si], box_rows)) != LSP_OK) return rc;
  }
  if ((rc = make_map(&op->b, dtype, X, K, M, p.bn)) != LSP_OK) return rc;
  // TMA-store epilogue when the output view can be described (else per-thread stores)
  p.out_tok = (p.m_pad % 32) ? 16 : 32;
  {
    const bool f32 = mode == EPI_F32 || mode == EPI_PARTIAL || dtype == LSP_DTYPE_F32;
    const int cols = mode == EPI_SWIGLU ? 64 : kTileRows;
    p.tma_out = make_out_map(&op->out, f32, Y, p.N, M, splits, ldy, cols, p.out_tok) == LSP_OK;
    if (!p.tma_out) op->out = op->b;       // unused placeholder
  }
  op->grid = dim3((unsigned)n_ctas, (unsigned)splits, 1);
  op->smem = (size_t)p.stages * stage_bytes + 1024 + 256;
  return LSP_OK;
}

template <typename T, int kOcc>
static int launch_t(const GemmOp* op, cudaStream_t s) {
  static std::once_flag once;
  std::call_once(once, [] {
    cudaFuncSetAttribute(gemm_kernel<T, kOcc>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget);
    if (kOcc > 1)   // room for kOcc CTAs' shared memory on one SM
      cudaFuncSetAttribute(gemm_kernel<T, kOcc>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
  });
  const cudaError_t e = launch_pdl(gemm_kernel<T, kOcc>, op->grid, dim3(kGemmThreads), op->smem, s,
                                   op->a[0], op->a[1], op->a[2], op->b, op->out, op->p);
  return e == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

int gemm_launch(const GemmOp* op, cudaStream_t s) {
  if (op->occ == 3) return op->dtype == LSP_DTYPE_BF16 ? launch_t<bf16, 3>(op, s) : launch_t<float, 3>(op, s);
  return op->dtype == LSP_DTYPE_BF16 ? launch_t<bf16, 1>(op, s) : launch_t<float, 1>(op, s);
}

int launch_sum_partials(const float* part, int splits, size_t n, float* y, cudaStream_t s) {
  const unsigned blocks = (unsigned)std::min<size_t>((n + 255) / 256, 4096);
  return launch_pdl(sum_partials_kernel, dim3(blocks), dim3(256), 0, s, part, splits, n, y) ==
                 cudaSuccess
             ? LSP_OK
             : LSP_ERR_CUDA;
}

}  // namespace lsp
