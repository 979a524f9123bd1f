// Fixed-context block attention of a draft layer on the tcgen05 tensor cores
// (Sec. 2.3, Eq. draft-context), with the q/k/v finalisation folded in:
// bf16 storage, head dim 128.
//
// One CTA (16 warps) per (request b, KV head g).  The rep = nq/nkv query
// heads of the group share the group's keys and values, so their 16-row
// query blocks are stacked on the UMMA M axis (128 rows) and every key is
// one column of a single score matrix:
//     key rows [0, 16)                    block keys of KV head g (rows >= B masked)
//     key rows [16, 16 + W)               window slots (slots >= count = min(t, W) masked)
//     key rows [16 + W, 16 + W + 16 rep)  summary keys G_h, 16 per query head
//                                         (a row sees only its own head's R entries)
// Before the grid-dependency wait: TMA loads of the window keys and values
// and of G (128-byte swizzled boxes), the summary values M_h converted to
// bf16.  After it: the q/k/v projection's split partials of the block rows
// are summed in split order, q and k RMS-normalised and rotated (the
// rotate-half form of the rotary embedding), and stored in the operand
// layouts.  S = Q K^T (fp32) lands in TMEM columns [0, nk).  Each TMEM lane
// quadrant is read by four warps (column quarters) holding their scores in
// registers; with at most four heads a head's 16 rows appear twice in its
// quadrant and the two copies take alternate 16-key chunks, so no softmax
// lane works on a padding row.  The row max and sum are exchanged through
// shared memory; P = 2^((s - max) log2(e) / sqrt(d)), rounded to bf16, is
// written to shared memory as the K-major A operand of O = P V, with V =
// [V^b ; V^w ; M_h] an MN-major B operand (rows of 128 dims contiguous).  O
// (TMEM columns [384, 512), the copies' partial sums added) / row sum is the
// head's output: one softmax over block, window and summary.
//
// Shared memory (128-byte swizzled, 8-row groups 1024 B apart; a row of 128
// dims is two 64-element k-blocks): Q [2][128 rows], K [2][nk rows], V
// [2][nk rows]; P [ceil(nk/64)][128 rows] reuses the Q and K space once the
// score MMAs have completed.
#include "common.cuh"
#include "lsp_internal.h"

namespace lsp {
namespace {

constexpr int kTcM = 128;         // UMMA M: stacked query rows
constexpr int kTcD = 128;         // head dim
constexpr int kTcOcol = 384;      // TMEM column of the O accumulator
constexpr int kTcCols = 512;      // TMEM columns allocated
constexpr int kTcThreads = 512;   // four warps per TMEM lane quadrant (column quarters)
constexpr int kTcMaxKeys = 352;   // S columns stay below kTcOcol; shared memory bound
constexpr int kTcMaxCh = 6;       // 16-column chunks per warp: ceil(352 / 16 / 4)
constexpr int kTcMaxItems = 5;    // summary value chunks per thread of the 480 non-TMA threads (rep <= 8)

struct TcLayout {
  int nk, qstride, dup;
  uint32_t off_k, off_v, off_x, off_bar, bytes;
};

__host__ __device__ inline TcLayout tc_layout(int W, int rep) {
  TcLayout L;
  L.nk = 16 + W + 16 * rep;
  // Head h's block rows start at row h * qstride, so the real rows spread over
  // the four TMEM lane quadrants (a multiple of 8 keeps TMA boxes 1024-B
  // aligned).  With at most four heads every head's 16 rows appear twice in
  // its quadrant (lanes 0-15 and 16-31): the two copies take alternate key
  // chunks, so no lane of the softmax works on a padding row.
  L.dup = rep <= 4 ? 2 : 1;
  L.qstride = L.dup == 2 ? 32 : min(32, (kTcM / rep) & ~7);
  L.off_k = kTcM * 256;                          // Q: 2 k-blocks x 128 rows x 128 B
  L.off_v = L.off_k + (uint32_t)L.nk * 256;      // K: 2 k-blocks x nk rows x 128 B
  L.off_x = L.off_v + (uint32_t)L.nk * 256;      // V: same
  L.off_bar = L.off_x + 4 * 2 * kTcM * 4;        // [quarter][max, sum][row] fp32
  L.bytes = L.off_bar + 64 + 1024;               // barriers, TMEM slot, 1024-B alignment slack
  return L;
}

// Byte offset of 16-byte chunk c8 (dims 8 c8 .. 8 c8 + 7) of row n in a
// [2 k-blocks][rows][128 B] region with 128-byte swizzling (the layout a TMA
// box with SWIZZLE_128B writes at a 1024-byte aligned address).
__device__ __forceinline__ uint32_t sw_off(int n, int c8, int rows) {
  return (uint32_t)((c8 >> 3) * rows * 128 + (n >> 3) * 1024 + (n & 7) * 128 +
                    (((c8 & 7) ^ (n & 7)) << 4));
}

__device__ __forceinline__ void st_shared_v4(uint32_t a, uint32_t x, uint32_t y, uint32_t z, uint32_t w) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(a), "r"(x), "r"(y), "r"(z), "r"(w)
               : "memory");
}

// Shared-memory descriptor of an MN-major operand with 128-byte swizzling:
// 64 contiguous N elements per 128-B row, 8 K rows per 1024-B group (SBO),
// `lbo` bytes between consecutive 64-element N blocks.
__device__ __forceinline__ uint64_t sdesc_sw128_mn(uint32_t saddr, uint32_t lbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)(1024u >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// kind::f16 instruction descriptor: bf16 A and B, fp32 D, M = 128, N = n;
// A K-major, B K-major or (b_mn) MN-major.
__device__ __forceinline__ uint32_t tc_idesc(int n, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (b_mn ? (1u << 16) : 0u) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(kTcM >> 4) << 24);
}

__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Non-suspending wait (test_wait in a loop): these phases complete within
// microseconds and every thread of the CTA polls them; bounded like mbar_wait.
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n"
      " mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_spin(uint32_t bar, uint32_t parity, unsigned* err) {
  if (mbar_test(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_test(bar, parity)) return true;
    if ((it & 255u) == 0 && global_ns() - t0 > kWaitLimitNs) {
      set_err(err, LSP_DEV_TIMEOUT);
      return false;
    }
  }
}

// 4 consecutive fp32 values of a bf16 vector (norm weights), one 8-byte load
__device__ __forceinline__ void ld_bf16x4(const void* p, float* v) {
  const uint2 u = *reinterpret_cast<const uint2*>(p);
  const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&u.x);
  const __nv_bfloat162 c = *reinterpret_cast<const __nv_bfloat162*>(&u.y);
  v[0] = __low2float(a); v[1] = __high2float(a); v[2] = __low2float(c); v[3] = __high2float(c);
}

template <int DUP>
__global__ void __launch_bounds__(kTcThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap mwk, const __grid_constant__ CUtensorMap mwv,
                   const __grid_constant__ CUtensorMap mg, const AttnParams p, const int wbox) {
  extern __shared__ uint8_t tsm_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(tsm_raw) + 1023) &
                                           ~static_cast<uintptr_t>(1023));
  const int rep = p.nq / p.nkv;
  const TcLayout L = tc_layout(p.W, rep);
  const int nk = L.nk, qs = L.qstride, B = p.B, W = p.W, R = p.R, l = p.layer;
  const uint32_t s_q = smem_u32(sm), s_k = s_q + L.off_k, s_v = s_q + L.off_v, s_p = s_q;
  float* sx = reinterpret_cast<float*>(sm + L.off_x);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L.off_bar);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 4);
  volatile int* s_abort = reinterpret_cast<volatile int*>(tslot + 1);
  const uint32_t bar_kv = smem_u32(bars), bar_s = smem_u32(bars + 2), bar_o = smem_u32(bars + 3);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int b = blockIdx.x / p.nkv, g = blockIdx.x % p.nkv;

  if (tid == 0) {
    for (int k = 0; k < 4; ++k) mbar_init(smem_u32(bars + k), 1);
    *s_abort = 0;
    fence_barrier_init();
    tma_prefetch_desc(&mwk);
    tma_prefetch_desc(&mwv);
  }
  if (warp == 0) tmem_alloc(smem_u32(tslot), kTcCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  griddep_launch();

  // The window, summary and t come from the view update at the start of the
  // round: the q/k/v projection before this kernel triggers its dependents
  // only after its own dependency wait, so every kernel before that
  // projection has completed and they are read before this kernel's wait.
  // Only the projection's partials wait for it.
  const long long t = p.t[b];
  const int count = (int)(t < W ? t : W);
  const int nwb = (count + wbox - 1) / wbox;           // window boxes (W % wbox == 0)
  if (warp == 1) {
    // ---- TMA: window keys / values as key rows 16 .., summary keys G_h as
    //      key rows 16 + W + 16 h (R rows each)
    const uint32_t bytes = 2u * 2u * (uint32_t)(nwb * wbox) * 128u + (R > 0 ? 2u * (uint32_t)(rep * R) * 128u : 0u);
    if (lane == 0) mbar_expect_tx(bar_kv, bytes);
    __syncwarp();
    const uint64_t pol_f = policy_evict_first(), pol_n = policy_evict_normal();
    const int wrow0 = ((b * p.L + l) * p.nkv + g) * W;
    const int items = 4 * nwb + (R > 0 ? 2 * rep : 0);
    for (int it = lane; it < items; it += 32) {
      if (it < 4 * nwb) {
        const int kv = it & 1, kb = (it >> 1) & 1, j = it >> 2;
        const uint32_t dst = (kv ? s_v : s_k) + (uint32_t)kb * (uint32_t)(nk * 128) + (uint32_t)(16 + j * wbox) * 128u;
        tma_load_2d(dst, kv ? &mwv : &mwk, bar_kv, kb * 64, wrow0 + j * wbox, pol_f);
      } else {
        const int k2 = it - 4 * nwb, kb = k2 & 1, h = k2 >> 1;
        const uint32_t dst = s_k + (uint32_t)kb * (uint32_t)(nk * 128) + (uint32_t)(16 + W + 16 * h) * 128u;
        tma_load_2d(dst, &mg, bar_kv, kb * 64, (l * p.nq + g * rep + h) * R, pol_n);
      }
    }
  } else {
    // warps 0 and 2-15: 480 threads, indices 0..479
    const int t0 = warp == 0 ? lane : tid - 32, nt = kTcThreads - 32;
    // ---- summary values M_h (fp32 -> bf16) as value rows 16 + W + 16 h + r
    //      (rows r >= R zero): every load of this thread issued before its stores
    const float* Mp = p.m + (((size_t)(b * p.L + l) * p.nq + (size_t)g * rep) * R) * kTcD;
    float4 mv[kTcMaxItems][2];
#pragma unroll
    for (int u = 0; u < kTcMaxItems; ++u) {
      const int idx = t0 + u * nt;
      const int hr = idx >> 4, c8 = idx & 15, hh = hr >> 4, r = hr & 15;
      if (idx < rep * 256 && r < R) {
        const float4* src = reinterpret_cast<const float4*>(Mp + ((size_t)hh * R + r) * kTcD + c8 * 8);
        mv[u][0] = src[0];
        mv[u][1] = src[1];
      }
    }
    // ---- zero values of the key rows no TMA box covers (P is 0 there, and
    //      0 x V must stay 0): block rows >= B, window rows past the last box
    const int wz = W - nwb * wbox;
    for (int idx = t0; idx < (wz + 16 - B) * 16; idx += nt) {
      const int k = idx >> 4, c8 = idx & 15;
      const int n = k < wz ? 16 + nwb * wbox + k : B + (k - wz);
      st_shared_v4(s_v + sw_off(n, c8, nk), 0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int u = 0; u < kTcMaxItems; ++u) {
      const int idx = t0 + u * nt;
      const int hr = idx >> 4, c8 = idx & 15, r = hr & 15;
      if (idx < rep * 256) {
        const uint32_t o = s_v + sw_off(16 + W + hr, c8, nk);
        if (r < R)
          st_shared_v4(o, pack_bf16(mv[u][0].x, mv[u][0].y), pack_bf16(mv[u][0].z, mv[u][0].w),
                       pack_bf16(mv[u][1].x, mv[u][1].y), pack_bf16(mv[u][1].z, mv[u][1].w));
        else
          st_shared_v4(o, 0u, 0u, 0u, 0u);
      }
    }
  }
  // ---- block q (rep heads), k, v of KV head g from the projection's split
  //      partials: summed in split order, q and k RMS-normalised and rotated,
  //      rounded to bf16 and stored in the operand layouts (q rows
  //      h * qs + 16 c + i for copy c < DUP, key / value rows i).  A warp
  //      takes three rows at a time, every partial of them in flight.
  griddep_wait();
  {
    const int heads = p.nq + 2 * p.nkv, nitems = (rep + 2) * B;
    const size_t ldq = (size_t)heads * kTcD, pstride = (size_t)p.C * B * ldq;
    for (int it0 = warp; it0 < nitems; it0 += 3 * (kTcThreads / 32)) {
      float x[3][4];
      int kind[3], ii[3];
      const float* src[3];
#pragma unroll
      for (int u = 0; u < 3; ++u) {
        const int it = it0 + u * (kTcThreads / 32);
        kind[u] = it / B;
        ii[u] = it % B;
        const int head = kind[u] < rep ? g * rep + kind[u] : (kind[u] == rep ? p.nq + g : p.nq + p.nkv + g);
        src[u] = p.part + (size_t)(b * B + ii[u]) * ldq + (size_t)head * kTcD + 4 * lane;
        x[u][0] = x[u][1] = x[u][2] = x[u][3] = 0.f;
      }
      for (int s0 = 0; s0 < p.splits; s0 += 3) {
        float4 y[3][3];
#pragma unroll
        for (int v = 0; v < 3; ++v)
#pragma unroll
          for (int u = 0; u < 3; ++u)
            if (s0 + v < p.splits && it0 + u * (kTcThreads / 32) < nitems)
              y[v][u] = __ldcs(reinterpret_cast<const float4*>(src[u] + (size_t)(s0 + v) * pstride));
#pragma unroll
        for (int v = 0; v < 3; ++v)
#pragma unroll
          for (int u = 0; u < 3; ++u)
            if (s0 + v < p.splits && it0 + u * (kTcThreads / 32) < nitems) {
              x[u][0] += y[v][u].x;
              x[u][1] += y[v][u].y;
              x[u][2] += y[v][u].z;
              x[u][3] += y[v][u].w;
            }
      }
#pragma unroll
      for (int u = 0; u < 3; ++u) {
        if (it0 + u * (kTcThreads / 32) >= nitems) break;          // warp-uniform
        if (kind[u] <= rep) {
          float w[4], cs[8];
          ld_bf16x4(static_cast<const bf16*>(kind[u] < rep ? p.q_norm : p.k_norm) + 4 * lane, w);
          const float* csp = p.rope + ((size_t)(b * B + ii[u]) * (kTcD / 2) + 4 * (lane & 15)) * 2;
          const float4 c0 = *reinterpret_cast<const float4*>(csp), c1 = *reinterpret_cast<const float4*>(csp + 4);
          cs[0] = c0.x; cs[1] = c0.y; cs[2] = c0.z; cs[3] = c0.w; cs[4] = c1.x; cs[5] = c1.y; cs[6] = c1.z; cs[7] = c1.w;
          float ss = 0.f;
#pragma unroll
          for (int e = 0; e < 4; ++e) ss += x[u][e] * x[u][e];
          const float rstd = rsqrtf(warp_sum(ss) / (float)kTcD + p.eps);
#pragma unroll
          for (int e = 0; e < 4; ++e) x[u][e] *= rstd * w[e];
          // rotate-half: dim j pairs with j + 64 (lane ^ 16)
          const float sg = lane < 16 ? -1.f : 1.f;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float partner = __shfl_xor_sync(0xffffffffu, x[u][e], 16);
            x[u][e] = x[u][e] * cs[2 * e] + sg * partner * cs[2 * e + 1];
          }
        }
        const uint32_t lo = pack_bf16(x[u][0], x[u][1]), hi = pack_bf16(x[u][2], x[u][3]);
        const int c8 = lane >> 1;
        const uint32_t sub = (uint32_t)(lane & 1) * 8u;
        if (kind[u] < rep) {
#pragma unroll
          for (int c = 0; c < DUP; ++c) {
            const uint32_t a = s_q + sw_off(kind[u] * qs + 16 * c + ii[u], c8, kTcM) + sub;
            asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(a), "r"(lo), "r"(hi) : "memory");
          }
        } else {
          const uint32_t a = (kind[u] == rep ? s_k : s_v) + sw_off(ii[u], c8, nk) + sub;
          asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(a), "r"(lo), "r"(hi) : "memory");
        }
      }
    }
  }
  fence_proxy_async_smem();          // the tensor cores read the generic-proxy stores
  __syncthreads();

  // ---- S = Q K^T: columns [0, 256) and [256, nk), eight 16-dim steps each
  if (tid == 0) {
    const bool ok = mbar_spin(bar_kv, 0, p.err);
    if (!ok) {
      *s_abort = 1;
    } else {
      tc_fence_after();
#pragma unroll 1
      for (int n0 = 0; n0 < nk; n0 += 256) {
        const int nw = min(256, nk - n0);
        const uint32_t idesc = tc_idesc(nw, false);
#pragma unroll
        for (int ks = 0; ks < kTcD / 16; ++ks) {
          const uint32_t kb = (uint32_t)(ks >> 2), within = (uint32_t)(ks & 3) * 32u;
          const uint64_t ad = sdesc_sw128(s_q + kb * (kTcM * 128) + within);
          const uint64_t bd =
              sdesc_sw128(s_k + kb * (uint32_t)(nk * 128) + (uint32_t)(n0 / 8) * 1024u + within);
          umma_f16(tmem + (uint32_t)n0, ad, bd, idesc, ks > 0 ? 1u : 0u);
        }
      }
      umma_commit(bar_s);
    }
  }
  __syncthreads();
  const bool go = *s_abort == 0;

  // ---- softmax: the thread of TMEM lane `row`, over its warp's column
  //      quarter (chunks ch0 .. ch0 + my - 1), scores held in registers.
  //      With DUP == 2 the copy `hid` of a row takes chunks u = 2k + hid.
  const int q4 = warp & 3, qt = warp >> 2;
  const int row = q4 * 32 + lane, hh = row / qs, within = row % qs;
  const int hid = DUP == 2 ? (within >> 4) : 0, i = DUP == 2 ? (within & 15) : within;
  const bool row_ok = hh < rep && i < B;
  const int nch = nk / 16, ch0 = qt * nch / 4, my = (qt + 1) * nch / 4 - ch0;
  const uint32_t trow = tmem + ((uint32_t)(q4 * 32) << 16);
  // valid columns of a 16-column chunk are a prefix of it: their count
  auto chunk_lim = [&](int u) -> int {
    if (!row_ok || u >= my) return 0;
    const int cc = (ch0 + u) * 16;
    if (cc < 16) return B;
    if (cc < 16 + W) return max(0, min(16, count - (cc - 16)));
    return ((cc - 16 - W) >> 4) == hh ? R : 0;
  };
  if (go && !mbar_spin(bar_s, 0, p.err)) *s_abort = 1;
  tc_fence_after();
  float v[kTcMaxCh][16];
#pragma unroll
  for (int u = 0; u < kTcMaxCh; u += 2) {
    if (u + 1 < my)
      tmem_ld32(trow + (uint32_t)((ch0 + u) * 16), v[u]);     // v[u], v[u + 1] are contiguous
    else if (u < my)
      tmem_ld16(trow + (uint32_t)((ch0 + u) * 16), v[u]);
  }
  constexpr int kIter = kTcMaxCh / DUP;
  float mx = -INFINITY;
#pragma unroll
  for (int k = 0; k < kIter; ++k) {
    const int u = k * DUP + hid;
    const int lim = chunk_lim(u);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const float x = (DUP == 2 && hid) ? v[k * DUP + 1][j] : v[k * DUP][j];
      if (j < lim) mx = fmaxf(mx, x);
    }
  }
  if (DUP == 2) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
  sx[qt * 2 * kTcM + row] = mx;
  __syncthreads();
  const float sl2 = 1.4426950408889634f * rsqrtf((float)kTcD);
  const float m = fmaxf(fmaxf(sx[row], sx[2 * kTcM + row]), fmaxf(sx[4 * kTcM + row], sx[6 * kTcM + row]));
  const float mb = (m == -INFINITY) ? 0.f : m * sl2;
  float sum = 0.f;
  const uint32_t prow = s_p + (uint32_t)(row >> 3) * 1024u + (uint32_t)(row & 7) * 128u;
#pragma unroll
  for (int k = 0; k < kIter; ++k) {
    const int u = k * DUP + hid;
    const int lim = chunk_lim(u);
    uint32_t w[8];
#pragma unroll
    for (int j = 0; j < 16; j += 2) {
      const float x0 = (DUP == 2 && hid) ? v[k * DUP + 1][j] : v[k * DUP][j];
      const float x1 = (DUP == 2 && hid) ? v[k * DUP + 1][j + 1] : v[k * DUP][j + 1];
      const float p0 = ex2f(j < lim ? fmaf(x0, sl2, -mb) : -INFINITY);
      const float p1 = ex2f(j + 1 < lim ? fmaf(x1, sl2, -mb) : -INFINITY);
      const __nv_bfloat162 pr = __floats2bfloat162_rn(p0, p1);
      sum += __low2float(pr) + __high2float(pr);
      w[j >> 1] = *reinterpret_cast<const uint32_t*>(&pr);
    }
    // keys cc .. cc + 15 of this row: two 16-byte chunks of its 64-key block;
    // with DUP == 2 the other copy's chunk of this row is zero
#pragma unroll
    for (int c = 0; c < DUP; ++c) {
      const int uu = k * DUP + c;
      if (uu < my) {
        const int cc = (ch0 + uu) * 16;
        const bool mine = DUP == 1 || c == hid;
        const uint32_t base = prow + (uint32_t)(cc >> 6) * (kTcM * 128);
        const int ca = (cc & 63) >> 3;
        st_shared_v4(base + (uint32_t)((ca ^ (row & 7)) << 4), mine ? w[0] : 0u, mine ? w[1] : 0u,
                     mine ? w[2] : 0u, mine ? w[3] : 0u);
        st_shared_v4(base + (uint32_t)(((ca + 1) ^ (row & 7)) << 4), mine ? w[4] : 0u, mine ? w[5] : 0u,
                     mine ? w[6] : 0u, mine ? w[7] : 0u);
      }
    }
  }
  if (DUP == 2) sum += __shfl_xor_sync(0xffffffffu, sum, 16);
  sx[qt * 2 * kTcM + kTcM + row] = sum;
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();

  // ---- O = P V: nk / 16 key steps; V is the MN-major B operand
  if (tid == 0 && *s_abort == 0) {
    tc_fence_after();
    const uint32_t idesc = tc_idesc(kTcD, true);
    const uint32_t lbo = (uint32_t)nk * 128u;      // dims 0-63 -> dims 64-127
#pragma unroll 1
    for (int j = 0; j < nk / 16; ++j) {
      const uint64_t ad = sdesc_sw128(s_p + (uint32_t)(j >> 2) * (kTcM * 128) + (uint32_t)(j & 3) * 32u);
      const uint64_t bd = sdesc_sw128_mn(s_v + (uint32_t)j * 2048u, lbo);
      umma_f16(tmem + (uint32_t)kTcOcol, ad, bd, idesc, j > 0 ? 1u : 0u);
    }
    umma_commit(bar_o);
  }
  // ---- O / row sum -> bf16: this warp's 32 dims of its rows (with DUP == 2
  //      the two copies' partial O add, each copy storing 16 of the dims)
  __syncwarp();
  const bool go2 = *s_abort == 0;
  if (go2 && !mbar_spin(bar_o, 0, p.err)) *s_abort = 1;
  tc_fence_after();
  {
    const float tot = (sx[kTcM + row] + sx[3 * kTcM + row]) + (sx[5 * kTcM + row] + sx[7 * kTcM + row]);
    const float inv = tot > 0.f ? 1.0f / tot : 0.f;
    float o[32];
    tmem_ld32(trow + (uint32_t)(kTcOcol + qt * 32), o);
    bf16* out = static_cast<bf16*>(p.out) + (size_t)(b * B + i) * p.nq * kTcD + (size_t)(g * rep + hh) * kTcD +
                qt * 32;
    if (DUP == 2) {
      float f[16];
#pragma unroll
      for (int c = 0; c < 16; ++c) {
        const float send = hid ? o[c] : o[c + 16];
        const float recv = __shfl_xor_sync(0xffffffffu, send, 16);
        f[c] = (hid ? o[c + 16] : o[c]) + recv;
      }
      if (go2 && row_ok) {
#pragma unroll
        for (int c = 0; c < 16; c += 8) {
          uint4 w4;
          w4.x = pack_bf16(f[c] * inv, f[c + 1] * inv);
          w4.y = pack_bf16(f[c + 2] * inv, f[c + 3] * inv);
          w4.z = pack_bf16(f[c + 4] * inv, f[c + 5] * inv);
          w4.w = pack_bf16(f[c + 6] * inv, f[c + 7] * inv);
          *reinterpret_cast<uint4*>(out + hid * 16 + c) = w4;
        }
      }
    } else if (go2 && row_ok) {
#pragma unroll
      for (int c = 0; c < 32; c += 8) {
        uint4 w4;
        w4.x = pack_bf16(o[c] * inv, o[c + 1] * inv);
        w4.y = pack_bf16(o[c + 2] * inv, o[c + 3] * inv);
        w4.z = pack_bf16(o[c + 4] * inv, o[c + 5] * inv);
        w4.w = pack_bf16(o[c + 6] * inv, o[c + 7] * inv);
        *reinterpret_cast<uint4*>(out + c) = w4;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kTcCols);
  }
}

}  // namespace

bool attn_tc_supported(int B, int W, int R, int nq, int nkv, int d) {
  if (nkv < 1 || nq % nkv) return false;
  const int rep = nq / nkv;
  if (d != kTcD || B < 1 || B > 16 || R < 0 || R > 16 || W < 0 || W > 256 || W % 16 || rep < 1 || rep > 8)
    return false;
  const TcLayout L = tc_layout(W, rep);
  return L.nk <= kTcMaxKeys && L.bytes <= 227 * 1024;
}

int attn_tc_plan(AttnTcPlan* pl, const AttnParams& p) {
  pl->ok = 0;
  if (!attn_tc_supported(p.B, p.W, p.R, p.nq, p.nkv, p.d)) return LSP_ERR_SHAPE;
  pl->wbox = p.W % 32 == 0 ? 32 : 16;
  const uint64_t wrows = (uint64_t)p.C * p.L * p.nkv * (p.W > 0 ? p.W : 1);
  int rc;
  if ((rc = tmap_2d_bf16_sw128(&pl->wk, p.win_k, kTcD, wrows, kTcD * 2, 64, pl->wbox)) != LSP_OK) return rc;
  if ((rc = tmap_2d_bf16_sw128(&pl->wv, p.win_v, kTcD, wrows, kTcD * 2, 64, pl->wbox)) != LSP_OK) return rc;
  const uint64_t grows = (uint64_t)p.L * p.nq * (p.R > 0 ? p.R : 1);
  if ((rc = tmap_2d_bf16_sw128(&pl->g, p.G, kTcD, grows, kTcD * 2, 64, p.R > 0 ? p.R : 1)) != LSP_OK) return rc;
  pl->ok = 1;
  return LSP_OK;
}

int launch_attention_tc(const AttnParams& p, const AttnTcPlan& pl, cudaStream_t s) {
  if (!pl.ok) return LSP_ERR_SHAPE;
  const TcLayout L = tc_layout(p.W, p.nq / p.nkv);
  static bool attr_set = false;
  if (!attr_set) {
    if (cudaFuncSetAttribute(attn_tc_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024) !=
            cudaSuccess ||
        cudaFuncSetAttribute(attn_tc_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024) !=
            cudaSuccess)
      return LSP_ERR_CUDA;
    attr_set = true;
  }
  const cudaError_t e =
      L.dup == 2 ? launch_pdl(attn_tc_kernel<2>, dim3(p.C * p.nkv), dim3(kTcThreads), (size_t)L.bytes, s, pl.wk,
                              pl.wv, pl.g, p, pl.wbox)
                 : launch_pdl(attn_tc_kernel<1>, dim3(p.C * p.nkv), dim3(kTcThreads), (size_t)L.bytes, s, pl.wk,
                              pl.wv, pl.g, p, pl.wbox);
  return e == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

}  // namespace lsp
