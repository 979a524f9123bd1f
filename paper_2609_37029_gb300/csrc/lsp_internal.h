// Internal host-side interfaces between the C-ABI layer and the kernel files.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/lsp.h"

namespace lsp {

// ------------------------------------------------------------------ launch helper
// Launch as a programmatic dependent of the preceding work in the stream: the
// kernel may start while its predecessor finishes and must call griddep_wait()
// before it reads the predecessor's outputs or writes anything it reads.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// ------------------------------------------------------------------ GEMM
enum EpiMode {
  EPI_F32 = 0,      // Y (float) = acc
  EPI_T = 1,        // Y (dtype) = acc
  EPI_PARTIAL = 2,  // Y (float) [split][M][ldy] = this split's partial sum (the consumer adds)
  EPI_SWIGLU = 3,   // Y (dtype) = silu(acc_gate) * acc_up
};

constexpr int kGemmThreads = 192;   // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr int kTileRows = 128;      // weight rows per tile (UMMA M)

struct GemmParams {
  int M, N, K;          // token rows, output features, reduction length
  int kblocks, splits, n_tiles;
  int mode;
  int seg_tile0[3];     // first tile index of each A segment
  int nseg;
  int bn, n_tok_tiles, m_pad, stages, tmem_cols;
  int tma_out;          // 1: the epilogue stages tiles in shared memory and TMA-stores them
  int out_tok;          // tokens per staged output chunk (16 or 32)
  int tok_groups;       // CTAs per weight tile, each over m_pad consecutive tokens
  int late_trigger;     // 1: let the next kernel launch only after this one's dependency wait
  void* Y;
  int ldy;
  unsigned* err;
};

struct GemmOp {
  CUtensorMap a[3];
  CUtensorMap b;
  CUtensorMap out;      // [splits][M][N] view of Y for the TMA-store epilogue
  GemmParams p;
  int dtype;
  dim3 grid;
  int occ;              // CTAs per SM the plan sizes for: 3 picks the register-bounded instance
  size_t smem;
};

// Plan Y = X W^T where W is the row-concatenation of `nseg` weight segments
// (each [seg_rows[i]][K]); for EPI_SWIGLU, segment 0 = gate and 1 = up, both
// [N][K].  EPI_PARTIAL writes `splits` fp32 partial sums [splits][M][ldy] for
// the consumer to add; other modes need splits == 1.  splits <= 0 chooses
// for `num_sms`.
int gemm_plan(GemmOp* op, int dtype, const void* X, int M, int K, const void* const* W,
              const int* seg_rows, int nseg, int mode, void* Y, int ldy, unsigned* err,
              int num_sms, int splits);
int gemm_launch(const GemmOp* op, cudaStream_t s);
// The split-K factor gemm_plan uses (input <= 0 = choose), and the token
// groups it splits M into (groups may be null).
void gemm_choose(int dtype, int M, int K, int n_tiles, int mode, int num_sms, int* splits,
                 int* groups = nullptr);
int gemm_tiles(int mode, const int* seg_rows, int nseg);
// Token rows one token group of M rows split G ways covers (a multiple of 16).
int gemm_group_rows(int M, int G);
// occ_max: CTAs one SM can hold (1-3) for this tile shape.
int gemm_auto_splits(int n_ctas, int kblocks, int num_sms, double per_split_cost, int max_splits,
                     int occ_max);
double gemm_partial_cost(int M, int N);
int gemm_kblocks(int K, int dtype);
// Deterministic sum of `splits` fp32 partials [splits][n] into y[n].
int launch_sum_partials(const float* part, int splits, size_t n, float* y, cudaStream_t s);

// ------------------------------------------------------------------ view update
struct ViewParams {
  const void* k_new;
  const void* v_new;
  const void* h_new;
  int rows;
  int h_rows;             // rows of h_new per (b, l): rows, or 1 = only the boundary row
  const int32_t* acc;
  const void* G;
  void* win_k;
  void* win_v;
  float* m;
  float* eta;
  void* h;
  int64_t* t;
  int* done;
  unsigned* err;
  int C, L, nq, nkv, d, H, W, R;
};
int launch_view_update(const ViewParams& p, int dtype, cudaStream_t s);

// ------------------------------------------------------------------ small ops
struct CombineParams {
  const int32_t* tokens;   // [C][B]
  const void* embed;       // [V][H]
  const void* pos;         // [B][H]
  const void* mask_emb;    // [H]
  const float* c;          // [splits][C][H] partial sums of c_t
  int c_splits;
  const void* norm_w;      // [H] first layer input norm
  float* x;                // [M][H]
  void* xn;                // [M][H]
  float* rope;             // [C][B][d/2][2]
  const int64_t* t;        // [C]
  unsigned* err;
  int C, B, H, V, d;
  float eps;
  double theta;
};
int launch_combine(const CombineParams& p, int dtype, cudaStream_t s);
// x += sum_s part[s] (s < splits, fp32 [splits][M][H]); out = RMSNorm(x) * w.
int launch_resid_norm(float* x, const float* part, int splits, const void* w, void* out, int M,
                      int H, float eps, int dtype, cudaStream_t s);

// ------------------------------------------------------------------ attention
// q | k | v of the block rows: sum of the projection's split-K partials, then
// per-head RMSNorm (q_norm / k_norm) and rotary embedding on q and k.
struct QkvParams {
  const float* part;      // [splits][M][(nq+2nkv)d] fp32
  int splits;
  const void* q_norm;     // [d]
  const void* k_norm;     // [d]
  const float* rope;      // [C][B][d/2][2]
  void* out;              // [M][(nq+2nkv)d] dtype
  int M, B, nq, nkv, d;
  float eps;
};
int launch_qkv_finalize(const QkvParams& p, int dtype, cudaStream_t s);

struct AttnParams {
  const void* qkv;        // [M][(nq+2nkv)d] dtype: normalised, rotated q, k; v
  const void* win_k;      // state window of the tapped layer's base: [C][L][nkv][W][d]
  const void* win_v;
  const void* G;          // [L][nq][R][d]
  const float* m;         // [C][L][nq][R][d]
  const int64_t* t;       // [C]
  void* out;              // [M][nq d]
  int C, B, L, nq, nkv, d, W, R, layer;
  float eps;
  unsigned* err;          // device error word (a bounded wait that gave up)
  // tcgen05 kernel only: the q/k/v projection's split partials, finalised
  // inside the attention (sum in split order, q/k RMSNorm, rotary embedding)
  const float* part;      // [splits][M][(nq+2nkv)d] fp32
  int splits;
  const void* q_norm;     // [d]
  const void* k_norm;     // [d]
  const float* rope;      // [C][B][d/2][2]
};
// Tensor maps of the tcgen05 attention (window K and V, summary keys G),
// built once per state: ok == 0 where the shape is not served
// (bf16, d = 128, B <= 16, R <= 16, W <= 256 with W % 16 == 0, nq/nkv <= 8,
// 16 + W + 16 nq/nkv <= 352).
struct AttnTcPlan {
  CUtensorMap wk, wv, g;
  int wbox;               // window rows per TMA box
  int ok;
};
int attn_tc_plan(AttnTcPlan* pl, const AttnParams& p);
bool attn_tc_supported(int B, int W, int R, int nq, int nkv, int d);
// tc: the state's plan (null or !ok: the mma.sync kernel).
int launch_attention(const AttnParams& p, int dtype, cudaStream_t s, const AttnTcPlan* tc);
int launch_attention_tc(const AttnParams& p, const AttnTcPlan& pl, cudaStream_t s);
// 2-D bf16 tensor map, 128-byte swizzle: rows x inner elements (row pitch
// row_bytes), box (box_inner <= 64, box_rows <= 256).
int tmap_2d_bf16_sw128(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t rows, uint64_t row_bytes,
                       uint32_t box_inner, uint32_t box_rows);

// ------------------------------------------------------------------ prefill
struct PrefillParams {
  const void* k;          // request b's prefix K: [L][rows][nkv][d] dtype
  const void* v;          // V, same layout
  const void* hid;        // hidden states [L][h_rows][H] dtype (h_rows = rows or 1: the last row only)
  int rows;               // t (>= 1)
  int h_rows;
  const void* G;          // [L][nq][R][d]
  void* win_k;            // state window [C][L][nkv][W][d]
  void* win_v;
  float* m;               // [C][L][nq][R][d]
  float* eta;             // [C][L][nq][R]
  void* h;                // [C][L][H]
  int64_t* t;             // [C]
  float* ws;              // prefill_ws_floats(L, nq) segment partials
  int b, L, nq, nkv, d, W, R, H;
};
constexpr int kPrefillMaxSeg = 64;   // prefix segments (CTAs per tapped layer x KV head)
size_t prefill_ws_floats(int L, int nq);
int launch_prefill(const PrefillParams& p, int dtype, cudaStream_t s);

// ------------------------------------------------------------------ verification
struct VerifyParams {
  const float* zt;          // target logits [C][B+1][V]
  const float* zq;          // draft logits [C][B][V]
  const int32_t* y;         // drafted tokens [C][B]
  int32_t* accepted;        // [C]
  int32_t* next_token;      // [C]
  float* st_a;              // chunk partials [C][2B+1][nst]: max of z log2(e) / T (T > 0), max of z (T = 0)
  float* st_b;              //   sum of 2^(x - max) (T > 0)
  int* st_i;                //   argmax index (T = 0)
  int nst;                  // chunks per row (set by launch_verify)
  float* part_val;          // draw partials [C][<= kVerMaxDrawChunks]
  int* part_idx;
  unsigned* ctr;            // [C] self-resetting counters (zero between calls)
  unsigned* err;
  int C, B, V;
  float temperature;
  uint32_t round;
  uint64_t seed;
};
constexpr int kVerMaxStatChunks = 32;
constexpr int kVerMaxDrawChunks = 128;
constexpr int kVerMaxB = 512;
int verify_max_stat_chunks(int V);
int launch_verify(const VerifyParams& p, int num_sms, cudaStream_t s);

// ------------------------------------------------------------------ sampler
struct SampleParams {
  const float* src;       // [C][B][V] base logits
  float* dst;             // [C][B][V] corrected logits or nullptr
  const int32_t* prev;    // y_0 source: element b * prev_stride
  int prev_stride;
  const void* Ec;
  const void* Wc;
  int32_t* out_tokens;    // [C][B]
  float* part_val;        // [2][nblk][C]   (per-step kernel)
  int* part_idx;          // [2][nblk][C]
  unsigned long long* sync;   // sample_sync_bytes(B): step keys + arrival counts (persistent
                              // kernel); all zero between launches
  unsigned* err;
  int C, B, V, rc, nblk;
  int num_sms;
  float temperature;
  uint32_t round;
  uint64_t seed;
  int b0;                 // global index of request 0 of this launch (the Philox counter's request word)
};
int sample_blocks(int num_sms);
size_t sample_sync_bytes(int B);
int launch_sample(const SampleParams& p, int dtype, cudaStream_t s);
// Kernel launches one launch_sample call issues for these shapes on this device.
int sample_launches(const SampleParams& p, int dtype);
int launch_philox_words(uint64_t seed, uint32_t round, uint32_t b, uint32_t i, uint32_t* out,
                        int count, cudaStream_t s);

}  // namespace lsp
