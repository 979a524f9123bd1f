// C ABI of the drafting round: state ownership, host-side validation and the
// launch sequence of one round (declarations and contracts: include/lsp.h).
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <new>

#include "lsp_internal.h"

namespace lsp {
size_t attn_smem_bytes(int B, int W, int nq, int nkv);
}

using namespace lsp;

namespace {

inline size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }
inline int esize(int dtype) { return dtype == LSP_DTYPE_BF16 ? 2 : 4; }

struct Layout {
  // interface (export order)
  size_t win, m, eta, h, t;
  // extras
  size_t G, err, done;
};

Layout interface_layout(const lsp_config& c) {
  const size_t es = esize(c.dtype);
  Layout l;
  l.win = (size_t)c.C * c.L * c.nkv * c.W * c.d * es;
  l.m = (size_t)c.C * c.L * c.nq * c.R * c.d * sizeof(float);
  l.eta = (size_t)c.C * c.L * c.nq * c.R * sizeof(float);
  l.h = (c.flags & LSP_NO_BOUNDARY) ? 0 : (size_t)c.C * c.L * c.H * es;
  l.t = (size_t)c.C * sizeof(int64_t);
  l.G = (size_t)c.L * c.nq * c.R * c.d * es;
  l.err = sizeof(unsigned);
  l.done = (size_t)c.C * sizeof(int);
  return l;
}

int layer_of(const lsp_config& c, int j) {
  return c.layer_map[j] >= 0 ? c.layer_map[j] : j * c.L / c.D;
}

struct PlanKey {
  lsp_weights w;
  float* out_logits;
};

}  // namespace

struct lsp_state {
  lsp_config cfg;
  int device = 0, num_sms = 0;
  bool initialized = false;
  // interface
  void* base = nullptr;
  void *win_k = nullptr, *win_v = nullptr, *h = nullptr, *G = nullptr;
  float *m = nullptr, *eta = nullptr;
  int64_t* t = nullptr;
  unsigned* err = nullptr;
  int* done = nullptr;
  // workspace
  void* ws = nullptr;
  float *x = nullptr, *logits = nullptr, *rope = nullptr, *part = nullptr;
  void *xn = nullptr, *qkv = nullptr, *o = nullptr, *act = nullptr;
  size_t part_bytes = 0;
  float* part_val = nullptr;
  int* part_idx = nullptr;
  float* prefill_ws = nullptr;       // prefill segment partials (bf16, d = 128 configs)
  float* ver_sa = nullptr;           // verification row partials and draw partials
  float* ver_sb = nullptr;
  int* ver_si = nullptr;
  float* ver_pv = nullptr;
  int* ver_pi = nullptr;
  unsigned* ver_ctr = nullptr;
  unsigned long long* sample_sync = nullptr;
  size_t sample_sync_bytes = 0;
  int nblk = 0;
  // cached projection plans
  AttnTcPlan attn_tc = {};
  bool have_plans = false;
  PlanKey key;
  GemmOp fuse, lm;
  GemmOp qkv_op[LSP_MAX_DRAFT_LAYERS], o_op[LSP_MAX_DRAFT_LAYERS], gu_op[LSP_MAX_DRAFT_LAYERS],
      down_op[LSP_MAX_DRAFT_LAYERS];
  // optional stage-boundary events (caller-owned)
  cudaEvent_t stage_ev[8 + 7 * LSP_MAX_DRAFT_LAYERS] = {};
  int n_stage_ev = 0;
};

namespace {
const char* kLayerStages[7] = {"qkv", "attention", "o_proj", "post_norm", "gate_up", "down", "next_norm"};
inline int stage_total(const lsp_config& c) { return 5 + 7 * c.D; }
// External records so that a captured round carries them as event-record nodes.
inline void mark(lsp_state* st, int k, cudaStream_t s) {
  if (k < st->n_stage_ev) cudaEventRecordWithFlags(st->stage_ev[k], s, cudaEventRecordExternal);
}
}  // namespace

extern "C" {

const char* lsp_status_string(int s) {
  switch (s) {
    case LSP_OK: return "ok";
    case LSP_ERR_ARG: return "invalid argument";
    case LSP_ERR_SHAPE: return "unsupported shape";
    case LSP_ERR_CUDA: return "CUDA error";
    case LSP_ERR_TIMEOUT: return "device wait timed out";
    case LSP_ERR_STATE: return "state not initialised or device error pending";
    case LSP_ERR_NOMEM: return "device allocation failed";
    case LSP_ERR_UNSUPPORTED: return "unsupported device or feature";
    default: return "unknown status";
  }
}

int lsp_config_check(const lsp_config* c) {
  if (!c) return LSP_ERR_ARG;
  if (c->C < 1 || c->B < 1 || c->L < 1 || c->D < 1 || c->H < 1 || c->nq < 1 || c->nkv < 1 ||
      c->d < 2 || c->F < 1 || c->V < 1 || c->W < 0 || c->R < 0 || c->rc < 1)
    return LSP_ERR_SHAPE;
  if (c->dtype != LSP_DTYPE_BF16 && c->dtype != LSP_DTYPE_F32) return LSP_ERR_ARG;
  if (c->flags & ~LSP_NO_BOUNDARY) return LSP_ERR_ARG;
  if (c->D > LSP_MAX_DRAFT_LAYERS || c->nq % c->nkv) return LSP_ERR_SHAPE;
  if (c->C * c->B > 512 || c->C > 64) return LSP_ERR_SHAPE;
  if (c->H % 128 || (c->nq * c->d) % 128 || (c->nkv * c->d) % 128 || c->F % 64) return LSP_ERR_SHAPE;
  if (c->H > 8192 || (c->H / c->nkv) % 8) return LSP_ERR_SHAPE;
  if (c->V % 16 || c->rc % 16 || c->rc > 256) return LSP_ERR_SHAPE;
  if (!(c->rope_theta > 0.f) || !(c->rms_eps >= 0.f)) return LSP_ERR_ARG;
  const int rep = c->nq / c->nkv;
  if (rep * c->R > 128) return LSP_ERR_SHAPE;                 // view-update queries per CTA
  if (c->d != 64 && c->d != 128) return LSP_ERR_SHAPE;        // view-update lane split
  if (c->dtype == LSP_DTYPE_BF16) {
    if (c->d != 128 || c->B > 16 || c->R > 16) return LSP_ERR_SHAPE;
    if (lsp::attn_smem_bytes(c->B, c->W, c->nq, c->nkv) > 227 * 1024) return LSP_ERR_SHAPE;
  } else {
    if ((size_t)(3 * c->B * c->d + c->B * (c->B + c->W + c->R) + 4 + 64 * c->d) * 4 > 227 * 1024) return LSP_ERR_SHAPE;
  }
  for (int j = 0; j < c->D; ++j)
    if (c->layer_map[j] >= c->L) return LSP_ERR_SHAPE;
  return LSP_OK;
}

size_t lsp_state_bytes(const lsp_config* c) {
  if (lsp_config_check(c) != LSP_OK) return 0;
  const Layout l = interface_layout(*c);
  return 2 * l.win + l.m + l.eta + l.h + l.t;
}

static void free_state(lsp_state* st) {
  if (!st) return;
  if (st->base) cudaFree(st->base);
  if (st->ws) cudaFree(st->ws);
  delete st;
}

// Projections that write split-K partials (summed by their consumer): their
// token rows, reduction length and output features, for sizing the buffer.
static void partial_shapes(const lsp_config& c, int* M, int* K, int* N, int* n) {
  const int Mt = c.C * c.B;
  int i = 0;
  M[i] = c.C; K[i] = c.L * c.H; N[i++] = c.H;                      // boundary fusion
  M[i] = Mt; K[i] = c.H; N[i++] = (c.nq + 2 * c.nkv) * c.d;        // q | k | v
  M[i] = Mt; K[i] = c.nq * c.d; N[i++] = c.H;                      // o
  M[i] = Mt; K[i] = c.F; N[i++] = c.H;                             // down
  *n = i;
}

int lsp_state_create(const lsp_config* cfg, lsp_state** out) {
  if (!cfg || !out) return LSP_ERR_ARG;
  *out = nullptr;
  int rc = lsp_config_check(cfg);
  if (rc != LSP_OK) return rc;
  lsp_state* st = new (std::nothrow) lsp_state();
  if (!st) return LSP_ERR_NOMEM;
  st->cfg = *cfg;
  lsp_config& c = st->cfg;
  for (int j = 0; j < c.D; ++j) c.layer_map[j] = layer_of(*cfg, j);
  if (cudaGetDevice(&st->device) != cudaSuccess) { free_state(st); return LSP_ERR_CUDA; }
  cudaDeviceProp prop;
  if (cudaGetDeviceProperties(&prop, st->device) != cudaSuccess) { free_state(st); return LSP_ERR_CUDA; }
  if (prop.major < 10) { free_state(st); return LSP_ERR_UNSUPPORTED; }
  st->num_sms = prop.multiProcessorCount;

  // ---- interface allocation
  const Layout l = interface_layout(c);
  size_t off = 0;
  const size_t o_wk = off; off = align256(off + l.win);
  const size_t o_wv = off; off = align256(off + l.win);
  const size_t o_m = off; off = align256(off + l.m);
  const size_t o_eta = off; off = align256(off + l.eta);
  const size_t o_h = off; off = align256(off + l.h);
  const size_t o_t = off; off = align256(off + l.t);
  const size_t o_G = off; off = align256(off + l.G);
  const size_t o_err = off; off = align256(off + l.err);
  const size_t o_done = off; off = align256(off + l.done);
  if (cudaMalloc(&st->base, off) != cudaSuccess) { free_state(st); return LSP_ERR_NOMEM; }
  char* b = static_cast<char*>(st->base);
  st->win_k = b + o_wk; st->win_v = b + o_wv;
  st->m = reinterpret_cast<float*>(b + o_m);
  st->eta = reinterpret_cast<float*>(b + o_eta);
  st->h = l.h ? b + o_h : nullptr;
  st->t = reinterpret_cast<int64_t*>(b + o_t);
  st->G = b + o_G;
  st->err = reinterpret_cast<unsigned*>(b + o_err);
  st->done = reinterpret_cast<int*>(b + o_done);

  // ---- workspace
  const size_t es = esize(c.dtype);
  const int M = c.C * c.B;
  int pm[8], pk[8], pn[8], np;
  partial_shapes(c, pm, pk, pn, &np);
  size_t pbytes = 0;
  for (int i = 0; i < np; ++i) {
    int splits = 0;
    const int rows[1] = {pn[i]};
    gemm_choose(c.dtype, pm[i], pk[i], gemm_tiles(EPI_PARTIAL, rows, 1), EPI_PARTIAL, st->num_sms, &splits);
    pbytes = std::max(pbytes, (size_t)splits * pm[i] * pn[i] * sizeof(float));
  }
  st->nblk = sample_blocks(st->num_sms);
  off = 0;
  const size_t w_x = off; off = align256(off + (size_t)M * c.H * 4);
  const size_t w_xn = off; off = align256(off + (size_t)M * c.H * es);
  const size_t w_qkv = off; off = align256(off + (size_t)M * (c.nq + 2 * c.nkv) * c.d * es);
  const size_t w_o = off; off = align256(off + (size_t)M * c.nq * c.d * es);
  const size_t w_act = off; off = align256(off + (size_t)M * c.F * es);
  const size_t w_log = off; off = align256(off + (size_t)M * c.V * 4);
  const size_t w_rope = off; off = align256(off + (size_t)M * (c.d / 2) * 2 * 4);
  const size_t w_part = off; off = align256(off + pbytes);
  const size_t w_pv = off; off = align256(off + (size_t)2 * st->nblk * c.C * 4);
  const size_t w_pi = off; off = align256(off + (size_t)2 * st->nblk * c.C * 4);
  const size_t w_sync = off; off = align256(off + sample_sync_bytes(c.B));
  const bool prefill_ok = c.dtype == LSP_DTYPE_BF16 && c.d == 128;
  const size_t w_pf = off; off = align256(off + (prefill_ok ? prefill_ws_floats(c.L, c.nq) * sizeof(float) : 0));
  const size_t ver_rows = (size_t)c.C * (2 * c.B + 1) * verify_max_stat_chunks(c.V);
  const size_t w_vsa = off; off = align256(off + ver_rows * sizeof(float));
  const size_t w_vsb = off; off = align256(off + ver_rows * sizeof(float));
  const size_t w_vsi = off; off = align256(off + ver_rows * sizeof(int));
  const size_t w_vpv = off; off = align256(off + (size_t)c.C * kVerMaxDrawChunks * sizeof(float));
  const size_t w_vpi = off; off = align256(off + (size_t)c.C * kVerMaxDrawChunks * sizeof(int));
  const size_t w_vc = off; off = align256(off + (size_t)c.C * sizeof(unsigned));
  if (cudaMalloc(&st->ws, off) != cudaSuccess) { free_state(st); return LSP_ERR_NOMEM; }
  char* w = static_cast<char*>(st->ws);
  st->x = reinterpret_cast<float*>(w + w_x);
  st->xn = w + w_xn;
  st->qkv = w + w_qkv;
  st->o = w + w_o;
  st->act = w + w_act;
  st->logits = reinterpret_cast<float*>(w + w_log);
  st->rope = reinterpret_cast<float*>(w + w_rope);
  st->part = reinterpret_cast<float*>(w + w_part);
  st->part_bytes = pbytes;
  st->part_val = reinterpret_cast<float*>(w + w_pv);
  st->part_idx = reinterpret_cast<int*>(w + w_pi);
  st->sample_sync = reinterpret_cast<unsigned long long*>(w + w_sync);
  st->prefill_ws = prefill_ok ? reinterpret_cast<float*>(w + w_pf) : nullptr;
  st->ver_sa = reinterpret_cast<float*>(w + w_vsa);
  st->ver_sb = reinterpret_cast<float*>(w + w_vsb);
  st->ver_si = reinterpret_cast<int*>(w + w_vsi);
  st->ver_pv = reinterpret_cast<float*>(w + w_vpv);
  st->ver_pi = reinterpret_cast<int*>(w + w_vpi);
  st->ver_ctr = reinterpret_cast<unsigned*>(w + w_vc);
  st->sample_sync_bytes = sample_sync_bytes(c.B);
  if (cudaMemset(st->ws, 0, off) != cudaSuccess || cudaMemset(st->base, 0, o_done + l.done) != cudaSuccess) {
    free_state(st);
    return LSP_ERR_CUDA;
  }
  *out = st;
  return LSP_OK;
}

void lsp_state_destroy(lsp_state* st) {
  if (!st) return;
  cudaDeviceSynchronize();
  free_state(st);
}

static inline cudaStream_t S(lsp_stream_t s) { return static_cast<cudaStream_t>(s); }

__global__ void state_reset_kernel(float* eta, size_t n_eta, int64_t* t, int C, unsigned* err,
                                   int* done) {
  const size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x;
  if (i < n_eta) eta[i] = -INFINITY;
  if (i < (size_t)C) { t[i] = 0; done[i] = 0; }
  if (i == 0) *err = 0;
}

int lsp_state_init(lsp_state* st, const void* G, lsp_stream_t stream) {
  if (!st) return LSP_ERR_ARG;
  const lsp_config& c = st->cfg;
  const Layout l = interface_layout(c);
  if (!G && l.G) return LSP_ERR_ARG;          // G is empty (may be null) when R = 0
  cudaStream_t s = S(stream);
  auto zero = [&](void* p, size_t n) { return n == 0 || cudaMemsetAsync(p, 0, n, s) == cudaSuccess; };
  if (!zero(st->win_k, l.win) || !zero(st->win_v, l.win) || !zero(st->m, l.m) || !zero(st->h, l.h) ||
      (l.G && cudaMemcpyAsync(st->G, G, l.G, cudaMemcpyDeviceToDevice, s) != cudaSuccess))
    return LSP_ERR_CUDA;
  const size_t n_eta = l.eta / sizeof(float);
  const size_t n = std::max(n_eta, (size_t)c.C);
  state_reset_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(st->eta, n_eta, st->t, c.C, st->err,
                                                                  st->done);
  if (cudaGetLastError() != cudaSuccess) return LSP_ERR_CUDA;
  st->initialized = true;
  return LSP_OK;
}

// rows of h per (b, l) that a feature struct describes (-1: invalid)
static int feats_h_rows(const lsp_target_feats* f) {
  if (f->h_rows == 0 || f->h_rows == f->rows) return f->rows;
  return f->h_rows == 1 ? 1 : -1;
}

int lsp_view_update(lsp_state* st, const lsp_target_feats* f, const int32_t* acc,
                    lsp_stream_t stream) {
  if (!st || !f || !acc || !f->k || !f->v || f->rows < 1 || feats_h_rows(f) < 0) return LSP_ERR_ARG;
  if (!f->h && st->h) return LSP_ERR_ARG;
  if (!st->initialized) return LSP_ERR_STATE;
  const lsp_config& c = st->cfg;
  ViewParams p;
  p.k_new = f->k; p.v_new = f->v; p.h_new = f->h; p.rows = f->rows; p.h_rows = feats_h_rows(f); p.acc = acc;
  p.G = st->G; p.win_k = st->win_k; p.win_v = st->win_v; p.m = st->m; p.eta = st->eta;
  p.h = st->h; p.t = st->t; p.done = st->done; p.err = st->err;
  p.C = c.C; p.L = c.L; p.nq = c.nq; p.nkv = c.nkv; p.d = c.d; p.H = c.H; p.W = c.W; p.R = c.R;
  mark(st, 0, S(stream));
  const int rc = launch_view_update(p, c.dtype, S(stream));
  mark(st, 1, S(stream));
  return rc;
}

int lsp_prefill(lsp_state* st, int b, const lsp_target_feats* f, lsp_stream_t stream) {
  if (!st || !f || !f->k || !f->v || f->rows < 1 || feats_h_rows(f) < 0) return LSP_ERR_ARG;
  if (!f->h && st->h) return LSP_ERR_ARG;
  if (!st->initialized) return LSP_ERR_STATE;
  const lsp_config& c = st->cfg;
  if (b < 0 || b >= c.C) return LSP_ERR_ARG;
  PrefillParams p;
  p.k = f->k; p.v = f->v; p.hid = f->h; p.rows = f->rows; p.h_rows = feats_h_rows(f); p.G = st->G;
  p.win_k = st->win_k; p.win_v = st->win_v; p.m = st->m; p.eta = st->eta; p.h = st->h; p.t = st->t;
  p.ws = st->prefill_ws;
  p.b = b; p.L = c.L; p.nq = c.nq; p.nkv = c.nkv; p.d = c.d; p.W = c.W; p.R = c.R; p.H = c.H;
  return launch_prefill(p, c.dtype, S(stream));
}

int lsp_verify(lsp_state* st, const float* target_logits, const float* draft_logits,
               const int32_t* draft_tokens, const lsp_sample_params* sp, int32_t* accepted_len,
               int32_t* next_token, lsp_stream_t stream) {
  if (!st || !target_logits || !draft_logits || !draft_tokens || !sp || !accepted_len || !next_token)
    return LSP_ERR_ARG;
  if (!(sp->temperature >= 0.f) || !std::isfinite(sp->temperature)) return LSP_ERR_ARG;
  if (((uintptr_t)target_logits | (uintptr_t)draft_logits) & 15) return LSP_ERR_ARG;
  const lsp_config& c = st->cfg;
  VerifyParams p;
  p.zt = target_logits; p.zq = draft_logits; p.y = draft_tokens;
  p.accepted = accepted_len; p.next_token = next_token;
  p.st_a = st->ver_sa; p.st_b = st->ver_sb; p.st_i = st->ver_si; p.nst = 1;
  p.part_val = st->ver_pv; p.part_idx = st->ver_pi;
  p.ctr = st->ver_ctr; p.err = st->err;
  p.C = c.C; p.B = c.B; p.V = c.V;
  p.temperature = sp->temperature; p.round = sp->round; p.seed = sp->seed;
  return launch_verify(p, st->num_sms, S(stream));
}

static int build_plans(lsp_state* st, const lsp_weights* w, float* out_logits) {
  const lsp_config& c = st->cfg;
  const int M = c.C * c.B;
  const int dt = c.dtype;
  int rc;
  auto plan = [&](GemmOp* op, const void* X, int Mx, int K, const void* const* W, const int* rows,
                  int nseg, int mode, void* Y, int ldy) {
    const int r = gemm_plan(op, dt, X, Mx, K, W, rows, nseg, mode, Y, ldy, st->err, st->num_sms, 0);
    if (r == LSP_OK && mode == EPI_PARTIAL &&
        (size_t)op->p.splits * Mx * op->p.N * sizeof(float) > st->part_bytes)
      return LSP_ERR_SHAPE;
    return r;
  };
  if (st->h) {
    if (!w->fuse) return LSP_ERR_ARG;
    const void* W[1] = {w->fuse};
    const int rows[1] = {c.H};
    if ((rc = plan(&st->fuse, st->h, c.C, c.L * c.H, W, rows, 1, EPI_PARTIAL, st->part, c.H)) != LSP_OK)
      return rc;
  }
  for (int j = 0; j < c.D; ++j) {
    const lsp_layer_weights& lw = w->layer[j];
    if (!lw.in_norm || !lw.wq || !lw.wk || !lw.wv || !lw.q_norm || !lw.k_norm || !lw.wo ||
        !lw.post_norm || !lw.w_gate || !lw.w_up || !lw.w_down)
      return LSP_ERR_ARG;
    const void* Wqkv[3] = {lw.wq, lw.wk, lw.wv};
    const int rqkv[3] = {c.nq * c.d, c.nkv * c.d, c.nkv * c.d};
    if ((rc = plan(&st->qkv_op[j], st->xn, M, c.H, Wqkv, rqkv, 3, EPI_PARTIAL, st->part,
                   (c.nq + 2 * c.nkv) * c.d)) != LSP_OK)
      return rc;
    const void* Wo[1] = {lw.wo};
    const int ro[1] = {c.H};
    if ((rc = plan(&st->o_op[j], st->o, M, c.nq * c.d, Wo, ro, 1, EPI_PARTIAL, st->part, c.H)) != LSP_OK)
      return rc;
    const void* Wgu[2] = {lw.w_gate, lw.w_up};
    const int rgu[2] = {c.F, c.F};
    if ((rc = plan(&st->gu_op[j], st->xn, M, c.H, Wgu, rgu, 2, EPI_SWIGLU, st->act, c.F)) != LSP_OK)
      return rc;
    const void* Wd[1] = {lw.w_down};
    const int rd[1] = {c.H};
    if ((rc = plan(&st->down_op[j], st->act, M, c.F, Wd, rd, 1, EPI_PARTIAL, st->part, c.H)) != LSP_OK)
      return rc;
  }
  {
    const void* W[1] = {w->lm_head};
    const int rows[1] = {c.V};
    if ((rc = plan(&st->lm, st->xn, M, c.H, W, rows, 1, EPI_F32, out_logits ? out_logits : st->logits,
                   c.V)) != LSP_OK)
      return rc;
  }
  {
    AttnParams ap = {};
    ap.qkv = st->qkv; ap.win_k = st->win_k; ap.win_v = st->win_v; ap.G = st->G; ap.m = st->m;
    ap.C = c.C; ap.B = c.B; ap.L = c.L; ap.nq = c.nq; ap.nkv = c.nkv; ap.d = c.d; ap.W = c.W; ap.R = c.R;
    st->attn_tc.ok = 0;
    if (dt == LSP_DTYPE_BF16 && (rc = attn_tc_plan(&st->attn_tc, ap)) != LSP_OK && rc != LSP_ERR_SHAPE)
      return rc;
    // the tcgen05 attention reads the view state before its dependency wait:
    // the q/k/v projection before it triggers only after its own wait
    for (int j = 0; j < c.D; ++j) st->qkv_op[j].p.late_trigger = st->attn_tc.ok;
  }
  st->key.w = *w;
  st->key.out_logits = out_logits;
  st->have_plans = true;
  return LSP_OK;
}

static int run_sampler(lsp_state* st, const float* src, float* dst, const int32_t* prev,
                       int prev_stride, const void* Ec, const void* Wc, const lsp_sample_params* sp,
                       int32_t* out_tokens, cudaStream_t s) {
  const lsp_config& c = st->cfg;
  SampleParams p = {};
  p.src = src; p.dst = dst; p.prev = prev; p.prev_stride = prev_stride; p.Ec = Ec; p.Wc = Wc;
  p.out_tokens = out_tokens; p.part_val = st->part_val; p.part_idx = st->part_idx;
  p.sync = st->sample_sync; p.err = st->err;
  p.C = c.C; p.B = c.B; p.V = c.V; p.rc = c.rc; p.nblk = st->nblk; p.num_sms = st->num_sms;
  p.temperature = sp->temperature; p.round = sp->round; p.seed = sp->seed;
  return launch_sample(p, c.dtype, s);
}

int lsp_draft(lsp_state* st, const int32_t* block_tokens, const lsp_weights* w,
              const lsp_sample_params* sp, int32_t* out_tokens, float* out_logits,
              lsp_stream_t stream) {
  if (!st || !block_tokens || !w || !sp || !out_tokens) return LSP_ERR_ARG;
  if (!w->embed || !w->final_norm || !w->lm_head || !w->fuse || !w->pos || !w->mask_emb || !w->Ec ||
      !w->Wc)
    return LSP_ERR_ARG;
  if (!(sp->temperature >= 0.f) || !std::isfinite(sp->temperature)) return LSP_ERR_ARG;
  if (!st->initialized) return LSP_ERR_STATE;
  const lsp_config& c = st->cfg;
  cudaStream_t s = S(stream);
  int rc;
  if (!st->have_plans || std::memcmp(&st->key.w, w, sizeof(lsp_weights)) != 0 ||
      st->key.out_logits != out_logits) {
    if ((rc = build_plans(st, w, out_logits)) != LSP_OK) return rc;
  }
  const int M = c.C * c.B;
  int ev = 2;   // stage boundaries after view_update's [0, 1]
  // boundary state c_t = W_fuse [h^l1; ...; h^lL] (absent with LSP_NO_BOUNDARY)
  if (st->h && (rc = gemm_launch(&st->fuse, s)) != LSP_OK) return rc;
  mark(st, ev++, s);
  // input slots + first input norm + rotary table
  CombineParams cp;
  cp.tokens = block_tokens; cp.embed = w->embed; cp.pos = w->pos; cp.mask_emb = w->mask_emb;
  cp.c = st->h ? st->part : nullptr; cp.c_splits = st->h ? st->fuse.p.splits : 0; cp.norm_w = w->layer[0].in_norm; cp.x = st->x; cp.xn = st->xn; cp.rope = st->rope;
  cp.t = st->t; cp.err = st->err; cp.C = c.C; cp.B = c.B; cp.H = c.H; cp.V = c.V; cp.d = c.d;
  cp.eps = c.rms_eps; cp.theta = (double)c.rope_theta;
  if ((rc = launch_combine(cp, c.dtype, s)) != LSP_OK) return rc;
  mark(st, ev++, s);
  for (int j = 0; j < c.D; ++j) {
    const lsp_layer_weights& lw = w->layer[j];
    if ((rc = gemm_launch(&st->qkv_op[j], s)) != LSP_OK) return rc;
    const bool tc_attn = c.dtype == LSP_DTYPE_BF16 && st->attn_tc.ok;
    if (!tc_attn) {               // the tcgen05 attention finalises q/k/v itself
      QkvParams qp = {};
      qp.part = st->part; qp.splits = st->qkv_op[j].p.splits; qp.q_norm = lw.q_norm; qp.k_norm = lw.k_norm;
      qp.rope = st->rope; qp.out = st->qkv; qp.M = M; qp.B = c.B; qp.nq = c.nq; qp.nkv = c.nkv; qp.d = c.d;
      qp.eps = c.rms_eps;
      if ((rc = launch_qkv_finalize(qp, c.dtype, s)) != LSP_OK) return rc;
    }
    mark(st, ev++, s);
    AttnParams ap = {};
    ap.qkv = st->qkv;
    ap.win_k = st->win_k; ap.win_v = st->win_v; ap.G = st->G; ap.m = st->m; ap.t = st->t;
    ap.out = st->o; ap.C = c.C; ap.B = c.B; ap.L = c.L; ap.nq = c.nq; ap.nkv = c.nkv; ap.d = c.d;
    ap.W = c.W; ap.R = c.R; ap.layer = c.layer_map[j]; ap.eps = c.rms_eps; ap.err = st->err;
    ap.part = st->part; ap.splits = st->qkv_op[j].p.splits; ap.q_norm = lw.q_norm; ap.k_norm = lw.k_norm;
    ap.rope = st->rope;
    if ((rc = launch_attention(ap, c.dtype, s, &st->attn_tc)) != LSP_OK) return rc;
    mark(st, ev++, s);
    if ((rc = gemm_launch(&st->o_op[j], s)) != LSP_OK) return rc;
    mark(st, ev++, s);
    if ((rc = launch_resid_norm(st->x, st->part, st->o_op[j].p.splits, lw.post_norm, st->xn, M, c.H,
                                c.rms_eps, c.dtype, s)) != LSP_OK)
      return rc;
    mark(st, ev++, s);
    if ((rc = gemm_launch(&st->gu_op[j], s)) != LSP_OK) return rc;
    mark(st, ev++, s);
    if ((rc = gemm_launch(&st->down_op[j], s)) != LSP_OK) return rc;
    mark(st, ev++, s);
    const void* next_norm = j + 1 < c.D ? w->layer[j + 1].in_norm : w->final_norm;
    if ((rc = launch_resid_norm(st->x, st->part, st->down_op[j].p.splits, next_norm, st->xn, M, c.H,
                                c.rms_eps, c.dtype, s)) != LSP_OK)
      return rc;
    mark(st, ev++, s);
  }
  // frozen LM head: z^(0) = W_lm RMSNorm_final(x)
  if ((rc = gemm_launch(&st->lm, s)) != LSP_OK) return rc;
  mark(st, ev++, s);
  float* z0 = out_logits ? out_logits : st->logits;
  rc = run_sampler(st, z0, out_logits, block_tokens, c.B, w->Ec, w->Wc, sp, out_tokens, s);
  mark(st, ev++, s);
  return rc;
}

int lsp_sample(lsp_state* st, const float* base_logits, const int32_t* prev_token, const void* Ec,
               const void* Wc, const lsp_sample_params* sp, int32_t* out_tokens, float* out_logits,
               lsp_stream_t stream) {
  if (!st || !base_logits || !prev_token || !Ec || !Wc || !sp || !out_tokens) return LSP_ERR_ARG;
  if (!(sp->temperature >= 0.f) || !std::isfinite(sp->temperature)) return LSP_ERR_ARG;
  return run_sampler(st, base_logits, out_logits, prev_token, 1, Ec, Wc, sp, out_tokens, S(stream));
}

int lsp_gemm_plan_info(int dtype, int M, int N, int K, int swiglu, int num_sms, int* splits,
                       int* tok_groups, int* tokens_per_group) {
  if (!splits || !tok_groups || !tokens_per_group || M < 1 || M > 512 || N < 1 || K < 1 || num_sms < 1)
    return LSP_ERR_ARG;
  if (dtype != LSP_DTYPE_BF16 && dtype != LSP_DTYPE_F32) return LSP_ERR_ARG;
  const int mode = swiglu ? EPI_SWIGLU : EPI_PARTIAL;
  const int rows[1] = {N};
  int s = 0, g = 1;
  gemm_choose(dtype, M, K, gemm_tiles(mode, rows, 1), mode, num_sms, &s, &g);
  *splits = s;
  *tok_groups = g;
  *tokens_per_group = gemm_group_rows(M, g);
  return LSP_OK;
}

size_t lsp_linear_workspace_bytes(int M, int N, int splits) {
  if (M < 1 || N < 1 || splits < 1) return 0;
  return splits == 1 ? 0 : (size_t)splits * M * N * sizeof(float);
}

int lsp_linear(const void* X, const void* W, float* Y, int M, int N, int K, int dtype, int splits,
               void* workspace, size_t workspace_bytes, lsp_stream_t stream) {
  if (!X || !W || !Y || M < 1 || N < 1 || K < 1 || splits < 1 || splits > 16) return LSP_ERR_ARG;
  if (dtype != LSP_DTYPE_BF16 && dtype != LSP_DTYPE_F32) return LSP_ERR_ARG;
  const int rows[1] = {N};
  if (splits > 1 && (!workspace || workspace_bytes < lsp_linear_workspace_bytes(M, N, splits)))
    return LSP_ERR_ARG;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return LSP_ERR_CUDA;
  GemmOp op;
  const void* Ws[1] = {W};
  float* part = static_cast<float*>(workspace);
  // one split writes Y directly; more write fp32 partials that a second kernel sums
  const bool direct = splits == 1;
  int rc = gemm_plan(&op, dtype, X, M, K, Ws, rows, 1, direct ? EPI_F32 : EPI_PARTIAL, direct ? Y : part, N,
                     nullptr, sms, splits);
  if (rc != LSP_OK) return rc;
  if (op.p.splits != splits) return LSP_ERR_SHAPE;
  if ((rc = gemm_launch(&op, S(stream))) != LSP_OK || direct) return rc;
  return launch_sum_partials(part, splits, (size_t)M * N, Y, S(stream));
}

int lsp_philox_words(uint64_t seed, uint32_t round, uint32_t b, uint32_t i, uint32_t* out,
                     int count, lsp_stream_t stream) {
  if (!out || count < 0) return LSP_ERR_ARG;
  return launch_philox_words(seed, round, b, i, out, count, S(stream));
}

int lsp_stage_count(lsp_state* st) { return st ? stage_total(st->cfg) : 0; }

int lsp_round_launches(lsp_state* st) {
  if (!st) return 0;
  const lsp_config& c = st->cfg;
  SampleParams p = {};
  p.C = c.C; p.B = c.B; p.V = c.V; p.rc = c.rc; p.num_sms = st->num_sms; p.sync = st->sample_sync;
  // view update, fuse, combine; per layer q/k/v GEMM, finalize (not with the
  // tcgen05 attention, which finalises q/k/v itself), attention, o, norm,
  // gate/up, down, norm; LM head; the sampler
  const int fuse = (c.flags & LSP_NO_BOUNDARY) ? 0 : 1;
  const int fin = (c.dtype == LSP_DTYPE_BF16 && attn_tc_supported(c.B, c.W, c.R, c.nq, c.nkv, c.d)) ? 0 : 1;
  return 2 + fuse + (7 + fin) * c.D + 1 + sample_launches(p, c.dtype);
}

const char* lsp_stage_name(lsp_state* st, int k) {
  if (!st || k < 0 || k >= stage_total(st->cfg)) return nullptr;
  if (k == 0) return "view_update";
  if (k == 1) return "fuse";
  if (k == 2) return "combine";
  const int n = stage_total(st->cfg);
  if (k == n - 2) return "lm_head";
  if (k == n - 1) return "sampler";
  return kLayerStages[(k - 3) % 7];
}

int lsp_set_stage_events(lsp_state* st, void* const* events, int n_events) {
  if (!st) return LSP_ERR_ARG;
  if (n_events == 0) { st->n_stage_ev = 0; return LSP_OK; }
  if (!events || n_events != stage_total(st->cfg) + 1) return LSP_ERR_ARG;
  for (int i = 0; i < n_events; ++i) {
    if (!events[i]) return LSP_ERR_ARG;
    st->stage_ev[i] = static_cast<cudaEvent_t>(events[i]);
  }
  st->n_stage_ev = n_events;
  return LSP_OK;
}

int lsp_get_error(lsp_state* st, uint32_t* dev_error, int clear, lsp_stream_t stream) {
  if (!st || !dev_error) return LSP_ERR_ARG;
  cudaStream_t s = S(stream);
  unsigned v = 0;
  if (cudaMemcpyAsync(&v, st->err, sizeof(unsigned), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return LSP_ERR_CUDA;
  if (clear && v && cudaMemsetAsync(st->err, 0, sizeof(unsigned), s) != cudaSuccess) return LSP_ERR_CUDA;
  // a sampler launch that gave up waiting leaves its step counters behind
  if (clear && (v & LSP_DEV_TIMEOUT) &&
      cudaMemsetAsync(st->sample_sync, 0, st->sample_sync_bytes, s) != cudaSuccess)
    return LSP_ERR_CUDA;
  *dev_error = v;
  if (v & LSP_DEV_TIMEOUT) return LSP_ERR_TIMEOUT;
  return v ? LSP_ERR_STATE : LSP_OK;
}

static int copy_interface(lsp_state* st, void* host, size_t bytes, bool to_host, cudaStream_t s) {
  const lsp_config& c = st->cfg;
  const Layout l = interface_layout(c);
  if (bytes != lsp_state_bytes(&c)) return LSP_ERR_ARG;
  char* hp = static_cast<char*>(host);
  void* dev[6] = {st->win_k, st->win_v, st->m, st->eta, st->h, st->t};
  const size_t sz[6] = {l.win, l.win, l.m, l.eta, l.h, l.t};
  for (int i = 0; i < 6; ++i) {
    if (sz[i] == 0) continue;
    cudaError_t e = to_host ? cudaMemcpyAsync(hp, dev[i], sz[i], cudaMemcpyDeviceToHost, s)
                            : cudaMemcpyAsync(dev[i], hp, sz[i], cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return LSP_ERR_CUDA;
    hp += sz[i];
  }
  return cudaStreamSynchronize(s) == cudaSuccess ? LSP_OK : LSP_ERR_CUDA;
}

int lsp_state_export(lsp_state* st, void* host_buf, size_t bytes, lsp_stream_t stream) {
  if (!st || !host_buf) return LSP_ERR_ARG;
  return copy_interface(st, host_buf, bytes, true, S(stream));
}

int lsp_state_import(lsp_state* st, const void* host_buf, size_t bytes, lsp_stream_t stream) {
  if (!st || !host_buf) return LSP_ERR_ARG;
  if (!st->initialized) return LSP_ERR_STATE;   // G comes from lsp_state_init
  return copy_interface(st, const_cast<void*>(host_buf), bytes, false, S(stream));
}

}  // extern "C"
