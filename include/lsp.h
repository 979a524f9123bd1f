/*
 * lsp.h -- C ABI of the fixed-cost drafting round (LongSpark, arxiv 2609.37029).
 *
 * One drafting round (Sec. 2.4 "Inference", Fig. 2):
 *   1. lsp_view_update: fold the target verification pass's newly accepted rows
 *      into the fixed-size context interface -- the global summary (Eq.
 *      global-summary maintained by the merge of App. A.2, Eq. summary-update),
 *      the recent KV window and the boundary hidden states (Sec. 2.2).
 *   2. lsp_draft: the block-diffusion drafter forward over [block; window;
 *      summary] (Sec. 2.3, Eq. draft-context, App. A.1), the frozen final norm
 *      and LM head (base logits z^(0)), then lsp_sample's correction+sampling.
 *   3. lsp_sample: the low-rank Markov correction (Eq. markov) and sequential
 *      sampling of the B proposals (Eq. proposal-factorization).
 *
 * Conventions shared by every call:
 *   - Every call returns an int status: LSP_OK (0) or a negative LSP_ERR_*.
 *     Argument and shape errors are detected on the host before any launch and
 *     nothing is enqueued then.  No exception or abort crosses the ABI.
 *   - All device work is enqueued on the caller's stream (lsp_stream_t is a
 *     cudaStream_t; NULL means the legacy default stream) and returns without
 *     synchronising, except where a call says otherwise.
 *   - Pointers documented as "device" must be device (or managed) memory owned
 *     by the caller, valid until the enqueued work completes.  The library owns
 *     only what lsp_state_create allocates.
 *   - Element type of every tensor argument documented as "dtype" is the
 *     config's dtype: LSP_DTYPE_BF16 (bfloat16) or LSP_DTYPE_F32 (float).
 *   - Errors a kernel detects (a token id out of range, accepted_len beyond the
 *     row capacity, a bounded wait that timed out) set bits of a device error
 *     word (LSP_DEV_*) read by lsp_get_error; kernels never trap.
 *   - Layouts are dense and row-major; linear weights are [out][in] with `in`
 *     contiguous (y = W x).
 *   - Concurrency: the device work of one state (its interface, workspace and
 *     synchronisation words) must be ordered -- one stream, or streams the
 *     caller synchronises; calls on different states, and lsp_linear calls
 *     with different workspaces, may overlap from any threads and streams.
 *     The one process-wide buffer is lsp_sample_noalloc's scratch (below).
 *   - No environment variable changes what the library computes or how.
 */
#ifndef LSP_H
#define LSP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define LSP_MAX_DRAFT_LAYERS 16

/* status codes */
#define LSP_OK 0
#define LSP_ERR_ARG (-1)          /* null pointer / invalid scalar argument */
#define LSP_ERR_SHAPE (-2)        /* config or size outside what the kernels support */
#define LSP_ERR_CUDA (-3)         /* a CUDA runtime or driver call failed */
#define LSP_ERR_TIMEOUT (-4)      /* a device wait gave up (see lsp_get_error) */
#define LSP_ERR_STATE (-5)        /* state not initialised or device error pending */
#define LSP_ERR_NOMEM (-6)        /* device allocation failed in lsp_state_create */
#define LSP_ERR_UNSUPPORTED (-7)  /* no sm_103a device / feature unavailable */

/* device error word bits (lsp_get_error) */
#define LSP_DEV_TIMEOUT 1u        /* a bounded mbarrier/flag wait expired */
#define LSP_DEV_BAD_TOKEN 2u      /* a token id outside [-1, V) (slot 0: outside [0, V)) */
#define LSP_DEV_BAD_DELTA 4u      /* accepted_len outside [0, row capacity] */

#define LSP_DTYPE_BF16 0
#define LSP_DTYPE_F32 1

/* lsp_config.flags.  LSP_NO_BOUNDARY: the "w/o boundary state" variant of the
 * ablation (Sec. 3.4, Fig. 5): the state keeps no boundary hidden state, the
 * boundary fusion is not run and the input slots are E[u_i] + P_i alone.  The
 * other two variants are shapes: w/o global summary is R = 0, w/o recent KV
 * window is W = 0. */
#define LSP_NO_BOUNDARY 1u

typedef void* lsp_stream_t;       /* cudaStream_t */
typedef struct lsp_state lsp_state; /* opaque, library-owned */

/*
 * Shapes of one drafter + target pairing.
 *   C   concurrency: requests processed together (state rows)
 *   B   draft block slots = proposals per round (Sec. 2.3)
 *   L   tapped target layers (the set of Sec. 2.2; App. B.1 uses 5)
 *   D   drafter layers (App. B.1: 5)
 *   H   hidden size; nq / nkv query / key-value heads of head dim d (the
 *       target's, since draft queries score target window keys)
 *   F   drafter MLP width; V vocabulary; rc rank of the Markov correction
 *   W   recent window rows per tapped layer (App. B.1: 256)
 *   R   summary queries per tapped layer and query head (App. B.1: 16)
 *   layer_map[j]  tapped-layer index draft layer j reads its window and summary
 *       from (Sec. 2.3 pairs draft layer j with tapped layer l(j)); a value < 0
 *       selects floor(j * L / D)
 *   rope_theta  rotary base of the drafter's block queries/keys; rms_eps RMSNorm eps
 *   flags  0 or LSP_NO_BOUNDARY
 * Supported: dtype BF16 with d == 128, B <= 16, nq % nkv == 0, nq/nkv <= 8;
 * dtype F32 with d <= 128 even; H, nq*d, nkv*d, F multiples of 64; C*B <= 512;
 * W >= 0 and R >= 0 (0 removes the window / the summary from the context).
 */
typedef struct lsp_config {
  int C, B, L, D, H, nq, nkv, d, F, V, W, R, rc;
  int dtype;
  int layer_map[LSP_MAX_DRAFT_LAYERS];
  float rope_theta;
  float rms_eps;
  unsigned flags;
} lsp_config;

/*
 * New target rows of one verification pass (Sec. 2.1, 2.4): for request b,
 * tapped layer l and new row j < accepted_len[b]:
 *   k[b][l][j][0..nkv)[0..d)   key rows as cached by the target (rotary applied)
 *   v[b][l][j][0..nkv)[0..d)   value rows
 *   h[b][l][j][0..H)           hidden state at that row (only row accepted_len-1 is read)
 * All three are device pointers of dtype with row capacity `rows` per (b, l);
 * h may be null (and is not read) with LSP_NO_BOUNDARY.
 * h_rows: rows of h per (b, l).  0 (the default when the struct is zeroed) or
 * `rows`: the layout above.  1: h[b][l][0..H) holds only the boundary row --
 * the hidden state at row accepted_len[b]-1 (for lsp_prefill: at row t-1) --
 * which is all the interface reads (Sec. 2.2), so a caller that stages the
 * rows from host memory copies C*L*H elements instead of C*L*rows*H.  Any
 * other value is LSP_ERR_ARG.
 */
typedef struct lsp_target_feats {
  const void* k;
  const void* v;
  const void* h;
  int rows;
  int h_rows;
} lsp_target_feats;

/* One Qwen3-style draft layer (App. B.1); device pointers of dtype. */
typedef struct lsp_layer_weights {
  const void* in_norm;    /* [H] */
  const void* wq;         /* [nq*d][H] */
  const void* wk;         /* [nkv*d][H] */
  const void* wv;         /* [nkv*d][H] */
  const void* q_norm;     /* [d] per-head RMSNorm of block queries */
  const void* k_norm;     /* [d] per-head RMSNorm of block keys */
  const void* wo;         /* [H][nq*d] */
  const void* post_norm;  /* [H] */
  const void* w_gate;     /* [F][H] */
  const void* w_up;       /* [F][H] */
  const void* w_down;     /* [H][F] */
} lsp_layer_weights;

/* Drafter weights (device pointers of dtype). The target's embedding, final
 * norm and LM head are reused frozen (Sec. 2.3, App. B.1). */
typedef struct lsp_weights {
  const void* embed;       /* [V][H] target token embedding */
  const void* final_norm;  /* [H] target final RMSNorm weight */
  const void* lm_head;     /* [V][H] target vocabulary head */
  const void* fuse;        /* [H][L*H] boundary fusion: c_t = fuse . [h^l1;...;h^lL] (Sec. 2.2);
                              may be null with LSP_NO_BOUNDARY */
  const void* pos;         /* [B][H] within-block positional encodings (Sec. 2.3) */
  const void* mask_emb;    /* [H] mask-token embedding of slots 1..B-1 */
  const void* Ec;          /* [V][rc] correction embedding E_c (Eq. markov) */
  const void* Wc;          /* [V][rc] correction output map W_c (Eq. markov) */
  lsp_layer_weights layer[LSP_MAX_DRAFT_LAYERS];
} lsp_weights;

/*
 * Sampling of the proposals (Eq. proposal-factorization).  temperature == 0:
 * greedy, y_i = argmax_v z_i[v].  temperature > 0: Gumbel-max,
 * y_i = argmax_v (z_i[v] / T + g) (z / T taken in fp32 as z * fl(1/T), exact at T = 1),
 * g = -log(-log u), u = ((x >> 9) + 0.5) * 2^-23,
 * x = word (v & 3) of Philox4x32-10 with key (seed lo32, seed hi32) and counter
 * (v >> 2, i, b, round).  Ties go to the lowest vocabulary index.
 */
typedef struct lsp_sample_params {
  float temperature;
  uint32_t round;
  uint64_t seed;
} lsp_sample_params;

/* Human-readable name of a status code (static string). */
const char* lsp_status_string(int status);

/* Bytes of the persistent per-state interface for `cfg` (window, summary
 * (m, eta), boundary h, counters), all C requests: a function of the shapes
 * only, never of the prefix length (Sec. 2.4 "Fixed-cost complexity").
 * Returns 0 for an invalid config. Host-only; needs no GPU. */
size_t lsp_state_bytes(const lsp_config* cfg);

/* Validate `cfg` on the host. LSP_OK or LSP_ERR_SHAPE / LSP_ERR_ARG. Needs no GPU. */
int lsp_config_check(const lsp_config* cfg);

/* Allocate a state on the current device: the interface (lsp_state_bytes) and
 * a fixed workspace for the drafter's activations, logits and sampler
 * partials.  Synchronous; the only call that allocates device memory.  The
 * state starts uninitialised (call lsp_state_init). */
int lsp_state_create(const lsp_config* cfg, lsp_state** out);

/* Free everything lsp_state_create allocated (synchronises the device first).
 * NULL is ignored. */
void lsp_state_destroy(lsp_state* st);

/* Reset the interface to the empty prefix -- m = 0, eta = -inf, empty window,
 * zero boundary, t = 0, device error word cleared -- and copy the summary
 * queries G (device, dtype, [L][nq][R][d]; Sec. 2.2, App. B.2 "Summary
 * queries", held fixed during inference) into the state.  The summary over a
 * prefix is then built by lsp_view_update calls over its rows in chunks of any
 * size (the merge of App. A.2 makes the chunking exact); this is the one-time
 * O(t) prefill the paper attributes to target prefill (Fig. 3). */
int lsp_state_init(lsp_state* st, const void* G, lsp_stream_t stream);

/* Fold accepted_len[b] new target rows of request b (device int32 [C], each in
 * [0, feats->rows]; 0 leaves request b untouched) into the interface:
 *  - summary: for every tapped layer l, query head h and summary query r,
 *    the attention statistics of g_r over the new keys of KV head h/(nq/nkv)
 *    are merged into (eta, m) by Eq. summary-update;
 *  - window: the new K/V rows enter the ring of the last W rows (row p of the
 *    prefix lives in slot p mod W);
 *  - boundary: h of the last new row replaces the boundary state;
 *  - t += accepted_len[b].
 * Reads only the new rows, never the prefix (Sec. 2.4). */
int lsp_view_update(lsp_state* st, const lsp_target_feats* feats,
                    const int32_t* accepted_len, lsp_stream_t stream);

/* One drafter forward for all C requests (Sec. 2.3, App. A.1) followed by the
 * sampler of lsp_sample.
 *   block_tokens  device int32 [C][B]: slot 0 = committed token a (also y_0 of
 *                 the Markov correction); slots >= 1: -1 for the mask embedding
 *                 or a token id to embed
 *   w             weights (host struct of device pointers)
 *   sp            sampling parameters (host struct)
 *   out_tokens    device int32 [C][B]: proposals y_1..y_B
 *   out_logits    device float [C][B][V] corrected logits z_i (the verification
 *                 distributions q_i = softmax(z_i)), or NULL to skip writing them
 * Rotary positions of slot i are t + i (t = rows folded so far).  Uses only
 * the state's fixed workspace; allocates nothing. */
int lsp_draft(lsp_state* st, const int32_t* block_tokens, const lsp_weights* w,
              const lsp_sample_params* sp, int32_t* out_tokens, float* out_logits,
              lsp_stream_t stream);

/* Correction + sampling alone (Eq. markov, Eq. proposal-factorization) on given
 * base logits, with the state's config (C, B, V, rc, dtype) and workspace:
 *   base_logits  device float [C][B][V] (z^(0); not modified)
 *   prev_token   device int32 [C]: y_0 = a of each request
 *   Ec, Wc       device dtype [V][rc]
 *   out_tokens   device int32 [C][B]; out_logits device float [C][B][V] or NULL
 * For i = 1..B in order: z_i = z_i^(0) + W_c E_c[y_{i-1}], y_i drawn per sp. */
int lsp_sample(lsp_state* st, const float* base_logits, const int32_t* prev_token,
               const void* Ec, const void* Wc, const lsp_sample_params* sp,
               int32_t* out_tokens, float* out_logits, lsp_stream_t stream);

/* Correction + sampling without a state and without any device allocation,
 * for callers that cannot allocate device memory where they sample (a loop
 * running under another framework's caching allocator that already reserved
 * the device, or code that must not create an lsp_state).  The paper has no
 * counterpart: this is a deployment variant of lsp_sample.
 *   Same computation and tensor arguments as lsp_sample; the shapes are passed
 *   explicitly (1 <= C <= 64, B >= 1, V and rc multiples of 16, rc <= 256) and
 *   dtype is LSP_DTYPE_BF16 or LSP_DTYPE_F32 for Ec / Wc.
 *   dev_error: optional device uint32 that receives LSP_DEV_* bits (OR-ed in;
 *   NULL skips error reporting).
 * Scratch: a fixed 512 KiB __device__ array inside the library, held by every
 * GPU that loads it until the process exits.  A call needs
 *   align256(16 * nblk * C) + align256(2048 * B + 4 * B) bytes of it,
 * with nblk = min(2 * SMs, 512) and align256(x) = x rounded up to 256, and
 * returns LSP_ERR_SHAPE beyond 512 KiB (on 152 SMs: C = 16 fits B <= 217,
 * C = 64 fits B <= 103).  The first successful call on a device looks up the
 * array's device address and the SM count (a failed lookup is retried by the
 * next call); make that first call before any stream capture on the device.
 * Every call shares the array: calls that overlap on the GPU (other streams
 * or threads) race, so the caller must serialise them.  The step counters are
 * cleared on the caller's stream before each launch.  Allocates nothing and
 * calls no allocating CUDA or library routine. */
int lsp_sample_noalloc(const float* base_logits, const int32_t* prev_token, const void* Ec,
                       const void* Wc, int dtype, int C, int B, int V, int rc,
                       const lsp_sample_params* sp, int32_t* out_tokens, float* out_logits,
                       uint32_t* dev_error, lsp_stream_t stream);

/* Prefill (Sec. 2.2, Eq. global-summary, App. A.2; Fig. 3: the summary is
 * initialised over the full prefix during target prefill): replace request
 * b's interface by the one its whole prefix of t = f->rows rows defines --
 * summary (eta, m) = attention of the R summary queries of every tapped layer
 * and query head over all t rows, window ring = the last min(t, W) rows
 * (prefix row p in slot p mod W), boundary = hidden state of row t-1, and t.
 *   f->k, f->v: device dtype [L][t][nkv][d] (request b only); f->h: device
 *   dtype [L][t][H]; borrowed for the call's duration on `stream`.
 * Equivalent to folding the t rows into an empty request with
 * lsp_view_update, but split over the whole GPU (segments of the prefix
 * merged in order with Eq. summary-update; deterministic).  Needs an
 * initialised state (G); bf16 storage with d = 128, 0 <= R <= 16, nq/nkv <= 8 (else
 * LSP_ERR_UNSUPPORTED: use lsp_view_update).  Other requests are untouched. */
int lsp_prefill(lsp_state* st, int b, const lsp_target_feats* f, lsp_stream_t stream);

/* Target-side verification of the drafted blocks (Sec. 2.1, Eq. acceptance,
 * Eq. residual): for each request the candidates y_1..y_B are tested in order,
 * y_i accepted with probability min(1, p_i(y_i) / q_i(y_i)); at the first
 * rejected position i a correction token is drawn from [p_i - q_i]_+; if all B
 * are accepted a bonus token is drawn from p_{B+1}.  p_i = softmax(target
 * logits_i / T), q_i = softmax(draft logits_i / T); T = 0 is greedy (accept
 * y_i iff y_i = argmax p_i, emit argmax p_{r+1}; ties to the lowest index).
 *   target_logits: device float [C][B+1][V] (position B: p(. | s, y_1..y_B));
 *   draft_logits: device float [C][B][V] (lsp_draft's out_logits);
 *   draft_tokens: device int32 [C][B] (lsp_draft's out_tokens);
 *   sp: the round's sampling parameters (the ones lsp_draft used);
 *   accepted_len: device int32 [C] = r in [0, B]; next_token: device int32 [C].
 *   16-byte aligned logits.  The round then advances each request by r + 1
 *   tokens (the next round's accepted_len is r + 1 and its committed token is
 *   next_token).
 * Randomness: Philox4x32-10 with key `seed`; acceptance uniform of position i =
 * word 0 of counter (0, 2^30 + i, b, round), u = ((x >> 9) + 1/2) 2^-23,
 * accepted iff u q_i(y_i) < p_i(y_i); the draw at position i is Gumbel-max with
 * the words of counters (v >> 2, 2^31 + i, b, round).  Drafted tokens outside
 * [0, V) set LSP_DEV_BAD_TOKEN.  Asynchronous on `stream`. */
int lsp_verify(lsp_state* st, const float* target_logits, const float* draft_logits,
               const int32_t* draft_tokens, const lsp_sample_params* sp, int32_t* accepted_len,
               int32_t* next_token, lsp_stream_t stream);

/* Dense projection Y = X W^T with the drafter's tensor-core GEMM (the kernel
 * every projection of lsp_draft uses), for checking it on its own.
 *   X device dtype [M][K]; W device dtype [N][K]; Y device float [M][N].
 *   M <= 512; K * element size a multiple of 16 bytes.
 *   splits: split-K factor (1..16, at most the number of K blocks).  With
 *   splits > 1 the kernel writes fp32 partial sums to `workspace` (device, at
 *   least lsp_linear_workspace_bytes(M, N, splits) bytes) and a second kernel
 *   sums them in split order into Y; with splits == 1 Y is written directly
 *   and `workspace` may be NULL. */
size_t lsp_linear_workspace_bytes(int M, int N, int splits);

/* Diagnostic, host only (needs no GPU): the launch plan the drafter's
 * projection GEMM takes for M token rows, N output features and reduction
 * length K on a device with num_sms SMs.
 *   swiglu = 0: a projection whose fp32 split-K partials a consumer sums
 *   (the q/k/v, o, down and boundary-fusion projections); swiglu = 1: the
 *   fused gate/up projection with N = F (gate and up each [F][K]).
 *   *splits: split-K factor; *tok_groups: CTAs per weight tile, each over
 *   *tokens_per_group consecutive token rows (a multiple of 16).
 * LSP_ERR_ARG for null outputs, M outside [1, 512], N, K or num_sms < 1 or
 * an unknown dtype. */
int lsp_gemm_plan_info(int dtype, int M, int N, int K, int swiglu, int num_sms, int* splits,
                       int* tok_groups, int* tokens_per_group);
int lsp_linear(const void* X, const void* W, float* Y, int M, int N, int K, int dtype,
               int splits, void* workspace, size_t workspace_bytes, lsp_stream_t stream);

/* Raw Philox4x32-10 words of the sampler stream, for checking the generator:
 * out[n] (device uint32) = word (v & 3) of block (v >> 2) with v = n, counter
 * (v >> 2, i, b, round) and key (seed lo32, seed hi32); n < count. */
int lsp_philox_words(uint64_t seed, uint32_t round, uint32_t b, uint32_t i,
                     uint32_t* out, int count, lsp_stream_t stream);

/* Stage timing hook (observability; no effect on results).  With n_events > 0,
 * lsp_view_update and lsp_draft record the caller's CUDA events (cudaEvent_t
 * handles, created by the caller with timing enabled, owned by the caller) at
 * stage boundaries on the call's stream: stage k runs between events[k] and
 * events[k+1].  Stages of one round, in order (lsp_stage_count / lsp_stage_name):
 *   0 view_update, 1 fuse, 2 combine, then per draft layer j: qkv, attention,
 *   o_proj, post_norm, gate_up, down, next_norm, then lm_head and sampler
 *   (with LSP_NO_BOUNDARY the fuse stage is empty).
 * n_events must be 0 (off) or lsp_stage_count(st) + 1.  Event records are
 * capturable, so a captured round carries them as graph nodes. */
int lsp_stage_count(lsp_state* st);
/* Number of kernel launches one round (lsp_view_update + lsp_draft) issues
 * for this state's config on the current device (the sampler is one launch
 * or B + 1 depending on the shape); 0 for a null state. */
int lsp_round_launches(lsp_state* st);
const char* lsp_stage_name(lsp_state* st, int k);
int lsp_set_stage_events(lsp_state* st, void* const* events, int n_events);

/* Read (and clear, if clear != 0) the state's device error word into
 * *dev_error (LSP_DEV_* bits).  Synchronises `stream`.  Returns LSP_OK,
 * or LSP_ERR_TIMEOUT / LSP_ERR_STATE when bits are set. */
int lsp_get_error(lsp_state* st, uint32_t* dev_error, int clear, lsp_stream_t stream);

/* Copy the interface (exactly lsp_state_bytes(cfg) bytes, including t) to /
 * from a host buffer, so a state can be checkpointed or built elsewhere.
 * Synchronous on `stream`. Layout (all per state, dense, in this order):
 *   win_k dtype [C][L][nkv][W][d], win_v dtype [C][L][nkv][W][d],
 *   m float [C][L][nq][R][d], eta float [C][L][nq][R], h dtype [C][L][H],
 *   t int64 [C]. */
int lsp_state_export(lsp_state* st, void* host_buf, size_t bytes, lsp_stream_t stream);
int lsp_state_import(lsp_state* st, const void* host_buf, size_t bytes, lsp_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* LSP_H */
