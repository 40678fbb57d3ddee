/*
 * dkv.h -- C ABI of the GB300 DensityKV bank library (libdkv.so).
 *
 * One handle (dkv_bank_t) holds the H per-head historical KV banks of one
 * Transformer layer (Eq. 4).  Four calls make up the hot path:
 *
 *   dkv_bank_admit     Steps 1-2 of the online update (Sec. 3.4; Alg. 1, App. C):
 *                      mean-normalised candidate scores (Eq. 6 / C.1), stable sort,
 *                      projected density growth for every prefix length
 *                      (Eqs. 8-9 / C.2-C.3), eviction budgets (Eq. 10) and the
 *                      largest prefix feasible for every head, r* (Eq. 11).
 *                      No state visible through the bank buffers changes.
 *   dkv_bank_compress  Step 3 (Sec. 3.4; Alg. 1): mandatory-then-densest eviction,
 *                      commit (Eq. 12), exact maintenance of the cached densities
 *                      (Eq. C.4) and frozen insertion baselines of the admitted
 *                      states (Eq. 5).  An empty bank admits the first min(N, M_h)
 *                      candidates in source order (Alg. 1, m = 0 branch).
 *   dkv_bank_attend    Softmax attention of the current block's queries over
 *                      [retained bank | local window], logits q.k / sqrt(d_k)
 *                      (Sec. 3.2; App. A Eq. "supp-logit"; Fig. 2 caption).
 *   dkv_bank_create    Binds caller-owned device buffers to a handle.
 *
 * Conventions
 *   - Every pointer named "device" is a CUDA device pointer on the current
 *     device; "host" pointers are ordinary host memory.  No torch types.
 *   - All tensors are dense, row-major, with the innermost dimension d.
 *     Keys/values/queries are bf16 (DKV_DTYPE_BF16) or fp32 (DKV_DTYPE_FP32),
 *     as fixed at create time.  d_k = d_v = d, d in {64, 128}.
 *   - Bank buffers and the workspace are OWNED BY THE CALLER and borrowed for
 *     the lifetime of the handle.  The library never allocates device memory
 *     on the hot path; dkv_bank_create allocates only host bookkeeping and
 *     CUDA events.
 *   - Work is enqueued on the given stream (cudaStream_t passed as void*,
 *     NULL = legacy default stream) and returns without synchronising.
 *     Occupancy, r* and every intermediate live on the device; no call on the
 *     hot path reads them back, so a whole update can be captured in a graph.
 *   - Argument and state errors are reported synchronously by the return
 *     value and enqueue nothing.  Device-side failures (a bounded wait that
 *     timed out, an inconsistent bank) set a sticky device error word that
 *     dkv_bank_sync() reports; CUDA launch errors are returned as
 *     DKV_ERR_CUDA by the call that saw them.
 *   - Calls on one handle must be ordered on one stream (or by the caller's
 *     own events).  admit must be followed by compress before the next admit
 *     (else DKV_ERR_STATE).  attend between admit and compress reads the
 *     pre-update bank: the update is atomic from the reader's point of view
 *     (App. C, "Decision granularity versus computational tiling").
 *   - The candidate buffers passed to admit must stay valid and unmodified
 *     until the compress that follows has completed on the stream.
 */
#ifndef DKV_H_
#define DKV_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct dkv_bank_s* dkv_bank_t;

typedef enum {
  DKV_OK = 0,
  DKV_ERR_ARG = 1,          /* null pointer, bad enum, bad parameter value               */
  DKV_ERR_SHAPE = 2,        /* size outside what the handle / library supports           */
  DKV_ERR_STATE = 3,        /* call out of order (admit twice, compress without admit)   */
  DKV_ERR_CUDA = 4,         /* a CUDA runtime call or launch failed                      */
  DKV_ERR_NOMEM = 5,        /* workspace smaller than dkv_bank_workspace_size_ex()       */
  DKV_ERR_TIMEOUT = 6,      /* a bounded device-side wait gave up (sticky, see sync)     */
  DKV_ERR_UNSUPPORTED = 7,  /* feature not available for this dtype / d / device         */
  DKV_ERR_DEVICE = 8        /* device-side consistency check failed (sticky, see sync)   */
} dkv_status_t;

typedef enum { DKV_DTYPE_BF16 = 0, DKV_DTYPE_FP32 = 1 } dkv_dtype_t;

/* How candidate/bank interactions are computed.
 * DKV_SCORE_TENSOR: tcgen05 bf16 tensor-core contraction (bf16 banks only),
 *                   fp32 accumulation and fp32 epilogue.
 * DKV_SCORE_FP32:   direct fp32 sum of squared differences on the CUDA cores
 *                   (the exactness mode; required for fp32 banks).           */
typedef enum { DKV_SCORE_TENSOR = 0, DKV_SCORE_FP32 = 1 } dkv_score_mode_t;

/* Update policy (Table 2(b) and App. E "Policy ablations"; the defaults are the
 * paper's method).  Candidate order: ascending Eq. 6 score (default) or source
 * order of the block (pi = identity; no score pass).  Eviction (Sec. 3.4 Step 3):
 * threshold crossers first, then decreasing rho~(r*) (default); only decreasing
 * rho~(r*) ("densest-only"); or threshold crossers first, then source order of the
 * bank, read as provenance order, oldest (step, src) first.  In every policy r* is
 * the largest prefix feasible under Eqs. 9-11 for the candidates in that order.    */
typedef enum { DKV_ORDER_SCORE = 0, DKV_ORDER_SOURCE = 1 } dkv_order_t;
typedef enum {
  DKV_EVICT_MANDATORY_DENSEST = 0,
  DKV_EVICT_DENSEST = 1,
  DKV_EVICT_MANDATORY_SOURCE = 2
} dkv_evict_t;

/* Retention descriptor (App. E "Retention geometry").  DKV_DESC_K: the post-RoPE key
 * (Sec. 3, default).  DKV_DESC_KV: the concatenation [k; v] of key and value, so every
 * interaction of Eqs. 2-12 uses ||k - k'||^2 + ||v - v'||^2 and, when sigma <= 0,
 * sigma = sqrt(2d / 2) = sqrt(d) (App. B's rule for the descriptor dimension 2d).
 * Attention still reads the keys and values as they are.                          */
typedef enum { DKV_DESC_K = 0, DKV_DESC_KV = 1 } dkv_descriptor_t;

/* Method parameters.  Defaults (dkv_params_default): tau = 2, sigma = sqrt(d/2),
 * p = 2, eps = 1, delta = 1e-6, shared cross-head prefix (Sec. 4.1; App. B
 * "Parameterization"; App. D "Default DensityKV configuration").           */
typedef struct {
  float tau;            /* allowed density-growth factor, tau > 1 (Eq. 9)             */
  float sigma;          /* bandwidth (Eq. 2); <= 0 selects sqrt(d/2) (App. B)         */
  float p;              /* decay exponent, p in {1, 2, 4} (Eq. 2; Table 2a range)      */
  float eps;            /* regulariser, eps > 0 (Eq. 2)                                */
  float delta;          /* baseline floor, delta > 0 (Eq. 5)                           */
  int32_t sync_heads;   /* 1: one prefix length r* for all heads (Eq. 11);
                           0: each head its own largest feasible prefix (App. E)      */
  int32_t score_mode;   /* dkv_score_mode_t                                            */
  int32_t order;        /* dkv_order_t                                                 */
  int32_t eviction;     /* dkv_evict_t                                                 */
  int32_t refresh_baselines; /* 0: baselines frozen at insertion (Eq. 5, default);
                           1: b = max(rho, delta) for every retained state after each
                           update (App. E "Density baseline" ablation)              */
  int32_t layer_heads;  /* 0: the H heads are one layer.  Else H is a multiple of it and
                           the handle holds H / layer_heads independent layers of
                           layer_heads heads each (rows [l * layer_heads, (l + 1) *
                           layer_heads) of every [H][..] buffer): each layer has its own
                           shared prefix r* (Eq. 11) and prefix range, and one call
                           updates or reads all layers with single kernel launches      */
  int32_t descriptor;   /* dkv_descriptor_t: the vectors whose geometry the density uses
                           (Eqs. 2-3).  DKV_DESC_KV needs the workspace of
                           dkv_bank_workspace_size_ex; knorm then holds ||k||^2 + ||v||^2 */
} dkv_params_t;

/* Caller-owned device buffers of the handle's H per-head banks (one layer, or
 * H / layer_heads layers stacked along heads).  M_max = max_h budgets[h];
 * head h's state lives in rows [h * M_max, h * M_max + budgets[h]).  Slots
 * [0, occupancy_h) of head h are the retained states; their order is not
 * meaningful (the bank is a set, Eq. 12).                                     */
typedef struct {
  void* k;              /* device [H][M_max][d] keys (post-RoPE), dtype             */
  void* v;              /* device [H][M_max][d] values, dtype                       */
  float* rho;           /* device [H][M_max] cached density rho_i (App. C)          */
  float* base;          /* device [H][M_max] frozen insertion baseline b_i (Eq. 5)  */
  float* knorm;         /* device [H][M_max] cached ||k_i||^2 (derived, fp32)       */
  int64_t* prov_step;   /* device [H][M_max] update step that admitted the state    */
  int32_t* prov_src;    /* device [H][M_max] source index within its block          */
  int32_t* occupancy;   /* device [H] number of retained states per head            */
  void* workspace;      /* device scratch, >= dkv_bank_workspace_size_ex() bytes for
                           the handle's parameters (= dkv_bank_workspace_size() with
                           the key descriptor), 256-byte aligned; contents are
                           private to the handle                                    */
  size_t workspace_bytes;
} dkv_buffers_t;

/* Per-update statistics (read back by dkv_bank_stats). */
typedef struct {
  int32_t r_star;       /* admitted prefix length (Eq. 11); per-head values below    */
  int32_t rmax;         /* largest prefix length tested, min(N, min_h M_h)           */
  int32_t n_candidates; /* N of the last admit                                        */
  int32_t empty_init;   /* 1 if every head took the empty-bank path                  */
} dkv_layer_stats_t;

typedef struct {
  int32_t occupancy_before;
  int32_t occupancy_after;
  int32_t admitted;       /* r_h                                                      */
  int32_t evicted;        /* |R^h| = e_{r_h} (Eq. 10)                                 */
  int32_t mandatory;      /* states with g(r_h) >= tau, evicted first (Step 3)        */
  int32_t pre_violators;  /* states with g(0) >= tau (rounding drift; never evicted
                             when r_h = 0)                                            */
} dkv_head_stats_t;

/* Status text; never NULL. */
const char* dkv_status_str(dkv_status_t status);

/* Library version (major * 10000 + minor * 100 + patch). */
int32_t dkv_version(void);

/* Fills *out with the paper's default parameters for head dimension d. */
dkv_status_t dkv_params_default(dkv_params_t* out, int32_t d);

/* Bytes of device workspace a handle needs for H heads of dimension d, budgets
 * budgets[0..H) (host array), at most n_max candidates per admit, keys of
 * `dtype`.  Returns 0 if the arguments are invalid.                          */
size_t dkv_bank_workspace_size(int32_t H, int32_t d, const int32_t* budgets,
                               int32_t n_max, int32_t dtype);

/* As dkv_bank_workspace_size for a handle created with *params (host pointer; NULL:
 * the defaults).  The [K; V] descriptor needs the values of the candidates in score
 * order and of the survivors and evicted states as well: H (n_max + M_max + n_max) d
 * elements more.  Returns 0 if the arguments are invalid.                        */
size_t dkv_bank_workspace_size_ex(int32_t H, int32_t d, const int32_t* budgets,
                                  int32_t n_max, int32_t dtype, const dkv_params_t* params);

/* Creates a handle over caller-owned buffers (see dkv_buffers_t).  budgets is a
 * host array of H per-head budgets M_h >= 1.  Create writes the workspace
 * header once, synchronously (budgets, a cleared error word); it does not
 * touch the bank buffers, so the caller must zero `occupancy` (or call
 * dkv_bank_reset) before the first admit.  Limits: 1 <= H <= 4096,
 * d in {64, 128}, 1 <= M_h <= 262144, 1 <= n_max <= 16384.
 * DKV_SCORE_TENSOR requires dtype bf16 and d = 128.                          */
dkv_status_t dkv_bank_create(dkv_bank_t* out, int32_t H, int32_t d, const int32_t* budgets,
                             int32_t n_max, int32_t dtype, const dkv_params_t* params,
                             const dkv_buffers_t* buffers);

/* Releases the handle (host bookkeeping only; caller buffers are untouched).
 * Safe on NULL. */
void dkv_bank_destroy(dkv_bank_t bank);

/* Empties every head (occupancy := 0) on `stream`: a new video (Sec. 4.1). */
dkv_status_t dkv_bank_reset(dkv_bank_t bank, void* stream);

/* Steps 1-2 for the finalized block leaving the window (Sec. 3.4).
 *   Kc, Vc : device [H][N][d] candidate keys / values in source order
 *            (source index = row within the block), dtype of the handle.
 *   N      : 1 <= N <= n_max.
 *   step   : provenance recorded for admitted states, 0 <= step < 2^31; it
 *            should differ between updates, so that (step, source index)
 *            identifies a state (fill-eviction ties are broken by it).
 * Enqueues work on `stream`; the bank buffers are not modified.              */
dkv_status_t dkv_bank_admit(dkv_bank_t bank, const void* Kc, const void* Vc, int32_t N,
                            int64_t step, void* stream);

typedef enum {
  DKV_ROPE_INTERLEAVED = 0,   /* rotation pair j = elements (2j, 2j + 1)  */
  DKV_ROPE_HALF = 1           /* rotation pair j = elements (j, j + d/2)  */
} dkv_rope_layout_t;

/* dkv_bank_admit for keys that still carry their temporal rotary position.
 * The backbones attend to nonlocal memory keys with the temporal RoPE coordinate
 * set to 0 and the spatial coordinates kept, and the bank stores exactly those
 * keys (App. A, "Attention-logit" setup).  Keys taken from a local window carry the
 * rotation of their frame's coordinate t_x instead; this call first rotates every
 * pair j with theta[j] != 0 back by the angle t_x * theta[j]:
 *     x0 = x cos a + y sin a,  y0 = y cos a - x sin a,   a = t_x theta_j,
 * stores the result rounded to nearest (ties to even) in the key type, and then
 * runs admit on the stored keys (scores, order, crossings and the keys committed
 * by the following compress are those of the re-zeroed keys).  Values are not
 * rotated.  The rounding is that of the exact rotation (fp32 evaluation with an
 * error bound, float64 where the bound cannot decide it).
 *   t_coord : device int32 [N], temporal coordinate of each candidate (shared by
 *             all heads and layers of the handle), 4-byte aligned.
 *   theta   : device fp32 [d/2], angular frequency of each rotation pair; 0 for
 *             pairs outside the temporal band (left bit for bit).
 *   layout  : dkv_rope_layout_t.
 * Both arrays are read during the call's work on `stream` only.  The re-zeroed
 * keys live in the workspace until the following compress, so Kc may be reused
 * once this call's work has completed.  Errors as dkv_bank_admit, plus
 * DKV_ERR_ARG for a null or misaligned t_coord / theta or an unknown layout.   */
dkv_status_t dkv_bank_admit_rope(dkv_bank_t bank, const void* Kc, const void* Vc, int32_t N,
                                 int64_t step, const int32_t* t_coord, const float* theta,
                                 int32_t layout, void* stream);

/* Step 3 + commit for the block given to the preceding admit (Sec. 3.4;
 * Alg. 1; Eq. 12; Eq. C.4).  After it completes on `stream`, occupancy,
 * k, v, rho, base, knorm and provenance describe the committed banks.
 * Equivalent to dkv_bank_evict followed by dkv_bank_commit on one stream.    */
dkv_status_t dkv_bank_compress(dkv_bank_t bank, void* stream);

/* First half of compress: rho~ at the shared prefix r* (Eq. C.2), the mandatory
 * and densest eviction sets (Sec. 3.4) and the workspace copies of survivors and
 * evicted keys.  Reads the bank but does not modify k, v, occupancy or provenance,
 * so bank-reading attention of the current step may still run concurrently on
 * another stream.  Valid only right after admit (else DKV_ERR_STATE).          */
dkv_status_t dkv_bank_evict(dkv_bank_t bank, void* stream);

/* Second half of compress: the commit of Eq. 12 (admitted candidates into the
 * evicted slots, then appended), density maintenance of the survivors (Eq. C.4)
 * and the frozen baselines of the admitted states (Eq. 5).  Overwrites k, v and
 * occupancy: every reader of the pre-update bank (attention on another stream)
 * must be ordered before it.  Valid only right after evict (else DKV_ERR_STATE).
 * The new baselines run on a stream owned by the handle, forked from and joined
 * back into `stream` by events (also under stream capture); work enqueued on
 * `stream` afterwards is ordered after all of it.                               */
dkv_status_t dkv_bank_commit(dkv_bank_t bank, void* stream);

/* Bank-reading attention (Sec. 3.2, Fig. 2):
 *   O[h] = softmax(Q[h] [Kbank_h ; Kw[h]]^T / sqrt(d)) [Vbank_h ; Vw[h]]
 * over the occupancy_h retained states followed by the W window states.
 *   Q  : device [H][Nq][d], Kw, Vw : device [H][W][d], O : device [H][Nq][d],
 *   all of the handle's dtype; 1 <= Nq <= 1<<20, 0 <= W <= 1<<20.
 * A head with no retained state and W = 0 gets O = 0.  Reads the current
 * committed bank; does not modify it.                                        */
dkv_status_t dkv_bank_attend(dkv_bank_t bank, const void* Q, int32_t Nq, const void* Kw,
                             const void* Vw, int32_t W, void* O, void* stream);

/* Within-block competition (App. E "Within-block competition"): sequential,
 * density-gated admission, so that earlier candidates of a block act on later
 * ones.  The block's order is fixed once against the bank at block start (the
 * order dkv_bank_admit would take); then, for j = 0 .. N-1, the j-th candidate of
 * every head is offered as a complete one-candidate update (growth gate of
 * Eqs. 8-11, eviction, commit of Eq. 12, density maintenance of Eq. C.4 and the
 * frozen baseline of Eq. 5), the state recording its source index in the block
 * as provenance.  A bank whose heads are all empty is initialised by the whole
 * block (Alg. 1, m = 0), exactly as dkv_bank_admit + compress would; a bank with
 * some empty heads returns DKV_ERR_STATE.
 *   Kc, Vc  : device [H][N][d] as for dkv_bank_admit.
 *   scratch : device, 256-byte aligned, >= dkv_sequential_scratch_size() bytes.
 * Synchronises with `stream` once (to read the occupancy) and enqueues about a
 * dozen launches per candidate: an ablation path, not the hot path.  Must not be
 * called between admit and commit (DKV_ERR_STATE).                              */
size_t dkv_sequential_scratch_size(int32_t H, int32_t d, int32_t n_max, int32_t dtype);
dkv_status_t dkv_bank_update_sequential(dkv_bank_t bank, const void* Kc, const void* Vc, int32_t N,
                                        int64_t step, void* scratch, size_t scratch_bytes, void* stream);

/* Declares that the caller has written bank contents directly (k, v, rho,
 * base, prov_*) and sets occupancy from the host array occupancy[0..H)
 * (0 <= occupancy[h] <= budgets[h]).  Recomputes the derived key norms.
 * Used for checkpoint restore and teacher-forced testing.  Must not be called
 * between admit and compress (DKV_ERR_STATE).                                 */
dkv_status_t dkv_bank_import(dkv_bank_t bank, const int32_t* occupancy, void* stream);

/* Checkpoint read, the inverse of dkv_bank_import (the bank of (K, V, rho, b,
 * provenance, occupancy) that Alg. 1 carries from one update to the next,
 * Sec. 3.4): waits for the work enqueued by this handle, then copies every
 * head's state into the caller's arrays in dst, laid out as in dkv_buffers_t
 * for this handle's H and M_max:
 *   k, v              [H][M_max][d] keys / values, dtype of the handle
 *   rho, base         [H][M_max] fp32 cached density rho_i, baseline b_i
 *   prov_step         [H][M_max] int64, prov_src [H][M_max] int32
 *   occupancy         [H] int32
 * Each of these may point to host memory (pageable or pinned) or device memory;
 * a NULL field is skipped.  knorm, workspace and workspace_bytes are ignored:
 * the key norms are derived, and dkv_bank_import recomputes them.  Only rows
 * [0, occupancy[h]) of head h are meaningful.  Synchronous: returns after the
 * copies have completed.  DKV_ERR_STATE between admit and compress; a failed
 * copy gives DKV_ERR_CUDA and leaves dst partly written.                      */
dkv_status_t dkv_bank_export(dkv_bank_t bank, const dkv_buffers_t* dst);

/* Waits for all work enqueued by this handle, then reports the sticky device
 * error word (DKV_ERR_TIMEOUT / DKV_ERR_DEVICE) or a CUDA error.  Clears the
 * word after reporting it.                                                    */
dkv_status_t dkv_bank_sync(dkv_bank_t bank);

/* Copies the statistics of the last update to host memory (synchronises with
 * the handle's last stream).  layer holds one entry per layer (H / layer_heads,
 * 1 when layer_heads = 0); heads may be NULL, else it holds H entries.        */
dkv_status_t dkv_bank_stats(dkv_bank_t bank, dkv_layer_stats_t* layer, dkv_head_stats_t* heads);

/* Copies the current per-head occupancy to host memory (synchronises).       */
dkv_status_t dkv_bank_occupancy(dkv_bank_t bank, int32_t* occupancy);

/* Read-only device views of the intermediates of the last update, for
 * inspection and parity testing.  Valid until the next admit on the handle.
 * Strides are in elements.  Entries beyond the current N / occupancy are
 * unspecified.                                                               */
typedef struct {
  const float* score;        /* [H][n_max]  Eq. 6 score s_h(x), source order          */
  const int32_t* perm;       /* [H][n_max]  pi_h: candidate index at sorted position   */
  const int32_t* cross;      /* [H][M_max]  min{r : g_i(r) >= tau} over r <= rmax,
                                            INT32_MAX when no such r                 */
  const float* rho_tilde;    /* [H][M_max]  rho~_i(r_h) (Eq. C.2), set by evict        */
  const int32_t* slot_new;   /* [H][n_max]  bank slot of the j-th admitted candidate   */
  int64_t n_max;
  int64_t M_max;
} dkv_intermediates_t;

dkv_status_t dkv_bank_intermediates(dkv_bank_t bank, dkv_intermediates_t* out);

/* Kernel timing: enable = 1 brackets every kernel the handle launches with
 * CUDA events on its stream, enable = 2 only the attention launches (0: off;
 * other values: DKV_ERR_ARG).  dkv_bank_kernel_times() returns, per kernel
 * name, the number of launches and the summed device milliseconds of the
 * launches whose events have completed (it synchronises); with enable = 2 the
 * other kernels are counted with 0 ms.  With enable = 1 the commit runs the
 * survivor and new-baseline passes one after the other on the caller's stream
 * (otherwise side by side on two streams), so that each launch's time is its
 * own.  Timing adds two event records per timed launch; keep it off when not
 * measuring.                                                                 */
dkv_status_t dkv_bank_set_timing(dkv_bank_t bank, int32_t enable);
dkv_status_t dkv_bank_kernel_times(dkv_bank_t bank, int32_t max_kernels, char* names /* [max][48] */,
                                   int32_t* launches, double* total_ms, int32_t* n_kernels);

/* Self-test of the bounded device-side waits (no paper counterpart; a diagnostic).
 * Launches one CTA that waits, through the library's own bounded-wait helper, on a
 * barrier nothing arrives on; after limit_us microseconds (1 .. 1e6) the wait gives
 * up, the kernel records the timeout and returns.  Returns DKV_ERR_TIMEOUT when the
 * wait gave up as designed (the expected result), and writes the measured wait
 * duration to *elapsed_ns (host).  Synchronises the device; allocates 16 bytes of
 * device memory for the duration of the call.  The context stays usable.          */
dkv_status_t dkv_selftest_wait_timeout(int32_t limit_us, int64_t* elapsed_ns);

/* Largest candidate count accepted by dkv_candidate_order_noalloc. */
#define DKV_NOALLOC_MAX_N 16384

/* Candidate scores and order for ONE head, without any device allocation.
 *
 * The paper has no counterpart of this call; it exists for callers that cannot
 * allocate device memory and so cannot provide the workspace of dkv_bank_create:
 * code inside a framework whose pool owns every device byte, hosts that forbid
 * allocation after start-up (real-time or embedded deployments), or plugins that
 * are handed only fixed input and output buffers.  It computes what the first half
 * of dkv_bank_admit computes for one head in the fp32 score mode: the Eq. 6 score
 * of every candidate and the stable ascending order of those scores (ties in source
 * order; an empty bank, m = 0, gives the source order and zero scores).
 *
 *   K_bank   : device [m][d] bank keys of the head, dtype
 *   base     : device [m] frozen baselines b_i (fp32)
 *   Kc       : device [N][d] candidate keys in source order, dtype
 *   params   : host; tau, sigma, p, eps, delta as for dkv_bank_create (the other
 *              fields are ignored)
 *   scores_out : device [N] fp32, or NULL
 *   perm_out : device [N] int32: perm_out[j] = candidate at sorted position j
 *
 * Limits: 1 <= N <= DKV_NOALLOC_MAX_N (else DKV_ERR_SHAPE, nothing is launched),
 * 0 <= m <= 262144, d in {64, 128}.
 * Arithmetic: that of the fp32 score mode of dkv_bank_admit, in the same order, so
 * the scores and the order are bit-identical to admit's in that mode.
 * Memory: the scores live in a fixed 64 KiB device array inside the library (one
 * per GPU that loads it, kept until the process exits); the call allocates nothing,
 * on the device or through any library.  The first successful call on each device
 * (made with that device current) looks up that array's device address and sets a
 * kernel attribute; make that first call before any stream capture.  If that set-up
 * fails the call returns DKV_ERR_CUDA and the next call on the device tries again.
 * Nothing in the array needs clearing: every entry a call reads is written earlier
 * in the same call.  All calls on a device share the array, so calls whose work
 * overlaps on the GPU (different streams without ordering between them) race;
 * order them on one stream.                                                      */
dkv_status_t dkv_candidate_order_noalloc(const void* K_bank, const float* base, int32_t m, const void* Kc,
                                         int32_t N, int32_t d, int32_t dtype, const dkv_params_t* params,
                                         float* scores_out, int32_t* perm_out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* DKV_H_ */
