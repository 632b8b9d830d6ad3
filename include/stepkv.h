/*
 * stepkv.h -- C ABI of the StepKV compression pass on GB300 (sm_103a).
 *
 * StepKV (arXiv 2609.22158) compresses an agent's KV cache at each completed-step boundary
 * (Sec. 3, Eq. 1): every prunable token i gets a retention priority P_i = alpha*T_i + beta*S_k
 * (Eq. 5), where T_i is attention-based token saliency and S_k the utility of the step k that
 * produced token i (Eqs. 2-4, Algorithm 1), and the B_t highest-priority tokens are kept.
 *
 * The pass has five stages, all computed by this library's CUDA kernels:
 *   1. score   -- T_i from the observation-window queries against all cached keys (stepkv_score)
 *   2. reduce  -- per-step aggregation of saliency, keyed by each token's step id
 *   3. fuse    -- Eqs. 2-5 (stages 2-5 of this list are in stepkv_select)
 *   4. select  -- exact global top-B over the prunable tokens under the budget
 *   5. compact -- gather of the retained K/V rows into a dense cache (stepkv_compact)
 * stepkv_compress runs all five for one or more trajectories.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Pointers are DEVICE pointers unless a comment says "host".  Arrays of per-layer tensors are
 *    HOST arrays of device pointers.
 *  - bf16 tensors are passed as void* holding IEEE bfloat16 values.
 *  - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream).  Every call
 *    only enqueues work on `stream` and returns; nothing synchronises the host.
 *  - The library never allocates or frees memory and keeps no state between calls; scratch
 *    memory is the caller's `ws` (size from the matching *_workspace_size function, 256-byte
 *    aligned).  Calls on different streams with different workspaces may run concurrently.
 *    The one exception is stepkv_select_static_scratch (below), which takes no workspace and uses
 *    a fixed scratch array compiled into the library instead.
 *  - CUDA graphs: the calls issue kernel launches only (no copies, memsets or synchronisation), so a
 *    call can be captured into a CUDA graph and replayed, with new data in the same buffers between
 *    replays.  The saliency kernel orders its blocks through flags in the workspace; the value a
 *    launch publishes mixes a per-call host value with an epoch kept in the workspace and advanced
 *    by every launch, so a replay never mistakes the previous launch's flags for its own.  The
 *    workspace needs no initialisation.  Make one ordinary call before capturing (it sets the
 *    kernels' shared-memory limits, which must not happen during a capture).
 *  - Errors: argument problems are detected on the host and returned (STEPKV_EINVAL,
 *    STEPKV_EUNSUPPORTED, STEPKV_ENOSPACE) before anything is enqueued.  A failed launch returns
 *    STEPKV_ECUDA.  Data-dependent problems found on the device (a step id out of range, kept_cap
 *    too small, a bounded device-side wait that ran out) are written to *dev_status with
 *    atomicCAS(0 -> code): the FIRST error wins and later calls never clear it.  dev_status is a
 *    device int32 the caller zeroes once and reads after its own synchronisation.  Kernels that
 *    hit such an error skip the affected work and return; they never trap.
 *  - Token order: slots 0..T-1 of a layer's cache.  Retained slots are reported in ascending
 *    original order, so with the protected prompt as a prefix the compacted cache is exactly
 *    C_prot || C_traj[K] of Eq. 1.
 *  - GQA: query head g reads KV head g / G, G = Hq / Hkv.
 */
#ifndef STEPKV_H
#define STEPKV_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define STEPKV_API __attribute__((visibility("default")))
#else
#define STEPKV_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  STEPKV_OK = 0,
  STEPKV_EINVAL = 1,        /* invalid argument (host check, nothing enqueued) */
  STEPKV_ECUDA = 2,         /* a CUDA runtime call or launch failed */
  STEPKV_ENOSPACE = 3,      /* workspace too small (host) / kept_cap < n_kept (device) */
  STEPKV_EUNSUPPORTED = 4,  /* shape or alignment outside what the kernels handle */
  STEPKV_EDATA = 5,         /* device: invalid data (step id out of [0, n_steps), bad kept index) */
  STEPKV_ETIMEOUT = 6       /* device: a bounded wait inside a kernel expired */
} stepkv_status_t;

enum { STEPKV_NORM_MAX = 0, STEPKV_NORM_NONE = 1 };
enum { STEPKV_POOL_MAX = 0, STEPKV_POOL_AVG = 1 };
#define STEPKV_MAX_POOL 63
enum { STEPKV_BUDGET_RATIO = 0, STEPKV_BUDGET_COUNT = 1 };

/* Hyper-parameters of Eqs. 2-5 (Table H defaults from stepkv_default_params). */
typedef struct {
  float lambda;   /* redundancy penalty in r_k (Eq. 2) */
  float w_r;      /* completion weight (Eq. 4) */
  float w_c;      /* reuse weight (Eq. 4) */
  float r_min;    /* inner clip of r_k (Eq. 4) */
  float r_max;
  float s_max;    /* outer clip of S_k (Eq. 4) */
  float eta;      /* reuse update scale (Eq. 3) */
  float alpha;    /* token-saliency weight (Eq. 5) */
  float beta;     /* step-utility weight (Eq. 5) */
  int32_t sal_norm; /* STEPKV_NORM_MAX: T_i divided by its maximum over prunable tokens (appendix,
                       "H_i normalised to [0, H_max]"); STEPKV_NORM_NONE: T_i used as is */
  int32_t sal_pool; /* SnapKV-style token-axis pooling of each saliency row before the mean over rows
                       (Sec. 4.2: T_i from an existing estimator such as SnapKV): odd width k in
                       [1, STEPKV_MAX_POOL], 1 = none.  Window [i - k/2, i + k/2] clipped to [0, T).
                       In stepkv_compress a width > 1 makes the saliency stage write its rows (one
                       launch per trajectory) and pool them, instead of summing them on the fly */
  int32_t sal_pool_mode; /* STEPKV_POOL_MAX: maximum over the window; STEPKV_POOL_AVG: mean of the
                            window's in-range values */
} stepkv_params_t;

/* KV budget (Eq. 1).  RATIO: B_t = max(1, floor(ratio_num * N_t / ratio_den)) of the N_t
 * prunable tokens (exact integer arithmetic); COUNT: B_t = count.  In both cases |K| = min(B_t, N_t),
 * and |K| = 0 when N_t = 0.  Protected tokens are kept on top of the budget. */
typedef struct {
  int32_t mode;
  int32_t ratio_num;
  int32_t ratio_den;
  int32_t count;
} stepkv_budget_t;

/* Per-step trajectory signals at the boundary after step t = n_steps-1 (0-based step ids).
 * All arrays are device float32 [n_steps].  valid/gain/red are the inputs of Eq. 2 for every step
 * (they do not change once a step is final); obs_sim[k] = sim(Obs_t, Obs_k) drives Eq. 3 for k < t
 * (obs_sim[t] is ignored; NULL = no Phase-2 update).  reuse_in holds c_k from the previous boundary
 * (reuse_in[t] is ignored: Algorithm 1 Phase 1 sets c_t = 0); reuse_out receives the updated c_k
 * (may alias reuse_in; NULL = not written). */
typedef struct {
  int32_t n_steps;
  const float* valid;
  const float* gain;
  const float* red;
  const float* obs_sim;
  const float* reuse_in;
  float* reuse_out;
} stepkv_steps_t;

/* Outputs of the selection stage.  kept_idx/n_kept are required, the rest may be NULL. */
typedef struct {
  int32_t* kept_idx;      /* [kept_cap]: retained slots (protected + selected), ascending */
  int32_t kept_cap;       /* capacity of kept_idx (and of the compacted caches) */
  int32_t* n_kept;        /* [1]: number of retained slots = n_protected + min(B_t, N_t) */
  int32_t* n_budget;      /* [2] or NULL: (N_t, B_t) */
  float* priority;        /* [T] or NULL: P_i (Eq. 5); -inf for protected tokens */
  float* token_sal;       /* [T] or NULL: normalised saliency T_i used in Eq. 5 */
  float* step_util;       /* [n_steps] or NULL: S_k (Eq. 4) after this boundary's update */
  int32_t* step_count;    /* [n_steps] or NULL: prunable tokens per step */
  float* step_sal_sum;    /* [n_steps] or NULL: sum of T_i over the step's prunable tokens */
  float* step_sal_max;    /* [n_steps] or NULL: max of T_i over the step's prunable tokens */
  int32_t* step_kept;     /* [n_steps] or NULL: retained prunable tokens per step */
} stepkv_select_out_t;

/* One trajectory for stepkv_compress. */
typedef struct {
  int32_t L, Hkv, Hq, d, T, W;
  int32_t n_sal_layers;            /* saliency from layers L-n_sal_layers .. L-1 (Table H: last 3) */
  const void* const* K;            /* host [L]: K of layer l, [Hkv][rows >= T][d] bf16 */
  const void* const* V;            /* host [L]: V of layer l, same layout */
  int64_t kv_head_stride;          /* elements between KV heads (>= T*d, multiple of 8) */
  const void* const* Q;            /* host [n_sal_layers]: window queries of layer L-n_sal_layers+i,
                                      [Hq][W][d] bf16; query w sits at slot T-W+w */
  int64_t q_head_stride;           /* elements between query heads (>= W*d, multiple of 8) */
  const int32_t* step_id;          /* [T]: step of each token; ignored for protected tokens */
  const uint8_t* prot;             /* [T]: 1 = protected (never pruned, always kept) */
  const int32_t* pos_in;           /* [T] or NULL: original position of each slot */
  stepkv_steps_t steps;
  stepkv_budget_t budget;
  void* const* K_out;              /* host [L]: compacted K, [Hkv][rows >= kept_cap][d].  When every
                                      K_out[l] is K[l] and every V_out[l] is V[l] (one head stride), the
                                      compaction runs in place by hole filling: rows [0, n_kept) end up
                                      holding the retained set, each retained slot below n_kept staying
                                      where it is and each hole receiving a retained row from a slot at or
                                      above n_kept, so the rows are no longer in slot order; step_id_out
                                      and pos_out give each row's step and original position.  Attention
                                      over the rows does not depend on their order. */
  void* const* V_out;              /* host [L] */
  int64_t out_head_stride;         /* elements (>= kept_cap*d, multiple of 8) */
  int32_t* step_id_out;            /* [kept_cap] or NULL: step_id of each retained slot */
  int32_t* pos_out;                /* [kept_cap] or NULL: pos_in (or the slot index) of each retained slot */
  stepkv_select_out_t sel;
  /* Where the caches live.  STEPKV_MEM_DEVICE (0, the default of a zeroed struct): K/V and
     K_out/V_out are device memory.  STEPKV_MEM_HOST: page-locked host memory (cudaHostAlloc or
     cudaHostRegister; checked with cudaPointerGetAttributes, else STEPKV_EINVAL) that the compaction
     reads or writes across the CPU-GPU link, moving only the retained rows: a cache offloaded to host
     memory is compressed straight into HBM (out_location DEVICE) or back into host memory.  With
     kv_location HOST the saliency stage reads K_sal instead of K. */
  int32_t kv_location;
  int32_t out_location;
  const void* const* K_sal;        /* host [n_sal_layers] of device pointers, required when kv_location is
                                      HOST: layer L-n_sal_layers+i's K in device memory, same layout and
                                      head stride as K; ignored otherwise */
  const float* const* sal_lse;     /* host [n_sal_layers] of device pointers, or NULL: each window query's
                                      natural-log log-sum-exp over its causal row, [Hq][W] float32 (what the
                                      Observation prefill's attention reports; Sec. 4.2 collects T_i during
                                      that prefill).  Given, the saliency stage skips its first pass; see
                                      stepkv_score_lse */
} stepkv_problem_t;

#define STEPKV_MEM_DEVICE 0
#define STEPKV_MEM_HOST 1

/* Table H defaults (appendix "Implementation Details"): lambda=0.3, w_r=0.85, w_c=0.15, r_min=-1,
 * r_max=2, S_max=8, eta=1.5, alpha=0.2, beta=0.8, max-normalised saliency. */
STEPKV_API void stepkv_default_params(stepkv_params_t* p);

/* Static text for a status code (never NULL). */
STEPKV_API const char* stepkv_status_string(int32_t status);

/* Library ABI version (major*1000 + minor). */
STEPKV_API int32_t stepkv_version(void);

/* Message of the last CUDA error seen by this thread inside the library ("" if none). */
STEPKV_API const char* stepkv_last_cuda_error(void);

/* ---------------------------------------------------------------------------------------------
 * Stage 1: token saliency (Sec. 4.2 "Token Saliency"; the attention-based T_i collected from the
 * observation-window queries of the last layers, Table H).
 *
 * For each of n_layers layers, KV head h and key slot j:
 *   sal[l][h][j] = (1/G) * sum_{g = hG}^{hG+G-1} sum_{w < W} softmax_{j' <= T-W+w}( q_{l,g,w} . k_{l,h,j'} / sqrt(d) )[j]
 * i.e. a causal scaled softmax of each window query over the whole visible context (protected
 * tokens included), summed over the window queries and averaged over the GQA group.
 *
 *  K[l]   host array of device pointers, [Hkv][rows][d] bf16 with head stride k_head_stride
 *         elements; rows >= T.  Base 16-byte aligned, k_head_stride % 8 == 0.
 *  Q[l]   host array, [Hq][W][d] bf16 with head stride q_head_stride (% 8 == 0).
 *  sal    [n_layers][Hkv][T] float32 output.
 *  Supported: d in {64, 128}; Hq % Hkv == 0; 1 <= W <= T; W <= 4096; 1 <= n_layers <= 8.
 *  Work: two tensor-core passes over K (row statistics, then saliency).
 */
STEPKV_API size_t stepkv_score_workspace_size(int32_t n_layers, int32_t Hkv, int32_t Hq, int32_t T, int32_t W);
STEPKV_API stepkv_status_t stepkv_score(int32_t n_layers, const void* const* K, int64_t k_head_stride,
                             const void* const* Q, int64_t q_head_stride,
                             int32_t Hkv, int32_t Hq, int32_t d, int32_t T, int32_t W,
                             float* sal, void* ws, size_t ws_bytes, int32_t* dev_status, void* stream);

/* stepkv_score with the rows' statistics supplied (Sec. 4.2: T_i "collected during the existing
 * observation prefill"): the prefill's attention already computes, for every window query, the
 * log-sum-exp of its causal row, so only the second pass (the per-key softmax mass) runs.
 *
 *  lse[l]  host array of device pointers, [Hq][W] float32: lse[g][w] = ln sum_{j <= T-W+w}
 *          exp(q_{l,g,w} . k_{l,g/G,j} / sqrt(d)), natural log, as flash-attention kernels report it.
 *  Everything else as stepkv_score (same workspace size).  The result equals stepkv_score's when lse is
 *  the exact log-sum-exp; an lse off by delta for one query row scales that row's contribution by
 *  exp(-delta).
 */
STEPKV_API stepkv_status_t stepkv_score_lse(int32_t n_layers, const void* const* K, int64_t k_head_stride,
                                 const void* const* Q, int64_t q_head_stride, const float* const* lse,
                                 int32_t Hkv, int32_t Hq, int32_t d, int32_t T, int32_t W,
                                 float* sal, void* ws, size_t ws_bytes, int32_t* dev_status, void* stream);

/* ---------------------------------------------------------------------------------------------
 * Stages 2-4: step reduction, fusion and selection (Eqs. 1-5, Algorithm 1 Phases 1-3).
 *
 *  sal       [n_sal][T] float32: saliency rows (e.g. stepkv_score's n_layers*Hkv rows);
 *            T_i = mean over the n_sal rows (each row first pooled over params->sal_pool tokens when
 *            that is > 1), then normalised per params->sal_norm.
 *  step_id   [T] int32: step of each token (must lie in [0, n_steps) for prunable tokens; a
 *            violation sets STEPKV_EDATA and no selection is written).
 *  prot      [T] uint8: 1 = protected.
 *  steps, params, budget: host structs (device arrays inside steps).
 *  out       host struct of device output pointers (see stepkv_select_out_t).
 *  Ranking: (P_i descending, slot index ascending) -- on equal priority the older token wins.
 *  Supported: 1 <= T <= 262144, 1 <= n_steps <= 65535, n_sal >= 1.
 */
STEPKV_API size_t stepkv_select_workspace_size(int32_t n_sal, int32_t T, int32_t n_steps);
STEPKV_API stepkv_status_t stepkv_select(const float* sal, int32_t n_sal, int32_t T,
                              const int32_t* step_id, const uint8_t* prot,
                              const stepkv_steps_t* steps, const stepkv_params_t* params,
                              const stepkv_budget_t* budget, const stepkv_select_out_t* out,
                              void* ws, size_t ws_bytes, int32_t* dev_status, void* stream);

/* ---------------------------------------------------------------------------------------------
 * Stages 2-4 without a caller workspace.  The paper has no counterpart: this is a library
 * convenience, not part of the method.
 *
 * Who needs it: callers that cannot allocate device memory at call time.  A serving loop whose
 * device memory is fully reserved up front (a KV-cache pool that holds nearly all of HBM) would
 * see a per-call cudaMalloc fail; a latency-bound loop cannot take the device-wide
 * synchronisation that cudaFree implies; a plain C host has no caching allocator to borrow a
 * workspace from.  Such callers allocate their outputs once and call this instead of
 * stepkv_select; it allocates nothing.
 *
 * Same arguments, results and errors as stepkv_select without (ws, ws_bytes).  The scratch is a
 * 256-byte-aligned array of 1,146,880 bytes in the library's device image (one per device,
 * created with the library's module), enough for the mean saliency row and the per-step
 * accumulators up to the limits below.
 *  - Limits: T <= STEPKV_STATIC_SCRATCH_MAX_T and n_steps <= STEPKV_STATIC_SCRATCH_MAX_STEPS.
 *    Larger problems return STEPKV_ENOSPACE before anything is enqueued; use stepkv_select with
 *    a workspace for them.
 *  - Set-up: the first call on each device looks up the scratch's device address
 *    (cudaGetSymbolAddress, which may load the library's module) and keeps it for the process.
 *    Make that first call before any stream capture.  The address is not refreshed after
 *    cudaDeviceReset.
 *  - Nothing in the scratch needs to start at zero: the mean kernel overwrites the saliency row
 *    and the selection kernel zeroes its accumulators before using them.
 *  - Calls whose work overlaps on the device (different streams, or threads enqueueing on
 *    different streams of the same device) share the one scratch and race.  Calls on one stream
 *    are ordered and safe.  dev_status is the caller's device int32, as for stepkv_select.
 */
#define STEPKV_STATIC_SCRATCH_MAX_T 262144
#define STEPKV_STATIC_SCRATCH_MAX_STEPS 4096
STEPKV_API stepkv_status_t stepkv_select_static_scratch(const float* sal, int32_t n_sal, int32_t T,
                              const int32_t* step_id, const uint8_t* prot,
                              const stepkv_steps_t* steps, const stepkv_params_t* params,
                              const stepkv_budget_t* budget, const stepkv_select_out_t* out,
                              int32_t* dev_status, void* stream);

/* ---------------------------------------------------------------------------------------------
 * Stage 5: compaction (Eq. 1, C_hat = C_prot || C_traj[K]).
 *
 * For every layer l < n_layers, KV head h and r < *n_kept:
 *   K_out[l][h][r][:] = K_in[l][h][kept_idx[r]][:]   (same for V; bit-exact copies)
 *   step_id_out[r] = step_id_in[kept_idx[r]],  pos_out[r] = pos_in ? pos_in[kept_idx[r]] : kept_idx[r]
 *  n_kept is read on the device (no host synchronisation); *n_kept > kept_cap or a kept index
 *  outside [0, T) sets STEPKV_ENOSPACE / STEPKV_EDATA and skips the bad rows.
 *  V_in/V_out may be NULL (keys only); step/pos pointers may be NULL.
 *  Rows are d bf16 values; d*2 bytes must be a multiple of 16 and d <= 256; bases 16-byte aligned;
 *  in/out head strides % 8 == 0.  In-place compaction (K_out == K_in) is not supported here; the fused
 *  pass (stepkv_compress) offers it by hole filling.
 */
STEPKV_API stepkv_status_t stepkv_compact(int32_t n_layers, const void* const* K_in, const void* const* V_in,
                               int64_t in_head_stride, int32_t Hkv, int32_t d, int32_t T,
                               const int32_t* kept_idx, const int32_t* n_kept, int32_t kept_cap,
                               void* const* K_out, void* const* V_out, int64_t out_head_stride,
                               const int32_t* step_id_in, const int32_t* pos_in,
                               int32_t* step_id_out, int32_t* pos_out,
                               int32_t* dev_status, void* stream);

/* ---------------------------------------------------------------------------------------------
 * Decode attention over a compacted cache: the reads an agent makes after a boundary, each new
 * token attending to the retained rows C_hat = C_prot || C_traj[K] (Eq. 1).  One query token per
 * layer; GQA as above (query head g reads KV head g / G).
 *
 * For every layer l < n_layers and query head g < Hq:
 *   out[l][g][:] = sum_{j < n} softmax_j( q[l][g] . K[l][g/G][j] / sqrt(d) ) V[l][g/G][j][:]
 *  q[l]     host array of device pointers, [Hq][d] bf16.
 *  K[l], V[l] host arrays of device pointers, [Hkv][rows >= n_cap][d] bf16, head stride
 *           kv_head_stride elements (% 8 == 0); bases 16-byte aligned.
 *  n        keys per head: *n_dev when n_dev is not NULL (read on the device, e.g. the n_kept of a
 *           compaction), else n_host.  A device value above n_cap sets STEPKV_ENOSPACE and n_cap rows
 *           are used; a value below 1 sets STEPKV_EDATA and the output is zero.
 *  out[l]   host array of device pointers, [Hq][d] fp32.
 *  ws       scratch of stepkv_decode_workspace_size bytes (256-byte aligned): per-split partials.
 *  Supported: d in {64, 128}; G = Hq / Hkv in {1, 2, 4, 5, 8}; 1 <= n_cap; n_host <= n_cap.
 *  Work: split-K over 512-key chunks (one chunk of one (layer, KV head) per CTA, all G heads of the
 *  group per key-row load), then a merge of the chunks in order (deterministic).
 */
STEPKV_API size_t stepkv_decode_workspace_size(int32_t n_layers, int32_t Hkv, int32_t Hq, int32_t d, int32_t n_cap);
STEPKV_API stepkv_status_t stepkv_decode(int32_t n_layers, const void* const* q, const void* const* K,
                              const void* const* V, int64_t kv_head_stride, int32_t Hkv, int32_t Hq,
                              int32_t d, const int32_t* n_dev, int32_t n_host, int32_t n_cap,
                              float* const* out, void* ws, size_t ws_bytes, int32_t* dev_status,
                              void* stream);

/* ---------------------------------------------------------------------------------------------
 * Decode attention that also accumulates attention mass: the H2O-style token saliency (Sec. 4.2: T_i
 * "can be supplied by existing token-level KV importance estimators"; H2O scores a token by the
 * attention it has received).  Same arguments, outputs and rules as stepkv_decode, plus:
 *
 *  mass[l]  host array of device pointers, [Hkv][mass_head_stride >= n_cap] float32, read and
 *           written (4-byte aligned): for every KV head h and key j < n the call ADDS
 *             (1/G) * sum_{g = hG}^{hG+G-1} softmax_j( q[l][g] . K[l][h][j] / sqrt(d) )
 *           i.e. the key's softmax weight averaged over the GQA group (each call adds a total of 1
 *           per head over the keys).  The caller zeroes the rows (e.g. after a boundary) and reads
 *           them as saliency rows, e.g. stepkv_select(sal = mass rows of chosen layers, n_sal =
 *           layers x Hkv): T_i is then the mean accumulated attention of token i (Eq. 5's T_i).
 *  ws       stepkv_decode_h2o_workspace_size bytes: the split partials and every key's logits.
 *  out is bit-identical to stepkv_decode's on the same inputs; the masses are deterministic (one
 *  writer per element and call, heads summed in a fixed order).
 */
STEPKV_API size_t stepkv_decode_h2o_workspace_size(int32_t n_layers, int32_t Hkv, int32_t Hq, int32_t d,
                                                   int32_t n_cap);
STEPKV_API stepkv_status_t stepkv_decode_h2o(int32_t n_layers, const void* const* q, const void* const* K,
                                  const void* const* V, int64_t kv_head_stride, int32_t Hkv, int32_t Hq,
                                  int32_t d, const int32_t* n_dev, int32_t n_host, int32_t n_cap,
                                  float* const* out, float* const* mass, int64_t mass_head_stride,
                                  void* ws, size_t ws_bytes, int32_t* dev_status, void* stream);

/* ---------------------------------------------------------------------------------------------
 * Step signals from evidence cues (Sec. 4.1: observation validity, evidence gain, action redundancy of
 * Eq. 2 and the similarity that drives Eq. 3).  Every field of a step (0 Thought, 1 Action,
 * 2 Observation) is given as up to STEPKV_MAX_CUES evidence cues: distinct 32-bit ids in strictly
 * increasing order (how cues are drawn from text is the caller's; the paper caps them at 64 per field).
 * sim(a, b) = |A n B| / |A u B| over cue sets (0 when both are empty); a concatenation of fields is the
 * union of their cues.  For every target step k in [k0, n_steps):
 *   gain[k] = 1 - max_{u<k} sim(Th_k || Obs_k, Th_u || Obs_u)     (1 for the first step)
 *   red[k]  = max_{u<k} sim(Act_k, Act_u)                          (0 for the first step)
 * and, when obs_sim is not NULL, for the newest step t = n_steps - 1:
 *   obs_sim[k] = sim(Obs_t, Obs_k) for k < t, obs_sim[t] = 0      (the input of Eq. 3)
 *  cues     [n_steps][3][STEPKV_MAX_CUES] uint32 (entries past a field's count are ignored)
 *  n_cues   [n_steps][3] int32 in [0, STEPKV_MAX_CUES]
 *  gain/red [n_steps] float32 or NULL (only entries k >= k0 are written); obs_sim [n_steps] or NULL.
 *  A count outside [0, 64] or a list that is not strictly increasing sets STEPKV_EDATA and the values
 *  that depend on it are not written.  1 <= n_steps <= 65535, 0 <= k0 <= n_steps.
 *  The outputs can be passed straight to stepkv_steps_t (valid stays the caller's: an empty or
 *  error-returning Observation is unusable).
 */
#define STEPKV_MAX_CUES 64
STEPKV_API stepkv_status_t stepkv_step_signals(const uint32_t* cues, const int32_t* n_cues, int32_t n_steps,
                                               int32_t k0, float* gain, float* red, float* obs_sim,
                                               int32_t* dev_status, void* stream);

/* Failure-detection self-test (no counterpart in the paper).  Runs the saliency kernel of stepkv_score
 * on the same arguments, except that the wait of its second pass (for every CTA's first-pass flag)
 * looks for a value no CTA ever publishes, so every CTA's wait runs out after wait_limit_ns
 * (1 us .. 1 s).  The kernel then records STEPKV_ETIMEOUT in *dev_status (caller-zeroed), drains its
 * own TMA copies and tensor-core operations, frees its tensor memory and returns: the CUDA context
 * stays usable and later calls on the stream run normally.  sal is left undefined.  Supported when
 * G * W <= 256 (one row group); else STEPKV_EUNSUPPORTED.  ws as for stepkv_score.
 */
STEPKV_API stepkv_status_t stepkv_selftest_score_timeout(int32_t n_layers, const void* const* K,
                                              int64_t k_head_stride, const void* const* Q,
                                              int64_t q_head_stride, int32_t Hkv, int32_t Hq, int32_t d,
                                              int32_t T, int32_t W, float* sal, void* ws, size_t ws_bytes,
                                              uint64_t wait_limit_ns, int32_t* dev_status, void* stream);

/* ---------------------------------------------------------------------------------------------
 * The fused pass (score -> reduce/fuse -> select -> compact) for n_traj independent trajectories
 * (one pruning boundary each, Algorithm 1).  probs is a host array; everything runs on `stream`:
 * the saliencies (consecutive trajectories of one head shape share a launch, up to 16), then the
 * selections of all trajectories in one launch (one 8-CTA cluster per trajectory, up to 16 per
 * launch), then the compactions (out-of-place ones share launches; an in-place one is a single move
 * launch that follows the hole-filling plan its selection wrote).  `ws` (size
 * from stepkv_compress_workspace_size over the same array) holds one shared region for the saliency
 * partials, a private region per trajectory, and one shared region for the saliency rows of a pooled
 * token saliency (params->sal_pool > 1: the rows of each trajectory are written, then pooled; the
 * region is sized for the largest trajectory whatever the params).  Caches in host memory (kv_location / out_location
 * STEPKV_MEM_HOST) are read and written in place over the CPU-GPU link by the compaction kernels;
 * their pointers are checked on the host before anything is enqueued.
 */
STEPKV_API size_t stepkv_compress_workspace_size(const stepkv_problem_t* probs, int32_t n_traj);
STEPKV_API stepkv_status_t stepkv_compress(const stepkv_problem_t* probs, int32_t n_traj,
                                const stepkv_params_t* params, void* ws, size_t ws_bytes,
                                int32_t* dev_status, void* stream);

/* ---------------------------------------------------------------------------------------------
 * Stage timing of the fused pass (profiling; the paper has no counterpart).  Sets, for the calling
 * thread, three caller-owned CUDA events (cudaEvent_t passed as void*, NULL = not recorded) that every
 * later stepkv_compress call of this thread records on its stream: `before` ahead of its first launch,
 * `after_select` between the selection and the compaction launches, `after` behind its last launch.
 * cudaEventElapsedTime between them gives the saliency + selection time and the compaction time of a
 * pass without changing its launches (the compaction follows the selection in plain stream order; no
 * event separates the saliency and selection kernels, which overlap by programmatic dependent
 * launch).  Call with three NULLs to stop.  The events must outlive the calls that record them.
 */
STEPKV_API void stepkv_set_stage_events(void* before, void* after_select, void* after);

#ifdef __cplusplus
}
#endif

#endif /* STEPKV_H */
