/*
 * commitkv.h — C ABI of the CommitKV hot path on one GB300 (sm_103a).
 *
 * CommitKV ("CommitKV: Lifecycle-Aware KV Cache Compression via Commit
 * Transitions for Multi-Turn Agents", arXiv 2608.07855) scores how much
 * deleting each event page of an agent's KV cache changes the attention
 * outputs of a probe window of queries, once before a tool-call commit and
 * once after the returned observation is in the cache (Section 3.2,
 * Eq. 5-8); classifies the pages' lifecycle states (Section 3.2, Eq. 9-10);
 * runs the greedy joint test on the completion candidates (Section 3.3,
 * Eq. 11); and at a compression checkpoint keeps a bounded set of pending
 * pages and fills the budget, applying one index set to keys, values and
 * absolute positions (Eq. 4, 12, 13).
 *
 * Conventions shared by every entry point
 *   - Memory: the caller owns all memory.  The library allocates nothing and
 *     keeps no global state (commitkv_compact_noalloc, at the end, is the
 *     one exception: it keeps a fixed scratch array).  Unless stated otherwise a pointer argument
 *     is device memory; arrays of per-trajectory pointers ("host array of
 *     device pointers") and every struct argument are host memory and are
 *     read before the call returns.
 *   - Streams: every call is asynchronous and stream-ordered on `stream`
 *     (a cudaStream_t; NULL = the legacy default stream).  Outputs are
 *     valid once the stream reaches the call.
 *   - Errors: arguments that can be checked on the host are checked before
 *     any launch and give COMMITKV_ERR_INVALID_ARG, COMMITKV_ERR_UNSUPPORTED
 *     or COMMITKV_ERR_WORKSPACE with nothing launched.  A failing CUDA launch
 *     gives COMMITKV_ERR_CUDA.  Problems only visible on the device (a page
 *     span outside the cache, unsorted pages, a bad page id, a NaN score, a
 *     bounded wait that ran out) are recorded in a status word inside the
 *     workspace; read it with commitkv_workspace_status.  The affected
 *     outputs are then unspecified, but the kernels stay in bounds and
 *     return.
 *   - Workspace: one caller-allocated device buffer of at least
 *     commitkv_workspace_size() bytes, 256-byte aligned, initialised once
 *     with commitkv_workspace_init.  Calls that share a workspace must not
 *     overlap on the GPU (use one workspace per stream).
 *   - Batches: each call takes n_traj independent trajectories
 *     (1 <= n_traj <= COMMITKV_MAX_TRAJ) and covers all of them with one
 *     launch sequence.
 *   - There is no CPU fallback.
 */
#ifndef COMMITKV_H
#define COMMITKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st;
typedef struct CUstream_st *cudaStream_t;

#define COMMITKV_ABI_VERSION 1
#define COMMITKV_MAX_TRAJ 64
/* Size of the fixed device scratch of commitkv_compact_noalloc (4 MiB). */
#define COMMITKV_NOALLOC_SCRATCH_BYTES (4u << 20)

typedef enum {
  COMMITKV_OK = 0,
  COMMITKV_ERR_INVALID_ARG = 1, /* host-checkable argument out of range */
  COMMITKV_ERR_UNSUPPORTED = 2, /* valid but not implemented (dtype, head_dim, ...) */
  COMMITKV_ERR_CUDA = 3,        /* a CUDA runtime call failed */
  COMMITKV_ERR_TIMEOUT = 4,     /* a bounded device-side wait ran out */
  COMMITKV_ERR_WORKSPACE = 5,   /* workspace missing, too small or misaligned */
  COMMITKV_ERR_DEVICE_INPUT = 6 /* device-resident input failed a device-side check */
} commitkv_status;

typedef enum { COMMITKV_F32 = 0, COMMITKV_BF16 = 1 } commitkv_dtype;

/* Model shape (Eq. 3): M layers, H KV heads of width d, and Hq = g * H
 * query heads; query head h reads KV head h / g (grouped-query attention).
 * K, V and Q share one dtype.  fp32 computes in fp32; bf16 inputs are
 * multiplied on the tensor cores with fp32 accumulation.
 * Supported: head_dim 64 or 128; any M >= 1, H >= 1, g >= 1.
 * softmax_scale 0 means 1/sqrt(head_dim). */
typedef struct {
  int32_t layers;    /* M */
  int32_t kv_heads;  /* H */
  int32_t q_heads;   /* Hq, a multiple of H */
  int32_t head_dim;  /* d */
  int32_t dtype;     /* commitkv_dtype of K, V and Q */
  float softmax_scale;
} commitkv_shape;

/* One trajectory: one resident cache and one probe window (Section 3.1-3.2).
 *   k, v        device; element (l, h, i, c) of K lives at
 *               k + l*stride_layer + h*stride_head + i*stride_tok + c
 *               (strides in elements; the d channels are contiguous).
 *               The pre-commit cache may be a prefix view of the post-commit
 *               cache (same pointers and strides, smaller S).
 *   pos         device [S] int32 absolute positions p_i (Eq. 4), strictly
 *               increasing.  Token i is visible to query p iff pos[i] <= p
 *               (the condition under the sums of Eq. 6).
 *   q           device [M][Hq][W][d] dense probe queries (already
 *               position-encoded), dtype of the shape.
 *   q_pos       device [W] int32 absolute positions of the probe queries
 *               (Q-c or Q+c of Eq. 5).
 *   page_start, page_len  device [P] int32: page E is the resident-index
 *               span [page_start[E], page_start[E] + page_len[E]).  Pages
 *               are sorted by start and do not overlap; 0 <= len, and the
 *               span lies inside [0, S) (checked on the device).
 */
typedef struct {
  const void *k;
  const void *v;
  int64_t stride_layer, stride_head, stride_tok;
  const int32_t *pos;
  int32_t S;
  const void *q;
  const int32_t *q_pos;
  int32_t W;
  const int32_t *page_start;
  const int32_t *page_len;
  int32_t P;
} commitkv_traj;

/* Thresholds of Eq. 9.  Require tau_dead < tau_use and rho_dead < rho_use. */
typedef struct {
  float tau_use, tau_dead, rho_use, rho_dead;
} commitkv_thresholds;

/* Size in bytes of the workspace every entry point below needs for these
 * trajectories (the maximum over the calls).  Pass the largest caches the
 * workspace will serve (normally the post-commit ones).  Returns 0 for
 * invalid arguments. */
size_t commitkv_workspace_size(const commitkv_shape *shape, int32_t n_traj,
                               const commitkv_traj *trajs);

/* Clears the workspace's device status word (stream-ordered).  Call once
 * after allocating a workspace. */
commitkv_status commitkv_workspace_init(void *workspace, size_t workspace_bytes,
                                        cudaStream_t stream);

/* Synchronises `stream`, then returns the first device-side error recorded
 * in the workspace since the last clear (COMMITKV_OK if none).  clear != 0
 * resets the word afterwards.  Returns COMMITKV_ERR_CUDA if the copy fails. */
commitkv_status commitkv_workspace_status(const void *workspace, size_t workspace_bytes,
                                          cudaStream_t stream, int32_t clear);

/* Static string naming a status code. */
const char *commitkv_status_string(commitkv_status status);

/* ------------------------------------------------------------------------
 * Page deletion effects, Section 3.2, Eq. 6-8.
 *
 * For every trajectory t, page E, layer l (selected by layer_mask), query
 * head h and probe query p of the window:
 *   a_pi  = softmax over visible i of softmax_scale * <q_p, k_i>
 *   o_p   = sum_i a_pi v_i
 *   o_p^{\E} = (o_p - sum_{i in E visible} a_pi v_i) / (1 - sum_{i in E visible} a_pi)
 *   r     = ||o_p - o_p^{\E}|| / ||o_p||                    (Eq. 6)
 *   R_out[t][E] = max over l, h, p of r                    (Eq. 7)
 * Called on the pre-commit cache with Q-c this is R-c; on the post-commit
 * cache with Q+c it is R+c (Eq. 8).  Degenerate rows, in this order: no
 * visible token of E -> 0; every visible token in E -> +inf; ||o_p|| = 0 ->
 * 0 if o_p^{\E} = o_p else +inf.  A row whose visible mass outside E
 * underflows in fp32 reports +inf.
 *
 *   layer_mask   host [M] (nonzero = layer takes part) or NULL = all layers.
 *   R_out        host array [n_traj] of device float [P_t]; fully written.
 *   head_R_out   NULL, or host array [n_traj] of device float [M][Hq][P_t]
 *                (NULL entries allowed): max over the window per (l, h);
 *                rows of unselected layers are written as 0.
 *   stats_out    NULL, or host array [n_traj] of device float
 *                [M][Hq][W_t][d + 4] (NULL entries allowed): per probe row
 *                m = max scaled score, l = sum exp(s - m), n = number of
 *                visible tokens (stored as float), 0, then o_p[0..d).
 *                commitkv_joint_test needs these for the post-commit pass.
 * -------------------------------------------------------------------- */
commitkv_status commitkv_page_effects(const commitkv_shape *shape, int32_t n_traj,
                                      const commitkv_traj *trajs, const uint8_t *layer_mask,
                                      float *const *R_out, float *const *head_R_out,
                                      float *const *stats_out, void *workspace,
                                      size_t workspace_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Page deletion effects from given row statistics (Section 3.2, Eq. 6-8),
 * one read of the page tokens.
 *
 * Eq. 6 needs, per probe row, the final softmax of the whole cache: the
 * normaliser and the output o_p.  An engine that already computed that
 * attention (its output and log-sum-exp for the probe queries) can pass
 * them here; the library then reads only the tokens of the pages (one pass)
 * instead of the whole cache and then the pages (two passes, as
 * commitkv_page_effects does).  Same definition, same degenerate cases and
 * same outputs as commitkv_page_effects.
 *
 *   stats_in     host array [n_traj] of device float [M][Hq][W_t][d + 4]
 *                (entries of trajectories with P = 0 or W = 0 may be NULL):
 *                per probe row m, l, (ignored), (ignored), o_p[0..d) with
 *                l = sum over visible i of exp(softmax_scale <q_p, k_i> - m)
 *                and o_p the normalised output.  From a log-sum-exp L: m = L,
 *                l = 1.  The stats_out of commitkv_page_effects on the same
 *                cache and window are valid stats_in.  Rows of unselected
 *                layers are not read.  Read only.
 *   R_out, head_R_out, layer_mask   as for commitkv_page_effects.
 * The number of visible tokens of each row is counted from pos and q_pos.
 * A row whose stats disagree with its cache gives effects of those stats.
 * -------------------------------------------------------------------- */
commitkv_status commitkv_page_effects_from_stats(const commitkv_shape *shape, int32_t n_traj,
                                                 const commitkv_traj *trajs, const uint8_t *layer_mask,
                                                 const float *const *stats_in, float *const *R_out,
                                                 float *const *head_R_out, void *workspace,
                                                 size_t workspace_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Per-token fill scores for a compression checkpoint (Section 3.3, Eq. 13:
 * the fill of the remaining budget).  The paper leaves the fill rule to an
 * appendix it does not include; this is window attention in the spirit of
 * SnapKV, whose probe windows the paper builds on:
 *   scores_out[t][i] = max over selected layers l, query heads h and probe
 *                      queries p with pos[i] <= q_pos[p] of
 *                      exp(s_pi - m_p) / l_p,   s_pi = softmax_scale <q_p, k_i>,
 * and 0 for a token that no probe query sees.  m_p and l_p are the row
 * statistics of the same cache and window: pass the stats_out of a
 * commitkv_page_effects call on this trajectory (a trajectory with P = 0
 * pages gives the statistics alone).  Larger scores keep a token first.
 *
 *   shape, n_traj, trajs   as for commitkv_page_effects; k, pos, S, q,
 *                          q_pos, W are read (v and the pages are not).
 *   layer_mask   optional host [M] u8, the layers that take part (NULL: all).
 *   stats        host array of n_traj device pointers, [M][Hq][W][d + 4]
 *                fp32 as written by commitkv_page_effects (m, l used; the
 *                rows of the selected layers are read).  Required when
 *                S_t > 0 and W_t > 0.
 *   scores_out   host array of n_traj device pointers, [S_t] fp32 each,
 *                overwritten (required when S_t > 0).
 *   workspace    at least 256 bytes, 256-byte aligned (the status word
 *                only; any workspace of the other calls will do).
 * Errors: INVALID_ARG for missing pointers or bad shapes, UNSUPPORTED for
 * head_dim other than 64 and 128.  Tensor cores for bf16, head_dim 128 and
 * 16-byte aligned rows (stats included); CUDA cores otherwise.
 * -------------------------------------------------------------------- */
commitkv_status commitkv_token_scores(const commitkv_shape *shape, int32_t n_traj, const commitkv_traj *trajs,
                                      const uint8_t *layer_mask, const float *const *stats,
                                      float *const *scores_out, void *workspace, size_t workspace_bytes,
                                      cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Lifecycle classification, Section 3.2, Eq. 9-10, and the candidate order
 * of Section 3.3.
 *
 * E_c = pages with eligible[E] != 0.  P-(E), P+(E) = #{F in E_c : R(F) <
 * R(E)} / |E_c| (ties share the lower rank).  H = (R >= tau_use and
 * P >= rho_use), L = (R <= tau_dead and P <= rho_dead), per window.
 * state_out[E]: 0 outside E_c, 1 completion candidate (H- and L+),
 * 2 dormant (L- and L+), 3 newly active (L- and H+), 4 still active (H-
 * and H+), 5 uncertain.  cand_out lists the candidates by increasing R+,
 * then decreasing R-, then increasing page index; n_cand_out[t] counts
 * them.
 *
 *   P            host [n_traj] page counts.
 *   R_pre, R_post, eligible   host arrays of device [P_t] (float, float, u8).
 *   thresholds   host; NULL = tau_use 0.05, tau_dead 0.01, rho_use 0.75,
 *                rho_dead 0.25 (the paper's settings).
 *   state_out    host array of device uint8 [P_t].
 *   cand_out     host array of device int32 [P_t]; first n_cand entries valid.
 *   n_cand_out   device int32 [n_traj].
 * A NaN effect is a device input error.
 * -------------------------------------------------------------------- */
commitkv_status commitkv_classify(int32_t n_traj, const int32_t *P, const float *const *R_pre,
                                  const float *const *R_post, const uint8_t *const *eligible,
                                  const commitkv_thresholds *thresholds, uint8_t *const *state_out,
                                  int32_t *const *cand_out, int32_t *n_cand_out, void *workspace,
                                  size_t workspace_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Classification variants: the ablations of Section 4.4 (Table 3).
 *
 * commitkv_classify with some of its steps removed; variant = 0 is
 * commitkv_classify.  Bits:
 *   COMMITKV_CLASSIFY_NO_PRECOMMIT   "w/o pre-commit state": the candidates
 *       are the pages with L+ (low after the commit) whatever their state
 *       before it, instead of H- and L+.  state_out is still the lifecycle
 *       state of Eq. 10; cand_out / n_cand_out list the L+ pages in the
 *       same order (increasing R+, then decreasing R-, then page index).
 *   COMMITKV_CLASSIFY_NO_PERCENTILE  "w/o percentile calibration": H = (R >=
 *       tau_use) and L = (R <= tau_dead) in both windows; rho_use and
 *       rho_dead are not used (they are still checked).
 * The paper's other ablations need no variant: "w/o joint validation"
 * retires every candidate (commitkv_joint_test with tau_joint = +inf),
 * "w/o transition protection" reserves no pending pages
 * (commitkv_compact with pending_cap_pages = 0), "w/o lifecycle mechanism"
 * retires nothing (no classify and joint test before commitkv_compact).
 * Unknown bits: COMMITKV_ERR_INVALID_ARG.  Otherwise as commitkv_classify.
 * -------------------------------------------------------------------- */
#define COMMITKV_CLASSIFY_NO_PRECOMMIT 1u
#define COMMITKV_CLASSIFY_NO_PERCENTILE 2u
commitkv_status commitkv_classify_variant(int32_t n_traj, const int32_t *P, const float *const *R_pre,
                                          const float *const *R_post, const uint8_t *const *eligible,
                                          const commitkv_thresholds *thresholds, uint32_t variant,
                                          uint8_t *const *state_out, int32_t *const *cand_out,
                                          int32_t *n_cand_out, void *workspace, size_t workspace_bytes,
                                          cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Greedy joint test, Section 3.3, Eq. 11 and the inner loop of Algorithm 1.
 *
 * Per trajectory, with A = {} and the candidates in the order given:
 * accept cand[j] iff R+(A u {cand[j]}) <= tau_joint, where R+(A) is Eq. 6-7
 * with every token of A deleted at once, maximised over the selected
 * layers, the query heads and the post-commit window.  A rejection does not
 * end the scan.
 *
 *   post         the post-commit caches and windows used for stats.
 *   stats        host array of device float [M][Hq][W_t][d + 4], the
 *                stats_out of commitkv_page_effects on the same post caches
 *                and layer_mask.
 *   cand, n_cand host array of device int32 [>= n_cand] / device int32
 *                [n_traj] (the outputs of commitkv_classify).
 *   accepted_out host array of device uint8 [P_t]: 1 for pages accepted at
 *                this commit, else 0 (every entry written).
 *   step_R_out   NULL, or host array of device float [P_t]: step_R[j] =
 *                R+(A u {cand[j]}) for the A accepted before step j.
 * -------------------------------------------------------------------- */
commitkv_status commitkv_joint_test(const commitkv_shape *shape, int32_t n_traj,
                                    const commitkv_traj *post, const uint8_t *layer_mask,
                                    const float *const *stats, const int32_t *const *cand,
                                    const int32_t *n_cand, float tau_joint,
                                    uint8_t *const *accepted_out, float *const *step_R_out,
                                    void *workspace, size_t workspace_bytes,
                                    cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Compression checkpoint, Section 3.3, Eq. 12-13, applied by Eq. 4.
 *
 * Per trajectory: tokens of retired pages (D_c) are excluded.  Pending
 * pages that are not retired are ordered by decreasing pending_priority
 * (their pre-commit effect R-), then increasing page index, and the longest
 * prefix with at most pending_cap_pages pages and at most pending_tokens_BN
 * tokens is protected (N_j).  The remaining budget B - |N_j| is filled with
 * the other non-retired tokens of highest fill_score (ties: higher index
 * first), or with all of them if they fit.  I_j is written in ascending
 * order, and K, V and positions are gathered with it.
 *
 *   cache        the caches to compact (their pages index retired/pending).
 *   retired      host array of device uint8 [P_t].
 *   pending      host array of device int32 [n_pending_t] distinct page ids
 *                (entries may be NULL when n_pending_t = 0).
 *   n_pending    host int32 [n_traj].
 *   pending_priority  host array of device float [P_t]: the pre-commit effect
 *                R- of every page (the R_out of the pre-commit pass); only the
 *                entries of pending pages are read.
 *   fill_score   host array of device float [S_t] (NaN is a device input error).
 *   budget_B >= 0, 0 <= pending_tokens_BN <= budget_B, pending_cap_pages >= 0.
 *   idx_out      host array of device int32 [budget_B].
 *   n_idx_out    device int32 [n_traj] = |I_j|.
 *   k_out, v_out NULL, or host arrays of device [M][H][budget_B][d] dense
 *                buffers (dtype of the shape); rows >= |I_j| are not written.
 *   pos_out      NULL, or host array of device int32 [budget_B].
 * -------------------------------------------------------------------- */
commitkv_status commitkv_compact(const commitkv_shape *shape, int32_t n_traj,
                                 const commitkv_traj *cache, const uint8_t *const *retired,
                                 const int32_t *const *pending, const int32_t *n_pending,
                                 const float *const *pending_priority,
                                 const float *const *fill_score, int32_t budget_B,
                                 int32_t pending_tokens_BN, int32_t pending_cap_pages,
                                 int32_t *const *idx_out, int32_t *n_idx_out,
                                 void *const *k_out, void *const *v_out, int32_t *const *pos_out,
                                 void *workspace, size_t workspace_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Compression checkpoint in place, Section 3.3, Eq. 12-13 and Eq. 4.
 *
 * The selection of commitkv_compact (same arguments and rules, same idx_out
 * and n_idx_out), with the gather done inside the cache: K and V row I_j of
 * every (layer, KV head) slice moves to row j of the same slice, in the
 * cache's own layout and strides, and pos[j] = pos[I_j], for j < |I_j|.  The
 * cache's k, v and pos buffers are overwritten (their const in
 * commitkv_traj notwithstanding); rows and positions at and after |I_j| keep
 * stale values, and the caller's cache length becomes |I_j|.  No second
 * cache-sized buffer is needed.  Because I_j is strictly increasing with
 * I_j >= j, the rows are moved in ascending chunks, each read whole before
 * any of its rows is written.
 *
 *   cache        the caches to compact: k, v and pos must be non-NULL when
 *                S_t > 0 (else COMMITKV_ERR_INVALID_ARG).
 *   other arguments as for commitkv_compact.
 * -------------------------------------------------------------------- */
commitkv_status commitkv_compact_in_place(const commitkv_shape *shape, int32_t n_traj,
                                          const commitkv_traj *cache, const uint8_t *const *retired,
                                          const int32_t *const *pending, const int32_t *n_pending,
                                          const float *const *pending_priority,
                                          const float *const *fill_score, int32_t budget_B,
                                          int32_t pending_tokens_BN, int32_t pending_cap_pages,
                                          int32_t *const *idx_out, int32_t *n_idx_out, void *workspace,
                                          size_t workspace_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * commitkv_compact without a workspace.  The paper has no counterpart: this
 * entry point exists for callers that cannot allocate device memory where
 * they compact.  A serving engine usually reserves nearly all device memory
 * for its own KV pool at start-up, so a later cudaMalloc fails or has to go
 * through an allocator that a plug-in cannot reach, and cudaFree
 * synchronises the whole device.  This call allocates nothing: no
 * cudaMalloc, no cudaFree, no allocating library routine.
 *
 * Same selection, outputs and host-side checks as commitkv_compact (all
 * arguments but the workspace mean the same); its scratch is a fixed array
 * of COMMITKV_NOALLOC_SCRATCH_BYTES (4 MiB) that the library keeps on every
 * GPU that loads it, until the process exits.  Unlike the rest of this
 * header, this is state held by the library:
 *   - Limit: 256 + sum over trajectories of S_t rounded up to 256 must not
 *     exceed COMMITKV_NOALLOC_SCRATCH_BYTES (one trajectory of up to
 *     4,194,048 resident tokens); larger requests return
 *     COMMITKV_ERR_WORKSPACE with nothing launched.
 *   - Set-up: the first call with a given device current looks up the
 *     array's device address (cudaGetSymbolAddress, which may also load the
 *     library's device code on that device).  Make that first call before
 *     any stream capture on that device.  A failed look-up returns
 *     COMMITKV_ERR_CUDA.  The address is kept for the life of the process:
 *     it belongs to the device's primary context, so a process that
 *     destroys that context (cudaDeviceReset) must not call this entry
 *     point on that device afterwards.
 *   - Sharing: every call on a device uses the same array.  Calls whose
 *     work can overlap on the GPU (different streams, different host
 *     threads) race on it and give wrong results; serialise them, for
 *     example by issuing them all on one stream.
 *   - Device-side errors: each call clears the array's status word first,
 *     then the kernels record device-side input errors in it (as in the
 *     workspace of commitkv_compact).  status_out, if not NULL, is a device
 *     int32 that receives that word (a commitkv_status) once the call's work
 *     is done on `stream`.
 * -------------------------------------------------------------------- */
commitkv_status commitkv_compact_noalloc(const commitkv_shape *shape, int32_t n_traj,
                                         const commitkv_traj *cache,
                                         const uint8_t *const *retired,
                                         const int32_t *const *pending, const int32_t *n_pending,
                                         const float *const *pending_priority,
                                         const float *const *fill_score, int32_t budget_B,
                                         int32_t pending_tokens_BN, int32_t pending_cap_pages,
                                         int32_t *const *idx_out, int32_t *n_idx_out,
                                         void *const *k_out, void *const *v_out,
                                         int32_t *const *pos_out, int32_t *status_out,
                                         cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* COMMITKV_H */
