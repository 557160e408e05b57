/*
 * liblast: GB300 (sm_103a) kernels for LAST's edge-side token selection
 * ("The Last Query Token Guides Visual Token Pruning ...", Sec. 3.2-3.4).
 *
 * The path, per request b of a ragged batch:
 *   1. last_scores  Eq. 6-8: the attention row of the last query position
 *                   p* = P_b - 1 (a full softmax over all P_b keys, visual and
 *                   text, including p* itself) is summed over every layer and
 *                   q-head at the visual positions and normalised over the
 *                   visual span: w~_i = s_i / sum_j s_j.
 *   2. last_select  Eq. 9-11: importance-weighted greedy k-center selection
 *                   under cosine distance on the encoder features X, budget k_b.
 *   3. last_gather  Eq. 12: the kept rows of X in ascending index order.
 *   last_prune runs 1-3 back to back on one stream.
 *
 * Variants the paper evaluates beside the method:
 *   last_select_topk  Table 5: keep the k_b highest scores (no diversity term).
 *   last_scores_rows  Table 4: scores from the attention rows of several query
 *                     positions (First, Middle, All Mean) instead of p* alone.
 * Deployment aids without a counterpart in the paper: last_prune_host (the
 * whole path on host buffers, copies included), last_scores_noalloc (scoring
 * without a caller workspace) and last_check_bounded_wait (exercises the
 * reporting of an expired device wait).
 *
 * Conventions shared by every entry point
 *   - All tensors are DEVICE pointers (caller-allocated, e.g. torch tensors),
 *     except those of last_prune_host; the library allocates no device memory.  Scratch lives in a caller
 *     workspace of at least last_workspace_size() bytes (256-byte aligned).
 *   - The offset arrays in last_problem are HOST arrays; each call validates
 *     them and copies a small plan into the workspace on `stream`.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *     default stream).  Successive calls on one stream may reuse one
 *     workspace; concurrent calls need distinct workspaces.
 *   - No entry point may be captured into a CUDA graph: each call copies its
 *     plan from pageable host memory that it owns and releases on return, so
 *     a captured copy would replay freed memory.  Launch-bound callers batch
 *     requests into one call instead (one launch per kernel for the batch).
 *   - Argument errors are detected on the host before any launch; the call
 *     returns a status and touches no output.  Device-side checks set a flag in
 *     the workspace that last_poll() reports: an out-of-range caller index
 *     (last_gather) or an expired bounded wait (every device wait has an
 *     iteration limit, so no call can hang the GPU).
 *   - The selection is deterministic and, given the same w~, bit-identical to
 *     the canonical fp32 arithmetic below on every run:
 *       dot(a,b): lane l in 0..31 owns coordinate groups g = l, l+32, l+64, ...
 *                 of 8 consecutive coordinates; it accumulates them in
 *                 increasing coordinate order with one fp32 fma each; the 32
 *                 lane sums are combined by an xor butterfly (offsets 16..1).
 *       r_i = dot(x_i,x_i) > 0 ? 1/sqrt(dot(x_i,x_i)) : 0  (IEEE div, sqrt)
 *       delta_i = min(delta_i, 1 - (dot(x_i,x_j) * r_i) * r_j),  p_i = w~_i * delta_i
 *       argmax ties go to the lowest index; selected tokens are excluded.
 *
 * Layouts (row-major, no padding)
 *   q      [batch][num_layers][num_q_heads][head_dim]      query of p* per layer
 *   k      [num_layers][cu_seqlens[batch]][num_kv_heads][head_dim]   packed keys
 *   x      [cu_vis[batch]][feat_dim]                       encoder features
 *   w      [cu_vis[batch]] fp32                            w~ (Eq. 8)
 *   idx    [cu_keep[batch]] int32, request-local, ascending per request
 *   x_out  [cu_keep[batch]][feat_dim], same dtype as x
 *   q-head h reads kv-head h / (num_q_heads / num_kv_heads).
 *
 * Limits (LAST_ERR_UNSUPPORTED beyond them; last_error_message() says which):
 *   scoring   G = num_q_heads / num_kv_heads in 1..8; head_dim * elem_bytes a
 *             multiple of 16; num_q_heads * head_dim fp32 values of q plus one
 *             chunk of logits within 100 KB of shared memory (e.g. up to 128
 *             q-heads of 128); num_layers * num_q_heads <= 6144.
 *   selection feat_dim a multiple of 8, at most 2048; the greedy selection
 *             (last_select, last_prune) keeps per-token state of a request in
 *             the shared memory of up to 16 clustered CTAs: about 120K tokens
 *             at feat_dim 64, 72K at bf16 feat_dim 2048, 13K at fp32 feat_dim
 *             2048.  A call of at most 4 requests past that bound runs them on
 *             every SM of the GPU instead (per-token state spread over all
 *             CTAs: millions of tokens); a call of more requests returns
 *             LAST_ERR_UNSUPPORTED for them.  Top-k and the gather have no
 *             such bound.
 */
#ifndef LAST_H_
#define LAST_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  LAST_OK = 0,
  LAST_ERR_INVALID_ARG = 1,          /* shape/offset/pointer check failed (host) */
  LAST_ERR_UNSUPPORTED = 2,          /* valid but outside the compiled limits */
  LAST_ERR_WORKSPACE_TOO_SMALL = 3,  /* ws_bytes < last_workspace_size() */
  LAST_ERR_CUDA = 4,                 /* a CUDA runtime call failed */
  LAST_ERR_DEVICE_INDEX = 5,         /* last_poll: a caller index was out of range */
  LAST_ERR_TIMEOUT = 6               /* last_poll: a bounded device wait expired; outputs invalid */
} last_status;

typedef enum { LAST_DTYPE_F32 = 0, LAST_DTYPE_BF16 = 1 } last_dtype;

/* Problem description (Eq. 2, Eq. 5-7).  Request b has P_b = cu_seqlens[b+1] -
 * cu_seqlens[b] positions whose last one is the query token p*; its N_b =
 * cu_vis[b+1] - cu_vis[b] visual tokens occupy positions vis_start[b] ..
 * vis_start[b] + N_b - 1 (which must end before p*); it keeps
 * k_b = cu_keep[b+1] - cu_keep[b] tokens, 0 <= k_b <= N_b (Eq. 2; see
 * last_budget).  All four arrays are host memory, read during the call only. */
typedef struct {
  int32_t batch;
  int32_t num_layers;      /* L: layers whose rows are summed (Eq. 7) */
  int32_t num_q_heads;     /* H in Eq. 7 */
  int32_t num_kv_heads;
  int32_t head_dim;
  int32_t feat_dim;        /* d_v in Eq. 1 */
  int32_t dtype;           /* last_dtype of q, k and x */
  float softmax_scale;     /* <= 0 selects 1/sqrt(head_dim) */
  const int32_t *cu_seqlens; /* [batch+1], cu_seqlens[0] == 0, non-decreasing */
  const int32_t *vis_start;  /* [batch] */
  const int32_t *cu_vis;     /* [batch+1] */
  const int32_t *cu_keep;    /* [batch+1] */
} last_problem;

/* Bytes of device workspace the entry points below need for `p`, except
 * last_scores_rows and last_prune_host, which are sized by
 * last_scores_rows_workspace_size and last_host_workspace_size.
 * Returns LAST_ERR_INVALID_ARG / LAST_ERR_UNSUPPORTED for a bad problem. */
last_status last_workspace_size(const last_problem *p, size_t *bytes);

/* Eq. 6-8.  w_out [cu_vis[batch]] fp32 receives w~ (sums to 1 per request). */
last_status last_scores(const last_problem *p, const void *q, const void *k, float *w_out,
                        void *ws, size_t ws_bytes, void *stream);

/* Eq. 9-12.  w [cu_vis[batch]] fp32 (e.g. from last_scores); idx_out
 * [cu_keep[batch]] receives sort(S_K) per request, request-local.  When x_out
 * is not NULL the kept rows are also written there (the fused form of
 * last_gather). */
last_status last_select(const last_problem *p, const float *w, const void *x,
                        int32_t *idx_out, void *x_out, void *ws, size_t ws_bytes,
                        void *stream);

/* Table 5, "LAST (Top-k)": the selection variant without the diversity term.
 * idx_out [cu_keep[batch]] receives, per request and in ascending order, the
 * k_b indices of highest w~ (ties between equal scores go to the lower index;
 * -0 equals +0).  When x_out is not NULL the kept rows of x are also written
 * there (x is then required; feat_dim a positive multiple of 8); x may be NULL
 * otherwise.  The problem's layer/head fields are not used.  Same ownership,
 * stream and error rules as last_select.  w must hold no NaN: the kept set is
 * then unspecified (but still k_b distinct valid indices). */
last_status last_select_topk(const last_problem *p, const float *w, const void *x,
                             int32_t *idx_out, void *x_out, void *ws, size_t ws_bytes,
                             void *stream);

/* Table 4 (attention sources: First, Middle, All Mean): Eq. 6-8 with the
 * attention rows of several query positions per request instead of p* alone.
 * Request b's query rows are cu_rows[b] .. cu_rows[b+1]-1 (HOST array, length
 * batch+1, cu_rows[0] = 0, at least one row per request); row r sits at the
 * request-local position row_pos[r] (HOST array), which must lie after the visual
 * span: vis_start[b] + N_b <= row_pos[r] <= P_b - 1; row r's softmax runs over the
 * keys 0 .. row_pos[r] (causal).  q_rows [cu_rows[batch]][num_layers][num_q_heads]
 * [head_dim] holds one query vector per row, layer and q-head; k as for
 * last_scores.  w_out [cu_vis[batch]] receives the visual probabilities summed
 * over rows, layers and q-heads and normalised per request (a mean over the rows
 * gives the same w~).  With one row per request (First, Middle, Last) the row
 * at position pos is the last-row computation on keys 0 .. pos, and the call
 * runs last_scores' kernels on the requests cut there (when G <= 8).
 * Limits: bf16 only; head_dim 64, 128, 192 or 256; rows x
 * (num_q_heads / num_kv_heads) <= 256 and rows x layers x q-heads <= 6144 per
 * request.  The workspace is sized by last_scores_rows_workspace_size. */
last_status last_scores_rows_workspace_size(const last_problem *p, const int32_t *cu_rows,
                                            const int32_t *row_pos, size_t *bytes);
last_status last_scores_rows(const last_problem *p, const int32_t *cu_rows,
                             const int32_t *row_pos, const void *q_rows, const void *k,
                             float *w_out, void *ws, size_t ws_bytes, void *stream);

/* Eq. 12.  x_out[r] = x[cu_vis[b] + idx[r]] for r in request b's output range.
 * An index outside [0, N_b) leaves its row unwritten and makes last_poll
 * return LAST_ERR_DEVICE_INDEX.  Any feat_dim that is a positive multiple of 8
 * is accepted (the selection's own feat_dim <= 2048 limit does not apply); the
 * workspace carries the plan and the device error word. */
last_status last_gather(const last_problem *p, const void *x, const int32_t *idx,
                        void *x_out, void *ws, size_t ws_bytes, void *stream);

/* The whole path: scores, selection, ordered gather.  w_out may be NULL (w~
 * is then kept in the workspace); x_out may be NULL (indices only). */
last_status last_prune(const last_problem *p, const void *q, const void *k, const void *x,
                       float *w_out, int32_t *idx_out, void *x_out,
                       void *ws, size_t ws_bytes, void *stream);

/* last_prune on HOST buffers: q, k and x are read from host memory and idx_out,
 * x_out (may be NULL) and w_out (may be NULL) are written to host memory, with
 * the layouts above.  The call enqueues on `stream` the host-to-device copies of
 * q, K and X into the device workspace, the whole path, and the device-to-host
 * copies of the results, and returns; the host buffers must stay valid and
 * unchanged until the stream has passed the call.  Pinned (page-locked) host
 * memory keeps every copy asynchronous, so a caller alternating two workspaces
 * on two streams overlaps one call's copies with another's kernels; pageable
 * memory works but the copies then block the host.  The device workspace holds
 * the plan and device copies of q, K, X, w~, the indices and the kept rows:
 * last_host_workspace_size() bytes, 256-byte aligned. */
last_status last_host_workspace_size(const last_problem *p, size_t *bytes);
last_status last_prune_host(const last_problem *p, const void *q_host, const void *k_host,
                            const void *x_host, float *w_out_host, int32_t *idx_out_host,
                            void *x_out_host, void *ws, size_t ws_bytes, void *stream);

/* last_scores without a caller workspace (the paper has no counterpart: this is
 * a deployment aid).  For callers that cannot allocate device memory at run time
 * -- e.g. an edge service that reserves all of its device memory at start-up and
 * treats later allocations as failures, or a program without a device allocator
 * of its own.  Same inputs, outputs and results as last_scores; the scratch lives
 * in a fixed 16 MiB array inside the library, held on every GPU that loads the
 * library until the process exits.  Each call looks up that array's device
 * address (cudaGetSymbolAddress, cached per device after the first call) with
 * the device current; like every entry point it cannot be captured into a CUDA
 * graph (the plan is copied from host memory the call releases).  All calls share
 * the array and it keeps the last call's contents: calls whose executions
 * overlap on the GPU race on it.  A problem needing more than 16 MiB of scratch
 * (last_workspace_size) returns LAST_ERR_UNSUPPORTED.  Allocates nothing. */
last_status last_scores_noalloc(const last_problem *p, const void *q, const void *k,
                                float *w_out, void *stream);

/* Diagnostic (no counterpart in the paper): runs one device-side bounded wait that
 * nothing completes, with a short iteration limit, so that the next last_poll on
 * `ws` (at least 256 bytes) returns LAST_ERR_TIMEOUT.  It exercises the path every
 * device wait of the library takes when a wait expires, without hanging or
 * faulting the GPU. */
last_status last_check_bounded_wait(void *ws, void *stream);

/* Synchronises `stream`, then reports the device-side flags of the last call
 * that used `ws`: LAST_OK, LAST_ERR_DEVICE_INDEX, or LAST_ERR_TIMEOUT (a wait
 * on an asynchronous copy gave up after its iteration limit instead of hanging;
 * the outputs of that call are then invalid). */
last_status last_poll(const void *ws, void *stream);

/* Eq. 2: k = ceil(num * n_vis / den) in exact integer arithmetic
 * (rho = num/den); -1 for n_vis < 0, num < 0 or den <= 0. */
int32_t last_budget(int32_t n_vis, int32_t num, int32_t den);

const char *last_status_string(last_status s);

/* Human-readable detail of the last non-OK status returned on this thread. */
const char *last_error_message(void);

#ifdef __cplusplus
}
#endif

#endif /* LAST_H_ */
