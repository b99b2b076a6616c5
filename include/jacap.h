/*
 * jacap.h - C ABI of libjacap: the prefill-time KV-cache eviction pass of
 * Jacap (Jacobian-capacity-aware eviction), Algorithm 1 of Sec. 3.4, on one
 * NVIDIA GB300 (sm_103a).
 *
 * For every unit = (request s, layer l, KV head g) with n_s cached tokens the
 * pass computes, per Algorithm 1 and Eqs. 8-10:
 *
 *   mu_h, lambda_h  mean and per-channel variance of the last w queries of
 *                   every query head h served by KV head g (Sec. 3.4, last
 *                   paragraph; diagonal Lambda_Q as in App. B.2);
 *   alpha_bar_h,i   softmax_i(k_i . mu_h / (tau sqrt(d)))  over all n_s tokens;
 *   w_i             (1/d) sum_h [alpha_bar_h,i (1 - alpha_bar_h,i)]^2 * kappa_h,i,
 *                   kappa_h,i = sum_c lambda_h,c k_i,c^2          (Eq. 8);
 *   A               I + sum_i w_i v_i v_i^T                     (Eq. 9);
 *   score_i         w_i v_i^T A^{-1} v_i                         (Eq. 10);
 *   C               the budget B highest scores (Alg. 1 step 5), ties to the
 *                   lower token index, listed in ascending order;
 *   K_out, V_out    the retained rows {(k_i, v_i)}_{i in C} (Sec. 3.1).
 *
 * Query head h is served by KV head h / (num_q_heads / num_kv_heads).
 *
 * Conventions for every entry point
 *  - Pointers named *_host are host memory; every other data pointer is device
 *    memory on the current CUDA device. The caller owns all memory; the library
 *    allocates nothing and keeps no mutable global state (the one exception is
 *    the static scratch of jacap_score_static).
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *    All work is enqueued asynchronously on it; nothing synchronises except
 *    jacap_device_status() and jacap_evict_host().
 *  - Host-side validation happens before anything is enqueued; on any error
 *    status nothing has been launched. A failed launch returns JACAP_ERR_CUDA.
 *  - Problems only the device can see (a malformed cu_seqlens array, a
 *    non-finite input or intermediate, a bounded wait that expired) are
 *    recorded in the status word kept at the start of the workspace; kernels
 *    that find it set return without work. Read it with jacap_device_status().
 *    No kernel traps or asserts.
 *  - Calls on different streams are safe when they use different workspaces.
 */
#ifndef JACAP_H
#define JACAP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  JACAP_OK = 0,
  JACAP_ERR_INVALID_ARG = 1, /* bad pointer, size, stride, alignment or layout   */
  JACAP_ERR_UNSUPPORTED = 2, /* head_dim != 128, group size above 8,
                                ridge = 0, or a device older than sm_103a       */
  JACAP_ERR_WORKSPACE = 3,   /* workspace too small or misaligned               */
  JACAP_ERR_CUDA = 4,        /* a CUDA runtime/driver call or launch failed     */
  JACAP_ERR_NONFINITE = 5,   /* (device) NaN/Inf met in an input or intermediate */
  JACAP_ERR_TIMEOUT = 6      /* (device) a bounded wait expired; the kernel quit */
} jacap_status;

typedef enum { JACAP_F32 = 0, JACAP_BF16 = 1 } jacap_dtype;

/*
 * Cache layout (Sec. 3.1: the KV cache {(k_i, v_i)} of every layer and head).
 *
 *  K, V    element (l, g, t, c) at  l*kv_stride_layer + g*kv_stride_head
 *          + t*kv_stride_token + c  (elements; channel c contiguous), for
 *          t in [0, total_tokens). Request s owns t in [cu[s], cu[s+1]).
 *  Q_win   the last `window` queries of every request, layer and query head:
 *          element (s, l, h, j, c) at s*q_stride_seq + l*q_stride_layer
 *          + h*q_stride_head + j*q_stride_pos + c.
 *  dtype   type of K, V and Q_win (all three share it).
 *
 * Requirements (else JACAP_ERR_INVALID_ARG / _UNSUPPORTED): head_dim == 128;
 * num_q_heads % num_kv_heads == 0 with a ratio G = num_q_heads / num_kv_heads
 * of 1 to 8 (e.g. G = 4 for Llama-3-8B, 5 for Qwen3-14B, 7 for Nemotron-7B;
 * larger groups give JACAP_ERR_UNSUPPORTED); window >= 1;
 * every stride a multiple of 8 elements (16-byte rows) and K, V, Q_win 16-byte
 * aligned; kv_stride_token >= head_dim; num_seqs >= 1; total_tokens >= 1 and
 * < 2^31; max_seqlen >= every n_s. cu_seqlens must satisfy cu[0] = 0,
 * cu[s] <= cu[s+1], cu[num_seqs] = total_tokens and n_s >= 1; the device
 * checks this and reports JACAP_ERR_INVALID_ARG through the status word.
 */
typedef struct {
  int32_t num_seqs;
  const int32_t* cu_seqlens; /* device, [num_seqs + 1] token offsets           */
  int32_t max_seqlen;        /* host upper bound of n_s                        */
  int64_t total_tokens;      /* N_tot = cu_seqlens[num_seqs]                   */
  int32_t num_layers;
  int32_t num_q_heads;
  int32_t num_kv_heads;
  int32_t head_dim;          /* d_k = d_o = 128                                */
  int32_t window;            /* w: queries per head used for (mu_Q, Lambda_Q)   */
  jacap_dtype dtype;
  int64_t kv_stride_layer, kv_stride_head, kv_stride_token;
  int64_t q_stride_seq, q_stride_layer, q_stride_head, q_stride_pos;
} jacap_layout;

/*
 * Method switches. Defaults {10.0f, 1, 1, 0, 0, 0, 0}:
 *  tau            temperature of the pool softmax (Sec. 3.4; Sec. 4.4 reports
 *                 the best accuracy near 10). Must be finite and > 0.
 *  weight_div_dk  1: keep the 1/d_k factor of Eq. 8; 0: drop it (Alg. 1 step 2
 *                 prints the weight without it).
 *  ridge          must be 1: the identity term of Eq. 9. (0 is an oracle-only
 *                 variant and returns JACAP_ERR_UNSUPPORTED.)
 *  cov_unbiased   0: lambda = population variance over the window (divide by
 *                 w); 1: divide by w - 1 (needs window >= 2).
 *  linear_weighting  0: the softmax-aware weight of Eq. 8; 1: the linear
 *                 surrogate S_C = I that App. A contrasts Jacap with, i.e.
 *                 rho_i = 1 and w_i = (1/d) sum_h kappa_h,i (a CapKV-style
 *                 weight; the logits and softmax statistics are then unused).
 *  full_covariance  0: the diagonal Lambda_Q of App. B.2 (the method as the
 *                 paper runs it); 1: the full covariance of the window queries,
 *                 kappa_h,i = (1/w) sum_j ((q_h,j - mu_h) . k_i)^2 (1/(w-1) with
 *                 cov_unbiased), the O(N d^2) variant of App. B.2. bf16 caches
 *                 with window in {8, 16, 32, 64} and G * window <= 128 use the
 *                 tensor cores inside the K pass (K is still read once); other
 *                 shapes and float32 caches a much slower CUDA-core kernel
 *                 after the K pass, which reads K a second time.
 *  schedule       how the Gram (Eq. 9), the factor of A and the scores (Eq. 10)
 *                 are run; every choice computes the same quantities (the
 *                 partial Grams may be summed in another order, within the
 *                 float32 rounding of the pass). 0: automatic (currently
 *                 the separate kernels, the faster schedule on GB300 for
 *                 every shape measured); 1: three separate kernels, each over
 *                 the whole cache; 2: fused, one persistent cooperative
 *                 launch whose CTAs take the three roles and hand each unit
 *                 from one role to the next as soon as it is ready, so that
 *                 part of the score role's read of V hits L2 (bf16 caches
 *                 only; float32 caches and jacap_score_out use separate
 *                 kernels whatever the value). Other values:
 *                 JACAP_ERR_INVALID_ARG.
 * Callers that zero-initialise the trailing fields get the method with the
 * automatic schedule.
 */
typedef struct {
  float tau;
  int32_t weight_div_dk;
  int32_t ridge;
  int32_t cov_unbiased;
  int32_t linear_weighting;
  int32_t full_covariance;
  int32_t schedule;
} jacap_params;

/* The schedule (jacap_params.schedule) that jacap_score, jacap_score_timed,
 * jacap_score_stats and jacap_evict_host would run for `layout` and `params`
 * on the current device: 1 (separate kernels) or 2 (fused). With the fused
 * schedule, roles[0..3] (if not NULL) receive its CTAs per role (factor, Gram,
 * score) and the V tiles per Gram work item loaded with the L2 evict_last
 * policy; zeros otherwise. Returns the schedule, or -(jacap_status) for an
 * invalid layout or params or an unsupported device. No GPU work. */
int32_t jacap_schedule_info(const jacap_layout* layout, const jacap_params* params, int32_t* roles);

/* Bytes of device workspace jacap_score/jacap_select need for `layout`
 * (budget is accepted for forward compatibility and may be any value >= 1).
 * Returns 0 if the layout is invalid. The workspace must be 256-byte aligned;
 * it holds the status word and every intermediate (mu, lambda, logits, kappa,
 * w, partial Grams, the factor of A): about 36 bytes per token and KV head of
 * every layer (G = 4) plus 192 KB per unit. Units are independent, so a caller
 * short of memory can run the calls over groups of layers (a layout with
 * num_layers = the group size and K, V, Q_win pointers advanced to the group's
 * first layer) with one workspace sized for a group. */
size_t jacap_workspace_size(const jacap_layout* layout, int32_t budget);

/*
 * Scores of every cached token (Algorithm 1 steps 1-4; Eqs. 8-10).
 *  q_win, k, v  device, layout above.
 *  scores       device float32 [num_layers][num_kv_heads][total_tokens]:
 *               score of token t of plane (l, g); r_i of Eq. 10.
 *  ws, ws_bytes device workspace of at least jacap_workspace_size() bytes.
 * Enqueues: a planning kernel (which also resets the status word), query
 * statistics, a streaming pass
 * over K (logits, kappa, softmax statistics), the merge of each unit's softmax
 * normaliser, the Eq. 8 weights (inside the weighted-Gram pass for bf16
 * caches), the weighted-Gram pass over V (tensor cores for bf16), the Cholesky
 * factor and inverse of A, and the quadratic forms (the last three as one
 * launch with the fused schedule).
 */
jacap_status jacap_score(const jacap_layout* layout, const jacap_params* params,
                         const void* q_win, const void* k, const void* v, float* scores,
                         void* ws, size_t ws_bytes, void* stream);

/*
 * jacap_score with timing hooks, for benchmarks: identical work, plus
 * cudaEventRecord(events[i], stream) before the i-th kernel of the pass and
 * events[num_events - 1] after the last one. `events` holds cudaEvent_t
 * handles (as void*) created by the caller; num_events must be 0 (no hooks)
 * or JACAP_SCORE_KERNELS + 1. Kernel order: plan, query statistics, K pass,
 * weights, Gram, factor, scores. The weights slot holds the merge of each
 * unit's softmax normaliser and, for float32 caches, the Eq. 8 weights (with
 * bf16 caches the Gram kernel computes them itself); with full_covariance the
 * K-pass slot also holds the CUDA-core kappa kernel when that one runs. With
 * the fused schedule (jacap_params.schedule) the Gram slot holds the one launch
 * that runs the Gram, the factor and the scores, and the factor and scores
 * slots are empty (their events are recorded back to back).
 */
#define JACAP_SCORE_KERNELS 7
jacap_status jacap_score_timed(const jacap_layout* layout, const jacap_params* params,
                               const void* q_win, const void* k, const void* v, float* scores,
                               void* ws, size_t ws_bytes, void* stream,
                               void* const* events, int32_t num_events);

/*
 * jacap_score with the true output directions u_i = W v_i of Sec. 3.1 (the
 * other entry points use the proxy u_i = v_i of Sec. 3.4), plus optional
 * timing hooks as in jacap_score_timed.
 *  out_factor  device float32 [num_layers][num_kv_heads][128][128], row-major,
 *              16-byte aligned, or NULL (then identical to jacap_score_timed):
 *              per plane a matrix F with F^T F = W^T W for the plane's output
 *              map W (d_o x 128; e.g. the R of a QR factorisation of W; how the
 *              W_O slices of the G query heads sharing a KV head form W is the
 *              caller's choice). The capacity matrix I + sum w u u^T (d_o x d_o,
 *              Eq. 9) reduces exactly to M = I + F G F^T, and
 *              r_i = w_i ||L_M^{-1} F v_i||^2 (Eq. 10).
 * Intermediates (jacap_workspace_offsets): gram is still G = sum w v v^T;
 * chol_inv holds T = L_M^{-1} F (a full matrix).
 */
jacap_status jacap_score_out(const jacap_layout* layout, const jacap_params* params,
                             const void* q_win, const void* k, const void* v,
                             const float* out_factor, float* scores,
                             void* ws, size_t ws_bytes, void* stream,
                             void* const* events, int32_t num_events);

/*
 * jacap_score for callers that cannot allocate device memory (the paper has no
 * counterpart; this is a deployment convenience). The workspace is a fixed
 * library-owned array of JACAP_STATIC_SCRATCH_BYTES in static device memory,
 * one per device; no call allocates. The work and results are those of
 * jacap_score with a caller workspace.
 *  - Layouts whose jacap_workspace_size() exceeds JACAP_STATIC_SCRATCH_BYTES
 *    are refused with JACAP_ERR_WORKSPACE before any CUDA call; an invalid
 *    or unsupported layout gives the status jacap_score would.
 *  - Set-up: the first call on a device (that device current) looks up the
 *    scratch address with cudaGetSymbolAddress, which loads the module's
 *    static memory, and caches it with the id of the current CUDA context; a
 *    call that finds another context current (after cudaDeviceReset, or a
 *    primary context released and retained again) looks it up afresh. Make
 *    the first call on each device before capturing a stream into a graph.
 *  - Footprint: every device context that loads libjacap's module holds the
 *    JACAP_STATIC_SCRATCH_BYTES array resident until the context ends, whether
 *    or not it ever calls this function (with CUDA_MODULE_LOADING=EAGER from
 *    the library's first use; with lazy loading once the module is loaded).
 *  - scratch_out (may be NULL) receives the scratch's device address; it is
 *    laid out as a workspace (see jacap_workspace_offsets) and can be passed
 *    as `ws` to jacap_select and jacap_device_status. Its status word is reset
 *    by every call; nothing else needs to start at zero.
 *  - Every call on a device shares that one scratch: calls (and any use of the
 *    returned address) that overlap in time race and corrupt each other's
 *    results. Serialise them, e.g. on one stream.
 */
#define JACAP_STATIC_SCRATCH_BYTES ((size_t)64 << 20)
jacap_status jacap_score_static(const jacap_layout* layout, const jacap_params* params,
                                const void* q_win, const void* k, const void* v, float* scores,
                                void* stream, void** scratch_out);

/*
 * TOP-B per unit (Algorithm 1 step 5). Reads `scores` as written by
 * jacap_score (non-negative float32). For unit (l, g, s):
 *  idx   device int32 [num_layers][num_kv_heads][num_seqs][budget]: the chosen
 *        token positions RELATIVE to the request start cu[s], ascending; ties
 *        in score go to the lower position; when n_s < budget all n_s
 *        positions are listed and the rest is -1.
 *  kept  device int32 [num_seqs]: min(n_s, budget).
 * budget >= 1. ws: the workspace used by jacap_score (its status word is
 * honoured and updated).
 */
jacap_status jacap_select(const jacap_layout* layout, const float* scores, int32_t budget,
                          int32_t* idx, int32_t* kept, void* ws, size_t ws_bytes, void* stream);

/*
 * Retained cache Z_C (Sec. 3.1): for every unit, copies rows idx[r] (relative
 * to cu[s]) of K and V, bit for bit, into
 *  k_out, v_out  device, dtype of the cache, dense [num_layers][num_kv_heads]
 *                [num_seqs][budget][head_dim]; rows whose idx is -1 are zeroed.
 * idx as produced by jacap_select; an entry that is -1 or not a position of
 * the request yields a zero row (no index value reads out of bounds). k_out and
 * v_out must be 16-byte aligned and
 * must not overlap k or v.
 */
jacap_status jacap_compact(const jacap_layout* layout, const void* k, const void* v,
                           const int32_t* idx, int32_t budget, void* k_out, void* v_out,
                           void* stream);

/*
 * jacap_select followed by jacap_compact in one launch (Algorithm 1 step 5 and
 * the retained cache Z_C of Sec. 3.1): each unit's kept rows are copied as
 * soon as its positions are known. Arguments, layouts, results and error
 * behaviour are those of the two calls: idx and kept as from jacap_select,
 * k_out and v_out as from jacap_compact with that idx (zero rows where idx is
 * -1). k, v, k_out and v_out must be 16-byte aligned and k_out, v_out must
 * overlap neither k, v, scores nor idx.
 */
jacap_status jacap_select_compact(const jacap_layout* layout, const float* scores, int32_t budget,
                                  int32_t* idx, int32_t* kept, const void* k, const void* v,
                                  void* k_out, void* v_out, void* ws, size_t ws_bytes, void* stream);

/*
 * Decoding-stage eviction (the paper's decoding experiments, Sec. 4; Sec. 3.4,
 * last paragraph: during decoding mu_Q and Lambda_Q are estimated from the
 * historical queries). Three calls on top of the ones above:
 *
 * jacap_stats_update merges new queries into running query statistics.
 *  q_new   device, the layout's Q_win strides and dtype; `window` (>= 1) is
 *          the number of new queries per (request, layer, query head).
 *  stats   device float32 [num_seqs][num_layers][num_q_heads][2][128],
 *          16-byte aligned: per channel the mean of every query merged so far
 *          and M2, the sum of their squared deviations from that mean.
 *  counts  device int32 [num_seqs][num_layers][num_q_heads]: how many queries
 *          have been merged (a negative count is read as 0).
 *  reset   1: discard the previous statistics and start from q_new;
 *          0: merge (Chan-Golub-LeVeque pairwise update, float32).
 * The caller owns both arrays. Only the layout's sizes, dtype and Q strides
 * are used (it must still pass the checks of jacap_score).
 */
jacap_status jacap_stats_update(const jacap_layout* layout, const void* q_new, int32_t reset,
                                float* stats, int32_t* counts, void* stream);

/*
 * jacap_score_timed with the query statistics taken from running statistics
 * (as kept by jacap_stats_update) instead of a query window: per query head
 * mu = mean and lambda = M2 / n (M2 / (n - 1) with cov_unbiased), n = counts.
 * q strides are unused and `window` only sizes the workspace (1 suffices).
 * A count below 1 (below 2 with cov_unbiased) records JACAP_ERR_INVALID_ARG in
 * the status word. full_covariance must be 0 (no running d x d covariance is
 * kept): 1 returns JACAP_ERR_UNSUPPORTED. The outputs and the other arguments
 * are those of jacap_score_timed.
 */
jacap_status jacap_score_stats(const jacap_layout* layout, const jacap_params* params,
                               const float* stats, const int32_t* counts,
                               const void* k, const void* v, float* scores,
                               void* ws, size_t ws_bytes, void* stream,
                               void* const* events, int32_t num_events);

/*
 * The retained cache in place: for every unit the kept rows idx[0 .. kept - 1]
 * (relative to cu[s], as produced by jacap_select) of K and V end up, bit for
 * bit, in rows 0 .. kept - 1 of the request's token range; rows from kept on
 * are left as they were (free for the next tokens). kept = min(n_s, budget).
 *  k, v  device, the layout; written in place.
 *  pos   device int32 or NULL: a per-token tag (e.g. the original position)
 *        moved with the rows, laid out like K with one int32 per token row:
 *        tag (l, g, t) at l*(kv_stride_layer/kv_stride_token)
 *        + g*(kv_stride_head/kv_stride_token) + t. For a dense K
 *        [num_layers][num_kv_heads][total_tokens][128] that is a dense
 *        [num_layers][num_kv_heads][total_tokens]; with pos the layer and head
 *        strides must be multiples of the token stride (else
 *        JACAP_ERR_INVALID_ARG).
 *  preserve_order
 *        1: row r receives idx[r] (ascending order, as jacap_compact); up to
 *           `kept` rows move, in chunks that are read whole before any row of
 *           the chunk is written, which cannot overwrite a row still to be
 *           read because idx[r] >= r.
 *        0: hole filling: kept rows below `kept` stay in place and the kept
 *           rows at or above `kept` move, in ascending order, into the evicted
 *           rows below `kept`, in ascending order; at most n_s - kept rows
 *           move (the order of a cache does not matter to attention once the
 *           positions are encoded in the keys; `pos` keeps them).
 *  ws    the workspace of jacap_score for this layout (status word).
 * The kept positions of every unit must ascend strictly within [0, n_s) (as
 * jacap_select emits them); a unit where they do not is left untouched and
 * JACAP_ERR_INVALID_ARG is recorded in the status word. Units run
 * concurrently.
 */
jacap_status jacap_compact_inplace(const jacap_layout* layout, void* k, void* v, int32_t* pos,
                                   const int32_t* idx, int32_t budget, int32_t preserve_order,
                                   void* ws, size_t ws_bytes, void* stream);

/*
 * jacap_select followed by jacap_compact_inplace in one launch: each unit's
 * kept rows are moved in place as soon as its positions are selected.
 * Arguments, layouts, results and error behaviour are those of the two calls
 * (idx and kept as from jacap_select; k, v and pos as after
 * jacap_compact_inplace with that idx and preserve_order). The positions
 * come from the selection itself, so no unit is refused for them. Hole filling
 * (preserve_order = 0) runs inside the selection kernel; the ascending-order
 * compaction, which moves every kept row, is enqueued as a second launch.
 */
jacap_status jacap_select_compact_inplace(const jacap_layout* layout, const float* scores, int32_t budget,
                                          int32_t* idx, int32_t* kept, void* k, void* v, int32_t* pos,
                                          int32_t preserve_order, void* ws, size_t ws_bytes, void* stream);

/*
 * Eviction of a cache held in host memory (an offloaded KV cache, Sec. 3.1):
 * the whole pass of jacap_score + jacap_select (+ jacap_compact) on caches that
 * stay in host memory, with the kept positions (and optionally the retained
 * rows Z_C) written back to host memory. Unlike the other entry points it
 * returns only when everything is done (both streams synchronised).
 *
 * The layers travel in groups of `group_layers` through two device buffers
 * carved from `dev_buf`: while group g is scored, selected and compacted on
 * `stream`, group g + 1 is copied host -> device on `copy_stream`, so the
 * device holds at most two groups and the pass overlaps the copies.
 *  layout       as for jacap_score, except: cu_seqlens is a HOST pointer
 *               (copied into dev_buf), and the host arrays must be dense:
 *               K, V [num_layers][num_kv_heads][total_tokens][128] and Q_win
 *               [num_seqs][num_layers][num_q_heads][window][128] (strides as
 *               those shapes give), else JACAP_ERR_INVALID_ARG.
 *  q_win_host, k_host, v_host  host memory; page-locked (cudaHostAlloc /
 *               cudaHostRegister) for the copies to overlap the pass.
 *  out_factor   device, optional: the per-plane factors of jacap_score_out
 *               (NULL: u = v).
 *  idx_host     host int32 [num_layers][num_kv_heads][num_seqs][budget], as
 *               jacap_select writes idx; kept_host host int32 [num_seqs].
 *  k_out_host, v_out_host  host [num_layers][num_kv_heads][num_seqs][budget][128]
 *               in the cache dtype, as jacap_compact writes them; both NULL to
 *               skip the rows (positions only), else both non-NULL.
 *  dev_buf      device memory the caller owns, 1024-byte aligned, at least
 *               jacap_host_buffer_size() bytes; holds the two group buffers,
 *               the workspace and the group outputs. The library allocates no
 *               device memory; it creates and destroys four CUDA events.
 *  copy_stream  a second stream for the host -> device copies; NULL (or equal
 *               to `stream`) runs everything in order on `stream`.
 * Returns the first error of the host checks, of a CUDA call, or of a group's
 * device status word (JACAP_ERR_INVALID_ARG, _NONFINITE, _TIMEOUT as from
 * jacap_device_status).
 */
size_t jacap_host_buffer_size(const jacap_layout* layout, int32_t budget, int32_t group_layers,
                              int32_t copy_rows);
jacap_status jacap_evict_host(const jacap_layout* layout, const jacap_params* params, int32_t budget,
                              int32_t group_layers, const void* q_win_host, const void* k_host,
                              const void* v_host, const float* out_factor, int32_t* idx_host,
                              int32_t* kept_host, void* k_out_host, void* v_out_host, void* dev_buf,
                              size_t dev_bytes, void* stream, void* copy_stream);

/* Synchronises `stream`, then reads the workspace status word: JACAP_OK or the
 * first device-side error recorded since the last jacap_score on `ws`. */
jacap_status jacap_device_status(const void* ws, void* stream);

/*
 * Self-test of the device-side failure detection (no counterpart in the
 * paper): enqueues one thread that clears the status word of `ws` and waits,
 * with the bounded wait every pipeline of the pass uses, on an mbarrier that
 * nothing ever arrives on. After limit_ns (1 us .. 10 s) the wait gives up,
 * sets JACAP_ERR_TIMEOUT in the status word and the kernel returns; nothing
 * faults and the context stays usable, so jacap_device_status then reports
 * JACAP_ERR_TIMEOUT and the next jacap_score starts clean. ws: >= 64 bytes,
 * 256-byte aligned (a workspace).
 */
jacap_status jacap_selftest_wait(void* ws, size_t ws_bytes, int64_t limit_ns, void* stream);

/* Static English text for a status code (never NULL). */
const char* jacap_status_string(jacap_status status);

/* Byte offsets of the intermediates inside the workspace, for tests and
 * debugging (all float32, row-major):
 *  mu_scaled  [num_seqs][num_layers][num_q_heads][128]   mu_h / (tau sqrt(d))
 *  lambda     [num_seqs][num_layers][num_q_heads][128]   diagonal of Lambda_Q
 *  weights    [num_layers][num_kv_heads][total_tokens]   w_i (Eq. 8 summed over the group)
 *  gram       [num_layers][num_kv_heads][num_seqs][128][128]  sum_i w_i v_i v_i^T
 *  chol_inv   [num_layers][num_kv_heads][num_seqs][128][128]  L^{-1}, A = L L^T
 * and, in a library built with JACAP_TRACE=1 (0 otherwise; uint64 words):
 *  trace_timeline  [units][8]  per unit, %globaltimer ns of the fused schedule's
 *                  first Gram tile, last Gram partial published, factor start,
 *                  factor published, first score image acquired, last score
 *                  tile, first score MMA (units = num_layers x num_kv_heads x
 *                  num_seqs, unit (l, g, s) at (l num_kv_heads + g) num_seqs + s)
 *  trace_cta       [5][1024][16]  per kernel (K pass 2, Gram 0, scores 1,
 *                  factor 3, selection 4) and CTA (the first 1024), ns its roles spent in
 *                  each wait and busy section of the last pass, summed over the
 *                  pass (the slots are documented where the kernels record them)
 * Returns JACAP_ERR_INVALID_ARG for an invalid layout. */
typedef struct {
  size_t mu_scaled, lambda, weights, gram, chol_inv;
  size_t trace_timeline, trace_cta;
} jacap_ws_offsets;
jacap_status jacap_workspace_offsets(const jacap_layout* layout, int32_t budget, jacap_ws_offsets* out);

#ifdef __cplusplus
}
#endif

#endif /* JACAP_H */
