/*
 * kvev.h -- C ABI of the GB300 layer-wise KV-cache eviction library (libkvev.so).
 *
 * The library executes a static layer-wise eviction plan (Sec. 3.1, Eq. 1 of
 * "Exploring a Layer-Wise Design Space for KV Cache Eviction"): every layer l
 * has, per inference phase, an operator r_l (a retention rule, or FULL = no
 * eviction in that phase) and a nominal retained-token capacity b_l.  At the
 * prefill eviction point it scores the prompt keys of every layer with the
 * rule that layer is routed to, selects the positions to keep per
 * (sequence, KV head) and gather-compacts K/V into a packed smaller cache.
 * The per-layer capacities can be produced by the allocator of Sec. 3.3
 * (Eq. 3 and its b_min clamping and largest-remainder rounding).
 *
 * Conventions shared by every entry point
 *   - Return value: KVEV_OK (0) or one of the KVEV_E* codes below.  Arguments
 *     are validated before any device work is enqueued; on a non-zero return
 *     nothing was enqueued.
 *   - Device buffers are caller-owned raw device pointers (16-byte aligned
 *     where noted); host arrays are plain host pointers read during the call
 *     and not retained.  The library never frees caller memory.
 *   - Device work is enqueued asynchronously on the caller's stream, passed as
 *     a `void *` holding a cudaStream_t (NULL = legacy default stream).
 *     Faults the kernels detect themselves (a bounded wait that ran out, a
 *     layout check) are recorded in a device status word read by kvev_status().
 *   - bf16 tensors are raw 16-bit patterns; layouts are row-major C order.
 *   - Threading: a plan may be used by one host thread at a time.
 */
#ifndef KVEV_H
#define KVEV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define KVEV_API __attribute__((visibility("default")))
#else
#define KVEV_API
#endif

/* ---- status codes ------------------------------------------------------ */
#define KVEV_OK 0
#define KVEV_EINVAL 1   /* bad argument: shape, pointer, alignment or rule parameter */
#define KVEV_ENOMEM 2   /* host or device allocation failed, or workspace too small */
#define KVEV_ECUDA 3    /* a CUDA runtime/driver call failed (e.g. no device) */
#define KVEV_ETIMEOUT 4 /* device: a bounded wait ran out (see kvev_status) */
#define KVEV_EDEVICE 5  /* device: an in-kernel consistency check failed */
#define KVEV_ENOTSUP 6  /* valid request outside what this build supports */

/* ---- operators (the retention rules a layer can be routed to) ----------- */
#define KVEV_FULL 0      /* no eviction in this phase (Sec. 3.1) */
#define KVEV_SNAPKV 1    /* observation-window attention + 1-D pooling, top-k (prefill) */
#define KVEV_H2O 2       /* accumulated attention heavy hitters + recent window (both phases) */
#define KVEV_STREAMING 3 /* attention sinks + most recent tokens (both phases) */
#define KVEV_TOVA 4      /* evict the token the current query attends to least (decode only) */

#define KVEV_POOL_MAX 0
#define KVEV_POOL_AVG 1

#define KVEV_T_IDENTITY 0 /* allocation transform for entropy scores (Sec. 3.3) */
#define KVEV_T_CAP_Q95 1  /* cap at the across-layer 95th percentile (PPL scores, Sec. 3.3) */

typedef struct kvev_plan kvev_plan;

/* ---- capacity allocation (host only; no GPU needed) ---------------------- */

/* Sec. 3.3, Eq. 3: per-layer capacities from layer scores s[0..L).
 *   t_l = T(s_l) (identity, or min(s_l, Q_0.95(s)) with type-7 interpolation);
 *   if min t <= 0 every t is shifted by -min t + 1e-6;
 *   w_l = t_l / sum t;  b~_l = B_total * w_l;
 *   layers with b~_l < b_min are fixed at b_min and the remaining capacity is
 *   re-split over the other layers in proportion to w, until none drops below;
 *   the result is rounded by largest remainder (ties to the lower layer).
 * Output: budget_out[0..L) with sum == B_total and every entry >= b_min.
 * EINVAL if L <= 0, b_min < 0, L*b_min > B_total, or any s is not finite. */
KVEV_API int kvev_alloc_from_scores(int32_t *budget_out, const double *s, int L, int64_t B_total,
                           int b_min, int transform);

/* Sec. 3.3 (budget sweep): scale a completed vector budget_in[0..L) to the
 * total B_target (b_l * B_target / sum budget_in) and round by largest
 * remainder; no b_min is re-applied.  EINVAL if the input sum is <= 0. */
KVEV_API int kvev_alloc_rescale(int32_t *budget_out, const int32_t *budget_in, int L, int64_t B_target);

/* ---- plan constructor: route profiles, TopRank, allocation scores -------- */
/* Host only (no GPU needed); every statistic is computed in fp64. */

#define KVEV_SCOPE_PREFILL 1 /* a route active in the prefill phase only (Sec. 3.1) */
#define KVEV_SCOPE_DECODE 2  /* ... in the decode phase only */
#define KVEV_SCOPE_BOTH 3    /* the tied both-phase candidate */

/* Sec. 3.2, representation-similarity profile: C[l][r] = cos(h_full_l, h_r_l).
 *   h_full   host fp32 [L][D]: FullKV's pooled attention-module output of layer l.
 *   h_cand   host fp32 [R][L][D]: the same with candidate operator r applied.
 *   C_out    host fp64 [L][R]; larger is closer to FullKV.
 * EINVAL: sizes <= 0, a NULL pointer, or a zero or non-finite norm. */
KVEV_API int kvev_profile_cosine(double *C_out, const float *h_full, const float *h_cand, int L, int R,
                                 int64_t D);

/* Sec. 3.3, PPL allocation score: s_l = max_r (ppl[l][r] - ppl_full), the
 * largest perplexity degradation of layer l over the profiled operators.
 *   ppl      host fp64 [L][R]: perplexity with operator r at layer l only.
 * EINVAL: sizes <= 0, a NULL pointer, or a non-finite value. */
KVEV_API int kvev_score_ppl(double *s_out, const double *ppl, double ppl_full, int L, int R);

/* Sec. 3.3, entropy allocation score: H_l = mean over the `rows` attention
 * rows of layer l (calibration sequences x heads x queries, flattened) of the
 * Shannon entropy in nats, -sum_k p log p (terms with p = 0 contribute 0).
 *   A        host fp32 [L][rows][K]: FullKV attention probabilities; masked
 *            keys are 0 and every row sums to 1 (within 1e-3).
 * EINVAL: sizes <= 0, a NULL pointer, a negative or non-finite entry, or a
 * row that is not a distribution. */
KVEV_API int kvev_score_entropy(double *H_out, const float *A, int L, int64_t rows, int K);

/* Sec. 3.2, Eq. (policy_routing): per layer, the operator with the best
 * profile statistic.
 *   g        host fp64 [L][R]: statistic of operator ops[r] at layer l.
 *   ops[R]   the operator ids (KVEV_*) of the profile's columns.
 *   covered  host uint8 [L][R] or NULL: 0 excludes an entry (the operator is
 *            not covered by the profile, or not compatible with the scope).
 *   higher_is_better  1 for the cosine profile, 0 for the PPL profile.
 * route_out[l] is ops of the best covered column; equal statistics keep the
 * column listed first; a layer with no covered column gets KVEV_FULL.
 * EINVAL: sizes <= 0, a NULL pointer, an unknown operator id, or a
 * non-finite covered entry. */
KVEV_API int kvev_route_toprank(int32_t *route_out, const double *g, int L, int R, const int32_t *ops,
                                const uint8_t *covered, int higher_is_better);

/* Sec. 3.2: install a route in the phases of a scope (KVEV_SCOPE_*): active
 * phases take route[l], inactive ones KVEV_FULL.  EINVAL if an operator is
 * not valid in an active phase (SnapKV is prefill only, TOVA decode only). */
KVEV_API int kvev_route_install(int32_t *route_prefill, int32_t *route_decode, const int32_t *route,
                                int L, int scope);

/* ---- plan ---------------------------------------------------------------- */

/* Create the static plan of Eq. 1 (host memory only; no device work).
 *   L, H_q, H_kv, d      model geometry; H_q must be a multiple of H_kv.
 *   route_prefill[L]     operator per layer at the prefill eviction point:
 *                        KVEV_FULL, KVEV_SNAPKV, KVEV_H2O or KVEV_STREAMING.
 *   route_decode[L]      operator per layer in the decode phase (KVEV_FULL,
 *                        KVEV_H2O, KVEV_TOVA, KVEV_STREAMING); NULL = all FULL.
 *   budget[L]            nominal capacity b_l (ignored for FULL layers).
 *   window               observation window W of the scoring rules (SnapKV, H2O).
 *   pool_kernel          SnapKV pooling width (odd, >= 1); pool_type KVEV_POOL_*.
 *   sink                 StreamingLLM attention-sink tokens.
 *   recent               StreamingLLM recent tokens; -1 = b_l - sink per layer,
 *                        otherwise min(recent, b_l - sink).
 *   h2o_recent           H2O protected recent window; -1 = floor(b_l / 2).
 * EINVAL: a SnapKV layer with b_l <= window, a StreamingLLM layer with
 * b_l <= sink, an H2O layer with b_l < 1 or h2o_recent > b_l, an even or
 * non-positive pool_kernel with a SnapKV layer, window < 1 with a scoring
 * layer, or a decode route that is not FULL/H2O/TOVA/STREAMING.
 * ENOTSUP: d not 64 or 128, G*window > 256 (G = H_q/H_kv) with a scoring
 * layer, or more than 64 scoring layers. */
KVEV_API int kvev_plan_create(kvev_plan **out, int L, int H_q, int H_kv, int d,
                     const int32_t *route_prefill, const int32_t *route_decode,
                     const int32_t *budget, int window, int pool_kernel, int pool_type,
                     int sink, int recent, int h2o_recent);

/* Sec. 3.4: a completed plan is serialised once and loaded at run time.
 * kvev_plan_save writes the plan's definition (geometry, routes, budgets,
 * rule parameters) to buf; with buf NULL it only stores the size in *bytes,
 * otherwise *bytes is the buffer's capacity on entry and the size written on
 * return.  The format is little-endian: the 8 bytes "KVEVPLN1", then 32-bit
 * words, then a 64-bit FNV-1a checksum of everything before it.
 * kvev_plan_load validates the magic, size and checksum and recreates the
 * plan through kvev_plan_create (same checks, same errors).
 * EINVAL: NULL pointers, a buffer too small (save), or a corrupt or
 * truncated buffer (load). */
KVEV_API int kvev_plan_save(const kvev_plan *plan, void *buf, size_t *bytes);
KVEV_API int kvev_plan_load(kvev_plan **out, const void *buf, size_t bytes);

/* Release the plan and the small device status buffer it may hold. */
KVEV_API void kvev_plan_destroy(kvev_plan *plan);

/* Sizes of the buffers kvev_evict_prefill() needs for a batch of B sequences
 * stored in caches of S_cap positions (any pointer may be NULL):
 *   out_kv_bytes    bytes of out_K (and, separately, of out_V): sum over
 *                   non-FULL layers of B*H_kv*b_l rows of d bf16;
 *   out_idx_bytes   bytes of out_idx (int32 per output row; also the size of
 *                   h2o_state in floats * 4);
 *   count_bytes     bytes of out_count (int32 [L][B][H_kv]);
 *   workspace_bytes device scratch for one call.
 * Worked example (App. E): L=32, b=512, B=1, H_kv=8, d=128 gives
 * 16,384 layer-token positions and 2*out_kv_bytes = 64.00 MiB of K+V. */
KVEV_API int kvev_plan_query(const kvev_plan *plan, int B, int S_cap, size_t *out_kv_bytes,
                    size_t *out_idx_bytes, size_t *count_bytes, size_t *workspace_bytes);

/* First packed output row of `layer` for a batch of B sequences; the row of
 * (layer, seq s, kv head h, slot j) is row_offset + (s*H_kv + h)*b_l + j.
 * FULL layers own no rows (the caller keeps their cache as it is). */
KVEV_API int kvev_plan_layer_offset(const kvev_plan *plan, int B, int layer, int64_t *row_offset);

/* Where a call leaves the window scores of a SnapKV/H2O layer: after
 * kvev_evict_prefill() returns (and its stream is synchronised), the bytes at
 * workspace + *byte_offset hold fp32 [B][H_kv][S_cap] scores of `layer`
 * (entry k of (s, h) valid for k < lens[s]; see the rule description below),
 * until the workspace is reused.  EINVAL if the layer has no scores. */
KVEV_API int kvev_plan_scores_offset(const kvev_plan *plan, int B, int S_cap, int layer,
                                     size_t *byte_offset);

/* Prefill eviction of every layer of the plan in grouped launches.
 *   K[L], V[L]     host arrays of pointers; layer l's cache is bf16
 *                  [B][H_kv][S_cap][d] (16-byte aligned).  Entries of FULL
 *                  layers may be NULL.  K of a SnapKV / H2O layer must be
 *                  device memory (it is streamed by the tensor-memory
 *                  accelerator); V of every layer and K of a StreamingLLM layer
 *                  are only read row by row at the kept positions and may also
 *                  be pinned host memory that the device addresses directly
 *                  (unified addressing), which is then read in place.
 *   Q_win[L]       host array of device pointers to the observation-window
 *                  queries, bf16 [B][H_q][W][d] (16-byte aligned); query i of
 *                  the window sits at position lens[s] - W + i.  Needed for
 *                  SnapKV and H2O layers, may be NULL elsewhere.
 *   lens_dev       device int32 [B]: valid length of each sequence, 0..S_cap.
 *   out_K, out_V   device bf16, packed rows (see kvev_plan_layer_offset): row
 *                  j of (l, s, h) is K[l][s][h][out_idx[row]]; slots past the
 *                  kept count hold zeros.  16-byte aligned.
 *   out_idx        device int32 per output row: kept positions in ascending
 *                  order, -1 in unused slots.
 *   out_count      device int32 [L][B][H_kv]: kept count (= min(b_l, lens[s])
 *                  for capacity-controlled layers; lens[s] for FULL layers).
 *   h2o_state      device fp32 per output row (nullable): for H2O layers the
 *                  window attention score of each kept token, the initial
 *                  accumulated-attention state of the decode phase.
 *   workspace      device scratch of at least the queried size (256-byte
 *                  aligned); contents need no initialisation.
 * The rules are the ones Sec. 2.1 cites, at the layer's capacity b_l:
 *   SnapKV: score[k] = (1/G) sum over the G query heads of the group and the
 *     W window rows of softmax(q K^T / sqrt(d))[k] (causal inside the window,
 *     normalised over every visible key); pooled over [0, n-W) with width
 *     pool_kernel (max, or average with zero padding divided by the width);
 *     keep the last W positions plus the top (b_l - W) pooled prefix scores.
 *   H2O: the same window score without pooling; keep the last h2o_recent
 *     positions plus the top (b_l - h2o_recent) scores before them.
 *   StreamingLLM: keep positions [0, sink) and the last `recent` positions.
 *   Any rule with b_l >= lens[s] keeps every position.
 * Top-k ties keep the lower position.
 * EINVAL on null/misaligned pointers or B < 0, S_cap < 1; ENOMEM if the
 * workspace is smaller than kvev_plan_query() reports.  The workspace holds,
 * among the rest, 4 bytes per position per (scoring layer, sequence, KV head)
 * for the selection's keys (rows padded to whole 128-position blocks). */
KVEV_API int kvev_evict_prefill(kvev_plan *plan, const void *const *K, const void *const *V,
                       const void *const *Q_win, const int32_t *lens_dev, int B, int S_cap,
                       void *out_K, void *out_V, int32_t *out_idx, int32_t *out_count,
                       float *h2o_state, void *workspace, size_t workspace_bytes, void *stream);

/* kvev_evict_prefill with the scores of chosen scoring layers supplied by the
 * caller: the fused form, where the caller's own prefill attention kernel
 * already forms the softmax rows and their column sums are the rules' scores.
 *   scores[L]  host array of device pointers; for a SnapKV or H2O layer NULL
 *              (the library scores it from Q_win) or fp32 [B][H_kv][S_cap]:
 *              raw[k] for k < lens[s] exactly as the layer's rule defines it
 *              (the group mean of the window rows' softmax weights; every
 *              prompt row's for H2O with kvev_plan_set_h2o_full_prompt).
 *              SnapKV's pooling, both rules' selection and H2O's decode seed
 *              (h2o_state) read it; Q_win[l] is not read for such a layer.
 *              Entries of other layers are ignored.  4-byte aligned.
 * Everything else as kvev_evict_prefill.  EINVAL if scores is NULL. */
KVEV_API int kvev_evict_prefill_scored(kvev_plan *plan, const void *const *K, const void *const *V,
                                       const void *const *Q_win, const float *const *scores,
                                       const int32_t *lens_dev, int B, int S_cap, void *out_K,
                                       void *out_V, int32_t *out_idx, int32_t *out_count,
                                       float *h2o_state, void *workspace, size_t workspace_bytes,
                                       void *stream);

/* kvev_evict_prefill with the window rows' softmax normalisers supplied by
 * the caller: the fused form, where the caller's own prefill attention has
 * already formed every query row's log-sum-exp (flash-attention-style kernels
 * return it).  The window scores of Sec. 2.1's rules need each window row's
 * normaliser over every visible key before any key's score is final; given
 * them, the library's score kernel makes one pass over K instead of two.
 *   lse_win[L]  host array of device pointers; for every SnapKV and H2O
 *               layer fp32 [B][H_q][W]: entry (s, q, i) is
 *               ln sum_{k <= t} exp(q_row . K[s][q / G][k] / sqrt(d)) for
 *               the window row of query head q at position t = lens[s] - W + i
 *               (the same scale and causal range as the scores; rows with
 *               t < 0 are not read).  For the H2O layers of a plan that
 *               scores them over the whole prompt
 *               (kvev_plan_set_h2o_full_prompt): fp32 [B][H_q][S_cap], the
 *               same for every prompt row t < lens[s] (the layout of a
 *               flash-attention softmax_lse), and the row pass is skipped.
 *               Entries of other layers are ignored.  4-byte aligned.
 * Q_win is still read (the scores need the rows' logits).  Everything else
 * as kvev_evict_prefill.  EINVAL if lse_win or an entry of a SnapKV / H2O
 * layer is NULL or misaligned. */
KVEV_API int kvev_evict_prefill_lse(kvev_plan *plan, const void *const *K, const void *const *V,
                                    const void *const *Q_win, const float *const *lse_win,
                                    const int32_t *lens_dev, int B, int S_cap, void *out_K,
                                    void *out_V, int32_t *out_idx, int32_t *out_count,
                                    float *h2o_state, void *workspace, size_t workspace_bytes,
                                    void *stream);

/* Sec. 2.1 (H2O's original scoring): with on = 1, the prefill scores of the
 * plan's H2O layers accumulate the attention of every prompt query row,
 *   raw[k] = (1/G) sum_g sum_{t=k}^{n-1} p_{g,t}(k),
 * p_{g,t} being query row (g, t)'s softmax over keys 0..t, instead of the
 * observation window's.  Q_win[l] of an H2O layer is then the whole prompt's
 * queries, bf16 [B][H_q][S_cap][d]; SnapKV layers keep their window queries.
 * Two extra launches compute it: a row pass (every row's log-sum-exp, kept in
 * the workspace) and a key pass (each key's sum over the rows that see it,
 * written once per key).  Cost grows with n^2.  Set it before
 * kvev_plan_query(): the workspace then also holds G * S_cap floats per H2O
 * (sequence, KV head).  EINVAL: NULL plan or on not 0/1. */
KVEV_API int kvev_plan_set_h2o_full_prompt(kvev_plan *plan, int on);

/* Synchronise the plan's last stream and read-and-clear the device status
 * word: *device_status receives KVEV_OK, KVEV_ETIMEOUT or KVEV_EDEVICE.
 * Returns ECUDA if the readback itself failed.  Status bits of
 * kvev_evict_prefill_noalloc() calls go to that call's own device_status
 * word and are never reported here. */
KVEV_API int kvev_status(kvev_plan *plan, int *device_status);

/* Bound (in nanoseconds) of every in-kernel wait; a wait that runs out
 * records KVEV_ETIMEOUT and the kernel finishes without producing valid
 * scores for the affected units.  Default 2e9 (2 s). */
KVEV_API int kvev_plan_set_wait_limit(kvev_plan *plan, int64_t ns);

/* Test hook: when `unit` >= 0 the score kernel never marks that scoring unit
 * as ready, so every wait on it runs out after the wait limit.  Used only to
 * exercise the timeout path; -1 disables it. */
KVEV_API int kvev_plan_debug_stall_unit(kvev_plan *plan, int unit);

/* ---- prefill eviction for callers that cannot allocate device memory ------ */

/* Size of the device scratch that kvev_evict_prefill_noalloc() uses instead of
 * a caller workspace (32 MiB; every GPU that loads the library holds it until
 * the process exits). */
#define KVEV_NOALLOC_SCRATCH_BYTES (32u << 20)

/* Same eviction as kvev_evict_prefill(), for callers that must not allocate:
 * code running where cudaMalloc is forbidden or unavailable (inside a memory
 * pool whose budget is already committed, in a custom allocator's own hooks,
 * under a framework that owns all device memory), or that has no workspace to
 * lend.  No counterpart in the paper: it is a deployment convenience.
 *   - The scratch is a fixed library-owned device array of
 *     KVEV_NOALLOC_SCRATCH_BYTES; a request whose kvev_plan_query()
 *     workspace_bytes exceeds it returns KVEV_ENOMEM before any device work.
 *   - The call allocates nothing: no cudaMalloc/cudaFree and no allocating
 *     library routine.  Inputs and outputs are the caller's, as for
 *     kvev_evict_prefill().
 *   - device_status: required device int32 (4-byte aligned; NULL is
 *     EINVAL) that the call zeroes on `stream` and in which the kernels
 *     record their status bits (1 = a bounded wait ran out, 2 = an in-kernel
 *     check failed).  It is the only place these calls report device-side
 *     errors: read it after the stream's work is done; any non-zero value
 *     means the outputs of that call are not valid.  kvev_status() never
 *     reports this entry point's calls.
 *   - The first call on each device looks up the scratch array's device
 *     address for that device (with that device current); make that first
 *     call before any stream capture on the device.
 *   - All calls in the process share the one array per device and each call
 *     starts by resetting the parts that must start at zero; calls whose GPU
 *     work overlaps (other streams, other host threads) race on it and must
 *     be serialised by the caller. */
KVEV_API int kvev_evict_prefill_noalloc(kvev_plan *plan, const void *const *K,
                                        const void *const *V, const void *const *Q_win,
                                        const int32_t *lens_dev, int B, int S_cap, void *out_K,
                                        void *out_V, int32_t *out_idx, int32_t *out_count,
                                        float *h2o_state, int32_t *device_status, void *stream);

/* ---- decode phase ---------------------------------------------------------- */

/* Decode arena: the retained caches kept across generated tokens, in
 * caller-owned device memory laid out by the plan.  Layer l with a retained
 * cache (prefill rule other than FULL) holds cap_l slots per (sequence, KV
 * head): cap_l = b_l for layers with a decode-phase rule (H2O, TOVA,
 * StreamingLLM) and b_l + growth for append-only layers (decode rule FULL).
 * Slot (s, h, j) of layer l is row row_offset(l) + (s*H_kv + h)*cap_l + j of
 * dec_K / dec_V (bf16 [rows][d]).  The state buffer (dec_state, 256-byte
 * aligned, kvev_decode_state_offsets) holds int32 lens[B] (sequence lengths,
 * advanced by every step), int32 count[units] (occupied slots), int32
 * evicted[units] (position evicted by the last step, -1 if none), int32
 * pos[rows] (position held by a slot, -1 = empty) and fp32 acc[rows] (H2O:
 * accumulated attention; TOVA: the last step's attention), where unit
 * unit_offset(l) + s*H_kv + h, and after them an internal step counter.  Slot
 * order carries no meaning.
 * EINVAL when a layer with a FULL prefill rule has a decode-phase rule (its
 * cache is the caller's own). */
KVEV_API int kvev_decode_query(const kvev_plan *plan, int B, int growth, int64_t *rows,
                               size_t *state_bytes);
KVEV_API int kvev_decode_layer(const kvev_plan *plan, int B, int growth, int layer,
                               int64_t *row_offset, int *cap, int *unit_offset);
/* offsets[5] = byte offsets in dec_state of lens, count, evicted, pos, acc. */
KVEV_API int kvev_decode_state_offsets(const kvev_plan *plan, int B, int growth, size_t *offsets);

/* Fill the arena from the output of kvev_evict_prefill() (same plan and B):
 * slot j < out_count of each unit takes packed row j (its K/V rows, its
 * position, and for H2O prefill layers its h2o_state score as the initial
 * acc, 0 elsewhere or when h2o_state is NULL); other slots are marked empty;
 * lens is copied from lens_dev.  Asynchronous on `stream`.  EINVAL on null or
 * misaligned pointers (rows 16-byte, state 256-byte). */
KVEV_API int kvev_decode_init(kvev_plan *plan, int B, int growth, const void *pre_K,
                              const void *pre_V, const int32_t *pre_idx, const int32_t *pre_count,
                              const float *h2o_state, const int32_t *lens_dev, void *dec_K,
                              void *dec_V, void *dec_state, void *stream);

/* One decode step (Sec. 2.1's cited rules in their decode phase; the new
 * token sits at position lens[s] and lens advances by one):
 *   k_new[L], v_new[L]  host arrays of device pointers, bf16 [B][H_kv][d]
 *                       (NULL for layers without an arena);
 *   q_new[L]            bf16 [B][H_q][d], the new token's queries (needed for
 *                       H2O and TOVA layers only).
 *   H2O:  p_j = (1/G) sum over the group's query heads of
 *         softmax_j(q . k_j / sqrt(d)) over the retained slots and the new
 *         token; acc += p; once b slots are held, the slot with the smallest
 *         acc among positions < lens+1-r (r = h2o_recent, or floor(b/2)) is
 *         evicted (ties: the higher position) and the new token takes it.
 *   TOVA: the same with acc = p (no accumulation) and r = 0, so the new token
 *         itself may be the one evicted.
 *   StreamingLLM: once sink + recent slots are held, the smallest position
 *         >= sink is evicted.
 *   FULL: append (count must stay <= cap, else the device status records an
 *         error).
 * Asynchronous; ENOTSUP if d is not 64/128 or G not 1, 2, 4 or 8. */
KVEV_API int kvev_decode_step(kvev_plan *plan, int B, int growth, void *dec_K, void *dec_V,
                              void *dec_state, const void *const *k_new, const void *const *v_new,
                              const void *const *q_new, void *stream);

/* The decode step with the attention supplied by the caller's own decode
 * attention kernel (the fused form of Sec. 2.1's H2O / TOVA decode rules: the
 * caller's attention already reads the retained K, so the step reads none).
 *   attn[L]  host array of device pointers; for every H2O / TOVA layer fp32
 *            [B][H_kv][cap_l + 1] (cap_l from kvev_decode_layer): for each
 *            unit (s, h) with count c, entries 0..c-1 are the group-mean
 *            softmax weights of the new token's queries on arena slots
 *            0..c-1 (slot order of the arena, as in dec_K) and entry c the
 *            weight on the new token itself, the softmax running over the
 *            retained slots and the new token; entries past c are not read.
 *            NULL for other layers.  4-byte aligned.
 * Everything else (append, acc update, eviction, StreamingLLM, FULL) is as in
 * kvev_decode_step; no queries are needed.  EINVAL if attn or an H2O / TOVA
 * layer's entry is NULL or misaligned. */
KVEV_API int kvev_decode_step_attn(kvev_plan *plan, int B, int growth, void *dec_K, void *dec_V,
                                   void *dec_state, const void *const *k_new,
                                   const void *const *v_new, const float *const *attn, void *stream);

/* ---- measurement ---------------------------------------------------------- */

/* Kernels of one kvev_evict_prefill() call, in launch order. */
#define KVEV_K_PROLOGUE 0
#define KVEV_K_SCORE 1
#define KVEV_K_SELECT 2
#define KVEV_K_GATHER 3
#define KVEV_NUM_KERNELS 4

/* When `on` is non-zero, every later kvev_evict_prefill() records a CUDA
 * event pair on the caller's stream around each of its kernel launches
 * (creates the events on first use; ECUDA if that fails). */
KVEV_API int kvev_plan_enable_timing(kvev_plan *plan, int on);

/* Device time in milliseconds of each kernel of the most recent timed call
 * (synchronises on its last event); ms[k] = -1 for a kernel that call did not
 * launch.  n = number of entries of ms (up to KVEV_NUM_KERNELS are written).
 * EINVAL if timing is off or no timed call was made. */
KVEV_API int kvev_plan_last_timings(kvev_plan *plan, float *ms, int n);

#ifdef __cplusplus
}
#endif
#endif /* KVEV_H */
