/*
 * provip.h - C ABI of the GB300 (sm_103a) ProViP token-pruning library.
 *
 * ProViP ("Not All Attention Heads Contribute to Critical Visual Token
 * Selection: Head-Aware Pruning Matters More") prunes visual tokens of a
 * vision-language model in two places:
 *   - before the LLM (Sec. 4.2-4.3): critical text tokens from the text
 *     self-similarity, text-guided cosine relevance of every visual token, a
 *     top-N1 keep set, and the pruned tokens merged into their nearest kept
 *     token;
 *   - inside the LLM (Sec. 4.4): attention probabilities from the text rows to
 *     the visual columns for a chosen set of heads, normalised over the full
 *     causal key range, averaged over heads and text rows, top-N2 kept, and the
 *     sequence (hidden states, K/V rows, position ids) compacted.
 *
 * Conventions shared by every call
 *   - Tensor pointers are DEVICE pointers owned by the caller, C-contiguous,
 *     row-major with the shapes given; the library never frees or retains them.
 *     Pointers marked "host" are read on the host during the call.
 *   - dtype is PROVIP_F32 or PROVIP_BF16 and applies to every floating-point
 *     input/output tensor of the call except scores, which are always fp32.
 *   - Every call is asynchronous on `stream` (a cudaStream_t; NULL is the
 *     legacy default stream) and allocates nothing: scratch memory comes from
 *     the caller's workspace `ws` of `ws_bytes` bytes (256-byte aligned), sized
 *     by the matching *_workspace_size() query with the same shape arguments.
 *     Workspace contents need not be initialised and are clobbered.
 *   - Return value: PROVIP_OK or a negative status. Arguments are validated on
 *     the host before anything is launched; on error nothing is enqueued.
 *     Values that live in device memory (lengths, indices) cannot be checked
 *     before launch: kernels that meet an out-of-range one skip it and set the
 *     device status word, read with provip_device_status().
 *   - Every wait inside a kernel is bounded (2 s); a wait that gives up sets
 *     PROVIP_DEVSTAT_TIMEOUT in the device status word instead of hanging.
 *   - Sequences are laid out per sample as [prefix rows | N_v visual rows |
 *     text rows | padding]: visual rows start at vis_start, a sample's rows
 *     beyond seq_len[b] are padding and never read.
 */
#ifndef PROVIP_H_
#define PROVIP_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* status codes */
#define PROVIP_OK 0
#define PROVIP_ERR_INVALID_ARG (-1) /* a host-checkable argument is out of range */
#define PROVIP_ERR_UNSUPPORTED (-2) /* dtype / shape / alignment not supported */
#define PROVIP_ERR_WORKSPACE (-3)   /* ws_bytes smaller than the size query */
#define PROVIP_ERR_CUDA (-4)        /* a CUDA call failed; see provip_last_error() */
#define PROVIP_ERR_TIMEOUT (-5)     /* returned by provip_device_status() */

/* element types */
#define PROVIP_F32 0
#define PROVIP_BF16 1

/* kernel families for provip_head_scores / provip_prune */
#define PROVIP_ALGO_AUTO 0    /* tensor cores for bf16, CUDA cores for fp32 */
#define PROVIP_ALGO_SIMT 1    /* CUDA-core FFMA kernels (fp32 and bf16) */
#define PROVIP_ALGO_TCGEN05 2 /* tcgen05 tensor cores (bf16 only): the streaming form
                                 when there are at least as many (sample, head, row
                                 block) units as SMs, else the cluster form */
#define PROVIP_ALGO_TCGEN05_TWOPASS 3 /* tcgen05, two kernels: chunk statistics, then
                                         probabilities (bf16 only) */
#define PROVIP_ALGO_TCGEN05_STREAM 4  /* tcgen05, one CTA per (sample, head, row block)
                                         streaming that head's keys through a TMA/TMEM
                                         pipeline: every key, then the visual keys again
                                         (from L2) (bf16 only) */
#define PROVIP_ALGO_TCGEN05_CLUSTER 5 /* tcgen05, one pass over K in a cluster per (head,
                                         sample), logits kept in TMEM (bf16 only); falls
                                         back to the two-pass form when L_max > 8192 or
                                         no cluster shape fits */
/* Different kernel families sum in different orders: results agree within the
 * floating-point tolerance, and are bit-identical between calls that take the
 * same family (the same algo and, for PROVIP_ALGO_TCGEN05, the same choice),
 * with or without head-confidence statistics. */

/* bits of the device status word */
#define PROVIP_DEVSTAT_TIMEOUT 1u  /* a bounded wait gave up */
#define PROVIP_DEVSTAT_BAD_ARG 2u  /* a device-resident argument was out of range */

/* ------------------------------------------------------------------------
 * Library status
 * ---------------------------------------------------------------------- */

/* Human-readable name of a status code (static string). */
const char *provip_status_string(int status);

/* Message of the last PROVIP_ERR_CUDA / INVALID_ARG / UNSUPPORTED returned on
 * the calling thread (static per thread; empty if none). */
const char *provip_last_error(void);

/* Library version as 10000*major + 100*minor + patch. */
int provip_version(void);

/* Process-wide switches of the library's kernel choice (tests and measurement
 * use them to reach every form); they apply to calls enqueued after the switch.
 *   PROVIP_OPT_MERGE_PAIRS: 1 (default) lets the bf16 nearest-centroid Gram of
 *   the merge (Sec. 4.3) run on pairs of SMs (tcgen05 cta_group::2, one M = 256
 *   MMA over two CTAs) where two-CTA clusters fit; 0 keeps it on single SMs.
 * Returns PROVIP_OK, or PROVIP_ERR_INVALID_ARG for an unknown option or a value
 * outside {0, 1}. */
#define PROVIP_OPT_MERGE_PAIRS 1
int provip_set_option(int option, int value);

/* Synchronises the current device, then returns the device status word of the
 * current device (PROVIP_DEVSTAT_* bits) in *bits and clears it when `clear`
 * is non-zero. Returns PROVIP_ERR_TIMEOUT if the TIMEOUT bit is set,
 * PROVIP_ERR_INVALID_ARG if BAD_ARG is set, PROVIP_OK otherwise. */
int provip_device_status(unsigned *bits, int clear);

/* Failure-detection self test: enqueues one CTA on `stream` whose first thread
 * waits, through the same bounded wait every kernel of the library uses, on an
 * mbarrier that nothing ever completes. After the wait budget (2 s) the wait
 * gives up, sets PROVIP_DEVSTAT_TIMEOUT in the device status word and the
 * kernel returns, so the context stays usable; provip_device_status() then
 * reports PROVIP_ERR_TIMEOUT. Returns PROVIP_OK once launched, or
 * PROVIP_ERR_CUDA. */
int provip_selftest_wait_timeout(void *stream);

/* ------------------------------------------------------------------------
 * Pre-LLM pass (Sec. 4.2-4.3)
 * ---------------------------------------------------------------------- */

/* Critical textual token selection (Sec. 4.2, equations for r and T):
 *   G = E_t E_t^T (no scaling), R = row-wise softmax of G,
 *   r_j = (1/N_t) sum_i R_ij,  T = { j : r_j > mean(r) };
 * over the text_len[b] valid rows of each sample. If no r_j exceeds the mean
 * (e.g. N_t = 1 or identical rows) T is every valid row.
 *   emb_t    [B, N_t_max, D] dtype; rows >= text_len[b] are not read.
 *   text_len [B] int32, 0 <= text_len[b] <= N_t_max.
 *   mask_out [B, N_t_max] uint8: 1 for j in T, 0 otherwise (and for padding).
 *   r_out    [B, N_t_max] fp32 or NULL: r (0 for padding).
 * Requires D % 8 == 0, N_t_max <= 4096. */
size_t provip_crit_text_workspace_size(int B, int N_t_max, int D);
int provip_crit_text(const void *emb_t, int B, int N_t_max, int D, const int *text_len,
                     int dtype, uint8_t *mask_out, float *r_out, void *ws, size_t ws_bytes,
                     void *stream);

/* Text-guided visual relevance (Sec. 4.3, equations for M, M-hat and p):
 *   M_ij = cos(E_t[i], E_v[j]) for i in T (crit_mask), j < N_v (0 for a zero row),
 *   p_j  = max_{i in T} ( M_ij - (1/N_v) sum_k M_ik ).
 *   emb_v [B, N_v, D], emb_t [B, N_t_max, D] dtype; crit_mask [B, N_t_max] uint8.
 *   p_out [B, N_v] fp32 (-inf for a sample without a critical row).
 * Requires D % 8 == 0. */
size_t provip_relevance_workspace_size(int B, int N_v, int D, int N_t_max);
int provip_relevance(const void *emb_v, int B, int N_v, int D, const void *emb_t,
                     const int *text_len, int N_t_max, const uint8_t *crit_mask, int dtype,
                     float *p_out, void *ws, size_t ws_bytes, void *stream);

/* Top-k per sample (Sec. 4.3 top N1 of p, Sec. 4.4 top N2 of v): the k
 * largest of scores[b][0..N), ties broken toward the lower index, written in
 * ascending index order to idx_out [B, k] int32. 1 <= k <= N <= 49152.
 * NaN sorts above +inf. No workspace. */
int provip_topk(const float *scores, int B, int N, int k, int *idx_out, void *stream);

/* Merge of pruned visual tokens into their nearest kept token (Sec. 4.3, last
 * paragraph; the paper defers the rule to ApET without stating it - this
 * library reads it as: each pruned row j goes to the kept row of largest
 * cosine, ties to the lower kept position; merged = uniform mean of the kept
 * row and its members).
 *   keep_idx   [B, keep] int32, strictly ascending visual indices (device).
 *   assign_out [B, N_v] int32: position in keep_idx of row j's centroid (kept
 *              rows map to their own position).
 *   merged_out [B, keep, D] dtype or NULL (assignment only). fp32 sums are
 *              accumulated in double, bf16 sums in float, both in ascending
 *              row order; the mean is rounded to nearest-even.
 * Requires D % 8 == 0, D <= 8192. */
size_t provip_merge_workspace_size(int B, int N_v, int D, int keep);
int provip_merge(const void *emb_v, int B, int N_v, int D, const int *keep_idx, int keep,
                 int dtype, int *assign_out, void *merged_out, void *ws, size_t ws_bytes,
                 void *stream);

/* The whole pre-LLM pass: critical text tokens (unless crit_mask_or_null is
 * given), relevance p, top keep_pre of p (idx_out, ascending), and the merge
 * (when merged_out_or_null is given). p_out_or_null / mask_out_or_null
 * receive the intermediate p [B, N_v] and T mask [B, N_t_max] when non-NULL;
 * assign_out_or_null [B, N_v] int32 receives the merge's assignment (as
 * provip_merge's assign_out) when non-NULL and the merge runs. */
size_t provip_similarity_reduce_workspace_size(int B, int N_v, int D, int N_t_max, int keep_pre);
int provip_similarity_reduce(const void *emb_v, int B, int N_v, int D, const void *emb_t,
                             const int *text_len, int N_t_max,
                             const uint8_t *crit_mask_or_null, int keep_pre, int dtype,
                             int *idx_out, void *merged_out_or_null, int *assign_out_or_null,
                             float *p_out_or_null, uint8_t *mask_out_or_null, void *ws,
                             size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * In-LLM head-aware pruning (Sec. 4.4)
 * ---------------------------------------------------------------------- */

/* Head-aware visual-token scores (Sec. 4.4, equations for S^vis and v):
 *   A_{h,j,i} = softmax over keys 0..t_j of q_{t_j,h} . k_{k,g(h)} / sqrt(d_h),
 *               taken at key vis_start + i  (t_j the absolute position of text
 *               row j, g(h) = h / (H_q / H_kv) its key/value head);
 *   v_i       = 1/(|V| |R|) sum_{h in V} sum_{j in R} A_{h,j,i}.
 * V = head_list (host int32[H_sel], distinct, in [0, H_q)), or every head
 * when head_list is NULL and H_sel == H_q (the paper's "all attention heads"
 * variant used at the middle pruning layer, Sec. 4.4); R = text rows
 * j < text_len[b] at positions text_start[b] + j, restricted to
 * row_mask_or_null[b][j] != 0 when given (e.g. the critical rows T).
 *   Q [B, L_max, H_q, d_h], K [B, L_max, H_kv, d_h] dtype (post-RoPE).
 *   text_start, text_len, seq_len [B] int32 (device).
 *   row_mask_or_null [B, N_t_max] uint8 or NULL.
 *   scores [B, N_v] fp32.
 * Only the selected heads are read; the attention matrix is never stored.
 * Requires d_h == 128, H_q % H_kv == 0, 1 <= H_sel <= 64, vis_start + N_v <=
 * seq_len[b], text_start[b] + text_len[b] <= seq_len[b] <= L_max.
 * algo: PROVIP_ALGO_* (TCGEN05 requires bf16). */
size_t provip_head_scores_workspace_size(int B, int L_max, int H_sel, int N_t_max, int N_v,
                                         int algo, int dtype);
int provip_head_scores(const void *Q, const void *K, int B, int L_max, int H_q, int H_kv,
                       int d_h, const int *head_list, int H_sel, const int *text_start,
                       const int *text_len, const uint8_t *row_mask_or_null, int N_t_max,
                       int vis_start, int N_v, const int *seq_len, int dtype, int algo,
                       float *scores, void *ws, size_t ws_bytes, void *stream);

/* provip_head_scores for callers that cannot allocate device memory (the
 * paper has no counterpart; this is a deployment convenience). Some hosts
 * cannot pass the library a workspace: a framework that owns every device
 * allocation and hands a plugin only its input and output tensors, or a
 * serving loop that allows no allocator call once it is running. This entry
 * point takes the same arguments as provip_head_scores minus the workspace and
 * keeps its scratch in a static device array of PROVIP_NOALLOC_SCRATCH_BYTES
 * (4 MiB) inside the library, which every GPU that loads the library holds
 * until the process exits. It allocates nothing.
 *   - A shape whose scratch (provip_head_scores_workspace_size) exceeds the
 *     array is rejected with PROVIP_ERR_UNSUPPORTED before anything is
 *     enqueued; use provip_head_scores with a workspace for it.
 *   - The first call on each device looks up the array's device address (with
 *     that device current); make that first call before any stream capture.
 *   - All calls on a device share the one array, which keeps what the last call
 *     left there (nothing in it needs to start at zero). Calls that overlap on
 *     the GPU - on different streams, or from different host threads without
 *     ordering - race on it and corrupt each other's results: issue them in
 *     order on one stream. */
#define PROVIP_NOALLOC_SCRATCH_BYTES (4u << 20)
int provip_head_scores_noalloc(const void *Q, const void *K, int B, int L_max, int H_q,
                               int H_kv, int d_h, const int *head_list, int H_sel,
                               const int *text_start, const int *text_len,
                               const uint8_t *row_mask_or_null, int N_t_max, int vis_start,
                               int N_v, const int *seq_len, int dtype, int algo, float *scores,
                               void *stream);

/* Survivor compaction given the kept indices (Sec. 4.1: pruned tokens are
 * excluded from all later computation). For every sample the output rows are
 *   [0, vis_start) ++ (vis_start + idx[b][a], a < keep) ++ [vis_start + N_v, seq_len[b])
 * gathered byte-exactly from hidden [B, L_max, D], K/V [B, L_max, H_kv, d_h]
 * (either may be NULL, both or neither) and pos [P, B, L_max] int32 (NULL
 * allowed) into hidden_out [B, L_out, D], K_out/V_out [B, L_out, H_kv, d_h],
 * pos_out [P, B, L_out] with L_out = L_max - N_v + keep. Position ids are
 * carried, not renumbered. seq_len_out [B] (may be NULL) = seq_len - N_v + keep.
 * Output rows >= seq_len_out[b] are left untouched.
 *   idx [B, keep] int32 ascending in [0, N_v) (device).
 * hidden, K, V, pos and the four outputs may each be device memory or host
 * memory the device can dereference (pinned and mapped, cudaHostAlloc):
 * host memory is detected (cudaPointerGetAttributes) and every row is then
 * copied with 16-byte loads and stores from the GPU's threads instead of bulk
 * copies, so that only the surviving rows cross the host link. Results are
 * the same.
 * Row sizes (D and H_kv*d_h elements) must be multiples of 16 bytes and every
 * tensor pointer 16-byte aligned. */
int provip_compact(const int *idx, int B, int N_v, int keep, const void *hidden, int D,
                   const void *K, const void *V, int H_kv, int d_h, const int *pos, int P,
                   const int *seq_len, int L_max, int vis_start, int dtype, void *hidden_out,
                   void *K_out, void *V_out, int *pos_out, int *seq_len_out, void *stream);

/* provip_topk on scores [B, N_v] (keep of them, idx_out ascending) followed by
 * provip_compact with that idx. No workspace. */
int provip_topk_compact(const float *scores, int B, int N_v, int keep, const void *hidden,
                        int D, const void *K, const void *V, int H_kv, int d_h, const int *pos,
                        int P, const int *seq_len, int L_max, int vis_start, int dtype,
                        void *hidden_out, void *K_out, void *V_out, int *pos_out,
                        int *idx_out, int *seq_len_out, void *stream);

/* Head-aware selection: provip_head_scores followed by the top `keep` of the
 * scores (ties to the lower index, idx_out [B, keep] ascending), with the
 * score reduction fused into the top-k kernel (the scores are bit-identical
 * to provip_head_scores'). scores_out_or_null receives v [B, N_v] when
 * non-NULL. Uses the workspace of provip_head_scores. N_v <= 49152. */
int provip_head_topk(const void *Q, const void *K, int B, int L_max, int H_q, int H_kv, int d_h,
                     const int *head_list, int H_sel, const int *text_start, const int *text_len,
                     const uint8_t *row_mask_or_null, int N_t_max, int vis_start, int N_v,
                     const int *seq_len, int keep, int dtype, int algo, int *idx_out,
                     float *scores_out_or_null, void *ws, size_t ws_bytes, void *stream);

/* The in-LLM pruning step end to end: provip_head_topk, then provip_compact
 * with its idx. Arguments as in the calls above; K is both the scored keys and
 * the compacted K. scores_out_or_null receives v [B, N_v] when non-NULL. Uses
 * the workspace of provip_head_scores.
 *
 * Kernels: the head scores, the top-k and the compaction run back to back on
 * the stream; the top-k and the compaction are launched as programmatic
 * dependents (the compaction copies the rows that do not depend on the kept
 * indices while the selection finishes).
 *
 * flags: 0, or a combination of the three below.
 * PROVIP_PRUNE_OVERLAP_PREVIOUS - the call's head-score kernel may start while
 * the kernel before it on the stream (typically the previous call's
 * compaction) is still running; it waits for that kernel only before it
 * completes (its workspace writes do not conflict with the previous call's
 * kernels, which have consumed the workspace by then). Pass it only when this
 * call's Q and K were not written by the kernel launched just before it on the
 * stream (for instance when pruning a stream of independent batches); other
 * kernels in between (e.g. the LLM layers that produce Q/K) make the flag
 * harmless. */
#define PROVIP_PRUNE_OVERLAP_PREVIOUS 1u
/* PROVIP_PRUNE_CONCURRENT - the caller runs other calls at the same time
 * on other streams (e.g. several independent batches side by side). The
 * compaction then takes only as many CTAs as the call's rows fill (at least
 * 160 KiB of rows each) and leaves the remaining SMs to the concurrent calls;
 * without the flag it spreads over every SM, which finishes a call that runs
 * alone soonest. Results are the same either way. */
#define PROVIP_PRUNE_CONCURRENT 2u
/* PROVIP_PRUNE_HOST_ROWS - hidden, V and pos, and the outputs hidden_out,
 * K_out, V_out and pos_out, may be host memory that is pinned and mapped into
 * the device's address space (cudaHostAlloc; any pointer the GPU can
 * dereference). The compaction then copies every kept row with 16-byte loads
 * and stores from the GPU's threads instead of bulk copies, which works for
 * device and mapped host memory alike, so a caller whose sequences live in
 * host memory moves only the surviving rows across the host link. Q and K must
 * still be device memory (the head scores read them through tensor maps), and
 * so must idx_out, seq_len_out and the scores. Results are the same. */
#define PROVIP_PRUNE_HOST_ROWS 4u
size_t provip_prune_workspace_size(int B, int L_max, int H_sel, int N_t_max, int N_v, int algo,
                                   int dtype);
int provip_prune(const void *Q, const void *K, const void *V, const void *hidden, int B,
                 int L_max, int H_q, int H_kv, int d_h, int D, const int *head_list, int H_sel,
                 const int *text_start, const int *text_len, const uint8_t *row_mask_or_null,
                 int N_t_max, int vis_start, int N_v, const int *seq_len, const int *pos, int P,
                 int keep, int dtype, int algo, void *hidden_out, void *K_out, void *V_out,
                 int *pos_out, int *idx_out, int *seq_len_out, float *scores_out_or_null,
                 void *ws, size_t ws_bytes, unsigned flags, void *stream);

/* ------------------------------------------------------------------------
 * Visual-head identification (Sec. 4.4, the head confidence C^h and the set
 * V_l of the N_vis most confident heads) and pruning with those heads
 * ---------------------------------------------------------------------- */

/* Head confidence over every query head h of the pruning layer:
 *   C[b][h] = sum over critical text rows j of Var_i(A_{h,j,i}),
 * A_{h,j,i} the cross-modal attention of provip_head_scores (softmax over the
 * full causal key range, taken at the N_v visual keys) and Var the population
 * variance over the N_v visual columns (1/N_v; the ranking is the same with
 * 1/(N_v - 1)). The critical rows are the text rows j < text_len[b] with
 * crit_mask_or_null[b][j] != 0 (the set T of Sec. 4.2, e.g. from
 * provip_crit_text); NULL takes every text row. Then, per sample, the N_vis
 * heads of largest C (ties to the lower head index) are the visual heads:
 *   vis_heads_out [B, N_vis] int32, ascending head indices (device);
 *   conf_out_or_null [B, H_q] fp32 receives C when non-NULL.
 * The selection is per sample (T and the attention maps are per input). An
 * empty critical set gives C = 0 for every head, hence heads 0..N_vis-1.
 * Every head is read once (all H_q heads' queries on the text rows, every
 * key/value head's keys). Requires H_q <= 64, 1 <= N_vis <= H_q and the shape
 * rules of provip_head_scores. Variances are accumulated per row in fp32 with
 * a pairwise (mean, M2) merge over column chunks.
 * Workspace: provip_visual_heads_workspace_size. */
size_t provip_visual_heads_workspace_size(int B, int L_max, int H_q, int N_t_max, int N_v,
                                          int N_vis, int algo, int dtype);
int provip_head_confidence(const void *Q, const void *K, int B, int L_max, int H_q, int H_kv,
                           int d_h, const int *text_start, const int *text_len,
                           const uint8_t *crit_mask_or_null, int N_t_max, int vis_start,
                           int N_v, const int *seq_len, int N_vis, int dtype, int algo,
                           float *conf_out_or_null, int *vis_heads_out, void *ws,
                           size_t ws_bytes, void *stream);

/* Shallow-layer pruning with visual heads only (Sec. 4.4): the confidence and
 * visual heads of provip_head_confidence, then v from the visual heads of each
 * sample over all its text rows (S^vis and v of Sec. 4.4), the top `keep` of v
 * (idx_out [B, keep] ascending, ties to the lower index) and the compaction of
 * provip_compact. One pass over the keys computes the attention statistics of
 * every head; with the same kernel family on both sides (algo STREAM, CLUSTER,
 * TWOPASS or SIMT) the scores of a sample's visual heads are bit-identical to
 * provip_prune called on that sample alone with head_list = its visual heads.
 * scores_out_or_null [B, N_v], vis_heads_out_or_null [B, N_vis] and
 * conf_out_or_null [B, H_q] receive v, the visual heads and C when non-NULL.
 * flags as in provip_prune. Workspace: provip_visual_heads_workspace_size. */
int provip_prune_visual_heads(const void *Q, const void *K, const void *V, const void *hidden,
                              int B, int L_max, int H_q, int H_kv, int d_h, int D,
                              const int *text_start, const int *text_len,
                              const uint8_t *crit_mask_or_null, int N_t_max, int vis_start,
                              int N_v, const int *seq_len, const int *pos, int P, int N_vis,
                              int keep, int dtype, int algo, void *hidden_out, void *K_out,
                              void *V_out, int *pos_out, int *idx_out, int *seq_len_out,
                              float *scores_out_or_null, int *vis_heads_out_or_null,
                              float *conf_out_or_null, void *ws, size_t ws_bytes,
                              unsigned flags, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* PROVIP_H_ */
