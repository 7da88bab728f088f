// Internal launch interface between the C-ABI layer (api.cu) and the kernel
// translation units. Not installed; the public interface is include/provip.h.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace provip {

constexpr int kMaxHeads = 64;
constexpr int kHeadDim = 128;  // d_h supported by the kernels
constexpr int kRowBlock = 128; // text rows per CTA row block

// ---------------------------------------------------------------------------
// head-aware scores (Sec. 4.4): two passes over the keys
//   pass 1 (stats): per text row and key chunk, the chunk max m_c and
//                   sum l_c of exp2(s - m_c) over the causal keys in the chunk;
//   pass 2 (probs): per visual key chunk, p = exp2(s - m) / l with the row's
//                   global (m, l), summed over the rows of the block ->
//                   partial[b][rb * H_sel + head][col].
// Scores are in the base-2 domain: s = <q, k> * log2(e) / sqrt(d_h).
// ---------------------------------------------------------------------------
struct HSArgs {
  const void* Q;  // [B, L_max, H_q, d_h]
  const void* K;  // [B, L_max, H_kv, d_h]
  int B, L_max, H_q, H_kv, d_h;
  int H_sel;
  int heads[kMaxHeads];
  const int* text_start;     // [B]
  const int* text_len;       // [B]
  const uint8_t* row_mask;   // [B, N_t_max] or null
  int N_t_max;
  int vis_start, N_v;
  const int* seq_len;        // [B]
  int n_rb;                  // row blocks: ceil(N_t_max / 128)
  int kc;                    // key chunk width of pass 1
  int n_kc;                  // ceil(L_max / kc)
  int vc;                    // visual chunk width of pass 2
  int n_vc;                  // ceil(N_v / vc)
  float scale_log2;          // log2(e) / sqrt(d_h)
  float2* stats;             // [B][n_rb][H_sel][n_kc][128]
  float* partial;            // [B][n_rb * H_sel][N_v]
  // head confidence (Sec. 4.4), optional: for every valid text row j with
  // conf_mask[b][j] != 0 (null: every valid row), the mean and the sum of
  // squared deviations (M2) of the row's visual probabilities over the columns
  // of each column chunk c the pass-2 kernels own:
  //   conf_part[((b * H_sel + head) * N_t_max + j) * conf_stride + c] = (mean, M2).
  // Chunk c covers the keys [conf_lo0 + c * conf_w, conf_lo0 + (c + 1) * conf_w)
  // intersected with the visual range (ConfGeom below).
  const uint8_t* conf_mask;
  float2* conf_part;         // null: no confidence statistics
  int conf_stride;           // chunk capacity per row
  unsigned* err;
};

// column chunks of the confidence statistics written by the path that ran
struct ConfGeom {
  int lo0;  // first key of chunk 0
  int w;    // keys per chunk
  int n;    // chunks
};

// geom (optional): the column chunks of the confidence statistics
cudaError_t hs_launch_simt(const HSArgs& a, int dtype, cudaStream_t s, ConfGeom* geom = nullptr);
// tcgen05 path (bf16): needs tensor maps over Q and K viewed as 2-D row tables.
cudaError_t hs_launch_tc(const HSArgs& a, const CUtensorMap* tmQ, const CUtensorMap* tmK,
                         cudaStream_t s, ConfGeom* geom = nullptr);
// one-pass tcgen05 path (clusters, TMEM-resident logits): writes the partials
// directly; *launched is false when no cluster shape fits this problem. pdl:
// launched as a programmatic dependent of the previous kernel on the stream
// (it reads Q/K at once and waits for that kernel only before writing).
// geom (optional): the confidence chunks of the launched shape.
cudaError_t hs_launch_fused(const HSArgs& a, const CUtensorMap* tmQ, const CUtensorMap* tmK,
                            cudaStream_t s, bool* launched, bool pdl = false,
                            ConfGeom* geom = nullptr);
// streaming tcgen05 path: one CTA per (row block x head, sample), keys through
// a TMA/TMEM pipeline, visual keys read a second time (from L2); no cluster.
cudaError_t hs_launch_stream(const HSArgs& a, const CUtensorMap* tmQ, const CUtensorMap* tmK,
                             cudaStream_t s, bool pdl = false, ConfGeom* geom = nullptr);
// largest number of confidence chunks the one-pass kernel uses (its cluster size)
constexpr int kFusedMaxChunks = 16;
// scores[b][i] = sum_u partial[b][u][i] / (H_sel * valid text rows of b)
cudaError_t hs_launch_reduce(const HSArgs& a, float* scores, cudaStream_t s);

// Head confidence and visual-head selection (Sec. 4.4): per sample,
//   C[head] = sum over confidence rows j of M2(j) / N_v (population variance of
//   the row's visual probabilities, its chunk statistics merged in chunk order),
// then the n_vis heads of largest C (ties to the lower position in the head
// list), in ascending list position:
//   sel_out[b][s]       position in the head list (for the partial sums),
//   vis_heads_out[b][s] head index (optional), conf_out[b][heads[i]] = C (optional).
// pdl: launched as a programmatic dependent of the head-score kernel.
struct ConfArgs {
  int n_vis;
  int* sel_out;        // [B][n_vis]
  int* vis_heads_out;  // [B][n_vis] or null
  float* conf_out;     // [B][H_q] or null
};
cudaError_t conf_select_launch(const HSArgs& a, const ConfGeom& g, const ConfArgs& c,
                               cudaStream_t s, bool pdl = false);

// ---------------------------------------------------------------------------
// top-k (ties to the lower index, ascending output)
// ---------------------------------------------------------------------------
struct TopkArgs {
  const float* scores;       // [B][N]; or null when reading head partials
  const float* partial;      // [B][n_part][N]
  int n_part;
  const int* text_len;       // used with partial: valid-row count per sample
  const uint8_t* row_mask;
  int N_t_max;
  int H_sel;
  // optional per-sample head subset [B][n_sel] (positions in the head list,
  // ascending): only those heads' partials are summed, divided by n_sel x rows
  const int* sel;
  int n_sel;
  float* scores_out;         // optional [B][N]
  int B, N, k;
  int* idx_out;              // [B][k]
  // optional (N above the rank kernel's range, see topk_writes_index): the
  // merge's index, kpos_out [B][N] (the output slot of a selected element,
  // else -1) and pruned_out [B][N - k] (the others, ascending)
  int* kpos_out;
  int* pruned_out;
  unsigned* err;
};
constexpr int kTopkMaxN = 49152;
// pdl: launched as a programmatic dependent of the previous kernel on the
// stream (the kernel waits for it before reading its inputs)
cudaError_t topk_launch(const TopkArgs& a, cudaStream_t s, bool pdl = false);
// whether topk_launch fills kpos_out / pruned_out for N keys (the block
// selects do; the cluster rank kernel for small N does not)
bool topk_writes_index(int N);

// ---------------------------------------------------------------------------
// compaction: rows [0, vis_start) ++ vis_start + idx ++ [vis_start + N_v, seq_len)
// ---------------------------------------------------------------------------
struct CompactArgs {
  const char* src[3];
  char* dst[3];
  long long row_bytes[3];
  int n_tensors;
  const int* pos;            // [P, B, L_max] or null
  int* pos_out;              // [P, B, L_out]
  int P;
  const int* idx;            // [B, keep]
  int keep, N_v, vis_start;
  const int* seq_len;        // [B]
  int* seq_len_out;          // [B] or null
  int B, L_max, L_out;
  unsigned* err;
};
// pdl: launched as a programmatic dependent of the previous kernel on the
// stream; rows that do not depend on idx are copied before waiting for it.
// allow_deep: the deeper slot ring may be used (it leaves room for a streaming
// head-score CTA per SM, not for the cluster form's larger one). concurrent:
// other calls run beside this one on other streams, so a small problem takes
// only the CTAs its bytes fill (otherwise it spreads over every SM).
// host_rows: sources or destinations may be mapped host memory, so every row is
// copied with 16-byte loads and stores (no bulk copies).
cudaError_t compact_launch(const CompactArgs& a, int num_sms, cudaStream_t s, bool pdl = false,
                           bool allow_deep = true, bool concurrent = false, bool host_rows = false);

// ---------------------------------------------------------------------------
// pre-LLM similarity pass (Sec. 4.2-4.3)
// ---------------------------------------------------------------------------
struct SimArgs {
  const void* emb_v;         // [B, N_v, D]
  const void* emb_t;         // [B, N_t_max, D]
  const int* text_len;       // [B]
  int B, N_v, D, N_t_max;
  int dtype;
  unsigned* err;
};
// Sec. 4.2: mask[b][j] (and r) from the text self-similarity. ws: G, max(1,
// crit_splits) x [B][Ntm][Ntm] f32.
cudaError_t crit_text_launch(const SimArgs& a, uint8_t* mask, float* r_out, float* G,
                             cudaStream_t s);
// inverse L2 norms of every visual row (0 for a zero row): inv_v [B][N_v]
cudaError_t vis_inv_norm_launch(const SimArgs& a, float* inv_v, cudaStream_t s);
// the same for the kept rows keep_idx [B][keep] only (inv_v[b][keep_idx[b][q]]),
// which is all the merge reads
cudaError_t kept_inv_norm_launch(const SimArgs& a, const int* keep_idx, int keep, float* inv_v,
                                 cudaStream_t s);
// Sec. 4.3: p[b][j] = max_{i in T} cos(t_i, v_j) - mu_i; also writes inv_v (the
// inverse norms of the visual rows, used again by the merge). ws_sum holds
// n_split partial sums over row chunks and their total.
// ws_sum holds max((n_split + 1) * B * D, relevance_fused_floats(B, N_v, N_t_max)) floats.
// mask_ready (optional): an event recorded where the mask is written (another
// stream); s waits for it before the first kernel that reads the mask, so that
// the kernels before that one run beside the mask's producer.
cudaError_t relevance_launch(const SimArgs& a, const uint8_t* mask, float* inv_v,
                             float* p, float* ws_sum, float* ws_mu, float* ws_invt,
                             int n_split, int num_sms, cudaStream_t s,
                             cudaEvent_t mask_ready = nullptr);
// Sec. 4.3 merge: assign[b][j] and merged[b][a][:]
// n_split: the SIMT split (sized by the caller); ws_pruned: [B][N_v] ints and
// ws_perm: [B][N_v][D] bf16 for the tcgen05 path (null: CUDA-core path);
// num_sms for its split choice
// index_ready: the kept-position map (in assign) and the pruned list (in
// ws_pruned) were written by the top-k that chose keep_idx (topk_writes_index)
cudaError_t merge_launch(const SimArgs& a, const int* keep_idx, int keep, const float* inv_v,
                         int* assign, void* merged, float* ws_best, int* ws_bidx,
                         int n_split, int* ws_pruned, void* ws_perm, int num_sms, cudaStream_t s,
                         bool index_ready = false);

// tcgen05 forms of the pre-LLM Grams (bf16), used by the launchers above
bool crit_gram_tc_supported(const SimArgs& a);
// K splits of the tcgen05 text Gram (0: not applicable); G holds that many
// [B][N_t_max][N_t_max] parts (at least one)
constexpr int kCritMaxSplits = 16;
int crit_splits(int N_t_max, int D, int dtype);
cudaError_t crit_gram_tc_launch(const SimArgs& a, float* G, cudaStream_t s);
bool relevance_tc_supported(const SimArgs& a);
// workspace floats of the tensor-core relevance (cosines + per-tile sums)
size_t relevance_fused_floats(int B, int N_v, int N_t_max);
// reads the text rows' inverse norms inv_t [B][N_t_max]; writes inv_v and p;
// ws holds relevance_fused_floats(...) floats
cudaError_t relevance_tc_launch(const SimArgs& a, const uint8_t* mask, const float* inv_t, float* inv_v,
                                float* p, float* ws, int num_sms, cudaStream_t s,
                                cudaEvent_t mask_ready = nullptr);
bool merge_tc_supported(const SimArgs& a, int keep, int n_split);
// pruned: the rows not kept, ascending ([B][N_v - keep], from merge_index_kernel)
// Writes the permuted copy perm, then runs the Gram on pairs of SMs when they
// are usable (*n_split_out = its column ranges), else on single SMs with n_split
// column splits (*n_split_out = n_split).
cudaError_t merge_argmax_tc_launch(const SimArgs& a, const int* keep_idx, int keep,
                                   const float* inv_v, const int* pruned, void* perm,
                                   int n_split, float* ws_best, int* ws_bidx, int num_sms,
                                   int* n_split_out, cudaStream_t s);
// N split of the tcgen05 merge Gram (fewest waves x tiles per CTA) and its upper bound
int merge_tc_split(int B, int N_v, int keep, int num_sms);
constexpr int kMergeMaxSplit = 16;

// the merge Gram on pairs of SMs (tcgen05 cta_group::2, merge_pair_tc.cu)
constexpr int kMergePairHeights = 4;
// A tile is (512-row group of one sample's pruned rows, range of its kept
// columns); groups x_hi .. Q-1 split the columns into n_lo ranges, groups
// 0 .. x_hi-1 into n_lo + 1.
struct MergePairPlan {
  int n_quads;  // 512-row groups of pruned rows per sample
  int Q;        // groups of the batch: B * n_quads
  int n_lo;     // column ranges of groups x_hi .. Q-1
  int x_hi;     // groups with n_lo + 1 ranges
  int T;        // tiles
  int P;        // clusters of two CTAs (pairs of SMs), at most T
  int n_slots;  // partial slots per row: n_lo + (x_hi > 0), <= kMergeMaxSplit
  int n_heights;                     // distinct B rows per CTA (N / 2) of the tiles
  int heights[kMergePairHeights];
};
bool merge_pair_plan(int B, int n_pruned, int keep, int D, int num_sms, MergePairPlan* p);
// bf16, the pair form enabled, and a two-CTA cluster of it fits on this device
bool merge_pair_usable(const SimArgs& a);
void merge_pair_enable(int on);
cudaError_t merge_argmax_pair_launch(const SimArgs& a, const int* keep_idx, int keep, const float* inv_v,
                                     const int* pruned, const void* perm, const MergePairPlan& plan,
                                     float* ws_best, int* ws_bidx, cudaStream_t s);

// host helper: encode a 2-D bf16 row table [rows, cols] (row stride in bytes)
// as a tensor map with 64 x box_rows boxes and 128-byte swizzle.
int make_tmap_bf16_2d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols,
                      uint64_t row_stride_bytes, uint32_t box_rows);

}  // namespace provip
