// Internal launch interface between the C-ABI layer and the kernel files.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "sense.h"

// Datastore handle (opaque to callers of the C ABI).
struct sense_datastore {
  const uint16_t* keys;  // bf16 [n, d] in use
  uint16_t* owned;       // normalised copy owned by the handle, or null
  const int32_t* spans;  // [n, m]
  int64_t n;
  int32_t d;
  int32_t m;
  int device;
};

namespace sense {

// The key scan visits rows in tiles of kTileRows.  Every kSampleStride-th
// tile forms the sample from which a per-query score threshold is taken;
// the remaining tiles are scanned against that threshold.
constexpr int kTileRows = 128;
constexpr int kSampleStride = 16;

enum ScanMode { SCAN_ALL = 0, SCAN_SAMPLE = 1, SCAN_REST = 2 };

// Number of sample rows / rest rows for n keys (including the padding rows
// of a partial last tile).
inline int64_t num_tiles(int64_t n) { return (n + kTileRows - 1) / kTileRows; }
inline int64_t sample_tiles(int64_t n) { return (num_tiles(n) + kSampleStride - 1) / kSampleStride; }
inline int64_t rest_tiles(int64_t n) { return num_tiles(n) - sample_tiles(n); }

// How one retrieval call splits its work and its workspace.
struct RetrievePlan {
  bool tc;           // tensor-core scan
  int group;         // queries per pass over the keys
  bool fused;        // single-pass scan with in-register top-k lists
  int fused_blocks;  // its grid size
  bool sampling;     // sample-threshold pass enabled
  int64_t s_rows;    // sample work rows
  int64_t r_rows;    // rest work rows
  int64_t pool_cap;  // pool slots per query
  size_t off_counts, off_thresh, off_sample, off_cand, off_pool, off_qpad, total;
};
RetrievePlan make_plan(const sense_datastore* ds, int q, int k);

// Runs one retrieval call with its workspace at `ws` (laid out by `p`).
sense_status run_retrieve(const RetrievePlan& p, const sense_datastore* ds,
                          const uint16_t* queries, int q, int k, float* out_scores,
                          int32_t* out_idx, char* ws, uint32_t* status, cudaStream_t s);

// Scan `n_work` work rows (mapped to key rows by `mode`) for q <= 8 queries.
// SCAN_SAMPLE writes every candidate key to out[qi * n_work + w];
// SCAN_ALL / SCAN_REST append keys >= thresh[qi] (0 if thresh is null) to
// out[qi * pool_cap + counts[qi]++].
sense_status launch_scan_gemv(const uint16_t* keys, int64_t n, int d, const uint16_t* queries,
                              int q, int mode, int64_t n_work, const uint64_t* thresh,
                              uint64_t* out, uint32_t* counts, int64_t pool_cap,
                              uint32_t* status, cudaStream_t s);

// Single-pass scan for q <= kFusedMaxQ queries and k <= kFusedMaxK: every
// warp keeps a sorted top-k list per query in registers, every block merges
// its warps' lists and writes its k best keys per query to
// cand[(qi * blocks + block) * k + r].  `blocks` must be the grid size the
// workspace was planned with (fused_blocks()).
constexpr int kFusedMaxQ = 4;
constexpr int kFusedMaxK = 128;
int fused_blocks();
inline size_t fused_smem_bytes(int q, int d, int k) {
  const int kpl = k <= 32 ? 1 : (k <= 64 ? 2 : 4);
  return (size_t)q * d * 2 + (size_t)q * 8 * kpl * 32 * sizeof(uint64_t);
}
sense_status launch_scan_gemv_topk(const uint16_t* keys, int64_t n, int d,
                                   const uint16_t* queries, int q, int k, int blocks,
                                   uint64_t* cand, cudaStream_t s);

// Same contract on tcgen05 tensor cores for qg <= nq <= 128 queries held in
// `qpad` ([nq, d] bf16, rows >= qg zero); the work set is n_half 128-row
// tiles selected by `mode`.
sense_status launch_scan_tc(const uint16_t* keys, int64_t n, int d, const uint16_t* qpad, int qg,
                            int nq, int mode, int64_t n_half, const uint64_t* thresh,
                            uint64_t* out, uint32_t* counts, int64_t pool_cap, uint32_t* status,
                            cudaStream_t s);
sense_status launch_selftest_wait(long long limit, uint32_t* status, cudaStream_t s);
// The single-query drafting tail fused in one kernel per query: merge of the
// single-pass scan's `nlists` lists, span gather, small-tree trie (k <=
// 128; draft_fused_fits(k, m)).  Outputs as launch_merge_lists,
// launch_gather (no anchor) and launch_tree.
bool draft_fused_fits(int k, int m);
sense_status launch_draft_fused(const uint64_t* lists, int nlists, int q, int k, float* out_scores,
                                int32_t* out_idx, const int32_t* spans, int64_t n, int m,
                                int32_t* out_spans, int cap, int mask_bits, int32_t* num_nodes,
                                int32_t* tokens, int32_t* parent, int32_t* depth, int32_t* gamma,
                                uint32_t* mask, uint32_t* status, cudaStream_t s);
// The approximate drafting tail fused in one kernel per query: the top k
// of the list scan's pool (short pools padded, as launch_merge_short), span
// gather, small-tree trie (draft_fused_fits(k, m)).
sense_status launch_pool_draft(const uint64_t* pool, const uint32_t* counts, int64_t pool_cap,
                               int q, int k, float* out_scores, int32_t* out_idx,
                               const int32_t* spans, int64_t n, int m, int32_t* out_spans, int cap,
                               int mask_bits, int32_t* num_nodes, int32_t* tokens,
                               int32_t* parent, int32_t* depth, int32_t* gamma, uint32_t* mask,
                               uint32_t* status, cudaStream_t s);
// DynSearch's tail: top k of each query's pool of pool_cap (= ring
// capacity) scored positions, then positions and spans of the winners.
sense_status launch_ctx_pool(const uint64_t* pool, const uint32_t* counts, int64_t pool_cap, int q,
                             int k, float* out_scores, int32_t* rel, const int64_t* count, int m,
                             const int32_t* ring, int64_t* out_pos, int32_t* out_spans,
                             uint32_t* status, cudaStream_t s);
// Span gather of k key indices per query and the small-tree trie fused in
// one kernel per query (draft_fused_fits(k, m)).
sense_status launch_span_draft(const int32_t* idx, int q, int k, const int32_t* spans, int64_t n,
                               int m, int32_t* out_spans, int cap, int mask_bits,
                               int32_t* num_nodes, int32_t* tokens, int32_t* parent,
                               int32_t* depth, int32_t* gamma, uint32_t* mask, uint32_t* status,
                               cudaStream_t s);
// Exact scores of a shortlist of n_cand key indices per query (-1 = empty),
// top k by (score desc, index asc).
sense_status launch_rescore(const uint16_t* keys, int64_t n, int d, const uint16_t* queries, int q,
                            const int32_t* cand, int n_cand, int k, float* out_scores,
                            int32_t* out_idx, uint32_t* status, cudaStream_t s);
sense_status launch_pad_queries(const uint16_t* src, int qg, int d, uint16_t* dst, int nq,
                                cudaStream_t s);
size_t scan_tc_smem_bytes(int d, int nq);
// The driver's cuTensorMapEncodeTiled (as a PFN_cuTensorMapEncodeTiled_v12000).
sense_status tensor_map_encoder(void** fn);

// Per query: exact k-th largest score code among the s_len sample keys ->
// thresh[qi] = code << 32; sample keys at or above it are appended to the
// pool.  `cand` holds q * chunk_count(s_len) * k keys of scratch.
int64_t chunk_count(int64_t s_len);
sense_status launch_threshold(const uint64_t* sample, int64_t s_len, int q, int k,
                              uint64_t* cand, uint64_t* thresh, uint64_t* pool, uint32_t* counts,
                              int64_t pool_cap, uint32_t* status, cudaStream_t s);

// Per query: the k largest keys of `nlists` descending-sorted lists of k
// keys ([q][nlists][k]), sorted descending -> scores, indices.
sense_status launch_merge_lists(const uint64_t* lists, int nlists, int q, int k,
                                float* out_scores, int32_t* out_idx, uint32_t* status,
                                cudaStream_t s);

// Per query: the k largest pool keys, sorted descending -> scores, indices.
// With counts == nullptr every one of the pool_cap slots is a candidate.
sense_status launch_merge(const uint64_t* pool, const uint32_t* counts, int64_t pool_cap, int q,
                          int k, float* out_scores, int32_t* out_idx, uint32_t* status,
                          cudaStream_t s);

// Same, but a query whose pool holds fewer than k keys is not an error: its
// remaining output slots get score -inf and index -1.
sense_status launch_merge_short(const uint64_t* pool, const uint32_t* counts, int64_t pool_cap,
                                int q, int k, float* out_scores, int32_t* out_idx,
                                uint32_t* status, cudaStream_t s);

sense_status launch_normalize(const float* src, int64_t n, int d, uint16_t* dst, cudaStream_t s);

sense_status launch_gather(const int32_t* spans, int64_t n, int m, const int32_t* idx, int q,
                           int k, const int32_t* anchor, int n_keep, int force,
                           int32_t* out_spans, uint32_t* status, cudaStream_t s);

sense_status launch_tree(const int32_t* spans, int q, int k, int m, int cap, int mask_bits,
                         int32_t* num_nodes, int32_t* tokens, int32_t* parent, int32_t* depth,
                         int32_t* gamma, uint32_t* mask, uint32_t* status, cudaStream_t s);

// Additive mask of App. C.6 Eq. 20 for q trees of capacity cap:
// out[q, cap, cache_len] f32 from the ancestor bit rows mask_bits
// [q, cap, ceil(cap/32)], the node counts and the committed lengths.
sense_status launch_tree_mask_full(const uint32_t* mask_bits, const int32_t* num_nodes,
                                   const int32_t* prefix_len, int q, int cap, int cache_len,
                                   float* out, uint32_t* status, cudaStream_t s);

struct GateArgs {
  const int32_t* tokens;
  const int32_t* parent;
  const int32_t* num_nodes;
  const int32_t* gamma;
  int q, k, m, cap;
  const float* root_logits;
  const float* node_logits;
  int vocab;
  const uint16_t* root_hidden;
  const uint16_t* node_hidden;
  int d;
  float thr;
  int kappa, window, tau;
  int unnormalized;
  int32_t* i_star;
  int32_t* L_star;
  int32_t* n_accept;
  int32_t* accepted;
  int32_t* next_node;
  int32_t* next_anchor;
  uint16_t* h_next;
  uint8_t* G;
  void* workspace;
  uint32_t* status;
};
size_t gate_workspace_bytes(int q, int cap, int kappa);
sense_status launch_gate(const GateArgs& a, cudaStream_t s);

}  // namespace sense
