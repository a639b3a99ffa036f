/*
 * sense.h - C ABI of libsense, a GB300 (sm_103a) library for the drafting
 * hot path of SENSE (Semantic Embedding Navigation with Soft-gated
 * Evaluation, arxiv 2606.00021):
 *
 *   hidden-state query --score--> top-k keys --gather--> candidate spans
 *   --loose trie--> draft tree --soft gate--> accepted prefix / next state
 *
 * Conventions shared by every call:
 *  - Every array argument is a DEVICE pointer on the current CUDA device,
 *    owned by the caller, contiguous row-major, unless stated otherwise.
 *  - bf16 values travel as uint16_t bit patterns.
 *  - Calls are asynchronous on the caller's stream (`sense_stream_t` is the
 *    same type as `cudaStream_t`; NULL is the legacy default stream).
 *    Outputs are valid once that stream has been synchronised.
 *  - Arguments are validated on the host before anything is launched; on
 *    any error nothing is launched and the outputs are untouched.  The
 *    functions return a status code, never throw, exit or abort.  A
 *    thread-local message describing the last error is available from
 *    sense_last_error().
 *  - Problems that only the device can see (an out-of-range key index, a
 *    negative token id, a wait that gave up) set bits in a per-device status
 *    word, read with sense_device_status().
 *  - No call synchronises the stream or allocates memory, except
 *    sense_datastore_build with SENSE_DS_NORMALIZE (allocates the normalised
 *    copy), sense_device_status (synchronises) and the first call of the
 *    library on a device (allocates the 256-byte status word).
 */
#ifndef SENSE_H_
#define SENSE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* sense_stream_t;
typedef struct sense_datastore sense_datastore;
typedef struct sense_ivf sense_ivf;
typedef struct sense_ctx sense_ctx;

typedef enum sense_status {
  SENSE_OK = 0,
  SENSE_ERR_INVALID_ARG = 1,   /* bad pointer, size, flag or workspace size  */
  SENSE_ERR_UNSUPPORTED = 2,   /* valid request outside the implemented range */
  SENSE_ERR_OOM = 3,           /* device allocation failed                    */
  SENSE_ERR_CUDA = 4,          /* a CUDA runtime call failed                  */
  SENSE_ERR_DEVICE_STATUS = 5, /* device status word has bits set            */
  SENSE_ERR_TIMEOUT = 6        /* a bounded device wait gave up               */
} sense_status;

/* Bits of the per-device status word. */
#define SENSE_DEVST_BAD_INDEX 0x1u   /* gather: key index outside [0, n)      */
#define SENSE_DEVST_BAD_TOKEN 0x2u   /* tree: negative token id in a span     */
#define SENSE_DEVST_TIMEOUT 0x4u     /* a pipeline wait hit its limit         */
#define SENSE_DEVST_INTERNAL 0x8u    /* an internal consistency check failed  */
#define SENSE_DEVST_BAD_LENGTH 0x10u /* tree mask: committed length + nodes
                                        outside [0, cache_len]               */

/* Key storage types for sense_datastore_build. */
#define SENSE_KEY_BF16 0
#define SENSE_KEY_F32 1

/* Datastore flags. */
#define SENSE_DS_BORROW 0x0u     /* keep the caller's bf16 keys (zero copy)   */
#define SENSE_DS_NORMALIZE 0x1u  /* f32 keys -> unit L2 norm -> bf16 copy     */

/* Gather flags. */
#define SENSE_GATHER_FORCE_ANCHOR 0x1u

/* Tree flags. */
#define SENSE_TREE_MASK_BITS 0x1u

/* Projection / k-means flags. */
#define SENSE_PROJECT_NORMALIZE 0x1u /* unit L2 norm of every projected row   */
#define SENSE_KMEANS_SPHERICAL 0x1u  /* inner-product assignment, unit centroids */

/* Gate flags. */
#define SENSE_GATE_UNNORMALIZED_ENTROPY 0x1u

/* Limits. */
#define SENSE_MAX_K 1024          /* retrieval top-k                          */
#define SENSE_MAX_RESCORE 1024    /* shortlist length of sense_rescore_topk   */
#define SENSE_MAX_M 32            /* span length                              */
#define SENSE_MAX_TREE_TOKENS 8192 /* k * m accepted by sense_build_tree      */
#define SENSE_MAX_KAPPA 16        /* gate top-k                               */
#define SENSE_MAX_WINDOW 64       /* gate lookahead window                    */
#define SENSE_MAX_PROJ_DIM 128    /* projected key dimension                  */

/* Library version, and the name of a status code (the paper has no
 * counterpart; these describe the library itself). */
int32_t sense_version(void);
const char* sense_status_string(sense_status s);
/* Message of the last error raised on the calling thread ("" if none; the
 * paper has no counterpart). */
const char* sense_last_error(void);

/*
 * Device-side failure reporting (the paper has no counterpart): reads the
 * status word of the current device, after synchronising `stream`; if
 * `clear` is non-zero the word is reset to 0 afterwards.
 * Returns SENSE_ERR_DEVICE_STATUS when any bit is set, else SENSE_OK.
 */
sense_status sense_device_status(sense_stream_t stream, uint32_t* out_bits, int32_t clear);

/* ---------------------------------------------------------------------- */
/* a1. Datastore                                                           */
/* ---------------------------------------------------------------------- */
/*
 * The static datastore C_s of Sec. 3.2.1 (Eq. 2, Eq. 6): n pairs
 * (key_i, span_i), key_i a d-dimensional hidden-state key, span_i the m
 * tokens that followed it.  App. E (Implementation Details) states that keys
 * are L2-normalised before indexing.
 *
 *   keys   [n, d] bf16 (key_dtype SENSE_KEY_BF16, flags SENSE_DS_BORROW):
 *          borrowed, must stay alive and unchanged while the datastore is
 *          used.  Or [n, d] f32 (SENSE_KEY_F32 with SENSE_DS_NORMALIZE):
 *          each row is scaled to unit L2 norm and rounded to bf16 (nearest,
 *          ties to even) into a copy owned by the datastore (a zero row
 *          stays zero).  The normalisation runs asynchronously on `stream`.
 *   spans  [n, m] int32, borrowed, token ids >= 0.
 *   Limits: 1 <= n <= 2^31 - 1, 8 <= d <= 65536 with d % 8 == 0,
 *   1 <= m <= SENSE_MAX_M; keys and spans 16-byte aligned.
 * *out receives an opaque host handle; release it with
 * sense_datastore_destroy (which frees the normalised copy, if any, after
 * synchronising the device).
 */
sense_status sense_datastore_build(const void* keys, int32_t key_dtype, int64_t n, int32_t d,
                                   const int32_t* spans, int32_t m, uint32_t flags,
                                   sense_stream_t stream, sense_datastore** out);
sense_status sense_datastore_destroy(sense_datastore* ds);
/* Device pointer of the bf16 keys in use (borrowed or owned). */
const uint16_t* sense_datastore_keys(const sense_datastore* ds);

/* ---------------------------------------------------------------------- */
/* a2 + a3. Scoring and top-k                                              */
/* ---------------------------------------------------------------------- */
/*
 * Exact inner-product search (Sec. 3.2.2 Eq. 7 and Eq. 8's sim(.,.); App. C.2
 * Alg. 2): for each query q, s[q, i] = <queries[q], key_i> accumulated in
 * fp32 from bf16 inputs, and the k largest scores are returned in the order
 * (score descending, key index ascending).
 *
 *   queries    [q, d] bf16, 16-byte aligned.
 *   out_scores [q, k] f32; out_idx [q, k] int32 (key indices).
 *   workspace  device scratch of at least
 *              sense_retrieve_workspace_bytes(ds, q, k) bytes, 256-byte
 *              aligned; its contents on entry do not matter.
 *   Limits: q >= 1, 1 <= k <= min(n, SENSE_MAX_K).
 * Paths: q <= 8 uses a CUDA-core streaming kernel; q > 8 uses tcgen05
 * tensor-core tiles (queries padded to a multiple of 16, processed in
 * groups of at most 128).
 */
size_t sense_retrieve_workspace_bytes(const sense_datastore* ds, int32_t q, int32_t k);
sense_status sense_retrieve_topk(const sense_datastore* ds, const uint16_t* queries, int32_t q,
                                 int32_t k, float* out_scores, int32_t* out_idx,
                                 void* workspace, size_t workspace_bytes, sense_stream_t stream);

/*
 * Sec. 3.2.2 Eq. 7's exact top-k, the same search as sense_retrieve_topk,
 * for callers that cannot allocate device memory and have no workspace to
 * pass: for example a serving
 * process whose device memory is all handed out in advance by another
 * allocator, or a plug-in whose host application exposes no device
 * allocator and forbids cudaMalloc (it can synchronise the device and fail
 * mid-request).  The paper has no counterpart to this entry point.
 *
 * Scratch comes from one file-scope device array of
 * SENSE_NOALLOC_SCRATCH_BYTES bytes, held by every GPU that loads the
 * library until the process exits.  This function calls no cudaMalloc,
 * cudaFree or other allocating routine.  Its first call on a device looks
 * up the array's device address (cudaGetSymbolAddress) with that device
 * current; make that first call before any stream capture.  A request whose
 * workspace (sense_retrieve_workspace_bytes) exceeds the array minus 256
 * bytes is rejected with SENSE_ERR_UNSUPPORTED.  All calls share the array,
 * which keeps the last call's contents (the counters that must start at zero
 * are cleared by every call); calls that overlap on the GPU race on it, so
 * order them on one stream.  The array's address is kept for the life of
 * the process: no call may span a cudaDeviceReset.  Device-side checks of
 * this function (SENSE_DEVST_INTERNAL, SENSE_DEVST_TIMEOUT) record into a
 * status word inside the array, not the one sense_device_status reads; every
 * call clears it first, and sense_retrieve_noalloc_status reads it.
 * Arguments, outputs and results are those of sense_retrieve_topk.
 */
#define SENSE_NOALLOC_SCRATCH_BYTES (32u << 20)
sense_status sense_retrieve_topk_noalloc(const sense_datastore* ds, const uint16_t* queries,
                                         int32_t q, int32_t k, float* out_scores,
                                         int32_t* out_idx, sense_stream_t stream);

/*
 * Device status of sense_retrieve_topk_noalloc on the current device (the
 * paper has no counterpart): synchronises `stream`, copies the status word
 * of the static array into *out_bits and, when `clear` is non-zero, zeroes
 * it.  Read it after a call and before the next one (each call clears it).
 * Allocates nothing.  Returns SENSE_ERR_TIMEOUT when SENSE_DEVST_TIMEOUT is
 * set, SENSE_ERR_DEVICE_STATUS for any other bit, SENSE_OK for none; a
 * non-OK result means that call's outputs must not be used.
 */
sense_status sense_retrieve_noalloc_status(sense_stream_t stream, uint32_t* out_bits,
                                           int32_t clear);

/*
 * Failure-detection self test of that status word (the paper has no
 * counterpart): the bounded-wait self test of sense_selftest_timeout, with
 * its SENSE_DEVST_TIMEOUT written into the static array's status word
 * instead of the device status word.  Read it with
 * sense_retrieve_noalloc_status.  Allocates nothing.
 */
sense_status sense_retrieve_noalloc_selftest(sense_stream_t stream, int64_t limit_cycles);

/* ---------------------------------------------------------------------- */
/* Approximate retrieval: PCA projection and an IVF / IVF-PQ index          */
/* ---------------------------------------------------------------------- */
/*
 * Sec. 3.2.2 Eq. 7 retrieves with ANN(k_t, C_db, N'); App. E builds it from
 * final-layer hidden states projected by PCA to 64 dimensions and
 * L2-normalised (Alg. 2: k = L2Norm(PCA(h))), indexed by FAISS IVF-PQ with
 * nlist = 4096 cells, nprobe = 32 and pq_m = 16 sub-quantizers.
 *
 * Arithmetic: fp32 without fused multiply-add, in a fixed order, so that
 * every decision (cell, code, probe, top-k index) is reproducible:
 * projected-space dot products and squared distances are summed term by
 * term in index order; the projection's length-d dot products are summed as
 * 32 interleaved partial sums (partial l takes the 4-column groups g with
 * g mod 32 = l, ascending) combined by an xor butterfly (16, 8, 4, 2, 1).
 * Every term of a projection sum thus passes through at most
 * h = 4 ceil(d / 128) + 5 additions, and each projected coordinate is within
 * (h + 2) 2^-24 sum_j |x_j - mu_j| |W_oj| of the exact value.
 */

/*
 * The key / query construction k = L2Norm(PCA(h)) of Alg. 2 and App. E:
 * y = (x - mean) W^T for bf16 rows x [n, d] and a basis W [v, d] f32 (rows =
 * principal axes); mean [d] f32 or NULL.  With SENSE_PROJECT_NORMALIZE each
 * row is then divided by its L2 norm (zero rows stay zero).  out [n, v] f32.
 * Limits: d % 8 == 0, 1 <= v <= SENSE_MAX_PROJ_DIM; x, basis, mean 16-byte
 * aligned.  The PCA basis itself is fitted offline by the caller.  For
 * small batches the rows are staged by bulk copies whose wait is bounded: a
 * copy that never lands sets SENSE_DEVST_TIMEOUT and leaves its row
 * unwritten.
 */
sense_status sense_project(const uint16_t* x, int64_t n, int32_t d, const float* basis, int32_t v,
                           const float* mean, uint32_t flags, float* out, sense_stream_t stream);

/*
 * Lloyd's k-means, the training of App. E's IVF-PQ index (its coarse
 * quantizer and its PQ codebooks, which the paper's FAISS trains): `iters` rounds of assignment (SENSE_KMEANS_SPHERICAL: largest
 * inner product, else smallest squared L2 distance; ties to the lowest
 * centroid) and update (member means accumulated as 2^-31 fixed-point
 * integers, divided in fp64, rounded to fp32; an empty cluster keeps its
 * centroid; spherical: then unit norm; spherical seeds are normalised
 * first).  x [n, dim] f32 with row stride ld floats (dim in {4, 8, 16, 32,
 * 64, 128}); init [k, dim] seeds; centroids [k, dim] out; out_assign [n]
 * (last round's assignment) or NULL.  workspace: at least
 * sense_kmeans_workspace_bytes(n, dim, k) bytes, 256-byte aligned.
 * Limits: 1 <= n < 2^31, 1 <= k <= 65536, iters >= 0.
 */
size_t sense_kmeans_workspace_bytes(int64_t n, int32_t dim, int32_t k);
sense_status sense_kmeans(const float* x, int64_t n, int32_t dim, int32_t ld, int32_t k,
                          int32_t iters, uint32_t flags, const float* init, float* centroids,
                          int32_t* out_assign, void* workspace, size_t workspace_bytes,
                          sense_stream_t stream);

/*
 * App. E's IVF-PQ encodes residuals: cell of each vector (largest inner
 * product with a centroid, ties to the lowest cell) and its residual
 * r = x - c_cell, for training PQ codebooks.
 * vecs [n, v] f32, centroids [nlist, v]; out_cell [n] int32,
 * out_residuals [n, v] f32.  v in {16, 32, 64, 128}, nlist <= 16384.
 */
sense_status sense_ivf_residuals(const float* vecs, int64_t n, int32_t v, const float* centroids,
                                 int32_t nlist, int32_t* out_cell, float* out_residuals,
                                 sense_stream_t stream);

/*
 * The index of Sec. 3.2.2 Eq. 7's ANN search as App. E sets it up (IVF or
 * IVF-PQ over L2-normalised PCA keys): builds an inverted-file index over
 * unit vectors vecs [n, v] f32 (copied; the index owns its memory,
 * allocated here, freed by sense_ivf_destroy).
 *  - cell of x = arg max_c <x, c> over centroids [nlist, v] (unit centroids:
 *    the nearest one);
 *  - lists in cell order, members in ascending key index;
 *  - codebooks NULL (pq_m = 0): the lists hold the vectors (IVF-flat);
 *    codebooks [pq_m, 256, v / pq_m] f32: the lists hold 8-bit codes of
 *    the residual x - c_cell, sub-vector m coded as its nearest codeword
 *    (squared L2, ties to the lowest index), as FAISS IVF-PQ encodes.
 * Synchronises `stream` (it reads the longest list length back).
 * Limits: n < 2^31, v in {16, 32, 64, 128}, nlist <= 16384, v / pq_m <= 16.
 */
sense_status sense_ivf_build(const float* vecs, int64_t n, int32_t v, const float* centroids,
                             int32_t nlist, const float* codebooks, int32_t pq_m,
                             sense_stream_t stream, sense_ivf** out);
sense_status sense_ivf_destroy(sense_ivf* ix);

/*
 * Read-only view of an index (inspection; the paper has no counterpart):
 * out_info [5] = {n, v, nlist, pq_m, longest
 * list}; device pointers to the list offsets [nlist + 1] int64, the key
 * index of each slot [n] int32 and the payload (flat: vectors [n, v] f32;
 * PQ: codes [n, pq_m] uint8), in list order.  Any output may be NULL.
 */
sense_status sense_ivf_arrays(const sense_ivf* ix, int64_t* out_info, const int64_t** out_offsets,
                              const int32_t** out_ids, const void** out_payload);

/*
 * Sec. 3.2.2 Eq. 7's ANN(k_t, C_db, N') with App. E's nprobe: top-k of the
 * approximate scores over the nprobe best cells, per query:
 *  - coarse score <q, c> for every cell; the nprobe largest are probed
 *    (ties to the lower cell); out_probes [q, nprobe] int32 or NULL;
 *  - IVF-flat: score = <q, x>; IVF-PQ: score = <q, c_cell> +
 *    sum_m <q_m, B_m[code_m]> (m ascending), the inner product decomposed
 *    over the residual;
 *  - out_scores [q, k] f32 / out_idx [q, k] int32 key indices, order (score
 *    desc, index asc); slots past the number of candidates in the probed
 *    lists get -inf / -1.
 * queries [q, v] f32 (projected, e.g. by sense_project).  workspace: at
 * least sense_ivf_search_workspace_bytes(ix, q, k, nprobe) bytes, 256-byte
 * aligned.  Limits: 1 <= q <= 65535, 1 <= k <= SENSE_MAX_K,
 * 1 <= nprobe <= min(nlist, SENSE_MAX_K).
 */
size_t sense_ivf_search_workspace_bytes(const sense_ivf* ix, int32_t q, int32_t k, int32_t nprobe);
sense_status sense_ivf_search(const sense_ivf* ix, const float* queries, int32_t q, int32_t k,
                              int32_t nprobe, float* out_scores, int32_t* out_idx,
                              int32_t* out_probes, void* workspace, size_t workspace_bytes,
                              sense_stream_t stream);

/*
 * Exact re-scoring of an approximate shortlist (Sec. 3.2.2 Eq. 8: the
 * composite score ranks the N' retrieved candidates D_ret by sim(h, k_i),
 * the similarity of the full hidden state to each candidate's key, and keeps
 * the top N).  For each query q, the score of candidate c is
 * <queries[q], keys[cand_idx[q, c]]> over the datastore's stored bf16 keys
 * with fp32 accumulation (the precision of sense_retrieve_topk; the
 * summation order differs, so a score may differ from that call's in the
 * last bits), and the k best candidates are written in the order (score
 * desc, key index asc).  A candidate that appears twice is scored and kept
 * twice.
 *
 * queries: bf16 [q, d] (the full hidden states), 16-byte aligned;
 * cand_idx: int32 [q, n_cand] key indices, -1 for an empty slot (what
 * sense_ivf_search writes when fewer than N' keys were found);
 * out_scores: f32 [q, k], out_idx: int32 [q, k]; slots beyond the valid
 * candidates get -inf / -1.  Device pointers owned by the caller; no
 * workspace.  Limits: 1 <= q <= 65535, 1 <= k <= n_cand <= SENSE_MAX_RESCORE.
 * An index outside [0, n) is treated as empty and sets
 * SENSE_DEVST_BAD_INDEX; a key-row copy that never lands sets
 * SENSE_DEVST_TIMEOUT and drops that warp's remaining candidates.
 * Asynchronous on `stream`.  A query runs on a cluster of 16 CTAs where the
 * device can hold one, else 8; SENSE_RESCORE_CLUSTER=8 in the environment
 * (read once per process) selects 8.
 */
sense_status sense_rescore_topk(const sense_datastore* ds, const uint16_t* queries, int32_t q,
                                const int32_t* cand_idx, int32_t n_cand, int32_t k,
                                float* out_scores, int32_t* out_idx, sense_stream_t stream);

/*
 * The approximate drafting step of one query batch in one call (App. E:
 * k = L2Norm(PCA(h)) searched in an IVF / IVF-PQ index, Sec. 3.2.2 Eq. 7
 * ANN; optionally Eq. 8's exact re-scoring of N' = rerank candidates; then
 * the D_ret span gather and the Sec. 3.2.3 Eq. 9 loose trie): the results,
 * bit for bit, of sense_project (normalised), sense_ivf_search (k, or
 * rerank candidates followed by sense_rescore_topk to k), sense_gather_drafts
 * without an anchor and sense_build_tree.  queries: bf16 [q, d] hidden
 * states with d = the datastore's d; basis [v, d] and mean [d] (nullable)
 * as for sense_project, v = the index's dimension; rerank = 0 (no
 * re-scoring) or in [k, SENSE_MAX_RESCORE].  The workspace is
 * sense_ann_draft_workspace_bytes(ix, q, k, nprobe, rerank) bytes, 256-byte
 * aligned; outputs as sense_draft.  Errors and device status are those of
 * the composed calls.
 */
size_t sense_ann_draft_workspace_bytes(const sense_ivf* ix, int32_t q, int32_t k, int32_t nprobe,
                                       int32_t rerank);
sense_status sense_ann_draft(const sense_ivf* ix, const sense_datastore* ds, const uint16_t* queries,
                             int32_t q, const float* basis, const float* mean, int32_t k,
                             int32_t nprobe, int32_t rerank, int32_t node_cap, uint32_t flags,
                             void* workspace, size_t workspace_bytes, float* out_scores,
                             int32_t* out_idx, int32_t* out_spans, int32_t* out_num_nodes,
                             int32_t* out_tokens, int32_t* out_parent, int32_t* out_depth,
                             int32_t* out_gamma, uint32_t* out_mask_bits, sense_stream_t stream);

/*
 * The approximate retrieval of sense_ann_draft without its gather and trie
 * (the static side of a hybrid step, Alg. 2): out_scores / out_idx [q, k]
 * exactly as sense_ann_draft writes them.  The workspace is
 * sense_ann_draft_workspace_bytes(ix, q, k, nprobe, rerank) bytes; the
 * datastore supplies the keys of the re-scoring (rerank > 0) and d.
 */
sense_status sense_ann_search(const sense_ivf* ix, const sense_datastore* ds,
                              const uint16_t* queries, int32_t q, const float* basis,
                              const float* mean, int32_t k, int32_t nprobe, int32_t rerank,
                              void* workspace, size_t workspace_bytes, float* out_scores,
                              int32_t* out_idx, sense_stream_t stream);

/* ---------------------------------------------------------------------- */
/* a4. Span gather                                                          */
/* ---------------------------------------------------------------------- */
/*
 * Candidate drafts D (Sec. 3.2.2, D_ret = {(k_i, s_i)}):
 * out_spans[q, r, :] = spans[idx[q, r], :].
 *
 *   idx       [q, k] int32 (as returned by sense_retrieve_topk).
 *   anchor    NULL, or [q] int32 anchor tokens x~.  With an anchor, the
 *             composite score of Eq. 8 (alpha >> beta) reorders the
 *             candidates: rows whose first token equals the anchor come
 *             first, each group keeping retrieval order; the first n_keep
 *             rows are written.  With SENSE_GATHER_FORCE_ANCHOR the first
 *             token of kept row 0 and of kept row n_keep-1 is set to the
 *             anchor (App. C.2 Alg. 2, forced anchor).
 *   n_keep    rows written per query: 1 <= n_keep <= k (must equal k when
 *             anchor is NULL).
 *   out_spans [q, n_keep, m] int32.
 * An index outside [0, n) produces a row of -1 and sets
 * SENSE_DEVST_BAD_INDEX; no out-of-range load is made.
 */
sense_status sense_gather_drafts(const sense_datastore* ds, const int32_t* idx, int32_t q,
                                 int32_t k, const int32_t* anchor, int32_t n_keep, uint32_t flags,
                                 int32_t* out_spans, sense_stream_t stream);

/* ---------------------------------------------------------------------- */
/* Dynamic context buffer and hybrid candidates                             */
/* ---------------------------------------------------------------------- */
/*
 * Sec. 3.2.1 Eq. 6: C_db = C_s u C_d, where the dynamic buffer C_d is filled
 * from the generation itself.  Alg. 1 appends (hidden state, token it
 * predicted) pairs with R.Update after prefill and after every accepted
 * step; Alg. 2 searches C_d with DynSearch, adds a boost delta to its scores
 * (s = [s_s; s_d + delta]) and reranks the union with Eq. 8.
 * Readings (the paper does not define DynSearch or a buffer size): an entry
 * is a position p with key L2Norm(h_p) stored as bf16 and span y_{p+1} ..
 * y_{p+M} (the tokens predicted by h_p .. h_{p+M-1}); it is searchable once
 * those M tokens have been appended; the buffer keeps the `capacity` most
 * recent positions as a ring; DynSearch is the exact inner-product top-k
 * (ties to the older position).
 */

/* The dynamic context buffer C_d of Sec. 3.2.1 (Eq. 6) and Alg. 1:
 * creates an empty buffer (allocates capacity * (2 d + 4) bytes on the
 * current device).  Limits: 1 <= m <= SENSE_MAX_M, m <= capacity <= 2^24,
 * d % 8 == 0. */
sense_status sense_ctx_create(int32_t capacity, int32_t d, int32_t m, sense_ctx** out);
sense_status sense_ctx_destroy(sense_ctx* ctx);
/* C_d's bookkeeping (Alg. 1 appends to it; the paper gives no reset or
 * count).  The buffer's position counter lives on the device, so that appends whose
 * length is only known there (sense_ctx_append_path) need no host round
 * trip.  sense_ctx_reset forgets every entry (asynchronous on `stream`);
 * sense_ctx_count synchronises `stream` and reads the number of positions
 * appended since creation or the last reset. */
sense_status sense_ctx_reset(sense_ctx* ctx, sense_stream_t stream);
sense_status sense_ctx_count(const sense_ctx* ctx, sense_stream_t stream, int64_t* out);

/*
 * R.Update: appends t positions.  hidden [t, d] bf16 (16-byte aligned):
 * the hidden state at each position; tokens [t] int32: the token that state
 * predicted (Alg. 1 passes H_align[i*, 0:L*+1] with the accepted tokens a).
 * When t > capacity only the last `capacity` rows are kept.  Asynchronous
 * on `stream`; later searches on the same stream see the new entries.
 */
sense_status sense_ctx_append(sense_ctx* ctx, const uint16_t* hidden, const int32_t* tokens,
                              int32_t t, sense_stream_t stream);

/*
 * R.Update after a verified step (Alg. 1): appends the accepted path
 * H_align[i*, 0:L*+1] with the accepted tokens a, entirely on the device.
 * Position j < n_accept gets the hidden state root_hidden [d] (j = 0) or
 * node_hidden[gamma[i*, j-1]] (node_hidden [n_nodes, d] bf16; gamma [k, m]
 * of this query's tree) and the token accepted[j]; i_star, n_accept and
 * accepted are device pointers (the outputs of sense_soft_gate for one
 * query).  An i* or a node outside its range sets SENSE_DEVST_BAD_INDEX and
 * that position is skipped.
 */
sense_status sense_ctx_append_path(sense_ctx* ctx, const uint16_t* root_hidden,
                                   const uint16_t* node_hidden, int32_t n_nodes,
                                   const int32_t* gamma, int32_t k, const int32_t* i_star,
                                   const int32_t* n_accept, const int32_t* accepted,
                                   sense_stream_t stream);

/*
 * Alg. 2's DynSearch over C_d (with the boost delta of its scores): per
 * query (queries [q, d] bf16, 16-byte aligned), the k
 * searchable entries with the largest <q, key> (fp32 accumulation), order
 * (score desc, position asc).  out_scores [q, k] f32 = score + delta;
 * out_pos [q, k] int64 positions; out_spans [q, k, m] int32.  Slots past the
 * number of searchable entries get -inf, -1 and a span of -1.  workspace:
 * sense_ctx_search_workspace_bytes(ctx, q, k) bytes, 256-byte aligned.
 * Limits: 1 <= q <= 65535, 1 <= k <= SENSE_MAX_K, delta finite.
 */
size_t sense_ctx_search_workspace_bytes(const sense_ctx* ctx, int32_t q, int32_t k);
sense_status sense_ctx_search(const sense_ctx* ctx, const uint16_t* queries, int32_t q, int32_t k,
                              float delta, float* out_scores, int64_t* out_pos,
                              int32_t* out_spans, void* workspace, size_t workspace_bytes,
                              sense_stream_t stream);

/*
 * Hybrid candidate drafts (Alg. 2, D_all = D_s u D_d and Eq. 8): per query,
 * the static results (static_scores [q, ks] f32 and static_idx [q, ks] key
 * indices of `ds`, e.g. from sense_retrieve_topk) and the dynamic results
 * (dyn_scores [q, kd] f32 already boosted, -inf = empty slot, dyn_spans
 * [q, kd, m] from sense_ctx_search) are ordered by score (desc; ties keep
 * static before dynamic and rank order within each).  With an anchor x~ per
 * query (anchor [q] or NULL) the candidates starting with x~ move first
 * (stable), the first n_keep rows are kept, and SENSE_GATHER_FORCE_ANCHOR
 * sets the first token of the first and of the last kept row to x~.  Rows
 * past the number of live candidates are -1.  out_spans [q, n_keep, m].
 * Limits: 1 <= ks + kd <= 2048, 1 <= n_keep <= ks + kd, m = the datastore's
 * span length.  A static index outside [0, n) sets SENSE_DEVST_BAD_INDEX and
 * that candidate is dropped.
 */
sense_status sense_hybrid_drafts(const sense_datastore* ds, const float* static_scores,
                                 const int32_t* static_idx, int32_t ks, const float* dyn_scores,
                                 const int32_t* dyn_spans, int32_t kd, int32_t q,
                                 const int32_t* anchor, int32_t n_keep, uint32_t flags,
                                 int32_t* out_spans, sense_stream_t stream);

/*
 * The hybrid drafting step's buffer side and tail in one call (Alg. 2:
 * DynSearch over the buffer with the delta boost, the union D_all with the
 * static results reranked by Eq. 8, then the Sec. 3.2.3 Eq. 9 loose trie of
 * the kept rows): the results, bit for bit, of sense_ctx_search(ctx,
 * queries, q, kd, delta) into dyn_scores [q, kd] f32, dyn_pos [q, kd] int64,
 * dyn_spans [q, kd, m] int32, then sense_hybrid_drafts(ds, static_scores,
 * static_idx, ks, ..., anchor, n_keep, flags) into out_spans [q, n_keep, m],
 * then sense_build_tree(out_spans, q, n_keep, m, node_cap, tree_flags) into
 * the tree outputs (as sense_build_tree).  The datastore and the buffer
 * share d and m.  workspace: sense_ctx_search_workspace_bytes(ctx, q, kd)
 * bytes, 256-byte aligned.  When n_keep <= 128 (and the trie fits shared
 * memory) it is two kernels: the buffer's scores, then one block per query
 * for the rest; otherwise the three calls' launches.  Errors and device
 * status are those of the composed calls.
 */
sense_status sense_dyn_draft(const sense_datastore* ds, const sense_ctx* ctx,
                             const uint16_t* queries, int32_t q, const float* static_scores,
                             const int32_t* static_idx, int32_t ks, int32_t kd, float delta,
                             const int32_t* anchor, int32_t n_keep, uint32_t flags,
                             int32_t node_cap, uint32_t tree_flags, void* workspace,
                             size_t workspace_bytes, float* dyn_scores, int64_t* dyn_pos,
                             int32_t* dyn_spans, int32_t* out_spans, int32_t* out_num_nodes,
                             int32_t* out_tokens, int32_t* out_parent, int32_t* out_depth,
                             int32_t* out_gamma, uint32_t* out_mask_bits, sense_stream_t stream);

/* ---------------------------------------------------------------------- */
/* a5. Loose trie (draft tree)                                              */
/* ---------------------------------------------------------------------- */
/*
 * Sorted-LCP loose trie of Sec. 3.2.3 Eq. 9 / App. C.3 Alg. 3: the distinct
 * non-empty prefixes of the k candidate spans of each query, numbered in
 * lexicographic preorder (the order of T_flat).
 *
 *   spans [q, k, m] int32 token ids (>= 0).
 *   node_cap  C > 0 keeps at most C nodes: each node is keyed by
 *             (smallest candidate rank containing it, depth) and the C
 *             smallest keys are kept (prefix-closed); 0 = no cap.
 *   Output capacity cap = node_cap if node_cap > 0 else k * m.
 *   out_num_nodes [q]; out_tokens, out_parent, out_depth [q, cap]
 *   (parent -1 = child of the current position; depth 0-based; slots past
 *   num_nodes are -1); out_gamma [q, k, m] = node id of candidate r's
 *   prefix of length j+1, in the candidates' input order (-1 when the cap
 *   dropped it).
 *   out_mask_bits (with SENSE_TREE_MASK_BITS, else may be NULL):
 *   [q, cap, ceil(cap/32)] uint32, bit b of row n set iff node b is an
 *   ancestor of n or n itself (Alg. 3's mask M).
 *   Limits: 1 <= k <= SENSE_MAX_K, 1 <= m <= SENSE_MAX_M,
 *   k * m <= SENSE_MAX_TREE_TOKENS.
 * A negative token sets SENSE_DEVST_BAD_TOKEN and that query gets
 * num_nodes = 0 with all outputs -1.
 */
sense_status sense_build_tree(const int32_t* spans, int32_t q, int32_t k, int32_t m,
                              int32_t node_cap, uint32_t flags, int32_t* out_num_nodes,
                              int32_t* out_tokens, int32_t* out_parent, int32_t* out_depth,
                              int32_t* out_gamma, uint32_t* out_mask_bits, sense_stream_t stream);

/*
 * The drafting step of one query batch in one call (the paper has no
 * separate counterpart: it is Sec. 3.2.2 Eq. 7 retrieval, the D_ret span
 * gather and the Sec. 3.2.3 Eq. 9 loose trie, composed): the same results,
 * bit for bit, as sense_retrieve_topk, then sense_gather_drafts without an
 * anchor (n_keep = k), then sense_build_tree on the gathered spans.
 * Arguments are those calls' arguments; out_spans is int32 [q, k, m] with
 * m = the datastore's span length, 16-byte aligned; the workspace is
 * sense_retrieve_workspace_bytes(ds, q, k) bytes, 256-byte aligned.  For
 * the single-pass retrieval (q <= 4, k <= 128, the exact scan's fused
 * lists) the merge, the gather and the trie run as one kernel per query;
 * otherwise the calls' own launches run in order.  Errors and device status
 * are those of the three calls.
 */
sense_status sense_draft(const sense_datastore* ds, const uint16_t* queries, int32_t q, int32_t k,
                         void* workspace, size_t workspace_bytes, int32_t node_cap, uint32_t flags,
                         float* out_scores, int32_t* out_idx, int32_t* out_spans,
                         int32_t* out_num_nodes, int32_t* out_tokens, int32_t* out_parent,
                         int32_t* out_depth, int32_t* out_gamma, uint32_t* out_mask_bits,
                         sense_stream_t stream);

/* ---------------------------------------------------------------------- */
/* Tree attention mask over a static KV cache                               */
/* ---------------------------------------------------------------------- */
/*
 * App. C.6 Eq. 20: the additive mask M_full with which the target model
 * verifies all L = num_nodes draft tokens in one forward pass over a static
 * KV cache.  The draft tokens occupy cache positions m .. m+L-1 behind the
 * m committed tokens.  For draft token i and cache position j:
 *   M_full[i, j] = 0     if j < m,
 *                = 0     if m <= j < m+L and node j-m is an ancestor of i
 *                        or i itself (Alg. 3's M, from sense_build_tree's
 *                        SENSE_TREE_MASK_BITS output),
 *                = -inf  otherwise.
 * Rows i >= L pad the fixed capacity: they get 0 on the m committed
 * columns and -inf elsewhere.
 *
 *   mask_bits [q, cap, ceil(cap/32)] uint32 (bit b of row n: M[n, b]);
 *   num_nodes [q] int32 (L); prefix_len [q] int32 (m);
 *   out [q, cap, cache_len] f32.
 *   Limits: q >= 1, 1 <= cap <= SENSE_MAX_TREE_TOKENS, cache_len >= 1;
 *   arrays 4-byte aligned (16-byte aligned out with cache_len % 4 == 0
 *   takes the vector store path).
 * A query with m < 0 or m + L > cache_len (or L outside [0, cap]) sets
 * SENSE_DEVST_BAD_LENGTH and gets rows of -inf.
 */
sense_status sense_tree_mask_full(const uint32_t* mask_bits, const int32_t* num_nodes, int32_t q,
                                  int32_t cap, const int32_t* prefix_len, int32_t cache_len,
                                  float* out, sense_stream_t stream);

/*
 * Tree-masked attention of the verify forward (Alg. 1: Forward(T, M_full,
 * K)) for one sequence, on tcgen05 tensor cores: per head h,
 *   out[h] = softmax(scale * Q[h] K[h]^T + M_full) V[h]
 * over the first prefix_len + L cache positions, where the L draft tokens
 * sit at positions prefix_len .. prefix_len + L - 1 and M_full is the mask
 * of Eq. 20 built on the fly from Alg. 3's ancestor bits (see
 * sense_tree_mask_full).
 *   q [heads, L, 128] bf16 (the draft tokens' queries);
 *   k_cache [heads, capacity, 128] bf16; vt_cache [heads, 128, capacity]
 *   bf16 (V stored transposed per head, so that both products read K-major
 *   tiles); positions past prefix_len + L are never used;
 *   mask_bits: L rows of mask_words uint32 (row n, bit b: node b is an
 *   ancestor of n or n itself), e.g. one query's rows of sense_build_tree's
 *   SENSE_TREE_MASK_BITS output;
 *   out [heads, L, 128] f32.  Probabilities are rounded to bf16 before the
 *   product with V (fp32 accumulation throughout).
 *   workspace: sense_tree_attention_workspace_bytes(heads, L, prefix_len)
 *   bytes, 256-byte aligned (used only when a head's keys are split over
 *   more than 8 CTAs; up to 8 splits merge on chip).
 * Limits: d_head == 128, 1 <= L <= 128, capacity % 128 == 0, prefix_len +
 * L <= capacity, scale > 0; q, caches and out 16-byte aligned.
 */
size_t sense_tree_attention_workspace_bytes(int32_t heads, int32_t L, int32_t prefix_len);
sense_status sense_tree_attention(const uint16_t* q, const uint16_t* k_cache,
                                  const uint16_t* vt_cache, int32_t heads, int32_t L,
                                  int32_t d_head, int32_t capacity, int32_t prefix_len,
                                  const uint32_t* mask_bits, int32_t mask_words, float scale,
                                  float* out, void* workspace, size_t workspace_bytes,
                                  sense_stream_t stream);

/* ---------------------------------------------------------------------- */
/* a6. Soft-gated evaluation                                                */
/* ---------------------------------------------------------------------- */
/*
 * Sec. 3.3 (Eqs. 12-19) and App. C.4 Alg. 4, per query:
 *  - position j of candidate i carries draft token D[i,j] = tokens[gamma[i,j]]
 *    and is predicted by P_align[i,j] = root_logits (j = 0) or the logits
 *    row of node gamma[i,j-1] (Eq. 11 alignment);
 *  - B_em = I(D == argmax P_align) (lowest index among equal maxima);
 *  - B_ent = I(E / log V > gamma), E the entropy of softmax(P_align) in nats
 *    (SENSE_GATE_UNNORMALIZED_ENTROPY: I(E > gamma), Eq. 14);
 *  - B_topk = I(D in top-kappa of P_align), order (logit desc, index asc);
 *  - B_con = I(#mismatches among positions j+1..j+W <= tau), positions past
 *    the span (and positions dropped by the node cap) counting as
 *    mismatches (Alg. 4's reading of Eq. 16: a strictly-future window);
 *  - G = B_em | (B_ent & (B_topk | B_con)); L_i = leading run of ones in
 *    G[i,:] minus 1; i* = lowest i with the largest L_i; L* = L_{i*}.
 * Positions whose node was dropped by the cap have G = 0.
 *
 *   tokens, parent [q, cap], num_nodes [q], gamma [q, k, m]: the tree from
 *   sense_build_tree (same cap).
 *   root_logits [q, vocab] f32 (p); node_logits [q, cap, vocab] f32 (the
 *   target logits at each tree node, P').  Only rows of the root, of nodes
 *   that have children, and of the chosen next node are read.
 *   root_hidden [q, d] bf16 (h); node_hidden [q, cap, d] bf16 (H').
 *   Outputs: out_i_star, out_L_star, out_n_accept (= L*+1), out_next_node
 *   (gamma[i*, L*], or -1 for the root when L* = -1), out_next_anchor
 *   (argmax of the next node's logits row, p_next of Eq. 19) [q] int32;
 *   out_accepted [q, m] int32 (D[i*, 0..L*], then -1);
 *   out_h_next [q, d] bf16 (h_next of Eq. 19);
 *   out_G [q, k, m] uint8 or NULL.
 *   params: gamma (threshold), topk (kappa, 1..SENSE_MAX_KAPPA), window W
 *   (1..SENSE_MAX_WINDOW), tau (>= 0), flags.  Paper defaults (App. E):
 *   gamma 0.05, kappa 3, W 6, tau 0.
 *   workspace: at least sense_soft_gate_workspace_bytes(q, cap, kappa)
 *   bytes of device scratch, 256-byte aligned, zero-filled before its
 *   first use and used by no other call: it holds per-query counters that
 *   let the last row of a query run the decision in the same launch, and
 *   every call leaves them zero.
 *   Limits: vocab >= kappa, vocab % 4 == 0; d % 8 == 0; k * m <=
 *   SENSE_MAX_TREE_TOKENS; logits 16-byte aligned.
 */
typedef struct sense_gate_params {
  float gamma;
  int32_t topk;
  int32_t window;
  int32_t tau;
  uint32_t flags;
} sense_gate_params;

size_t sense_soft_gate_workspace_bytes(int32_t q, int32_t cap, int32_t kappa);
sense_status sense_soft_gate(const int32_t* tokens, const int32_t* parent,
                             const int32_t* num_nodes, const int32_t* gamma, int32_t q, int32_t k,
                             int32_t m, int32_t cap, const float* root_logits,
                             const float* node_logits, int32_t vocab, const uint16_t* root_hidden,
                             const uint16_t* node_hidden, int32_t d,
                             const sense_gate_params* params, int32_t* out_i_star,
                             int32_t* out_L_star, int32_t* out_n_accept, int32_t* out_accepted,
                             int32_t* out_next_node, int32_t* out_next_anchor,
                             uint16_t* out_h_next, uint8_t* out_G, void* workspace,
                             size_t workspace_bytes, sense_stream_t stream);

/* ---------------------------------------------------------------------- */
/* Diagnostics                                                              */
/* ---------------------------------------------------------------------- */
/*
 * Failure-detection self test (the paper has no counterpart): one block
 * waits on a shared-memory barrier that nothing arrives on, through the same
 * bounded wait the tensor-core pipeline uses, with a limit of limit_cycles
 * SM clocks (1 .. 2^34).  The wait gives up, sets SENSE_DEVST_TIMEOUT in the
 * device status word and the kernel returns; the context stays usable.
 * Read the result with sense_device_status.
 */
sense_status sense_selftest_timeout(sense_stream_t stream, int64_t limit_cycles);

/* ---------------------------------------------------------------------- */
/* Launch profiling                                                         */
/* ---------------------------------------------------------------------- */
/*
 * Instrumentation (the paper has no counterpart).  When enabled, every
 * kernel launch of the library is bracketed by two CUDA events recorded on
 * the launching stream.  sense_profile_enable(1) clears
 * earlier records.  sense_profile_query synchronises on the recorded events
 * and returns, for the kernel family `name` (see sense_profile_name), the
 * summed device time in milliseconds and the number of launches.
 */
sense_status sense_profile_enable(int32_t on);
/*
 * Instrumentation, continued (no counterpart in the paper).  Restricts the
 * bracketing to the comma-separated kernel families in
 * `names` (NULL or "" = every family) until the next sense_profile_enable,
 * which selects every family again.  Each bracketed launch adds two event
 * records to its stream; filtering keeps them off the launches that are not
 * being measured.  SENSE_ERR_INVALID_ARG for an unknown family name.
 */
sense_status sense_profile_filter(const char* names);
/* The kernel families (count, i-th name) and the summed time of one family
 * (instrumentation; no counterpart in the paper). */
int32_t sense_profile_count(void);
const char* sense_profile_name(int32_t i);
sense_status sense_profile_query(const char* name, double* total_ms, int64_t* launches);

#ifdef __cplusplus
}
#endif
#endif /* SENSE_H_ */
