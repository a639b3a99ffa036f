// Exact top-k selection over candidate keys (Sec. 3.2.2 Eq. 7, top-N' by
// similarity; ties to the lower key index).
//
// A candidate key packs (score code, ~index) into 64 bits so that the total
// order (score desc, index asc) is plain unsigned order.  Selection is an
// MSD radix select: a 256-bin shared-memory histogram per 8-bit digit
// (warp-aggregated with __match_any_sync, since candidates share their high
// digits), a warp scan to find the digit holding the k-th largest key, and
// early exit once that digit's bin holds exactly the keys still needed.
// Keys are read from shared memory when they fit, else from global memory.
//  - chunk_topk: sample keys are cut into chunks of kChunk; one block per
//    (chunk, query) keeps the chunk's k largest keys.  The k largest of the
//    whole sample are among the union of these lists, and a key left out of
//    its chunk's list has k larger keys beside it, so it can be neither in
//    the final top-k nor needed by the threshold below;
//  - threshold: per query, the k-th largest score code of the lists gives
//    the per-query threshold (a lower bound of the final k-th score: the
//    sample is a subset of the keys); list keys at or above it enter the
//    query's pool;
//  - merge: per query, the k largest pool keys, bitonic-sorted in shared
//    memory, become the output scores and indices.
#include "common.cuh"
#include "draft_dev.cuh"
#include "launch.h"
#include "select_dev.cuh"
#include "tc_ptx.cuh"

namespace sense {
namespace {

constexpr int kChunk = 8192;  // keys per first-level block (64 KB)

__global__ void __launch_bounds__(kSelThreads, 1)
chunk_topk_kernel(const uint64_t* __restrict__ sample, int64_t s_len, int k, int n_chunks,
                  uint64_t* __restrict__ cand, uint32_t* status) {
  extern __shared__ uint64_t s_keys[];
  __shared__ unsigned hist[256];
  __shared__ Digit dig;
  __shared__ unsigned n_sel;
  const int c = blockIdx.x, q = blockIdx.y;
  const int64_t lo = (int64_t)c * kChunk;
  const int cnt = (int)min((int64_t)kChunk, s_len - lo);
  const uint64_t* src = sample + (int64_t)q * s_len + lo;
  uint64_t* dst = cand + ((int64_t)q * n_chunks + c) * k;
  if (cnt <= k) {
    for (int i = threadIdx.x; i < k; i += blockDim.x) dst[i] = (i < cnt) ? src[i] : 0ull;
    return;
  }
  for (int i = threadIdx.x; i < cnt; i += blockDim.x) s_keys[i] = src[i];
  __syncthreads();
  uint64_t prefix, pmask;
  const bool ok = radix_select([&](int64_t i) { return s_keys[i]; }, cnt, k, 0, hist, &dig,
                               &prefix, &pmask);
  if (!ok) {
    if (threadIdx.x == 0) raise_status(status, SENSE_DEVST_INTERNAL);
    return;
  }
  if (threadIdx.x == 0) n_sel = 0;
  __syncthreads();
  for (int i = threadIdx.x; i < cnt; i += blockDim.x) {
    const uint64_t key = s_keys[i];
    if ((key & pmask) >= prefix) {
      const unsigned p = atomicAdd(&n_sel, 1u);
      if (p < (unsigned)k) dst[p] = key;
    }
  }
}

__global__ void __launch_bounds__(kSelThreads, 1)
threshold_kernel(const uint64_t* __restrict__ lists, int64_t len, int k,
                 uint64_t* __restrict__ thresh, uint64_t* __restrict__ pool,
                 uint32_t* __restrict__ counts, int64_t pool_cap, uint32_t* status) {
  extern __shared__ uint64_t s_keys[];
  __shared__ unsigned hist[256];
  __shared__ Digit dig;
  const int q = blockIdx.x;
  const uint64_t* src = lists + (int64_t)q * len;
  const bool staged = len <= kSmemKeys;
  if (staged) {
    for (int64_t i = threadIdx.x; i < len; i += blockDim.x) s_keys[i] = src[i];
    __syncthreads();
  }
  auto get = [&](int64_t i) { return staged ? s_keys[i] : src[i]; };
  uint64_t prefix, pmask;
  // Score codes only (bits 63..32): the threshold needs no index order.
  const bool ok = radix_select(get, len, k, 32, hist, &dig, &prefix, &pmask);
  if (!ok && threadIdx.x == 0) raise_status(status, SENSE_DEVST_INTERNAL);
  // Keys whose masked high word is >= the prefix number at least k; the
  // threshold keeps them all (prefix's unselected low bits are zero).
  const uint64_t t0 = ok ? prefix : 0ull;
  if (threadIdx.x == 0) thresh[q] = t0;
  uint64_t* dst = pool + (int64_t)q * pool_cap;
  for (int64_t i0 = 0; i0 < len; i0 += blockDim.x) {
    const int64_t i = i0 + threadIdx.x;
    const uint64_t c = (i < len) ? get(i) : 0ull;
    const bool want = (i < len) && c != 0ull && (c >= t0);
    const uint32_t pos = warp_append(&counts[q], want);
    if (want) {
      if ((int64_t)pos < pool_cap) dst[pos] = c;
      else raise_status(status, SENSE_DEVST_INTERNAL);
    }
  }
}

__global__ void __launch_bounds__(kSelThreads, 1)
merge_kernel(const uint64_t* __restrict__ pool, const uint32_t* __restrict__ counts,
             int64_t pool_cap, int k, float* __restrict__ out_scores,
             int32_t* __restrict__ out_idx, uint32_t* status, int pad_short) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  extern __shared__ uint64_t s_keys[];
  merge_pool_block(pool, counts, pool_cap, k, out_scores, out_idx, status, pad_short, blockIdx.x,
                   s_keys);
}

// Exact top-k of `nlists` lists of k keys per query, each list sorted in
// descending order (the per-block output of the single-pass scan).  The
// k-th largest list head is a lower bound T of the k-th largest key (k lists
// each hold a key >= T), so only list prefixes >= T are candidates; they are
// gathered into shared memory, selected and sorted.  If the gathered set
// would not fit, every key of every list is used instead.
//
// Small merges (the lists fit in kFastKeys keys, at most kRankHeads lists)
// take a short path: one bulk copy brings every list into shared memory, T
// is the head of rank k - 1 (ranks counted against warp-sorted groups of
// heads by binary search), and each gathered candidate's rank among the
// candidates is its output slot, so no radix passes or block-wide sorting
// network run.  Nonzero keys are distinct (a key row lives in one list),
// which makes the ranks a permutation.
constexpr int kGather = 4096;
constexpr int kFastKeys = 20480;   // list keys staged by the short path (160 KB)
constexpr int kFastCand = 1024;    // candidates it ranks
constexpr int kRankHeads = 1024;   // lists it ranks
constexpr long long kCopyWaitCycles = 4000000000LL;

__device__ __forceinline__ bool wait_copy(uint32_t bar) {
  if (ptx::mbar_try_wait(bar, 0)) return true;
  const long long t0 = clock64();
  while (!ptx::mbar_try_wait(bar, 0)) {
    if (clock64() - t0 > kCopyWaitCycles) return false;
  }
  return true;
}

// The short path; returns false (block-uniform) when the candidates do not
// suit it, leaving the general path to run.  On a timed-out copy it marks the
// outputs and status and returns true.
__device__ bool merge_lists_short(const uint64_t* __restrict__ src, int nlists, int k,
                                  float* __restrict__ out_scores, int32_t* __restrict__ out_idx,
                                  uint32_t* status, uint64_t* s_keys) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint64_t s_t;
  __shared__ unsigned s_got;
  __shared__ int s_ok;
  uint64_t* s_cand = s_keys + kFastKeys;
  uint64_t* s_grp = s_cand + kFastCand;  // heads in sorted groups of 32
  const int total = nlists * k;
  const uint32_t b = ptx::smem_u32(&bar);
  if (threadIdx.x == 0) {
    ptx::mbar_init(b, 1);
    ptx::fence_barrier_init();
    const uint32_t bytes = (uint32_t)total * 8u;
    ptx::mbar_arrive_expect_tx(b, bytes);
    const uint64_t pol = ptx::policy_evict_first();
    for (uint32_t off = 0; off < bytes; off += 32768u)
      ptx::bulk_load(ptx::smem_u32(s_keys) + off, reinterpret_cast<const char*>(src) + off,
                     min(32768u, bytes - off), b, pol);
    s_t = 0ull;
    s_got = 0u;
  }
  __syncthreads();
  const bool arrived = wait_copy(b);
  if (!__syncthreads_and(arrived)) {
    if (threadIdx.x == 0) {
      raise_status(status, SENSE_DEVST_TIMEOUT);
      wait_copy(b);  // give the copy a second bound before the block leaves
    }
    for (int r = threadIdx.x; r < k; r += blockDim.x) {
      out_scores[r] = 0.0f;
      out_idx[r] = -1;
    }
    __syncthreads();
    return true;
  }
  // T: the k-th largest nonzero head (0 when fewer than k heads are
  // nonzero; nonzero keys are distinct).  Heads are cut into groups of 32,
  // each sorted (descending) by one warp with a bitonic network over
  // shuffles; a head's rank is the sum over groups of the heads above it,
  // found by binary search.
  if (nlists >= k) {
    const int lane = threadIdx.x & 31;
    const int ngroups = (nlists + 31) >> 5;
    for (int g = threadIdx.x >> 5; g < ngroups; g += blockDim.x >> 5) {
      const int i = g * 32 + lane;
      uint64_t h = (i < nlists) ? s_keys[(int64_t)i * k] : 0ull;
#pragma unroll
      for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
          const uint64_t o = __shfl_xor_sync(0xffffffffu, h, stride);
          const bool keep_max = ((lane & stride) == 0) == ((lane & size) == 0);
          h = keep_max ? (h > o ? h : o) : (h < o ? h : o);
        }
      }
      s_grp[i] = h;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < nlists; i += blockDim.x) {
      const uint64_t h = s_keys[(int64_t)i * k];
      if (h == 0ull) continue;
      int rank = 0;
      for (int g = 0; g < ngroups; ++g) {
        const uint64_t* grp = s_grp + g * 32;
        // heads of group g above h (a prefix, the group being descending):
        // the longest prefix of at most 31 found by halving steps, then slot 31
        int lo = 0;
#pragma unroll
        for (int step = 16; step > 0; step >>= 1)
          if (grp[lo + step - 1] > h) lo += step;
        rank += lo + ((lo == 31 && grp[31] > h) ? 1 : 0);
      }
      if (rank == k - 1) s_t = h;
    }
  }
  __syncthreads();
  const uint64_t t = s_t;
  for (int l = threadIdx.x; l < nlists; l += blockDim.x) {
    const uint64_t* lb = s_keys + (int64_t)l * k;
    for (int r = 0; r < k; ++r) {
      const uint64_t c = lb[r];
      if (c < t || c == 0ull) break;
      const unsigned p = atomicAdd(&s_got, 1u);
      if (p < (unsigned)kFastCand) s_cand[p] = c;
    }
  }
  __syncthreads();
  const int got = (int)s_got;
  if (threadIdx.x == 0) s_ok = (got >= k && got <= kFastCand);
  __syncthreads();
  if (!s_ok) return false;
  for (int i = threadIdx.x; i < got; i += blockDim.x) {
    const uint64_t c = s_cand[i];
    int rank = 0;
    for (int j = 0; j < got; ++j) {
      const uint64_t o = s_cand[j];
      rank += (o > c) || (o == c && j < i);
    }
    if (rank < k) {
      out_scores[rank] = code_score((uint32_t)(c >> 32));
      out_idx[rank] = (int32_t)cand_index(c);
    }
  }
  return true;
}

// Merge of query q's nlists sorted lists of k keys into its top k, by one
// block of kSelThreads threads; s_keys holds kSmemKeys keys.
__device__ void merge_lists_block(const uint64_t* __restrict__ lists, int nlists, int k,
                                  float* __restrict__ out_scores, int32_t* __restrict__ out_idx,
                                  uint32_t* status, int q, uint64_t* s_keys) {
  __shared__ unsigned hist[256];
  __shared__ Digit dig;
  __shared__ unsigned n_sel, n_got;
  __shared__ uint64_t sel[SENSE_MAX_K];
  const uint64_t* src = lists + (int64_t)q * nlists * k;
  if ((int64_t)nlists * k <= kFastKeys && nlists <= kRankHeads && ((nlists * k) & 1) == 0 &&
      (reinterpret_cast<uintptr_t>(src) & 15) == 0) {
    if (merge_lists_short(src, nlists, k, out_scores + (int64_t)q * k, out_idx + (int64_t)q * k,
                          status, s_keys))
      return;
  }
  // 1. lower bound from the list heads
  for (int b = threadIdx.x; b < nlists; b += blockDim.x) s_keys[b] = src[(int64_t)b * k];
  __syncthreads();
  uint64_t t = 0ull;
  if (nlists >= k) {
    uint64_t prefix, pmask;
    if (radix_select([&](int64_t i) { return s_keys[i]; }, nlists, k, 0, hist, &dig, &prefix,
                     &pmask))
      t = prefix;
  }
  // 2. gather list prefixes >= t
  if (threadIdx.x == 0) n_got = 0;
  __syncthreads();
  for (int b = threadIdx.x; b < nlists; b += blockDim.x) {
    const uint64_t* lb = src + (int64_t)b * k;
    for (int r = 0; r < k; ++r) {
      const uint64_t c = lb[r];
      if (c < t || c == 0ull) break;
      const unsigned p = atomicAdd(&n_got, 1u);
      if (p < (unsigned)kGather) s_keys[p] = c;
    }
  }
  __syncthreads();
  const bool small = n_got <= (unsigned)kGather;
  const int64_t cnt = small ? (int64_t)n_got : (int64_t)nlists * k;
  if (!small) {  // too many ties near the bound: use every key
    for (int64_t i = threadIdx.x; i < cnt && i < kSmemKeys; i += blockDim.x) s_keys[i] = src[i];
    __syncthreads();
  }
  auto get = [&](int64_t i) { return (i < kSmemKeys) ? s_keys[i] : src[i]; };
  uint64_t prefix, pmask;
  const bool ok = radix_select(get, cnt, k, 0, hist, &dig, &prefix, &pmask);
  if (!ok) {
    if (threadIdx.x == 0) raise_status(status, SENSE_DEVST_INTERNAL);
    for (int r = threadIdx.x; r < k; r += blockDim.x) {
      out_scores[(int64_t)q * k + r] = 0.0f;
      out_idx[(int64_t)q * k + r] = -1;
    }
    return;
  }
  if (threadIdx.x == 0) n_sel = 0;
  __syncthreads();
  for (int64_t i = threadIdx.x; i < cnt; i += blockDim.x) {
    const uint64_t c = get(i);
    if ((c & pmask) >= prefix) {
      const unsigned p = atomicAdd(&n_sel, 1u);
      if (p < (unsigned)k) sel[p] = c;
    }
  }
  __syncthreads();
  int kp = 1;
  while (kp < k) kp <<= 1;
  for (int i = threadIdx.x; i < kp; i += blockDim.x)
    if (i >= k) sel[i] = 0ull;
  __syncthreads();
  for (int size = 2; size <= kp; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < kp; i += blockDim.x) {
        const int j = i ^ stride;
        if (j > i) {
          const bool desc = ((i & size) == 0);
          const uint64_t a = sel[i], b = sel[j];
          if (desc ? (a < b) : (a > b)) {
            sel[i] = b;
            sel[j] = a;
          }
        }
      }
      __syncthreads();
    }
  }
  for (int r = threadIdx.x; r < k; r += blockDim.x) {
    const uint64_t c = sel[r];
    out_scores[(int64_t)q * k + r] = code_score((uint32_t)(c >> 32));
    out_idx[(int64_t)q * k + r] = (int32_t)cand_index(c);
  }
}

__global__ void __launch_bounds__(kSelThreads, 1)
merge_lists_kernel(const uint64_t* __restrict__ lists, int nlists, int k,
                   float* __restrict__ out_scores, int32_t* __restrict__ out_idx,
                   uint32_t* status) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  extern __shared__ uint64_t s_keys[];  // [kSmemKeys]
  merge_lists_block(lists, nlists, k, out_scores, out_idx, status, blockIdx.x, s_keys);
}

// The single-query drafting tail in one block per query: the merge of the
// scan's per-block lists into the top k, the span gather of those k keys
// and the small-tree trie of the gathered spans, one after the other.  Each
// phase reads what the previous one wrote to global memory (visible inside
// the block after a barrier); the trie reuses the merge's shared memory.
__global__ void __launch_bounds__(kSelThreads, 1)
draft_fused_kernel(const uint64_t* __restrict__ lists, int nlists, int k,
                   float* __restrict__ out_scores, int32_t* __restrict__ out_idx,
                   const int32_t* __restrict__ spans, int64_t n, int m, int32_t* out_spans,
                   int cap, int mask_words, int32_t* __restrict__ num_nodes,
                   int32_t* __restrict__ tokens, int32_t* __restrict__ parent,
                   int32_t* __restrict__ depth, int32_t* __restrict__ gamma,
                   uint32_t* __restrict__ mask, uint32_t* status) {
  extern __shared__ uint64_t s_keys[];  // [kSmemKeys]
  __shared__ int scratch[32];
  __shared__ int sv[3];
  const int q = blockIdx.x;
  pdl_wait();  // the scan's lists are complete
  pdl_launch_dependents();
  merge_lists_block(lists, nlists, k, out_scores, out_idx, status, q, s_keys);
  __syncthreads();
  gather_block(spans, n, m, out_idx, k, nullptr, k, 0, out_spans, status, q, scratch);
  __syncthreads();
  tree_small_block(out_spans, k, m, cap, mask_words, num_nodes, tokens, parent, depth, gamma,
                   mask, status, q, reinterpret_cast<int*>(s_keys), scratch, sv);
}

// The approximate drafting tail in one block per query: the top k of the
// list scan's pool (a short pool padded with -inf / -1), the span gather of
// those keys and the small-tree trie, one after the other, as in
// draft_fused_kernel.
__global__ void __launch_bounds__(kSelThreads, 1)
pool_draft_kernel(const uint64_t* __restrict__ pool, const uint32_t* __restrict__ counts,
                  int64_t pool_cap, int k, float* __restrict__ out_scores,
                  int32_t* __restrict__ out_idx, const int32_t* __restrict__ spans, int64_t n,
                  int m, int32_t* out_spans, int cap, int mask_words,
                  int32_t* __restrict__ num_nodes, int32_t* __restrict__ tokens,
                  int32_t* __restrict__ parent, int32_t* __restrict__ depth,
                  int32_t* __restrict__ gamma, uint32_t* __restrict__ mask, uint32_t* status) {
  extern __shared__ uint64_t s_keys[];  // [kSmemKeys]
  __shared__ int scratch[32];
  __shared__ int sv[3];
  const int q = blockIdx.x;
  pdl_wait();  // the scan's pool is complete
  pdl_launch_dependents();
  merge_pool_block(pool, counts, pool_cap, k, out_scores, out_idx, status, 1, q, s_keys);
  __syncthreads();
  gather_block(spans, n, m, out_idx, k, nullptr, k, 0, out_spans, status, q, scratch);
  __syncthreads();
  tree_small_block(out_spans, k, m, cap, mask_words, num_nodes, tokens, parent, depth, gamma,
                   mask, status, q, reinterpret_cast<int*>(s_keys), scratch, sv);
}

// DynSearch's tail in one block per query: the top k of the query's pool of
// buffered positions (a short pool padded with -inf / -1), then each
// winner's absolute position and its span from the token ring.  Entry e of
// the pool is position lo + e, lo = max(0, count - cap) the oldest position
// the ring still holds.
__global__ void __launch_bounds__(kSelThreads, 1)
ctx_pool_kernel(const uint64_t* __restrict__ pool, const uint32_t* __restrict__ counts,
                int64_t pool_cap, int k, float* __restrict__ out_scores,
                int32_t* __restrict__ rel, const int64_t* __restrict__ count, int m,
                const int32_t* __restrict__ ring, int64_t* __restrict__ out_pos,
                int32_t* __restrict__ out_spans, uint32_t* status) {
  extern __shared__ uint64_t s_keys[];  // [kSmemKeys]
  const int q = blockIdx.x;
  pdl_wait();  // the scores are complete
  pdl_launch_dependents();
  merge_pool_block(pool, counts, pool_cap, k, out_scores, rel, status, 1, q, s_keys);
  __syncthreads();
  const int64_t cnt = *count;
  const int64_t cap = pool_cap;  // the pool holds one slot per ring position
  const int64_t lo = cnt > cap ? cnt - cap : 0;
  for (int t = threadIdx.x; t < k * m; t += blockDim.x) {
    const int r = t / m, j = t - r * m;
    const int64_t slot = (int64_t)q * k + r;
    const int e = rel[slot];
    const int64_t p = lo + e;
    if (j == 0) out_pos[slot] = e < 0 ? -1 : p;
    out_spans[slot * m + j] = e < 0 ? -1 : ring[(p + j) % cap];
  }
}

// The span gather of k given key indices and the small-tree trie in one
// block per query (the tail after a shortlist re-scoring).
__global__ void __launch_bounds__(kSelThreads, 1)
span_draft_kernel(const int32_t* __restrict__ idx, int k, const int32_t* __restrict__ spans,
                  int64_t n, int m, int32_t* out_spans, int cap, int mask_words,
                  int32_t* __restrict__ num_nodes, int32_t* __restrict__ tokens,
                  int32_t* __restrict__ parent, int32_t* __restrict__ depth,
                  int32_t* __restrict__ gamma, uint32_t* __restrict__ mask, uint32_t* status) {
  extern __shared__ uint64_t s_keys[];  // [kSmemKeys], the trie's scratch
  __shared__ int scratch[32];
  __shared__ int sv[3];
  const int q = blockIdx.x;
  pdl_wait();  // the indices are complete
  pdl_launch_dependents();
  gather_block(spans, n, m, idx, k, nullptr, k, 0, out_spans, status, q, scratch);
  __syncthreads();
  tree_small_block(out_spans, k, m, cap, mask_words, num_nodes, tokens, parent, depth, gamma,
                   mask, status, q, reinterpret_cast<int*>(s_keys), scratch, sv);
}

template <class K>
sense_status set_smem(K kern, size_t bytes) {
  return cuda_check(func_smem(reinterpret_cast<const void*>(kern), (int)bytes),
                    "cudaFuncSetAttribute(select)");
}

}  // namespace

int64_t chunk_count(int64_t s_len) { return (s_len + kChunk - 1) / kChunk; }

sense_status launch_threshold(const uint64_t* sample, int64_t s_len, int q, int k,
                              uint64_t* cand, uint64_t* thresh, uint64_t* pool, uint32_t* counts,
                              int64_t pool_cap, uint32_t* status, cudaStream_t s) {
  const int64_t nch = chunk_count(s_len);
  const size_t chunk_smem = kChunk * sizeof(uint64_t);
  sense_status st = set_smem(chunk_topk_kernel, chunk_smem);
  if (st != SENSE_OK) return st;
  {
    LaunchScope ls(K_THRESHOLD, s);
    chunk_topk_kernel<<<dim3((unsigned)nch, q), kSelThreads, chunk_smem, s>>>(
        sample, s_len, k, (int)nch, cand, status);
    st = cuda_check(cudaGetLastError(), "launch chunk_topk");
    if (st != SENSE_OK) return st;
  }
  const int64_t len = nch * k;
  const size_t smem = (len <= kSmemKeys) ? (size_t)len * sizeof(uint64_t) : 0;
  st = set_smem(threshold_kernel, kSmemKeys * sizeof(uint64_t));
  if (st != SENSE_OK) return st;
  LaunchScope ls(K_THRESHOLD, s);
  threshold_kernel<<<q, kSelThreads, smem, s>>>(cand, len, k, thresh, pool, counts, pool_cap,
                                                status);
  return cuda_check(cudaGetLastError(), "launch threshold");
}

sense_status launch_merge_lists(const uint64_t* lists, int nlists, int q, int k,
                                float* out_scores, int32_t* out_idx, uint32_t* status,
                                cudaStream_t s) {
  sense_status st = set_smem(merge_lists_kernel, kSmemKeys * sizeof(uint64_t));
  if (st != SENSE_OK) return st;
  LaunchScope ls(K_MERGE, s);
  return cuda_check(launch_pdl(merge_lists_kernel, dim3(q), dim3(kSelThreads),
                              kSmemKeys * sizeof(uint64_t), s, lists, nlists, k, out_scores,
                              out_idx, status),
                    "launch merge_lists");
}

sense_status launch_draft_fused(const uint64_t* lists, int nlists, int q, int k, float* out_scores,
                                int32_t* out_idx, const int32_t* spans, int64_t n, int m,
                                int32_t* out_spans, int cap, int mask_bits, int32_t* num_nodes,
                                int32_t* tokens, int32_t* parent, int32_t* depth, int32_t* gamma,
                                uint32_t* mask, uint32_t* status, cudaStream_t s) {
  sense_status st = set_smem(draft_fused_kernel, kSmemKeys * sizeof(uint64_t));
  if (st != SENSE_OK) return st;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)q);
  cfg.blockDim = dim3(kSelThreads);
  cfg.dynamicSmemBytes = kSmemKeys * sizeof(uint64_t);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  LaunchScope ls(K_DRAFT, s);
  return cuda_check(cudaLaunchKernelEx(&cfg, draft_fused_kernel, lists, nlists, k, out_scores,
                                       out_idx, spans, n, m, out_spans, cap, (cap + 31) / 32,
                                       num_nodes, tokens, parent, depth, gamma,
                                       mask_bits ? mask : nullptr, status),
                    "launch draft_fused");
}

sense_status launch_pool_draft(const uint64_t* pool, const uint32_t* counts, int64_t pool_cap,
                               int q, int k, float* out_scores, int32_t* out_idx,
                               const int32_t* spans, int64_t n, int m, int32_t* out_spans, int cap,
                               int mask_bits, int32_t* num_nodes, int32_t* tokens,
                               int32_t* parent, int32_t* depth, int32_t* gamma, uint32_t* mask,
                               uint32_t* status, cudaStream_t s) {
  sense_status st = set_smem(pool_draft_kernel, kSmemKeys * sizeof(uint64_t));
  if (st != SENSE_OK) return st;
  LaunchScope ls(K_DRAFT, s);
  return cuda_check(launch_pdl(pool_draft_kernel, dim3((unsigned)q), dim3(kSelThreads),
                              kSmemKeys * sizeof(uint64_t), s, pool, counts, pool_cap, k,
                              out_scores, out_idx, spans, n, m, out_spans, cap, (cap + 31) / 32,
                              num_nodes, tokens, parent, depth, gamma, mask_bits ? mask : nullptr,
                              status),
                    "launch pool_draft");
}

sense_status launch_ctx_pool(const uint64_t* pool, const uint32_t* counts, int64_t pool_cap, int q,
                             int k, float* out_scores, int32_t* rel, const int64_t* count, int m,
                             const int32_t* ring, int64_t* out_pos, int32_t* out_spans,
                             uint32_t* status, cudaStream_t s) {
  sense_status st = set_smem(ctx_pool_kernel, kSmemKeys * sizeof(uint64_t));
  if (st != SENSE_OK) return st;
  LaunchScope ls(K_CTX, s);
  return cuda_check(launch_pdl(ctx_pool_kernel, dim3((unsigned)q), dim3(kSelThreads),
                              kSmemKeys * sizeof(uint64_t), s, pool, counts, pool_cap, k,
                              out_scores, rel, count, m, ring, out_pos, out_spans, status),
                    "launch ctx pool");
}

sense_status launch_span_draft(const int32_t* idx, int q, int k, const int32_t* spans, int64_t n,
                               int m, int32_t* out_spans, int cap, int mask_bits,
                               int32_t* num_nodes, int32_t* tokens, int32_t* parent,
                               int32_t* depth, int32_t* gamma, uint32_t* mask, uint32_t* status,
                               cudaStream_t s) {
  sense_status st = set_smem(span_draft_kernel, kSmemKeys * sizeof(uint64_t));
  if (st != SENSE_OK) return st;
  LaunchScope ls(K_DRAFT, s);
  return cuda_check(launch_pdl(span_draft_kernel, dim3((unsigned)q), dim3(kSelThreads),
                              kSmemKeys * sizeof(uint64_t), s, idx, k, spans, n, m, out_spans, cap,
                              (cap + 31) / 32, num_nodes, tokens, parent, depth, gamma,
                              mask_bits ? mask : nullptr, status),
                    "launch span_draft");
}

bool draft_fused_fits(int k, int m) {
  return k <= kTreeSmallK && sizeof(int) * ((size_t)3 * k * m + (size_t)5 * k) <=
                                 kSmemKeys * sizeof(uint64_t);
}

sense_status launch_merge(const uint64_t* pool, const uint32_t* counts, int64_t pool_cap, int q,
                          int k, float* out_scores, int32_t* out_idx, uint32_t* status,
                          cudaStream_t s) {
  sense_status st = set_smem(merge_kernel, kSmemKeys * sizeof(uint64_t));
  if (st != SENSE_OK) return st;
  LaunchScope ls(K_MERGE, s);
  return cuda_check(launch_pdl(merge_kernel, dim3(q), dim3(kSelThreads),
                              kSmemKeys * sizeof(uint64_t), s, pool, counts, pool_cap, k,
                              out_scores, out_idx, status, 0),
                    "launch merge");
}

sense_status launch_merge_short(const uint64_t* pool, const uint32_t* counts, int64_t pool_cap,
                                int q, int k, float* out_scores, int32_t* out_idx,
                                uint32_t* status, cudaStream_t s) {
  sense_status st = set_smem(merge_kernel, kSmemKeys * sizeof(uint64_t));
  if (st != SENSE_OK) return st;
  LaunchScope ls(K_MERGE, s);
  return cuda_check(launch_pdl(merge_kernel, dim3(q), dim3(kSelThreads),
                              kSmemKeys * sizeof(uint64_t), s, pool, counts, pool_cap, k,
                              out_scores, out_idx, status, 1),
                    "launch merge");
}

}  // namespace sense
