// Exact top-k selection over candidate keys (Sec. 3.2.2 Eq. 7, top-N' by
// similarity; ties to the lower key index).
//
// A candidate key packs (score code, ~index) into 64 bits so that the total
// order (score desc, index asc) is plain unsigned order.  Both kernels run
// one 1024-thread block per query and select by MSD radix: a 256-bin
// shared-memory histogram per 8-bit digit (warp-aggregated with
// __match_any_sync, since candidates share their high digits), a warp scan
// to find the digit holding the k-th largest key, and early exit once that
// digit's bin holds exactly the keys still needed.
//  - threshold: k-th largest score code of the sample -> per-query threshold;
//    sample keys at or above it are copied into the query's pool;
//  - merge: the k largest keys of the pool, bitonic-sorted in shared memory.
#include "common.cuh"
#include "launch.h"

namespace sense {
namespace {

constexpr int kSelThreads = 1024;

struct Digit {
  int bucket;
  int above;
};

// Histogram add for one value per thread (active lanes only).
__device__ __forceinline__ void hist_add(unsigned* hist, bool active, unsigned bin) {
  const unsigned am = __ballot_sync(0xffffffffu, active);
  if (active) {
    const unsigned grp = __match_any_sync(am, bin);
    const int lane = threadIdx.x & 31;
    if (lane == __ffs(grp) - 1) atomicAdd(&hist[bin], (unsigned)__popc(grp));
  }
}

// Finds the bin b (scanning from 255 down) where the running count first
// reaches `remaining`; writes (b, count strictly above b) to *out.
__device__ void find_digit(const unsigned* hist, int remaining, Digit* out) {
  if (threadIdx.x >= 32) return;
  const int lane = threadIdx.x;
  int c[8];
  int sum = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    c[i] = (int)hist[255 - 8 * lane - i];
    sum += c[i];
  }
  int incl = sum;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += t;
  }
  const int excl = incl - sum;
  if (excl < remaining && remaining <= incl) {
    int acc = excl;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      if (acc + c[i] >= remaining) {
        out->bucket = 255 - 8 * lane - i;
        out->above = acc;
        break;
      }
      acc += c[i];
    }
  }
}

__global__ void __launch_bounds__(kSelThreads)
threshold_kernel(const uint64_t* __restrict__ sample, int64_t s_len, int k,
                 uint64_t* __restrict__ thresh, uint64_t* __restrict__ pool,
                 uint32_t* __restrict__ counts, int64_t pool_cap, uint32_t* status) {
  __shared__ unsigned hist[256];
  __shared__ Digit dig;
  const int q = blockIdx.x;
  const uint64_t* src = sample + (int64_t)q * s_len;
  uint32_t prefix = 0, pmask = 0;
  int remaining = k;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    if (threadIdx.x == 0) dig.bucket = -1;
    __syncthreads();
    for (int64_t i0 = 0; i0 < s_len; i0 += blockDim.x) {
      const int64_t i = i0 + threadIdx.x;
      const uint32_t hi = (i < s_len) ? (uint32_t)(src[i] >> 32) : 0u;
      const bool act = (i < s_len) && ((hi & pmask) == prefix);
      hist_add(hist, act, (hi >> shift) & 255u);
    }
    __syncthreads();
    find_digit(hist, remaining, &dig);
    __syncthreads();
    if (dig.bucket < 0) {  // fewer than k sample keys: cannot happen when s_len >= k
      if (threadIdx.x == 0) raise_status(status, SENSE_DEVST_INTERNAL);
      prefix = 0;
      pmask = 0;
      break;
    }
    remaining -= dig.above;
    prefix |= (uint32_t)dig.bucket << shift;
    pmask |= 255u << shift;
    const bool exact = (int)hist[dig.bucket] == remaining;
    __syncthreads();
    if (exact) break;  // every key with this prefix is needed: prefix is a valid bound
  }
  // Keys whose high word matches the prefix (or exceeds it) number >= k.
  const uint64_t t0 = (uint64_t)prefix << 32;
  if (threadIdx.x == 0) thresh[q] = t0;
  uint64_t* dst = pool + (int64_t)q * pool_cap;
  for (int64_t i0 = 0; i0 < s_len; i0 += blockDim.x) {
    const int64_t i = i0 + threadIdx.x;
    const uint64_t c = (i < s_len) ? src[i] : 0ull;
    const bool want = (i < s_len) && (c >= t0);
    const uint32_t pos = warp_append(&counts[q], want);
    if (want) {
      if ((int64_t)pos < pool_cap) dst[pos] = c;
      else raise_status(status, SENSE_DEVST_INTERNAL);
    }
  }
}

__global__ void __launch_bounds__(kSelThreads)
merge_kernel(const uint64_t* __restrict__ pool, const uint32_t* __restrict__ counts,
             int64_t pool_cap, int k, float* __restrict__ out_scores,
             int32_t* __restrict__ out_idx, uint32_t* status) {
  __shared__ unsigned hist[256];
  __shared__ Digit dig;
  __shared__ unsigned n_sel;
  __shared__ uint64_t sel[SENSE_MAX_K];
  const int q = blockIdx.x;
  const uint64_t* src = pool + (int64_t)q * pool_cap;
  int64_t cnt = counts[q];
  if (cnt > pool_cap) cnt = pool_cap;

  uint64_t prefix = 0, pmask = 0;
  int remaining = k;
  bool ok = true;
  for (int shift = 56; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    if (threadIdx.x == 0) dig.bucket = -1;
    __syncthreads();
    for (int64_t i0 = 0; i0 < cnt; i0 += blockDim.x) {
      const int64_t i = i0 + threadIdx.x;
      const uint64_t c = (i < cnt) ? src[i] : 0ull;
      const bool act = (i < cnt) && ((c & pmask) == prefix);
      hist_add(hist, act, (unsigned)(c >> shift) & 255u);
    }
    __syncthreads();
    find_digit(hist, remaining, &dig);
    __syncthreads();
    if (dig.bucket < 0) {
      ok = false;
      break;
    }
    remaining -= dig.above;
    prefix |= (uint64_t)dig.bucket << shift;
    pmask |= 255ull << shift;
    const bool exact = (int)hist[dig.bucket] == remaining;
    __syncthreads();
    if (exact) break;
  }
  if (!ok) {  // fewer than k candidates: internal error, outputs marked
    if (threadIdx.x == 0) raise_status(status, SENSE_DEVST_INTERNAL);
    for (int r = threadIdx.x; r < k; r += blockDim.x) {
      out_scores[(int64_t)q * k + r] = 0.0f;
      out_idx[(int64_t)q * k + r] = -1;
    }
    return;
  }
  // Collect the keys whose masked prefix is >= the selected prefix: exactly k.
  if (threadIdx.x == 0) n_sel = 0;
  __syncthreads();
  for (int64_t i = threadIdx.x; i < cnt; i += blockDim.x) {
    const uint64_t c = src[i];
    if ((c & pmask) >= prefix) {
      const unsigned p = atomicAdd(&n_sel, 1u);
      if (p < (unsigned)k) sel[p] = c;
    }
  }
  __syncthreads();
  int kp = 1;
  while (kp < k) kp <<= 1;
  for (int i = threadIdx.x; i < kp; i += blockDim.x) {
    if (i >= k) sel[i] = 0ull;
  }
  __syncthreads();
  // Bitonic sort, descending.
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

}  // namespace

sense_status launch_threshold(const uint64_t* sample, int64_t s_len, int q, int k,
                              uint64_t* thresh, uint64_t* pool, uint32_t* counts,
                              int64_t pool_cap, uint32_t* status, cudaStream_t s) {
  LaunchScope ls(K_THRESHOLD, s);
  threshold_kernel<<<q, kSelThreads, 0, s>>>(sample, s_len, k, thresh, pool, counts, pool_cap,
                                             status);
  return cuda_check(cudaGetLastError(), "launch threshold");
}

sense_status launch_merge(const uint64_t* pool, const uint32_t* counts, int64_t pool_cap, int q,
                          int k, float* out_scores, int32_t* out_idx, uint32_t* status,
                          cudaStream_t s) {
  LaunchScope ls(K_MERGE, s);
  merge_kernel<<<q, kSelThreads, 0, s>>>(pool, counts, pool_cap, k, out_scores, out_idx, status);
  return cuda_check(cudaGetLastError(), "launch merge");
}

}  // namespace sense
