// Block-level top-k selection over 64-bit candidate keys (score code,
// inverted index), shared by the selection kernels (select.cu) and the
// fused kernels that end in a selection (ivf.cu): radix select, the
// group-head short path, the binned path for large k, and the block merge
// of one query's pool that chooses among them.
#pragma once

#include "common.cuh"
#include "draft_dev.cuh"

namespace sense {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kSmemKeys = 24576;      // keys staged in shared memory (192 KB)

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

// Radix select over keys get(0..cnt): finds the digits of the k-th largest
// key from bit 63 down to bit `low`.  On return the keys whose masked bits
// are >= prefix are the ones to keep: exactly k of them when the search
// stopped early or went down to bit 0 (keys distinct), at least k otherwise.
// Returns false if fewer than k keys exist.  All threads must call it.
template <class Get>
__device__ bool radix_select(Get get, int64_t cnt, int k, int low, unsigned* hist, Digit* dig,
                             uint64_t* out_prefix, uint64_t* out_mask) {
  uint64_t prefix = 0, pmask = 0;
  int remaining = k;
  for (int shift = 56; shift >= low; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    if (threadIdx.x == 0) dig->bucket = -1;
    __syncthreads();
    for (int64_t i0 = 0; i0 < cnt; i0 += blockDim.x) {
      const int64_t i = i0 + threadIdx.x;
      const uint64_t c = (i < cnt) ? get(i) : 0ull;
      const bool act = (i < cnt) && ((c & pmask) == prefix);
      hist_add(hist, act, (unsigned)(c >> shift) & 255u);
    }
    __syncthreads();
    find_digit(hist, remaining, dig);
    __syncthreads();
    if (dig->bucket < 0) {
      *out_prefix = prefix;
      *out_mask = pmask;
      return false;
    }
    remaining -= dig->above;
    prefix |= (uint64_t)dig->bucket << shift;
    pmask |= 255ull << shift;
    const bool exact = (int)hist[dig->bucket] == remaining;
    __syncthreads();
    if (exact) break;
  }
  *out_prefix = prefix;
  *out_mask = pmask;
  return true;
}

// Short path of merge_kernel for a pool of distinct nonzero keys (at most
// 32 * kPoolGroups of them).  The pool is cut into
// groups of at most 32; a group's maximum is a head, and the k-th largest head T
// bounds the k-th largest key from below (k groups hold a key >= T).  Heads
// are ranked against warp-sorted groups of heads by binary search; the keys
// >= T (a few dozen for a random pool) are then placed by their rank among
// themselves.  Returns false (block-uniform) when the candidates do not
// suit it, leaving the radix path to run.
constexpr int kPoolGroups = 1024;  // heads ranked by the short path
constexpr int kPoolCand = 512;     // candidates placed by rank (in `sel`), O(c^2 / threads)
constexpr int kPoolAll = 256;      // pools this small are ranked whole

// The keys are read where they are, in the pool (L2 loads, eight per thread
// in flight; a fused caller writes the pool earlier in the same launch):
// both passes over them are coalesced, so no staging copy is needed.
// Group g of the ngr = ceil(cnt / 32) groups holds the keys g, g + ngr,
// g + 2 ngr, ... (at most 32); its head (maximum) is formed by a team of
// adjacent lanes in registers.  Any partition into groups gives the same
// guarantee: the k-th largest head T has k distinct keys at or above it,
// so every key of the top k is >= T and is collected.
template <bool SMEM = false>  // SMEM: the keys are in shared memory
__device__ bool merge_pool_short(const uint64_t* __restrict__ keys, int cnt, int k, int pad_short,
                                 uint64_t* cand, float* __restrict__ out_scores,
                                 int32_t* __restrict__ out_idx) {
  auto key_at = [&](int i) -> uint64_t {
    if constexpr (SMEM) return keys[i];
    else return __ldcg(keys + i);
  };
  __shared__ uint64_t s_heads[kPoolGroups];  // group maxima, then sorted in groups of 32
  __shared__ uint64_t s_t;
  __shared__ unsigned s_got;
  __shared__ int s_ok;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const int ngr = (cnt + 31) >> 5;
  if (threadIdx.x == 0) {
    s_t = 0ull;
    s_got = 0u;
  }
  // heads: a team of `team` adjacent lanes (a power of two, as many as the
  // block has threads per group) forms each group's maximum, lane `sub` of
  // the team taking keys sub, sub + team, ... of the group; then the heads
  // are sorted descending within each group of 32 heads; past the pool 0
  const int nhg = (ngr + 31) >> 5;
  int team = 1;
  while (team < 32 && 2 * team * ngr <= (int)blockDim.x) team <<= 1;
  for (int s0 = 0; s0 < ngr * team; s0 += blockDim.x) {  // block-uniform trip count
    const int sl = s0 + threadIdx.x;
    const int g = sl / team, sub = sl - g * team;
    uint64_t m = 0ull;
    for (int j0 = sub; j0 < 32; j0 += 8 * team) {
      uint64_t x[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int j = j0 + u * team;
        const int i = g + j * ngr;
        x[u] = (g < ngr && j < 32 && i < cnt) ? key_at(i) : 0ull;
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) m = x[u] > m ? x[u] : m;
    }
    for (int off = team >> 1; off > 0; off >>= 1) {
      const uint64_t o = __shfl_xor_sync(0xffffffffu, m, off);
      m = o > m ? o : m;
    }
    if (sub == 0 && g < ngr) s_heads[g] = m;
  }
  for (int g = ngr + threadIdx.x; g < nhg * 32; g += blockDim.x) s_heads[g] = 0ull;
  __syncthreads();
  for (int hg = warp; hg < nhg; hg += nwarps) {
    uint64_t h = s_heads[hg * 32 + lane];
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
      for (int stride = size >> 1; stride > 0; stride >>= 1) {
        const uint64_t o = __shfl_xor_sync(0xffffffffu, h, stride);
        const bool keep_max = ((lane & stride) == 0) == ((lane & size) == 0);
        h = keep_max ? (h > o ? h : o) : (h < o ? h : o);
      }
    }
    s_heads[hg * 32 + lane] = h;
  }
  __syncthreads();
  // T: the head of rank k - 1 among the nonzero heads (0 when fewer than k)
  for (int i = threadIdx.x; i < nhg * 32; i += blockDim.x) {
    const uint64_t h = s_heads[i];
    if (h == 0ull) continue;
    int rank = 0;
    for (int hg = 0; hg < nhg; ++hg) {
      const uint64_t* grp = s_heads + hg * 32;
      int lo = 0;
#pragma unroll
      for (int step = 16; step > 0; step >>= 1)
        if (grp[lo + step - 1] > h) lo += step;
      rank += lo + ((lo == 31 && grp[31] > h) ? 1 : 0);
    }
    if (rank == k - 1) s_t = h;
  }
  __syncthreads();
  // every key >= T, appended with one shared atomic per warp and load batch
  const uint64_t t = s_t;
  for (int b0 = 0; b0 < cnt; b0 += 8 * (int)blockDim.x) {  // block-uniform trip count
    uint64_t x[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int i = b0 + u * (int)blockDim.x + (int)threadIdx.x;
      x[u] = i < cnt ? key_at(i) : 0ull;
    }
    unsigned take = 0u;  // bit u: x[u] is a candidate
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (x[u] != 0ull && x[u] >= t) take |= 1u << u;
    const unsigned mine = (unsigned)__popc(take);
    unsigned incl = mine;  // inclusive prefix of the lanes' counts
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const unsigned o = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += o;
    }
    const unsigned total = __shfl_sync(0xffffffffu, incl, 31);
    if (total == 0u) continue;  // warp-uniform
    unsigned base = 0u;
    if (lane == 31) base = atomicAdd(&s_got, total);
    base = __shfl_sync(0xffffffffu, base, 31) + incl - mine;
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      if ((take >> u) & 1u) {
        if (base < (unsigned)kPoolCand) cand[base] = x[u];
        ++base;
      }
    }
  }
  __syncthreads();
  const int got = (int)s_got;
  if (threadIdx.x == 0) s_ok = got <= kPoolCand && (got >= k || pad_short);
  __syncthreads();
  if (!s_ok) return false;
  for (int i = threadIdx.x; i < got; i += blockDim.x) {
    const uint64_t c = cand[i];
    int rank = 0;
    for (int j = 0; j < got; ++j) {
      const uint64_t o = cand[j];
      rank += (o > c) || (o == c && j < i);
    }
    if (rank < k) {
      out_scores[rank] = code_score((uint32_t)(c >> 32));
      out_idx[rank] = (int32_t)cand_index(c);
    }
  }
  for (int r = got + threadIdx.x; r < k; r += blockDim.x) {  // a short pool: -inf, -1
    out_scores[r] = -__int_as_float(0x7f800000);
    out_idx[r] = -1;
  }
  return true;
}

// Selection for pools much longer than k that the group-head bound cannot
// prune (k above the number of 32-key groups): keys are binned by their
// score code, (code - min) >> sh with sh chosen so that the range spans at
// most kBins bins, which keeps bins in code order.  A suffix count of the
// bin histogram finds the bin B holding the k-th largest key; the keys of
// bins >= B are scattered bucket by bucket into shared memory, and each
// key's rank is the count of keys in higher bins plus the larger keys of its
// own bucket (equal keys ordered by position).  Ranks below k are written,
// sorted.  Uses the shared memory past the pool: 2 kBins words of counts and
// cursors, then kBinCap keys.  Returns false (block-uniform) when the
// selected bins hold more than kBinCap keys (codes bunched in a few bins).
constexpr int kBins = 2 * kSelThreads;  // two bins per thread in the scan
constexpr int kBinCap = 4096;

__device__ bool merge_pool_binned(const uint64_t* s_keys, int cnt, int k,
                                  float* __restrict__ out_scores,
                                  int32_t* __restrict__ out_idx) {
  __shared__ uint32_t s_lo, s_hi;
  __shared__ int s_bin, s_above;
  __shared__ int scan_scratch[32];
  uint32_t* count = reinterpret_cast<uint32_t*>(const_cast<uint64_t*>(s_keys) + cnt);  // [kBins]
  uint32_t* start = count + kBins;                                     // [kBins]
  uint64_t* buf = reinterpret_cast<uint64_t*>(start + kBins);          // [kBinCap]
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    s_lo = 0xffffffffu;
    s_hi = 0u;
    s_bin = -1;
    s_above = 0;
  }
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) count[b] = 0u;
  __syncthreads();
  uint32_t lo = 0xffffffffu, hi = 0u;
  for (int i = threadIdx.x; i < cnt; i += blockDim.x) {
    const uint32_t c = (uint32_t)(s_keys[i] >> 32);
    lo = min(lo, c);
    hi = max(hi, c);
  }
  lo = __reduce_min_sync(0xffffffffu, lo);
  hi = __reduce_max_sync(0xffffffffu, hi);
  if (lane == 0) {
    atomicMin(&s_lo, lo);
    atomicMax(&s_hi, hi);
  }
  __syncthreads();
  const uint32_t clo = s_lo;
  const uint32_t range = s_hi - clo;  // codes span [clo, clo + range]
  int sh = 0;
  while (sh < 32 && (range >> sh) >= (uint32_t)kBins) ++sh;
  auto bin_of = [&](uint64_t key) { return (int)(((uint32_t)(key >> 32) - clo) >> sh); };
  for (int i = threadIdx.x; i < cnt; i += blockDim.x) atomicAdd(&count[bin_of(s_keys[i])], 1u);
  __syncthreads();
  // thread t holds bins kBins-1-2t and kBins-2-2t: the scan runs from the top bin down
  const int d0 = kBins - 1 - 2 * (int)threadIdx.x, d1 = d0 - 1;
  const int c0 = (int)count[d0], c1 = (int)count[d1];
  int total = 0;
  const int ex = block_exclusive_scan(c0 + c1, scan_scratch, &total);
  start[d0] = (uint32_t)ex;
  start[d1] = (uint32_t)(ex + c0);
  if (ex < k && k <= ex + c0) {
    s_bin = d0;
    s_above = ex;
  } else if (ex + c0 < k && k <= ex + c0 + c1) {
    s_bin = d1;
    s_above = ex + c0;
  }
  __syncthreads();
  const int B = s_bin;
  if (B < 0 || s_above + (int)count[B] > kBinCap) return false;  // block-uniform
  for (int i = threadIdx.x; i < cnt; i += blockDim.x) {
    const uint64_t key = s_keys[i];
    const int b = bin_of(key);
    if (b >= B) buf[atomicAdd(&start[b], 1u)] = key;  // start[b] ends at the bucket's end
  }
  __syncthreads();
  const int nsel = s_above + (int)count[B];
  for (int p = threadIdx.x; p < nsel; p += blockDim.x) {
    const uint64_t key = buf[p];
    const int b = bin_of(key);
    const int e = (int)start[b], s0 = e - (int)count[b];
    int r = s0;  // keys in higher bins
    for (int j = s0; j < e; ++j) {
      const uint64_t o = buf[j];
      r += (o > key) || (o == key && j < p);
    }
    if (r < k) {
      out_scores[r] = code_score((uint32_t)(key >> 32));
      out_idx[r] = (int32_t)cand_index(key);
    }
  }
  return true;
}

// Top k of query q's pool into out_scores / out_idx rows q (one block per
// query; s_keys: smem_keys keys of shared memory, kSmemKeys for the merge
// kernels).  With `in_smem` the pool_cap keys are already in s_keys (pool
// and counts unused).  The binned path runs only with kSelThreads threads.
// Every return is block-uniform, so a caller may continue after a block
// barrier.
__device__ void merge_pool_block(const uint64_t* __restrict__ pool,
                                 const uint32_t* __restrict__ counts, int64_t pool_cap, int k,
                                 float* __restrict__ out_scores, int32_t* __restrict__ out_idx,
                                 uint32_t* status, int pad_short, int q, uint64_t* s_keys,
                                 int smem_keys = kSmemKeys, bool in_smem = false) {
  __shared__ unsigned hist[256];
  __shared__ Digit dig;
  __shared__ unsigned n_sel;
  __shared__ uint64_t sel[SENSE_MAX_K];
  const uint64_t* src = in_smem ? s_keys : pool + (int64_t)q * pool_cap;
  int64_t cnt = (counts && !in_smem) ? (int64_t)counts[q] : pool_cap;  // else every slot is used
  if (cnt > pool_cap) cnt = pool_cap;
  // the short path (pool read where it is) needs a pruning threshold (k
  // group heads) or a tiny pool; past k = 128 it also wants 4 k groups, or
  // the keys above the k-th head overflow its kPoolCand candidates (a
  // 256-key shortlist of a 9,400-key pool did, every time)
  const int64_t ngr = (cnt + 31) / 32;
  const bool short_ok = cnt > 0 && cnt <= 32 * kPoolGroups &&
                        (cnt <= kPoolAll || (ngr >= (int64_t)k && (k <= 128 || ngr >= 4 * (int64_t)k)));
  if (short_ok &&
      (in_smem ? merge_pool_short<true>(src, (int)cnt, k, pad_short, sel, out_scores + (int64_t)q * k,
                                        out_idx + (int64_t)q * k)
               : merge_pool_short<false>(src, (int)cnt, k, pad_short, sel,
                                         out_scores + (int64_t)q * k, out_idx + (int64_t)q * k)))
    return;
  const bool staged = in_smem || cnt <= smem_keys;
  if (staged && !in_smem) {
    // L2 loads (a fused caller's pool was written earlier in the same
    // launch), eight per thread in flight before their stores
    for (int64_t i0 = threadIdx.x; i0 < cnt; i0 += 8 * (int64_t)blockDim.x) {
      uint64_t v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int64_t i = i0 + u * (int64_t)blockDim.x;
        v[u] = i < cnt ? __ldcg(src + i) : 0ull;
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int64_t i = i0 + u * (int64_t)blockDim.x;
        if (i < cnt) s_keys[i] = v[u];
      }
    }
    __syncthreads();
  }
  if (staged && cnt >= k && (int)blockDim.x == kSelThreads && cnt + kBins + kBinCap <= smem_keys &&
      merge_pool_binned(s_keys, (int)cnt, k, out_scores + (int64_t)q * k, out_idx + (int64_t)q * k))
    return;
  auto get = [&](int64_t i) { return staged ? s_keys[i] : __ldcg(src + i); };
  uint64_t prefix, pmask;
  bool ok = radix_select(get, cnt, k, 0, hist, &dig, &prefix, &pmask);
  if (!ok && pad_short) {  // fewer than k candidates allowed: keep them all
    prefix = 0ull;
    pmask = 0ull;
    ok = true;
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
    const uint64_t c = get(i);
    if ((c & pmask) >= prefix) {
      const unsigned p = atomicAdd(&n_sel, 1u);
      if (p < (unsigned)k) sel[p] = c;
    }
  }
  __syncthreads();
  int kp = 1;
  while (kp < k) kp <<= 1;
  const int got = min((int)n_sel, k);  // k, or the whole pool when it is short
  for (int i = threadIdx.x; i < kp; i += blockDim.x) {
    if (i >= got) sel[i] = 0ull;
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
    const bool real = r < got;  // slots past a short pool: -inf, -1
    out_scores[(int64_t)q * k + r] = real ? code_score((uint32_t)(c >> 32)) : -__int_as_float(0x7f800000);
    out_idx[(int64_t)q * k + r] = real ? (int32_t)cand_index(c) : -1;
  }
}

}  // namespace
}  // namespace sense
