// Block-level bodies of the span gather and the small-tree trie (draft.cu),
// shared with the fused drafting kernel (select.cu): each is run by one
// block for one query.
#pragma once

#include "common.cuh"

namespace sense {
namespace {

// Block-wide exclusive prefix sum of one int per thread (blockDim <= 1024).
// `scratch` holds at least 32 ints.  Returns the exclusive prefix; *total
// receives the block sum.
__device__ int block_exclusive_scan(int v, int* scratch, int* total) {
  const int lane = threadIdx.x & 31;
  const int wid = threadIdx.x >> 5;
  const int nw = (blockDim.x + 31) >> 5;
  int x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += t;
  }
  __syncthreads();
  if (lane == 31) scratch[wid] = x;
  __syncthreads();
  if (wid == 0) {
    int y = (lane < nw) ? scratch[lane] : 0;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, y, off);
      if (lane >= off) y += t;
    }
    scratch[lane] = y;  // inclusive per warp
  }
  __syncthreads();
  const int warp_base = (wid > 0) ? scratch[wid - 1] : 0;
  *total = scratch[nw - 1];
  const int r = warp_base + x - v;
  __syncthreads();
  return r;
}

// Rank of the set entries of flag[0..len): flag[i] != 0 becomes the number
// of set entries before i, flag[i] == 0 becomes -1; returns the set count.
// Each thread scans a contiguous run, then one block scan joins the runs.
__device__ int block_rank_flags(int* flag, int len, int* scratch) {
  const int per = (len + blockDim.x - 1) / blockDim.x;
  const int lo = min(len, (int)threadIdx.x * per);
  const int hi = min(len, lo + per);
  int cnt = 0;
  for (int i = lo; i < hi; ++i) cnt += flag[i] != 0;
  int total = 0;
  int run = block_exclusive_scan(cnt, scratch, &total);
  for (int i = lo; i < hi; ++i) {
    const int f = flag[i];
    flag[i] = f ? run : -1;
    run += f != 0;
  }
  __syncthreads();
  return total;
}

// Span gather of query q by one block (thread r copies rank r; every thread
// of the block takes part in the prefix count).  `scratch` holds 32 ints.
__device__ void gather_block(const int32_t* __restrict__ spans, int64_t n, int m,
                             const int32_t* __restrict__ idx, int k,
                             const int32_t* __restrict__ anchor, int n_keep, int force,
                             int32_t* __restrict__ out, uint32_t* status, int q, int* scratch) {
  const int r = threadIdx.x;
  int64_t i = -1;
  bool valid = false;
  if (r < k) {
    i = __ldcg(idx + (int64_t)q * k + r);  // L2: a fused caller wrote idx in this launch
    valid = (i >= 0 && i < n);
    if (!valid) raise_status(status, SENSE_DEVST_BAD_INDEX);
  }
  int pos = r;
  if (anchor) {
    const int a = anchor[q];
    const bool match = (r < k) && valid && spans[i * m] == a;
    int total = 0;
    const int before = block_exclusive_scan(match ? 1 : 0, scratch, &total);
    pos = match ? before : total + (r - before);
  }
  int32_t* dst = out + ((int64_t)q * n_keep + pos) * m;
  if (r < k && pos < n_keep) {
    if (valid) {
      const int32_t* srow = spans + i * m;
      if ((m & 3) == 0) {
        for (int j = 0; j < m; j += 4)
          *reinterpret_cast<int4*>(dst + j) = __ldg(reinterpret_cast<const int4*>(srow + j));
      } else {
        for (int j = 0; j < m; ++j) dst[j] = __ldg(srow + j);
      }
    } else {
      for (int j = 0; j < m; ++j) dst[j] = -1;
    }
  }
  if (anchor && force) {
    __syncthreads();
    if (r == 0) {
      const int a = anchor[q];
      out[((int64_t)q * n_keep) * m] = a;
      out[((int64_t)q * n_keep + n_keep - 1) * m] = a;
    }
  }
}


// Small trees (k <= kTreeSmallK): the same trie from ranks instead of a
// sorting network and prefix-max passes, in a handful of block barriers.
//   1. one warp per candidate row a, lanes over rows b: the LCP of (a, b)
//      decides their lexicographic order (ties by row index), so a's sorted
//      position is the count of rows before it; the largest LCP of a with a
//      lower-ranked row, mll[a], is kept too;
//   2. LCP with the sorted predecessor and the preorder bases (a warp's
//      prefix scan);
//   3. node of (sorted row p, depth j): walk back to the last row p' <= p
//      with lcp[p'] <= j (its creator);
//   4. node cap: the node of row r at depth j is first reached by rank r iff
//      j >= mll[r]; its key (r, j) then has rank
//      sum_{r' < r} (m - mll[r']) + (j - mll[r]) among all node keys, so the
//      kept test needs no table; kept nodes are renumbered by one prefix count;
//   5. outputs as in tree_kernel; each node writes its own mask row (its
//      ancestors' ids increase with depth).
constexpr int kTreeSmallK = 128;
constexpr int kTreeSmallThreads = 256;

// The small-tree trie of query q by one block (any multiple of 32 threads);
// `sm` holds (3 k m + 5 k) ints, `scratch` 32 ints, `sv` 3 ints.
__device__ void tree_small_block(const int32_t* __restrict__ spans, int k, int m, int cap,
                                 int mask_words, int32_t* __restrict__ num_nodes,
                                 int32_t* __restrict__ tokens, int32_t* __restrict__ parent,
                                 int32_t* __restrict__ depth, int32_t* __restrict__ gamma,
                                 uint32_t* __restrict__ mask, uint32_t* status, int q, int* sm,
                                 int* scratch, int* sv) {
  const int km = k * m;
  int* s_tok = sm;             // [k*m] candidate tokens
  int* s_own = s_tok + km;     // [k*m] node (uncapped preorder id) of (sorted row, depth)
  int* s_nid = s_own + km;     // [k*m] kept flag, then new id, per node
  int* s_ord = s_nid + km;     // [k] candidate row at sorted position
  int* s_lcp = s_ord + k;      // [k] LCP with the sorted predecessor
  int* s_mll = s_lcp + k;      // [k] largest LCP with a lower-ranked row
  int* s_base = s_mll + k;     // [k] preorder id of sorted row p's first new node
  int* s_pre = s_base + k;     // [k] nodes first reached by ranks below r
  int& s_bad = sv[0];
  int& s_total = sv[1];
  int& s_kept = sv[2];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int nwarps = blockDim.x >> 5;

  const int32_t* src = spans + (int64_t)q * km;
  if (threadIdx.x == 0) s_bad = 0;
  __syncthreads();
  for (int i = threadIdx.x; i < km; i += blockDim.x) {
    const int t = __ldcg(src + i);  // L2: a fused caller wrote the spans in this launch
    s_tok[i] = t;
    if (t < 0) s_bad = 1;
  }
  __syncthreads();

  int32_t* o_tok = tokens + (int64_t)q * cap;
  int32_t* o_par = parent + (int64_t)q * cap;
  int32_t* o_dep = depth + (int64_t)q * cap;
  int32_t* o_gam = gamma + (int64_t)q * km;
  uint32_t* o_mask = mask ? mask + (int64_t)q * cap * mask_words : nullptr;

  if (s_bad) {
    if (threadIdx.x == 0) {
      raise_status(status, SENSE_DEVST_BAD_TOKEN);
      num_nodes[q] = 0;
    }
    for (int i = threadIdx.x; i < cap; i += blockDim.x) {
      o_tok[i] = -1;
      o_par[i] = -1;
      o_dep[i] = -1;
    }
    for (int i = threadIdx.x; i < km; i += blockDim.x) o_gam[i] = -1;
    if (o_mask)
      for (int64_t i = threadIdx.x; i < (int64_t)cap * mask_words; i += blockDim.x) o_mask[i] = 0u;
    return;
  }

  // 1. sorted position and mll of every row
  for (int a = wid; a < k; a += nwarps) {
    const int* ra = s_tok + a * m;
    int before = 0, mll = 0;
    for (int b0 = 0; b0 < k; b0 += 32) {
      const int b = b0 + lane;
      bool prec = false;
      if (b < k && b != a) {
        const int* rb = s_tok + b * m;
        int l = 0;
        while (l < m && ra[l] == rb[l]) ++l;
        prec = (l < m) ? (rb[l] < ra[l]) : (b < a);
        if (b < a) mll = max(mll, l);
      }
      before += __popc(__ballot_sync(0xffffffffu, prec));
    }
    mll = __reduce_max_sync(0xffffffffu, mll);
    if (lane == 0) {
      s_ord[before] = a;
      s_mll[a] = mll;
    }
  }
  __syncthreads();
  // 2. LCP with the sorted predecessor
  for (int p = threadIdx.x; p < k; p += blockDim.x) {
    int l = 0;
    if (p > 0) {
      const int* ra = s_tok + s_ord[p - 1] * m;
      const int* rb = s_tok + s_ord[p] * m;
      while (l < m && ra[l] == rb[l]) ++l;
    }
    s_lcp[p] = l;
  }
  __syncthreads();
  //    bases: nodes created by sorted rows before p; nodes first reached by
  //    ranks before r (exclusive prefix sums by warp 0, 32 rows a step)
  if (wid == 0) {
    int cb = 0, cp = 0;  // sums of the rows before this step's
    for (int i0 = 0; i0 < k; i0 += 32) {
      const int i = i0 + lane;
      const int vb = i < k ? m - s_lcp[i] : 0, vp = i < k ? m - s_mll[i] : 0;
      int xb = vb, xp = vp;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int tb = __shfl_up_sync(0xffffffffu, xb, off);
        const int tp = __shfl_up_sync(0xffffffffu, xp, off);
        if (lane >= off) {
          xb += tb;
          xp += tp;
        }
      }
      if (i < k) {
        s_base[i] = cb + xb - vb;
        s_pre[i] = cp + xp - vp;
      }
      cb += __shfl_sync(0xffffffffu, xb, 31);
      cp += __shfl_sync(0xffffffffu, xp, 31);
    }
    if (lane == 0) s_total = cb;
  }
  __syncthreads();
  const int U = s_total;
  const bool capped = cap < U;
  // 3-4. node of every (sorted p, j); kept flag at each node's first-rank entry
  for (int e = threadIdx.x; e < km; e += blockDim.x) {
    const int p = e / m, j = e - p * m;
    int pc = p;
    while (s_lcp[pc] > j) --pc;  // s_lcp[0] == 0 ends the walk
    const int u = s_base[pc] + j - s_lcp[pc];
    s_own[e] = u;
    const int r = s_ord[p];
    if (capped && j >= s_mll[r]) s_nid[u] = (s_pre[r] + j - s_mll[r] < cap) ? 1 : 0;
  }
  __syncthreads();
  if (capped) {
    const int nk = block_rank_flags(s_nid, U, scratch);
    if (threadIdx.x == 0) s_kept = nk;
  } else {
    if (threadIdx.x == 0) s_kept = U;
  }
  __syncthreads();
  const int kept = s_kept;
  auto new_id = [&](int u) { return capped ? s_nid[u] : u; };

  // 5. outputs
  if (threadIdx.x == 0) num_nodes[q] = kept;
  for (int i = kept + threadIdx.x; i < cap; i += blockDim.x) {
    o_tok[i] = -1;
    o_par[i] = -1;
    o_dep[i] = -1;
  }
  if (o_mask)
    for (int64_t i = (int64_t)kept * mask_words + threadIdx.x; i < (int64_t)cap * mask_words;
         i += blockDim.x)
      o_mask[i] = 0u;
  for (int e = threadIdx.x; e < km; e += blockDim.x) {
    const int p = e / m, j = e - p * m;
    const int nid = new_id(s_own[e]);
    o_gam[s_ord[p] * m + j] = nid;
    if (s_lcp[p] <= j && nid >= 0) {
      o_tok[nid] = s_tok[s_ord[p] * m + j];
      o_dep[nid] = j;
      o_par[nid] = (j > 0) ? new_id(s_own[e - 1]) : -1;
      if (o_mask) {
        uint32_t* row = o_mask + (int64_t)nid * mask_words;
        int jj = 0;
        for (int w = 0; w < mask_words; ++w) {
          uint32_t bits = 0u;
          while (jj <= j) {
            const int b = new_id(s_own[p * m + jj]);
            if ((b >> 5) != w) break;
            bits |= 1u << (b & 31);
            ++jj;
          }
          row[w] = bits;
        }
      }
    }
  }
}

}  // namespace
}  // namespace sense
