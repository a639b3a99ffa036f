// Candidate drafts and the loose trie.
//
// gather (Sec. 3.2.2, D_ret = {(k_i, s_i)}; Eq. 8 rerank; App. C.2 Alg. 2
// forced anchor): one block per query, one thread per retrieved rank.  The
// anchor-first reordering of Eq. 8 (alpha >> beta) is a stable partition
// computed with a block-wide prefix count of anchor matches.
//
// tree (Sec. 3.2.3 Eq. 9; App. C.3 Alg. 3): one block per query builds the
// trie entirely in shared memory:
//   1. bitonic sort of the candidate rows in lexicographic order;
//   2. LCP of each sorted row with its predecessor: row p creates nodes at
//      depths lcp[p]..m-1 (Alg. 3's `unique`), and an exclusive scan of the
//      counts numbers the nodes in preorder (Eq. 9's T_flat);
//   3. node of (sorted row p, depth j) = node created by the last row
//      p' <= p with lcp[p'] <= j: a prefix-max over p per column (Alg. 3's
//      running column maximum);
//   4. node cap: key (first candidate rank containing the node, depth) -
//      segmented minimum by shared-memory atomicMin, then the cap smallest
//      keys are kept (keys are distinct integers < k*m, so a prefix count
//      over a presence table ranks them); kept nodes are renumbered in
//      preorder by a second prefix count;
//   5. outputs: tokens/parent/depth, gamma back in the candidates' order,
//      optional ancestor bit mask.
// Trees of at most 128 candidates take tree_small_kernel, which computes the
// same outputs from pairwise ranks in a few block barriers.
//
// tree mask (App. C.6 Eq. 20): the additive attention mask of the draft
// tokens over a static KV cache, written from the ancestor bit rows.  One
// block per output row (grid-stride); the row's mask words are staged in
// shared memory and the row is written with 16-byte stores.
#include <algorithm>

#include "common.cuh"
#include "draft_dev.cuh"
#include "launch.h"

namespace sense {
namespace {

__global__ void gather_kernel(const int32_t* __restrict__ spans, int64_t n, int m,
                              const int32_t* __restrict__ idx, int k,
                              const int32_t* __restrict__ anchor, int n_keep, int force,
                              int32_t* __restrict__ out, uint32_t* status) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  __shared__ int scratch[32];
  gather_block(spans, n, m, idx, k, anchor, n_keep, force, out, status, blockIdx.x, scratch);
}

constexpr int kTreeThreads = 1024;

// Lexicographic comparison of rows a and b of s (m tokens each); equal rows
// are ordered by row index so that the order is total.
__device__ __forceinline__ bool row_less(const int* s, int m, int a, int b) {
  const int* ra = s + a * m;
  const int* rb = s + b * m;
  for (int j = 0; j < m; ++j) {
    if (ra[j] != rb[j]) return ra[j] < rb[j];
  }
  return a < b;
}

__global__ void __launch_bounds__(kTreeThreads)
tree_kernel(const int32_t* __restrict__ spans, int k, int m, int cap, int mask_words,
            int32_t* __restrict__ num_nodes, int32_t* __restrict__ tokens,
            int32_t* __restrict__ parent, int32_t* __restrict__ depth,
            int32_t* __restrict__ gamma, uint32_t* __restrict__ mask, uint32_t* status) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  extern __shared__ int sm[];
  const int km = k * m;
  int kp = 1;
  while (kp < k) kp <<= 1;
  int* s_tok = sm;            // [k*m] candidate tokens
  int* s_own = s_tok + km;    // [k*m] node of (sorted row, depth); later scratch
  int* s_aux = s_own + km;    // [k*m] first-rank per node / key table
  int* s_new = s_aux + km;    // [k*m] kept-node new id
  int* s_ord = s_new + km;    // [kp] sorted row order
  int* s_lcp = s_ord + kp;    // [k]
  int* s_base = s_lcp + k;    // [k]
  __shared__ int scratch[32];
  __shared__ int s_bad, s_total, s_kept;

  const int q = blockIdx.x;
  const int32_t* src = spans + (int64_t)q * km;
  if (threadIdx.x == 0) s_bad = 0;
  __syncthreads();
  for (int i = threadIdx.x; i < km; i += blockDim.x) {
    const int t = src[i];
    s_tok[i] = t;
    if (t < 0) s_bad = 1;
  }
  for (int i = threadIdx.x; i < kp; i += blockDim.x) s_ord[i] = i;
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

  // 1. Bitonic sort of row indices (padding indices >= k sort last).
  for (int size = 2; size <= kp; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < kp; i += blockDim.x) {
        const int j = i ^ stride;
        if (j > i) {
          const bool up = ((i & size) == 0);
          const int a = s_ord[i], b = s_ord[j];
          bool b_first;  // true when b must precede a
          if (a >= k) b_first = (b < k) || (b < a);
          else if (b >= k) b_first = false;
          else b_first = row_less(s_tok, m, b, a);
          if (up ? b_first : !b_first) {
            s_ord[i] = b;
            s_ord[j] = a;
          }
        }
      }
      __syncthreads();
    }
  }

  // 2. LCP with the previous sorted row, node counts, preorder bases.
  int cnt = 0;
  if (threadIdx.x < k) {
    const int p = threadIdx.x;
    int l = 0;
    if (p > 0) {
      const int* ra = s_tok + s_ord[p - 1] * m;
      const int* rb = s_tok + s_ord[p] * m;
      while (l < m && ra[l] == rb[l]) ++l;
    }
    s_lcp[p] = l;
    cnt = m - l;
  }
  int total = 0;
  const int base = block_exclusive_scan(cnt, scratch, &total);
  if (threadIdx.x < k) s_base[threadIdx.x] = base;
  if (threadIdx.x == 0) s_total = total;
  // 3. Creator row per (p, j): prefix max over p of (lcp[p] <= j ? p : -1).
  for (int e = threadIdx.x; e < km; e += blockDim.x) {
    const int p = e / m, j = e - p * m;
    s_own[e] = (s_lcp[p] <= j) ? p : -1;
  }
  __syncthreads();
  // Hillis-Steele prefix max over p, ping-ponging between s_own and s_aux.
  int* pm_in = s_own;
  int* pm_out = s_aux;
  for (int off = 1; off < k; off <<= 1) {
    for (int e = threadIdx.x; e < km; e += blockDim.x) {
      const int p = e / m;
      int v = pm_in[e];
      if (p >= off) v = max(v, pm_in[e - off * m]);
      pm_out[e] = v;
    }
    __syncthreads();
    int* t = pm_in;
    pm_in = pm_out;
    pm_out = t;
  }
  // node id of (sorted p, j) = base[p'] + j - lcp[p'], p' the creator.
  for (int e = threadIdx.x; e < km; e += blockDim.x) {
    const int p = e / m, j = e - p * m;
    const int pc = pm_in[e];
    s_own[e] = s_base[pc] + j - s_lcp[pc];
  }
  __syncthreads();
  const int U = s_total;

  // 4. Node cap.
  const bool capped = cap < U;
  if (capped) {
    for (int u = threadIdx.x; u < U; u += blockDim.x) s_aux[u] = 0x7fffffff;
    __syncthreads();
    for (int e = threadIdx.x; e < km; e += blockDim.x) {
      const int p = e / m;
      atomicMin(&s_aux[s_own[e]], s_ord[p]);
    }
    __syncthreads();
    // key = first_rank * m + depth; mark presence in s_new (as a key table).
    for (int i = threadIdx.x; i < km; i += blockDim.x) s_new[i] = 0;
    __syncthreads();
    for (int e = threadIdx.x; e < km; e += blockDim.x) {
      const int p = e / m, j = e - p * m;
      if (s_lcp[p] <= j) {  // the creator entry of node s_own[e]
        const int u = s_own[e];
        s_new[s_aux[u] * m + j] = 1;
      }
    }
    __syncthreads();
    // rank of every present key
    block_rank_flags(s_new, km, scratch);
    // kept flag per node (u in preorder): rank of its key < cap.
    for (int e = threadIdx.x; e < km; e += blockDim.x) {
      const int p = e / m, j = e - p * m;
      if (s_lcp[p] <= j) {
        const int u = s_own[e];
        const int rk = s_new[s_aux[u] * m + j];
        s_aux[u] = (rk < cap) ? 1 : 0;  // s_aux now holds kept flags
      }
    }
    __syncthreads();
    // new ids: prefix count of kept flags in preorder
    for (int u = threadIdx.x; u < U; u += blockDim.x) s_new[u] = s_aux[u];
    __syncthreads();
    const int nk = block_rank_flags(s_new, U, scratch);
    if (threadIdx.x == 0) s_kept = nk;
  } else {
    for (int u = threadIdx.x; u < U; u += blockDim.x) s_new[u] = u;
    if (threadIdx.x == 0) s_kept = U;
  }
  __syncthreads();
  const int kept = s_kept;

  // 5. Outputs.
  if (threadIdx.x == 0) num_nodes[q] = kept;
  for (int i = kept + threadIdx.x; i < cap; i += blockDim.x) {
    o_tok[i] = -1;
    o_par[i] = -1;
    o_dep[i] = -1;
  }
  for (int e = threadIdx.x; e < km; e += blockDim.x) {
    const int p = e / m, j = e - p * m;
    const int u = s_own[e];
    const int nid = s_new[u];
    o_gam[s_ord[p] * m + j] = nid;
    if (s_lcp[p] <= j && nid >= 0) {
      o_tok[nid] = s_tok[s_ord[p] * m + j];
      o_dep[nid] = j;
      o_par[nid] = (j > 0) ? s_new[s_own[e - 1]] : -1;
    }
  }
  if (o_mask) {
    for (int64_t i = threadIdx.x; i < (int64_t)cap * mask_words; i += blockDim.x) o_mask[i] = 0u;
    __syncthreads();
    for (int e = threadIdx.x; e < km; e += blockDim.x) {
      const int p = e / m, j = e - p * m;
      if (s_lcp[p] <= j) {
        const int nid = s_new[s_own[e]];
        if (nid >= 0) {
          uint32_t* row = o_mask + (int64_t)nid * mask_words;
          for (int jj = 0; jj <= j; ++jj) {
            const int b = s_new[s_own[p * m + jj]];
            atomicOr(&row[b >> 5], 1u << (b & 31));
          }
        }
      }
    }
  }
}


__global__ void __launch_bounds__(kTreeSmallThreads)
tree_small_kernel(const int32_t* __restrict__ spans, int k, int m, int cap, int mask_words,
                  int32_t* __restrict__ num_nodes, int32_t* __restrict__ tokens,
                  int32_t* __restrict__ parent, int32_t* __restrict__ depth,
                  int32_t* __restrict__ gamma, uint32_t* __restrict__ mask, uint32_t* status) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  extern __shared__ int sm[];
  __shared__ int scratch[32];
  __shared__ int sv[3];
  tree_small_block(spans, k, m, cap, mask_words, num_nodes, tokens, parent, depth, gamma, mask,
                   status, blockIdx.x, sm, scratch, sv);
}

// Row r = (query qi, draft token i) of the [q, cap, cache_len] mask.
template <bool VEC>
__global__ void __launch_bounds__(256)
tree_mask_full_kernel(const uint32_t* __restrict__ mask_bits, const int32_t* __restrict__ num_nodes,
                      const int32_t* __restrict__ prefix_len, int q, int cap, int words,
                      int cache_len, float* __restrict__ out, uint32_t* status) {
  __shared__ uint32_t s_w[SENSE_MAX_TREE_TOKENS / 32];
  const float NEG = -__int_as_float(0x7f800000);
  const int64_t rows = (int64_t)q * cap;
  for (int64_t r = blockIdx.x; r < rows; r += gridDim.x) {
    const int qi = (int)(r / cap), i = (int)(r - (int64_t)qi * cap);
    const int L = num_nodes[qi], m = prefix_len[qi];
    const bool bad = m < 0 || L < 0 || L > cap || (int64_t)m + L > cache_len;
    if (bad && i == 0 && threadIdx.x == 0) raise_status(status, SENSE_DEVST_BAD_LENGTH);
    const bool tree_row = !bad && i < L;
    __syncthreads();  // s_w of the previous row is no longer read
    if (tree_row)
      for (int w = threadIdx.x; w < words; w += blockDim.x)
        s_w[w] = mask_bits[r * words + w];
    __syncthreads();
    const int lo = bad ? 0 : m;          // columns [0, lo) are 0
    const int hi = tree_row ? m + L : 0;  // tree columns [lo, hi) follow the bits
    auto val = [&](int c) -> float {
      if (c < lo) return 0.0f;
      if (c < hi) {
        const int b = c - m;
        return ((s_w[b >> 5] >> (b & 31)) & 1u) ? 0.0f : NEG;
      }
      return NEG;
    };
    float* row = out + r * cache_len;
    if (VEC) {
      for (int c = 4 * threadIdx.x; c < cache_len; c += 4 * blockDim.x)
        *reinterpret_cast<float4*>(row + c) = make_float4(val(c), val(c + 1), val(c + 2), val(c + 3));
    } else {
      for (int c = threadIdx.x; c < cache_len; c += blockDim.x) row[c] = val(c);
    }
  }
}

}  // namespace

sense_status launch_gather(const int32_t* spans, int64_t n, int m, const int32_t* idx, int q,
                           int k, const int32_t* anchor, int n_keep, int force,
                           int32_t* out_spans, uint32_t* status, cudaStream_t s) {
  const int threads = ((k + 31) / 32) * 32;
  LaunchScope ls(K_GATHER, s);
  return cuda_check(launch_pdl(gather_kernel, dim3(q), dim3(threads), 0, s, spans, n, m, idx, k,
                              anchor, n_keep, force, out_spans, status),
                    "launch gather");
}

size_t tree_smem_bytes(int k, int m) {
  int kp = 1;
  while (kp < k) kp <<= 1;
  return sizeof(int) * ((size_t)4 * k * m + kp + 2 * (size_t)k);
}

sense_status launch_tree(const int32_t* spans, int q, int k, int m, int cap, int mask_bits,
                         int32_t* num_nodes, int32_t* tokens, int32_t* parent, int32_t* depth,
                         int32_t* gamma, uint32_t* mask, uint32_t* status, cudaStream_t s) {
  const int words = (cap + 31) / 32;
  if (k <= kTreeSmallK) {
    const size_t smem = sizeof(int) * ((size_t)3 * k * m + (size_t)5 * k);
    cudaError_t e = func_smem(reinterpret_cast<const void*>(tree_small_kernel), (int)smem);
    if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(tree_small)");
    LaunchScope ls(K_TREE, s);
    return cuda_check(launch_pdl(tree_small_kernel, dim3(q), dim3(kTreeSmallThreads), smem, s,
                                 spans, k, m, cap, words, num_nodes, tokens, parent, depth, gamma,
                                 mask_bits ? mask : nullptr, status),
                      "launch tree_small");
  }
  const size_t smem = tree_smem_bytes(k, m);
  cudaError_t e = func_smem(reinterpret_cast<const void*>(tree_kernel), (int)smem);
  if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(tree)");
  LaunchScope ls(K_TREE, s);
  // one thread per candidate row at least; fewer threads make the many
  // block barriers of a small tree cheaper
  int threads = 128;
  while (threads < k) threads <<= 1;
  return cuda_check(launch_pdl(tree_kernel, dim3(q), dim3(threads), smem, s, spans, k, m, cap,
                              words, num_nodes, tokens, parent, depth, gamma,
                              mask_bits ? mask : nullptr, status),
                    "launch tree");
}

sense_status launch_tree_mask_full(const uint32_t* mask_bits, const int32_t* num_nodes,
                                   const int32_t* prefix_len, int q, int cap, int cache_len,
                                   float* out, uint32_t* status, cudaStream_t s) {
  const int words = (cap + 31) / 32;
  const int64_t rows = (int64_t)q * cap;
  const int grid = (int)std::min<int64_t>(rows, (int64_t)sm_count() * 16);
  const bool vec = (cache_len % 4 == 0) && (reinterpret_cast<uintptr_t>(out) % 16 == 0);
  LaunchScope ls(K_TREE_MASK, s);
  if (vec)
    tree_mask_full_kernel<true><<<grid, 256, 0, s>>>(mask_bits, num_nodes, prefix_len, q, cap,
                                                     words, cache_len, out, status);
  else
    tree_mask_full_kernel<false><<<grid, 256, 0, s>>>(mask_bits, num_nodes, prefix_len, q, cap,
                                                      words, cache_len, out, status);
  return cuda_check(cudaGetLastError(), "launch tree mask");
}

}  // namespace sense
