// Dynamic context buffer C_d and the hybrid static + dynamic candidate list.
//
// Sec. 3.2.1 Eq. 6 joins a static corpus C_s and a dynamic buffer C_d filled
// from the generation itself: Alg. 1 calls R.Update(h, y) after prefill and
// R.Update(H_align[i*, 0:L*+1], a) after each accepted step, i.e. it appends
// (hidden state, the token that state predicted) pairs.  Alg. 2 searches the
// buffer with DynSearch, boosts its scores by delta and reranks the union
// with Eq. 8.  Readings (the paper leaves DynSearch and the buffer size
// open): an entry is a position p with key L2Norm(h_p) (bf16, like the
// static keys) and span y_{p+1} .. y_{p+M}; it is searchable once its M
// continuation tokens exist; the buffer is a ring over the C most recent
// positions; DynSearch is the exact inner-product top-k (ties to the older
// position).
// The position counter lives in device memory, so that appends whose length
// is only known on the device (the accepted prefix of a step) need no host
// round trip and a whole decode step can be captured in a CUDA graph.
//  - ctx_append_kernel: one warp per appended row: fp64 norm, bf16 key into
//    ring slot p mod C, token into the token ring (rows: a host-given block,
//    or the accepted path H_align[i*, 0:L*+1] read through Gamma);
//  - ctx_bump_kernel: advances the counter after host-given rows are
//    written (the accepted path's kernel advances it itself);
//  - ctx_score_kernel: one warp per (entry, query): fp32 dot product of the
//    bf16 key and query + delta -> candidate key in the query's pool;
//  - ctx_pool_kernel (select.cu): the exact top-k of the pool (the shared
//    merge), then the winners' positions and spans, one block per query;
//  - hybrid_kernel: one block per query sorts the union of static and
//    dynamic candidates by (score desc, union index asc), applies the
//    anchor-first stable partition and the forced anchor, and copies the
//    kept spans.
#include <cuda_bf16.h>

#include <algorithm>

#include "common.cuh"
#include "draft_dev.cuh"
#include "launch.h"
#include "select_dev.cuh"

struct sense_ctx {
  int32_t cap;
  int32_t d;
  int32_t m;
  int device;
  uint16_t* keys;    // [cap, d] bf16 ring
  int32_t* tokens;   // [cap] ring: tokens[p mod cap] = y_{p+1}
  int64_t* count;    // device: positions appended so far (stream-ordered)
};

namespace sense {
namespace {

constexpr int kHybridMax = 2048;  // static + dynamic candidates per query
constexpr size_t kDynDraftSmemMax = 180 * 1024;  // dyn_draft_kernel: + 42 KB static

// Writes the key and token of one position; `x` is its bf16 hidden state.
__device__ void append_row(const uint16_t* __restrict__ x, int32_t token, int64_t slot, int d,
                           uint16_t* __restrict__ keys, int32_t* __restrict__ ring) {
  const int lane = threadIdx.x & 31;
  double ss = 0.0;
  for (int j = lane; j < d; j += 32) {
    const double v = (double)__uint_as_float((uint32_t)x[j] << 16);
    ss = fma(v, v, ss);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
  const double nrm = sqrt(ss);
  __nv_bfloat16* y = reinterpret_cast<__nv_bfloat16*>(keys + slot * d);
  for (int j = lane; j < d; j += 32) {
    const double v = (double)__uint_as_float((uint32_t)x[j] << 16);
    y[j] = nrm > 0.0 ? __double2bfloat16(v / nrm) : __double2bfloat16(0.0);
  }
  if (lane == 0) ring[slot] = token;
}

// Host-given rows: one warp per row i in [first, t).
__global__ void __launch_bounds__(256)
ctx_append_kernel(const uint16_t* __restrict__ hidden, const int32_t* __restrict__ tok, int t,
                  int first, const int64_t* __restrict__ count, int cap, int d,
                  uint16_t* __restrict__ keys, int32_t* __restrict__ ring) {
  const int i = first + (int)(((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  if (i >= t) return;  // warp-uniform
  append_row(hidden + (int64_t)i * d, tok[i], (*count + i) % cap, d, keys, ring);
}

// Accepted path of one step, one block of m warps: warp j < n_accept
// appends H_align[i*, j] (the root state for j = 0, else the state of node
// Gamma[i*, j-1]) with the accepted token a_j; then thread 0 advances the
// counter by n_accept clamped to [0, m].
__global__ void __launch_bounds__(1024)
ctx_append_path_kernel(const uint16_t* __restrict__ root, const uint16_t* __restrict__ nodes,
                       int n_nodes, const int32_t* __restrict__ gamma, int k, int m,
                       const int32_t* __restrict__ i_star, const int32_t* __restrict__ n_accept,
                       const int32_t* __restrict__ accepted, int64_t* __restrict__ count,
                       int cap, int d, uint16_t* __restrict__ keys, int32_t* __restrict__ ring,
                       uint32_t* status) {
  pdl_wait();  // the gate's outputs are complete
  pdl_launch_dependents();
  const int j = threadIdx.x >> 5;
  const int na = *n_accept, is = *i_star;
  const int64_t base = *count;
  if (j < na && j < m) {  // warp-uniform
    bool ok = !(is < 0 || is >= k || na > m);
    const uint16_t* x = root;
    if (ok && j > 0) {
      const int node = gamma[(int64_t)is * m + j - 1];
      if (node < 0 || node >= n_nodes) ok = false;
      else x = nodes + (int64_t)node * d;
    }
    if (!ok) {
      if ((threadIdx.x & 31) == 0) raise_status(status, SENSE_DEVST_BAD_INDEX);
    } else {
      append_row(x, accepted[j], (base + j) % cap, d, keys, ring);
    }
  }
  __syncthreads();  // every row read the counter before it moves
  if (threadIdx.x == 0) *count = base + (na < 0 ? 0 : (na > m ? m : na));
}

// count += t (host value) or += *t_dev (clamped to [0, m_max]).
__global__ void ctx_bump_kernel(int64_t* count, int64_t t, const int32_t* t_dev, int m_max) {
  if (t_dev) {
    int v = *t_dev;
    t = v < 0 ? 0 : (v > m_max ? m_max : v);
  }
  *count += t;
}

// Searchable positions [lo, lo + n_valid) after `count` appended positions.
__device__ __forceinline__ void ctx_range_dev(int64_t count, int cap, int m, int64_t* lo,
                                              int* n_valid) {
  const int64_t l = count > cap ? count - cap : 0;
  const int64_t hi = count - m + 1;  // exclusive
  *lo = l;
  *n_valid = hi > l ? (int)(hi - l) : 0;
}

// Grid-stride over (query, entry) pairs, one warp each; also records the
// number of searchable entries as every query's pool count.  A lane's
// sixteen 16-byte key loads of a row piece (a whole 4096-dimensional row)
// are issued together; its chunks j = lane, lane + 32, ... are summed in
// increasing order.
__global__ void __launch_bounds__(256)
ctx_score_kernel(const uint16_t* __restrict__ keys, const uint16_t* __restrict__ queries, int q,
                 int d, int cap, int m, const int64_t* __restrict__ count, float delta,
                 uint64_t* __restrict__ pool, uint32_t* __restrict__ counts) {
  pdl_wait();  // the buffer and the query are complete
  pdl_launch_dependents();
  constexpr int kBatch = 16;
  const int lane = threadIdx.x & 31;
  int64_t lo;
  int n_valid;
  ctx_range_dev(*count, cap, m, &lo, &n_valid);
  const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  if (gw < q && lane == 0) counts[gw] = (uint32_t)n_valid;
  const int chunks = d >> 3;
  for (int64_t w = gw; w < (int64_t)n_valid * q; w += nw) {
    const int qi = (int)(w / n_valid);
    const int e = (int)(w - (int64_t)qi * n_valid);
    const uint4* kr = reinterpret_cast<const uint4*>(keys + ((lo + e) % cap) * d);
    const uint4* qr = reinterpret_cast<const uint4*>(queries + (int64_t)qi * d);
    float acc = 0.0f;
    for (int j0 = 0; j0 < chunks; j0 += 32 * kBatch) {
      uint4 kv[kBatch];
#pragma unroll
      for (int t = 0; t < kBatch; ++t) {
        const int j = j0 + 32 * t + lane;
        kv[t] = j < chunks ? ld_stream_v4(kr + j) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int t = 0; t < kBatch; ++t) {
        const int j = j0 + 32 * t + lane;
        if (j < chunks) {
          const uint4 a = kv[t], b = __ldg(qr + j);
          acc = fmaf(bf_lo(a.x), bf_lo(b.x), acc);
          acc = fmaf(bf_hi(a.x), bf_hi(b.x), acc);
          acc = fmaf(bf_lo(a.y), bf_lo(b.y), acc);
          acc = fmaf(bf_hi(a.y), bf_hi(b.y), acc);
          acc = fmaf(bf_lo(a.z), bf_lo(b.z), acc);
          acc = fmaf(bf_hi(a.z), bf_hi(b.z), acc);
          acc = fmaf(bf_lo(a.w), bf_lo(b.w), acc);
          acc = fmaf(bf_hi(a.w), bf_hi(b.w), acc);
        }
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    if (lane == 0) pool[(int64_t)qi * cap + e] = cand_key(acc + delta, (uint32_t)e);
  }
}

// Query qi by one block (any multiple of 32 threads).  Union index u < ks:
// static rank u; u >= ks: dynamic rank u - ks.  The dynamic lists are read
// from L2 (a fused caller writes them earlier in the same launch).
__device__ void hybrid_block(const int32_t* __restrict__ spans, int64_t n, int m,
                             const float* __restrict__ s_scores, const int32_t* __restrict__ s_idx,
                             int ks, const float* d_scores, const int32_t* d_spans, int kd,
                             const int32_t* __restrict__ anchor, int n_keep, int force,
                             int32_t* __restrict__ out, uint32_t* status, int qi) {
  __shared__ uint64_t key[kHybridMax];
  __shared__ int dest[kHybridMax];
  __shared__ int n_live;
  const int tot = ks + kd;
  int pw = 1;
  while (pw < tot) pw <<= 1;
  const bool has_anchor = anchor != nullptr;
  const int a = has_anchor ? anchor[qi] : 0;
  if (threadIdx.x == 0) n_live = 0;
  __syncthreads();
  for (int u = threadIdx.x; u < pw; u += blockDim.x) {
    uint64_t kk = 0ull;
    if (u < ks) {
      const int idx = s_idx[(int64_t)qi * ks + u];
      if (idx >= 0 && idx < n) kk = cand_key(s_scores[(int64_t)qi * ks + u], (uint32_t)u);
      else raise_status(status, SENSE_DEVST_BAD_INDEX);
    } else if (u < tot) {
      const float s = __ldcg(d_scores + (int64_t)qi * kd + (u - ks));
      if (s > -__int_as_float(0x7f800000)) kk = cand_key(s, (uint32_t)u);
    }
    if (kk) atomicAdd(&n_live, 1);
    key[u] = kk;
  }
  __syncthreads();
  // bitonic sort, descending: (score desc, union index asc); empty keys last
  for (int size = 2; size <= pw; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < pw; i += blockDim.x) {
        const int j = i ^ stride;
        if (j > i) {
          const bool desc = (i & size) == 0;
          const uint64_t x = key[i], y = key[j];
          if (desc ? (x < y) : (x > y)) {
            key[i] = y;
            key[j] = x;
          }
        }
      }
      __syncthreads();
    }
  }
  const int live = n_live;
  auto first_token = [&](int u) -> int {
    if (u < ks) return spans[(int64_t)s_idx[(int64_t)qi * ks + u] * m];
    return __ldcg(d_spans + ((int64_t)qi * kd + (u - ks)) * m);
  };
  // stable partition (anchor matches first), one warp, 32 candidates a step
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    int base = 0;
    for (int pass = 0; pass < (has_anchor ? 2 : 1); ++pass) {
      for (int r0 = 0; r0 < live; r0 += 32) {
        const int r = r0 + lane;
        bool take = false;
        int u = 0;
        if (r < live) {
          u = (int)cand_index(key[r]);
          const bool match = has_anchor && first_token(u) == a;
          take = has_anchor ? (pass == 0 ? match : !match) : true;
        }
        const unsigned b = __ballot_sync(0xffffffffu, take);
        if (take) dest[base + __popc(b & ((1u << lane) - 1u))] = u;
        base += __popc(b);
      }
    }
  }
  __syncthreads();
  const int64_t obase = (int64_t)qi * n_keep * m;
  for (int e = threadIdx.x; e < n_keep * m; e += blockDim.x) {
    const int o = e / m, j = e - o * m;
    int v = -1;
    if (o < live) {
      const int u = dest[o];
      v = (u < ks) ? spans[(int64_t)s_idx[(int64_t)qi * ks + u] * m + j]
                   : __ldcg(d_spans + ((int64_t)qi * kd + (u - ks)) * m + j);
    }
    if (force && has_anchor && j == 0 && (o == 0 || o == n_keep - 1)) v = a;
    out[obase + e] = v;
  }
}

__global__ void __launch_bounds__(1024)
hybrid_kernel(const int32_t* __restrict__ spans, int64_t n, int m,
              const float* __restrict__ s_scores, const int32_t* __restrict__ s_idx, int ks,
              const float* __restrict__ d_scores, const int32_t* __restrict__ d_spans, int kd,
              const int32_t* __restrict__ anchor, int n_keep, int force,
              int32_t* __restrict__ out, uint32_t* status) {
  pdl_wait();  // both candidate lists are complete
  pdl_launch_dependents();
  hybrid_block(spans, n, m, s_scores, s_idx, ks, d_scores, d_spans, kd, anchor, n_keep, force, out,
               status, blockIdx.x);
}

// The hybrid drafting tail of one query by one block of 1024 threads: the
// top kd of the buffer's scored positions (the pool merge) with their
// positions and spans, the union with the static results reranked
// (hybrid_block) and the small-tree trie of the kept spans, each phase
// reading the previous one's global writes after a block barrier; the trie
// reuses the merge's shared memory.
__global__ void __launch_bounds__(1024, 1)
dyn_draft_kernel(const uint64_t* __restrict__ pool, const uint32_t* __restrict__ counts,
                 int cap, int kd, float* __restrict__ dyn_scores, int32_t* __restrict__ rel,
                 const int64_t* __restrict__ count, const int32_t* __restrict__ ring,
                 int64_t* __restrict__ dyn_pos, int32_t* __restrict__ dyn_spans,
                 const int32_t* __restrict__ spans, int64_t n, int m,
                 const float* __restrict__ s_scores, const int32_t* __restrict__ s_idx, int ks,
                 const int32_t* __restrict__ anchor, int n_keep, int force,
                 int32_t* __restrict__ out_spans, int node_cap, int mask_words,
                 int32_t* __restrict__ num_nodes, int32_t* __restrict__ tokens,
                 int32_t* __restrict__ parent, int32_t* __restrict__ depth,
                 int32_t* __restrict__ gamma, uint32_t* __restrict__ mask, int smem_keys,
                 uint32_t* status) {
  extern __shared__ uint64_t s_keys[];
  __shared__ int scratch[32];
  __shared__ int sv[3];
  const int q = blockIdx.x;
  pdl_wait();  // the buffer's scores and the static results are complete
  pdl_launch_dependents();
  merge_pool_block(pool, counts, cap, kd, dyn_scores, rel, status, 1, q, s_keys, smem_keys);
  __syncthreads();
  {  // positions and spans of the dynamic winners (as ctx_pool_kernel)
    const int64_t cnt = *count;
    const int64_t lo = cnt > cap ? cnt - cap : 0;
    for (int t = threadIdx.x; t < kd * m; t += blockDim.x) {
      const int r = t / m, j = t - r * m;
      const int64_t slot = (int64_t)q * kd + r;
      const int e = rel[slot];
      const int64_t p = lo + e;
      if (j == 0) dyn_pos[slot] = e < 0 ? -1 : p;
      dyn_spans[slot * m + j] = e < 0 ? -1 : ring[(p + j) % cap];
    }
  }
  __syncthreads();
  hybrid_block(spans, n, m, s_scores, s_idx, ks, dyn_scores, dyn_spans, kd, anchor, n_keep, force,
               out_spans, status, q);
  __syncthreads();
  tree_small_block(out_spans, n_keep, m, node_cap, mask_words, num_nodes, tokens, parent, depth,
                   gamma, mask, status, q, reinterpret_cast<int*>(s_keys), scratch, sv);
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

int current_device() {
  int dev = 0;
  cudaGetDevice(&dev);
  return dev;
}

bool aligned(const void* ptr, size_t a) { return (reinterpret_cast<uintptr_t>(ptr) % a) == 0; }

}  // namespace
}  // namespace sense

using namespace sense;

extern "C" {

sense_status sense_ctx_create(int32_t capacity, int32_t d, int32_t m, sense_ctx** out) {
  if (!out) return fail(SENSE_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (m < 1 || m > SENSE_MAX_M) return fail(SENSE_ERR_INVALID_ARG, "m=%d outside [1, %d]", m, SENSE_MAX_M);
  if (capacity < m || capacity > (1 << 24))
    return fail(SENSE_ERR_INVALID_ARG, "capacity=%d outside [m, 2^24]", capacity);
  if (d < 8 || d % 8) return fail(SENSE_ERR_INVALID_ARG, "d=%d must be a positive multiple of 8", d);
  auto* c = new sense_ctx{};
  c->cap = capacity;
  c->d = d;
  c->m = m;
  c->device = current_device();
  if (cudaMalloc(&c->keys, (size_t)capacity * d * 2) != cudaSuccess ||
      cudaMalloc(&c->tokens, (size_t)capacity * 4) != cudaSuccess ||
      cudaMalloc(&c->count, sizeof(int64_t)) != cudaSuccess ||
      cudaMemset(c->count, 0, sizeof(int64_t)) != cudaSuccess) {
    cudaGetLastError();
    cudaFree(c->keys);
    cudaFree(c->tokens);
    cudaFree(c->count);
    delete c;
    return fail(SENSE_ERR_OOM, "context buffer allocation failed");
  }
  *out = c;
  return SENSE_OK;
}

sense_status sense_ctx_destroy(sense_ctx* c) {
  if (!c) return SENSE_OK;
  cudaFree(c->keys);
  cudaFree(c->tokens);
  cudaFree(c->count);
  delete c;
  return SENSE_OK;
}

sense_status sense_ctx_reset(sense_ctx* c, sense_stream_t stream) {
  if (!c) return fail(SENSE_ERR_INVALID_ARG, "ctx is NULL");
  return cuda_check(cudaMemsetAsync(c->count, 0, sizeof(int64_t),
                                    reinterpret_cast<cudaStream_t>(stream)), "reset ctx");
}

sense_status sense_ctx_count(const sense_ctx* c, sense_stream_t stream, int64_t* out) {
  if (!c || !out) return fail(SENSE_ERR_INVALID_ARG, "ctx and out must be non-NULL");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  sense_status st = cuda_check(cudaStreamSynchronize(s), "cudaStreamSynchronize");
  if (st != SENSE_OK) return st;
  return cuda_check(cudaMemcpy(out, c->count, sizeof(int64_t), cudaMemcpyDeviceToHost), "read count");
}

sense_status sense_ctx_append(sense_ctx* c, const uint16_t* hidden, const int32_t* tokens, int32_t t,
                              sense_stream_t stream) {
  if (!c) return fail(SENSE_ERR_INVALID_ARG, "ctx is NULL");
  if (t < 0) return fail(SENSE_ERR_INVALID_ARG, "t=%d must be >= 0", t);
  if (t == 0) return SENSE_OK;
  if (!hidden || !tokens) return fail(SENSE_ERR_INVALID_ARG, "hidden and tokens must be non-NULL");
  if (!aligned(hidden, 16) || !aligned(tokens, 4)) return fail(SENSE_ERR_INVALID_ARG, "hidden must be 16-byte aligned");
  if (current_device() != c->device) return fail(SENSE_ERR_INVALID_ARG, "ctx lives on device %d", c->device);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int first = t > c->cap ? t - c->cap : 0;  // earlier rows would be overwritten
  const int64_t warps = t - first;
  {
    LaunchScope ls(K_CTX, s);
    ctx_append_kernel<<<(unsigned)((warps * 32 + 255) / 256), 256, 0, s>>>(
        hidden, tokens, t, first, c->count, c->cap, c->d, c->keys, c->tokens);
  }
  LaunchScope ls(K_CTX, s);
  ctx_bump_kernel<<<1, 1, 0, s>>>(c->count, t, nullptr, 0);
  return cuda_check(cudaGetLastError(), "launch ctx append");
}

sense_status sense_ctx_append_path(sense_ctx* c, const uint16_t* root_hidden,
                                   const uint16_t* node_hidden, int32_t n_nodes,
                                   const int32_t* gamma, int32_t k, const int32_t* i_star,
                                   const int32_t* n_accept, const int32_t* accepted,
                                   sense_stream_t stream) {
  if (!c) return fail(SENSE_ERR_INVALID_ARG, "ctx is NULL");
  if (!root_hidden || !node_hidden || !gamma || !i_star || !n_accept || !accepted)
    return fail(SENSE_ERR_INVALID_ARG, "arrays must be non-NULL");
  if (k < 1 || n_nodes < 1) return fail(SENSE_ERR_INVALID_ARG, "k=%d and n_nodes=%d must be >= 1", k, n_nodes);
  if (!aligned(root_hidden, 16) || !aligned(node_hidden, 16))
    return fail(SENSE_ERR_INVALID_ARG, "hidden states must be 16-byte aligned");
  if (current_device() != c->device) return fail(SENSE_ERR_INVALID_ARG, "ctx lives on device %d", c->device);
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  LaunchScope ls(K_CTX, s);
  return cuda_check(launch_pdl(ctx_append_path_kernel, dim3(1), dim3((unsigned)(c->m * 32)), 0, s,
                               root_hidden, node_hidden, n_nodes, gamma, k, c->m, i_star,
                               n_accept, accepted, c->count, c->cap, c->d, c->keys, c->tokens,
                               status),
                    "launch ctx append path");
}

size_t sense_ctx_search_workspace_bytes(const sense_ctx* c, int32_t q, int32_t k) {
  if (!c || q < 1 || k < 1) return 0;
  return align256((size_t)q * c->cap * 8) + align256((size_t)q * 4) + align256((size_t)q * k * 4);
}

}  // extern "C"

namespace {
// Validation of a DynSearch and its scoring launch (ctx_score_kernel): every
// query's pool of scored positions is left in the workspace.
sense_status ctx_score(const sense_ctx* c, const uint16_t* queries, int32_t q, int32_t k,
                       float delta, void* workspace, size_t workspace_bytes, cudaStream_t s,
                       uint64_t** pool_out, uint32_t** counts_out, int32_t** rel_out) {
  if (!c) return fail(SENSE_ERR_INVALID_ARG, "ctx is NULL");
  if (!queries || !workspace)
    return fail(SENSE_ERR_INVALID_ARG, "queries, outputs and workspace must be non-NULL");
  if (q < 1 || q > 65535) return fail(SENSE_ERR_INVALID_ARG, "q=%d outside [1, 65535]", q);
  if (k < 1 || k > SENSE_MAX_K) return fail(SENSE_ERR_INVALID_ARG, "k=%d outside [1, %d]", k, SENSE_MAX_K);
  if (!(delta == delta) || delta > 1e30f || delta < -1e30f) return fail(SENSE_ERR_INVALID_ARG, "delta must be finite");
  if (!aligned(queries, 16)) return fail(SENSE_ERR_INVALID_ARG, "queries must be 16-byte aligned");
  if (!aligned(workspace, 256)) return fail(SENSE_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  if (workspace_bytes < sense_ctx_search_workspace_bytes(c, q, k))
    return fail(SENSE_ERR_INVALID_ARG, "workspace of %zu bytes < %zu", workspace_bytes,
                sense_ctx_search_workspace_bytes(c, q, k));
  if (current_device() != c->device) return fail(SENSE_ERR_INVALID_ARG, "ctx lives on device %d", c->device);
  char* ws = static_cast<char*>(workspace);
  auto* pool = reinterpret_cast<uint64_t*>(ws);
  auto* counts = reinterpret_cast<uint32_t*>(ws + align256((size_t)q * c->cap * 8));
  auto* rel = reinterpret_cast<int32_t*>(ws + align256((size_t)q * c->cap * 8) + align256((size_t)q * 4));
  LaunchScope ls(K_CTX, s);
  const int64_t want = ((int64_t)q * c->cap * 32 + 255) / 256;
  const int64_t floor_q = ((int64_t)q * 32 + 255) / 256;  // at least one warp per query
  const int64_t blocks = std::max(floor_q, std::min<int64_t>(want, (int64_t)sm_count() * 16));
  sense_status st = cuda_check(
      launch_pdl(ctx_score_kernel, dim3((unsigned)blocks), dim3(256), 0, s, c->keys, queries, q,
                 c->d, c->cap, c->m, (const int64_t*)c->count, delta, pool, counts),
      "launch ctx score");
  *pool_out = pool;
  *counts_out = counts;
  *rel_out = rel;
  return st;
}

// Validation of a hybrid rerank's arguments (sense_hybrid_drafts).
sense_status check_hybrid(const sense_datastore* ds, const float* static_scores,
                          const int32_t* static_idx, int32_t ks, const float* dyn_scores,
                          const int32_t* dyn_spans, int32_t kd, int32_t q, const int32_t* anchor,
                          int32_t n_keep, uint32_t flags, const int32_t* out_spans) {
  if (!ds) return fail(SENSE_ERR_INVALID_ARG, "ds is NULL");
  if (q < 1 || q > 65535) return fail(SENSE_ERR_INVALID_ARG, "q=%d outside [1, 65535]", q);
  if (ks < 0 || kd < 0 || ks + kd < 1 || ks + kd > kHybridMax)
    return fail(SENSE_ERR_INVALID_ARG, "ks=%d, kd=%d: need 1 <= ks + kd <= %d", ks, kd, kHybridMax);
  if ((ks && (!static_scores || !static_idx)) || (kd && (!dyn_scores || !dyn_spans)) || !out_spans)
    return fail(SENSE_ERR_INVALID_ARG, "candidate arrays and out_spans must be non-NULL");
  if (n_keep < 1 || n_keep > ks + kd)
    return fail(SENSE_ERR_INVALID_ARG, "n_keep=%d outside [1, ks + kd]", n_keep);
  if (flags & ~SENSE_GATHER_FORCE_ANCHOR) return fail(SENSE_ERR_INVALID_ARG, "unknown flags 0x%x", flags);
  if ((flags & SENSE_GATHER_FORCE_ANCHOR) && !anchor)
    return fail(SENSE_ERR_INVALID_ARG, "SENSE_GATHER_FORCE_ANCHOR needs anchor");
  return SENSE_OK;
}
}  // namespace

extern "C" {

sense_status sense_ctx_search(const sense_ctx* c, const uint16_t* queries, int32_t q, int32_t k,
                              float delta, float* out_scores, int64_t* out_pos, int32_t* out_spans,
                              void* workspace, size_t workspace_bytes, sense_stream_t stream) {
  if (!c) return fail(SENSE_ERR_INVALID_ARG, "ctx is NULL");
  if (!queries || !out_scores || !out_pos || !out_spans || !workspace)
    return fail(SENSE_ERR_INVALID_ARG, "queries, outputs and workspace must be non-NULL");
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  uint64_t* pool = nullptr;
  uint32_t* counts = nullptr;
  int32_t* rel = nullptr;
  sense_status st = ctx_score(c, queries, q, k, delta, workspace, workspace_bytes, s, &pool,
                              &counts, &rel);
  if (st != SENSE_OK) return st;
  // top k of each pool, then the winners' positions and spans, one block per query
  return launch_ctx_pool(pool, counts, c->cap, q, k, out_scores, rel, c->count, c->m, c->tokens,
                         out_pos, out_spans, status, s);
}

sense_status sense_hybrid_drafts(const sense_datastore* ds, const float* static_scores,
                                 const int32_t* static_idx, int32_t ks, const float* dyn_scores,
                                 const int32_t* dyn_spans, int32_t kd, int32_t q,
                                 const int32_t* anchor, int32_t n_keep, uint32_t flags,
                                 int32_t* out_spans, sense_stream_t stream) {
  sense_status st = check_hybrid(ds, static_scores, static_idx, ks, dyn_scores, dyn_spans, kd, q,
                                 anchor, n_keep, flags, out_spans);
  if (st != SENSE_OK) return st;
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  LaunchScope ls(K_CTX, s);
  return cuda_check(launch_pdl(hybrid_kernel, dim3((unsigned)q), dim3(1024), 0, s,
                               (const int32_t*)ds->spans, ds->n, ds->m, static_scores, static_idx,
                               ks, dyn_scores, dyn_spans, kd, anchor, n_keep,
                               (flags & SENSE_GATHER_FORCE_ANCHOR) ? 1 : 0, out_spans, status),
                    "launch hybrid drafts");
}

sense_status sense_dyn_draft(const sense_datastore* ds, const sense_ctx* c,
                             const uint16_t* queries, int32_t q, const float* static_scores,
                             const int32_t* static_idx, int32_t ks, int32_t kd, float delta,
                             const int32_t* anchor, int32_t n_keep, uint32_t flags,
                             int32_t node_cap, uint32_t tree_flags, void* workspace,
                             size_t workspace_bytes, float* dyn_scores, int64_t* dyn_pos,
                             int32_t* dyn_spans, int32_t* out_spans, int32_t* out_num_nodes,
                             int32_t* out_tokens, int32_t* out_parent, int32_t* out_depth,
                             int32_t* out_gamma, uint32_t* out_mask_bits, sense_stream_t stream) {
  if (!ds || !c) return fail(SENSE_ERR_INVALID_ARG, "datastore and buffer must be non-NULL");
  if (ds->m != c->m || ds->d != c->d)
    return fail(SENSE_ERR_INVALID_ARG, "datastore and buffer must share d and m");
  if (!dyn_scores || !dyn_pos || !dyn_spans || !out_num_nodes || !out_tokens || !out_parent ||
      !out_depth || !out_gamma)
    return fail(SENSE_ERR_INVALID_ARG, "outputs must be non-NULL");
  const int m = c->m;
  sense_status st = check_hybrid(ds, static_scores, static_idx, ks, dyn_scores, dyn_spans, kd, q,
                                 anchor, n_keep, flags, out_spans);
  if (st != SENSE_OK) return st;
  if ((int64_t)n_keep * m > SENSE_MAX_TREE_TOKENS)
    return fail(SENSE_ERR_INVALID_ARG, "n_keep*m=%d exceeds %d", n_keep * m, SENSE_MAX_TREE_TOKENS);
  if (node_cap < 0) return fail(SENSE_ERR_INVALID_ARG, "node_cap=%d must be >= 0", node_cap);
  if (tree_flags & ~SENSE_TREE_MASK_BITS)
    return fail(SENSE_ERR_INVALID_ARG, "unknown tree flags 0x%x", tree_flags);
  const bool bits = (tree_flags & SENSE_TREE_MASK_BITS) != 0;
  if (bits && !out_mask_bits) return fail(SENSE_ERR_INVALID_ARG, "SENSE_TREE_MASK_BITS needs out_mask_bits");
  const size_t trie_bytes = sizeof(int) * ((size_t)3 * n_keep * m + (size_t)5 * n_keep);
  const size_t smem = std::max((size_t)c->cap * 8, trie_bytes);
  if (!draft_fused_fits(n_keep, m) || smem > kDynDraftSmemMax) {  // the calls one by one
    st = sense_ctx_search(c, queries, q, kd, delta, dyn_scores, dyn_pos, dyn_spans, workspace,
                          workspace_bytes, stream);
    if (st != SENSE_OK) return st;
    st = sense_hybrid_drafts(ds, static_scores, static_idx, ks, dyn_scores, dyn_spans, kd, q,
                             anchor, n_keep, flags, out_spans, stream);
    if (st != SENSE_OK) return st;
    return sense_build_tree(out_spans, q, n_keep, m, node_cap, tree_flags, out_num_nodes,
                            out_tokens, out_parent, out_depth, out_gamma, out_mask_bits, stream);
  }
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  uint64_t* pool = nullptr;
  uint32_t* counts = nullptr;
  int32_t* rel = nullptr;
  st = ctx_score(c, queries, q, kd, delta, workspace, workspace_bytes, s, &pool, &counts, &rel);
  if (st != SENSE_OK) return st;
  st = cuda_check(func_smem(reinterpret_cast<const void*>(dyn_draft_kernel), (int)smem),
                  "cudaFuncSetAttribute(dyn_draft)");
  if (st != SENSE_OK) return st;
  const int cap_nodes = node_cap > 0 ? node_cap : n_keep * m;
  LaunchScope ls(K_CTX, s);
  return cuda_check(
      launch_pdl(dyn_draft_kernel, dim3((unsigned)q), dim3(1024), smem, s, (const uint64_t*)pool,
                 (const uint32_t*)counts, c->cap, kd, dyn_scores, rel, (const int64_t*)c->count,
                 (const int32_t*)c->tokens, dyn_pos, dyn_spans, (const int32_t*)ds->spans, ds->n,
                 m, static_scores, static_idx, ks, anchor, n_keep,
                 (flags & SENSE_GATHER_FORCE_ANCHOR) ? 1 : 0, out_spans, cap_nodes,
                 (cap_nodes + 31) / 32, out_num_nodes, out_tokens, out_parent, out_depth,
                 out_gamma, bits ? out_mask_bits : nullptr, (int)(smem / 8), status),
      "launch dyn draft");
}

}  // extern "C"
