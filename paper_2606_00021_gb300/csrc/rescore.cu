// Exact re-scoring of an approximate shortlist (Sec. 3.2.2 Eq. 8).
//
// The approximate search returns N' candidates D_ret scored in the projected
// space; Eq. 8 ranks them by sim(h, k_i), the similarity of the full hidden
// state to each candidate's key, and keeps the top N.  This kernel computes
// that similarity exactly over the stored bf16 keys (fp32 accumulation, the
// same arithmetic as the exact scan) and selects the top k of the shortlist
// in the order (score desc, key index asc).
//
// A query's shortlist is a gather of N' scattered key rows (2 MB for 256
// rows of 4096 dims), so one query is spread over a cluster of kRsCtas CTAs:
// CTA r scores every kRsCtas-th candidate, one warp per candidate with the
// whole row's 16-byte loads of a lane issued together (the query stays in
// L1), and keeps the candidate keys (score code, inverted index) in its
// shared memory.  CTA 0 then gathers the cluster's keys through distributed
// shared memory, sorts them with a block bitonic network and writes the top
// k.  Slots with index -1 (fewer candidates than N') are empty; an index
// outside [0, n) is empty too and sets SENSE_DEVST_BAD_INDEX.
#include <cooperative_groups.h>
#include <cuda_bf16.h>

#include "common.cuh"
#include "launch.h"

namespace sense {
namespace {

constexpr int kRsCtas = 8;       // CTAs per query (one cluster)
constexpr int kRsThreads = 512;  // 16 warps
constexpr int kRsMaxPer = (SENSE_MAX_RESCORE + kRsCtas - 1) / kRsCtas;
constexpr int kRsBatch = 16;     // 16-byte loads in flight per lane

__device__ __forceinline__ float dot8(uint4 kv, uint4 qv, float acc) {
  acc = fmaf(bf_lo(kv.x), bf_lo(qv.x), acc);
  acc = fmaf(bf_hi(kv.x), bf_hi(qv.x), acc);
  acc = fmaf(bf_lo(kv.y), bf_lo(qv.y), acc);
  acc = fmaf(bf_hi(kv.y), bf_hi(qv.y), acc);
  acc = fmaf(bf_lo(kv.z), bf_lo(qv.z), acc);
  acc = fmaf(bf_hi(kv.z), bf_hi(qv.z), acc);
  acc = fmaf(bf_lo(kv.w), bf_lo(qv.w), acc);
  acc = fmaf(bf_hi(kv.w), bf_hi(qv.w), acc);
  return acc;
}

__global__ void __launch_bounds__(kRsThreads)
rescore_kernel(const uint16_t* __restrict__ keys, int64_t n, int d,
               const uint16_t* __restrict__ queries, const int32_t* __restrict__ cand,
               int n_cand, int n2, int k, float* __restrict__ out_scores,
               int32_t* __restrict__ out_idx, uint32_t* status) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  namespace cg = cooperative_groups;
  cg::cluster_group cl = cg::this_cluster();
  __shared__ uint64_t s_mine[kRsMaxPer];
  __shared__ uint64_t s_all[SENSE_MAX_RESCORE];
  const int r = (int)cl.block_rank();
  const int qi = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nw = blockDim.x >> 5;
  const int per = (n_cand + kRsCtas - 1) / kRsCtas;
  const uint16_t* qrow = queries + (int64_t)qi * d;
  const int chunks = d >> 3;  // 8 bf16 per 16-byte chunk
  for (int i = threadIdx.x; i < per; i += blockDim.x) s_mine[i] = 0ull;
  __syncthreads();
  for (int i = warp; i < per; i += nw) {
    const int c = r + kRsCtas * i;
    if (c >= n_cand) break;  // warp-uniform
    const int32_t idx = cand[(int64_t)qi * n_cand + c];
    if (idx < 0) continue;  // warp-uniform
    if ((int64_t)idx >= n) {
      if (lane == 0) raise_status(status, SENSE_DEVST_BAD_INDEX);
      continue;
    }
    const uint16_t* krow = keys + (int64_t)idx * d;
    float acc = 0.0f;
    for (int j0 = 0; j0 < chunks; j0 += 32 * kRsBatch) {
      uint4 kv[kRsBatch];
#pragma unroll
      for (int t = 0; t < kRsBatch; ++t) {
        const int j = j0 + 32 * t + lane;
        kv[t] = j < chunks ? ld_stream_v4(krow + 8 * j) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int t = 0; t < kRsBatch; ++t) {
        const int j = j0 + 32 * t + lane;
        if (j < chunks)
          acc = dot8(kv[t], __ldg(reinterpret_cast<const uint4*>(qrow + 8 * j)), acc);
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    if (lane == 0) s_mine[i] = cand_key(acc, (uint32_t)idx);
  }
  cl.sync();
  if (r == 0) {
    for (int c = threadIdx.x; c < n2; c += blockDim.x) {
      uint64_t v = 0ull;
      if (c < n_cand) v = *cl.map_shared_rank(s_mine + c / kRsCtas, (unsigned)(c % kRsCtas));
      s_all[c] = v;
    }
    __syncthreads();
    // bitonic sort of n2 keys, largest first
    for (int size = 2; size <= n2; size <<= 1) {
      for (int stride = size >> 1; stride > 0; stride >>= 1) {
        for (int i = threadIdx.x; i < n2 / 2; i += blockDim.x) {
          const int lo = 2 * i - (i & (stride - 1));
          const int hi = lo + stride;
          const bool desc = ((lo & size) == 0);
          const uint64_t a = s_all[lo], b = s_all[hi];
          if ((a < b) == desc) {
            s_all[lo] = b;
            s_all[hi] = a;
          }
        }
        __syncthreads();
      }
    }
    const float NEG = -__int_as_float(0x7f800000);
    for (int t = threadIdx.x; t < k; t += blockDim.x) {
      const uint64_t key = s_all[t];
      out_scores[(int64_t)qi * k + t] = key ? code_score((uint32_t)(key >> 32)) : NEG;
      out_idx[(int64_t)qi * k + t] = key ? (int32_t)cand_index(key) : -1;
    }
  }
  cl.sync();  // the other CTAs' shared memory stays alive until it is read
}

}  // namespace

sense_status launch_rescore(const uint16_t* keys, int64_t n, int d, const uint16_t* queries, int q,
                            const int32_t* cand, int n_cand, int k, float* out_scores,
                            int32_t* out_idx, uint32_t* status, cudaStream_t s) {
  int n2 = 2;
  while (n2 < n_cand) n2 <<= 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kRsCtas, (unsigned)q);
  cfg.blockDim = dim3(kRsThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kRsCtas;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  LaunchScope ls(K_RESCORE, s);
  return cuda_check(cudaLaunchKernelEx(&cfg, rescore_kernel, keys, n, d, queries, cand, n_cand, n2,
                                       k, out_scores, out_idx, status),
                    "launch rescore");
}

}  // namespace sense
