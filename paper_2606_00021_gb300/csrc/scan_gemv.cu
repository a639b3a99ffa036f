// Key scoring for small query batches (q <= 8): a streaming GEMV over the
// bf16 datastore on CUDA cores, fused with the candidate filter of the top-k.
//
// Sec. 3.2.2 (Eq. 7, Eq. 8 sim) scores every key against the query; with q
// this small the scan is a matrix-vector product whose cost is one read of
// the n x d x 2-byte key matrix, so the kernel is built to stream HBM:
//  - one warp per key row; lane l reads 16-byte chunks l, l+32, ... of the
//    row with non-allocating 128-bit loads, up to 16 chunks in flight per
//    lane (8 KB per warp), two 256-thread blocks per SM;
//  - queries sit in shared memory as bf16, products accumulate in fp32;
//  - a butterfly shuffle reduction gives every lane the full dot products;
//  - lane qi turns score qi into a candidate key and either stores it (sample
//    tiles) or appends it to the query's pool when it reaches the threshold.
#include "common.cuh"
#include "launch.h"

namespace sense {
namespace {

template <int MODE>
__device__ __forceinline__ int64_t work_row(int64_t w) {
  if (MODE == SCAN_SAMPLE) {
    const int64_t t = (w / kTileRows) * kSampleStride;
    return t * kTileRows + (w % kTileRows);
  } else if (MODE == SCAN_REST) {
    const int64_t j = w / kTileRows;
    const int64_t t = j + j / (kSampleStride - 1) + 1;
    return t * kTileRows + (w % kTileRows);
  }
  return w;
}

__device__ __forceinline__ float dot8(const uint4 k, const uint4 q, float acc) {
  acc = fmaf(bf_lo(k.x), bf_lo(q.x), acc);
  acc = fmaf(bf_hi(k.x), bf_hi(q.x), acc);
  acc = fmaf(bf_lo(k.y), bf_lo(q.y), acc);
  acc = fmaf(bf_hi(k.y), bf_hi(q.y), acc);
  acc = fmaf(bf_lo(k.z), bf_lo(q.z), acc);
  acc = fmaf(bf_hi(k.z), bf_hi(q.z), acc);
  acc = fmaf(bf_lo(k.w), bf_lo(q.w), acc);
  acc = fmaf(bf_hi(k.w), bf_hi(q.w), acc);
  return acc;
}

template <int Q, int MODE, int UNROLL>
__global__ void __launch_bounds__(256, 2)
scan_gemv_kernel(const uint16_t* __restrict__ keys, int64_t n, int d,
                 const uint16_t* __restrict__ queries, int64_t n_work,
                 const uint64_t* __restrict__ thresh, uint64_t* __restrict__ out,
                 uint32_t* __restrict__ counts, int64_t pool_cap, uint32_t* status) {
  extern __shared__ uint4 s_q[];  // [Q][C] bf16 chunks
  __shared__ uint64_t s_thr[Q];
  const int C = d >> 3;
  const uint4* qsrc = reinterpret_cast<const uint4*>(queries);
  for (int i = threadIdx.x; i < Q * C; i += blockDim.x) s_q[i] = qsrc[i];
  if (threadIdx.x < Q) s_thr[threadIdx.x] = thresh ? thresh[threadIdx.x] : 0ull;
  __syncthreads();

  const int lane = threadIdx.x & 31;
  const int64_t warp0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;

  for (int64_t w = warp0; w < n_work; w += nwarps) {
    const int64_t row = work_row<MODE>(w);
    float acc[Q];
#pragma unroll
    for (int qi = 0; qi < Q; ++qi) acc[qi] = 0.0f;
    if (row < n) {  // uniform across the warp
      const uint4* kr = reinterpret_cast<const uint4*>(keys + row * (int64_t)d);
      for (int c0 = 0; c0 < C; c0 += 32 * UNROLL) {
        uint4 kv[UNROLL];
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
          const int c = c0 + u * 32 + lane;
          kv[u] = (c < C) ? ld_stream_v4(kr + c) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
          const int c = c0 + u * 32 + lane;
          if (c < C) {
#pragma unroll
            for (int qi = 0; qi < Q; ++qi) acc[qi] = dot8(kv[u], s_q[qi * C + c], acc[qi]);
          }
        }
      }
    }
#pragma unroll
    for (int qi = 0; qi < Q; ++qi) {
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) acc[qi] += __shfl_xor_sync(0xffffffffu, acc[qi], off);
    }
    if (MODE == SCAN_SAMPLE) {
#pragma unroll
      for (int qi = 0; qi < Q; ++qi) {
        if (lane == qi) {
          out[(int64_t)qi * n_work + w] = (row < n) ? cand_key(acc[qi], (uint32_t)row) : 0ull;
        }
      }
    } else if (row < n) {
#pragma unroll
      for (int qi = 0; qi < Q; ++qi) {
        if (lane == qi) {
          const uint64_t c = cand_key(acc[qi], (uint32_t)row);
          if (c >= s_thr[qi]) {
            const uint32_t pos = atomicAdd(&counts[qi], 1u);
            if ((int64_t)pos < pool_cap) {
              out[(int64_t)qi * pool_cap + pos] = c;
            } else {
              raise_status(status, SENSE_DEVST_INTERNAL);
            }
          }
        }
      }
    }
  }
}

// Single pass: the GEMV scan of scan_gemv_kernel with the top-k kept in
// per-warp register lists instead of a threshold filter.  Scores are
// warp-uniform after the reduction, so list updates never diverge.  At the
// end the block sorts its warps' lists (bitonic, shared memory) and writes
// its k best keys per query.
template <int Q, int KPL, int UNROLL>
__global__ void __launch_bounds__(256, 2)
scan_gemv_topk_kernel(const uint16_t* __restrict__ keys, int64_t n, int d,
                      const uint16_t* __restrict__ queries, int k,
                      uint64_t* __restrict__ cand) {
  constexpr int K = KPL * 32;   // list length per warp
  constexpr int L = 8 * K;      // entries per query per block (8 warps)
  extern __shared__ uint4 s_q[];  // [Q][C] bf16 chunks, then the lists
  pdl_launch_dependents();      // the merge may be scheduled; it waits for this grid
  const int C = d >> 3;
  const uint4* qsrc = reinterpret_cast<const uint4*>(queries);
  for (int i = threadIdx.x; i < Q * C; i += blockDim.x) s_q[i] = qsrc[i];
  uint64_t* s_list = reinterpret_cast<uint64_t*>(s_q + Q * C);  // [Q][L]
  __syncthreads();

  const int lane = threadIdx.x & 31;
  const int wid = threadIdx.x >> 5;
  const int64_t warp0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  uint64_t v[Q][KPL];
  uint64_t lmin[Q];
#pragma unroll
  for (int qi = 0; qi < Q; ++qi) {
    lmin[qi] = 0ull;
#pragma unroll
    for (int s = 0; s < KPL; ++s) v[qi][s] = 0ull;
  }

  for (int64_t row = warp0; row < n; row += nwarps) {
    float acc[Q];
#pragma unroll
    for (int qi = 0; qi < Q; ++qi) acc[qi] = 0.0f;
    const uint4* kr = reinterpret_cast<const uint4*>(keys + row * (int64_t)d);
    for (int c0 = 0; c0 < C; c0 += 32 * UNROLL) {
      uint4 kv[UNROLL];
#pragma unroll
      for (int u = 0; u < UNROLL; ++u) {
        const int c = c0 + u * 32 + lane;
        kv[u] = (c < C) ? ld_stream_v4(kr + c) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < UNROLL; ++u) {
        const int c = c0 + u * 32 + lane;
        if (c < C) {
#pragma unroll
          for (int qi = 0; qi < Q; ++qi) acc[qi] = dot8(kv[u], s_q[qi * C + c], acc[qi]);
        }
      }
    }
#pragma unroll
    for (int qi = 0; qi < Q; ++qi) {
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) acc[qi] += __shfl_xor_sync(0xffffffffu, acc[qi], off);
      const uint64_t c = cand_key(acc[qi], (uint32_t)row);
      if (c > lmin[qi]) {  // warp-uniform
        list_insert<KPL>(v[qi], c, lane);
        lmin[qi] = __shfl_sync(0xffffffffu, v[qi][KPL - 1], 31);
      }
    }
  }
  // block merge: lists of all warps per query, sorted descending
#pragma unroll
  for (int qi = 0; qi < Q; ++qi) {
#pragma unroll
    for (int s = 0; s < KPL; ++s) s_list[qi * L + wid * K + s * 32 + lane] = v[qi][s];
  }
  __syncthreads();
  for (int size = 2; size <= L; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int t = threadIdx.x; t < Q * L; t += blockDim.x) {
        const int i = t % L, base = t - i;
        const int j = i ^ stride;
        if (j > i) {
          const bool desc = ((i & size) == 0);
          const uint64_t a = s_list[base + i], b = s_list[base + j];
          if (desc ? (a < b) : (a > b)) {
            s_list[base + i] = b;
            s_list[base + j] = a;
          }
        }
      }
      __syncthreads();
    }
  }
  for (int t = threadIdx.x; t < Q * k; t += blockDim.x) {
    const int qi = t / k, r = t - qi * k;
    cand[((int64_t)qi * gridDim.x + blockIdx.x) * k + r] = s_list[qi * L + r];
  }
}

template <int Q, int KPL>
sense_status launch_topk_q(const uint16_t* keys, int64_t n, int d, const uint16_t* queries, int k,
                           int blocks, uint64_t* cand, cudaStream_t s) {
  constexpr int UNROLL = (Q <= 2) ? 16 : 8;
  auto kern = scan_gemv_topk_kernel<Q, KPL, UNROLL>;
  const size_t smem = fused_smem_bytes(Q, d, KPL * 32);
  if (smem > 48 * 1024) {
    cudaError_t e = func_smem(reinterpret_cast<const void*>(kern), (int)smem);
    if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(scan_gemv_topk)");
  }
  LaunchScope ls(K_SCAN_GEMV, s);
  kern<<<blocks, 256, smem, s>>>(keys, n, d, queries, k, cand);
  return cuda_check(cudaGetLastError(), "launch scan_gemv_topk");
}

template <int Q>
sense_status launch_topk_kpl(const uint16_t* keys, int64_t n, int d, const uint16_t* queries,
                             int k, int blocks, uint64_t* cand, cudaStream_t s) {
  if (k <= 32) return launch_topk_q<Q, 1>(keys, n, d, queries, k, blocks, cand, s);
  if (k <= 64) return launch_topk_q<Q, 2>(keys, n, d, queries, k, blocks, cand, s);
  return launch_topk_q<Q, 4>(keys, n, d, queries, k, blocks, cand, s);
}

template <int Q, int MODE>
sense_status launch_q_mode(const uint16_t* keys, int64_t n, int d, const uint16_t* queries,
                           int64_t n_work, const uint64_t* thresh, uint64_t* out, uint32_t* counts,
                           int64_t pool_cap, uint32_t* status, cudaStream_t s) {
  constexpr int UNROLL = (Q <= 2) ? 16 : 8;
  auto kern = scan_gemv_kernel<Q, MODE, UNROLL>;
  const size_t smem = (size_t)Q * d * 2;
  if (smem > 48 * 1024) {
    cudaError_t e = func_smem(reinterpret_cast<const void*>(kern), (int)smem);
    if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(scan_gemv)");
  }
  int per_sm = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 256, smem);
  if (e != cudaSuccess) return cuda_check(e, "occupancy(scan_gemv)");
  if (per_sm < 1) per_sm = 1;
  int64_t blocks = (int64_t)sm_count() * per_sm;
  const int64_t need = (n_work + 7) / 8;  // 8 warps per block
  if (blocks > need) blocks = need > 0 ? need : 1;
  LaunchScope ls(K_SCAN_GEMV, s);
  kern<<<(unsigned)blocks, 256, smem, s>>>(keys, n, d, queries, n_work, thresh, out, counts,
                                           pool_cap, status);
  return cuda_check(cudaGetLastError(), "launch scan_gemv");
}

template <int Q>
sense_status launch_q(const uint16_t* keys, int64_t n, int d, const uint16_t* queries, int mode,
                      int64_t n_work, const uint64_t* thresh, uint64_t* out, uint32_t* counts,
                      int64_t pool_cap, uint32_t* status, cudaStream_t s) {
  switch (mode) {
    case SCAN_SAMPLE:
      return launch_q_mode<Q, SCAN_SAMPLE>(keys, n, d, queries, n_work, thresh, out, counts,
                                           pool_cap, status, s);
    case SCAN_REST:
      return launch_q_mode<Q, SCAN_REST>(keys, n, d, queries, n_work, thresh, out, counts,
                                         pool_cap, status, s);
    default:
      return launch_q_mode<Q, SCAN_ALL>(keys, n, d, queries, n_work, thresh, out, counts,
                                        pool_cap, status, s);
  }
}

}  // namespace

int fused_blocks() { return 2 * sm_count(); }

sense_status launch_scan_gemv_topk(const uint16_t* keys, int64_t n, int d,
                                   const uint16_t* queries, int q, int k, int blocks,
                                   uint64_t* cand, cudaStream_t s) {
  if (k < 1 || k > kFusedMaxK) return fail(SENSE_ERR_UNSUPPORTED, "fused scan needs k <= %d", kFusedMaxK);
  switch (q) {
    case 1: return launch_topk_kpl<1>(keys, n, d, queries, k, blocks, cand, s);
    case 2: return launch_topk_kpl<2>(keys, n, d, queries, k, blocks, cand, s);
    case 3: return launch_topk_kpl<3>(keys, n, d, queries, k, blocks, cand, s);
    case 4: return launch_topk_kpl<4>(keys, n, d, queries, k, blocks, cand, s);
    default: return fail(SENSE_ERR_UNSUPPORTED, "fused scan supports 1..%d queries", kFusedMaxQ);
  }
}

sense_status launch_scan_gemv(const uint16_t* keys, int64_t n, int d, const uint16_t* queries,
                              int q, int mode, int64_t n_work, const uint64_t* thresh,
                              uint64_t* out, uint32_t* counts, int64_t pool_cap,
                              uint32_t* status, cudaStream_t s) {
  switch (q) {
#define SENSE_GEMV_CASE(QQ) \
  case QQ:                  \
    return launch_q<QQ>(keys, n, d, queries, mode, n_work, thresh, out, counts, pool_cap, status, s);
    SENSE_GEMV_CASE(1)
    SENSE_GEMV_CASE(2)
    SENSE_GEMV_CASE(3)
    SENSE_GEMV_CASE(4)
    SENSE_GEMV_CASE(5)
    SENSE_GEMV_CASE(6)
    SENSE_GEMV_CASE(7)
    SENSE_GEMV_CASE(8)
#undef SENSE_GEMV_CASE
    default:
      return fail(SENSE_ERR_UNSUPPORTED, "GEMV scan supports 1..8 queries, got %d", q);
  }
}

}  // namespace sense
