// Approximate retrieval over projected keys: PCA projection, k-means, and an
// inverted-file index with flat vectors or product-quantised residuals.
//
// Sec. 3.2.2 Eq. 7 retrieves the top-N' by ANN(k_t, C_db, N'); App. E sets it
// up: hidden states projected by PCA to 64 dimensions and L2-normalised
// (Alg. 2, k = L2Norm(PCA(h))), a FAISS IVF-PQ index with nlist = 4096,
// nprobe = 32 and pq_m = 16.  Every step here ends in an integer decision (a
// cell, a code, a probe, a top-k index), so the arithmetic follows one fixed
// fp32 evaluation order, with no fused multiply-add (__fmul_rn / __fadd_rn):
//  - projected-space dot products and squared distances (dimension <= 128)
//    are summed term by term, index ascending, by one thread;
//  - the projection's long dot products (dimension d) are summed by the 32
//    lanes of a warp: lane l owns the 4-column groups g with g mod 32 = l,
//    in ascending order, and the lane sums are combined by an xor butterfly
//    (offsets 16, 8, 4, 2, 1);
//  - k-means sums are 2^-31 fixed-point integers (order-free atomics),
//    divided in fp64.
// Kernels:
//  project_bulk_kernel   one or a few query rows: x, the mean and each
//                        warp's row of W arrive by one bulk copy each, one
//                        warp per output; with normalisation the row's
//                        blocks form a cluster and block 0 normalises the
//                        gathered outputs (distributed shared memory)
//  project_rows_kernel   row staged in shared memory, one warp per output:
//                        query batches
//  project_tile_kernel   16 rows x 32 outputs per block, 16 warps, each lane
//                        holding 4 x 8 partial sums: key stores
//  normalize_rows_kernel one thread per row
//  assign_kernel<D,MODE> one thread per vector, centroids staged in shared
//                        memory: k-means and cell assignment (arg max inner
//                        product or arg min L2) and the coarse scores of a
//                        search (thread per cell, queries staged)
//  kmeans_accum / kmeans_finish: fixed-point member sums, new centroids
//  list kernels          stable counting sort of the cells (per-block
//                        histograms, a column scan, one warp placing each
//                        block's ids in order)
//  pq_encode_kernel      residual sub-vector -> nearest of 256 codewords
//  coarse_lut_kernel     a search's coarse keys and PQ lookup tables in one
//                        launch (blocks of cells, then blocks of codebooks)
//  project_coarse_kernel the approximate drafting step's query side: the
//                        normalised projection cluster, then its blocks
//                        write the coarse keys and lookup tables
//  ivf_scan_kernel       one block per (probe, query): flat dot products or
//                        LUT sums, candidates appended to the query's pool;
//                        the exact top-k of the pool is the existing merge.
#include <cooperative_groups.h>

#include <algorithm>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "launch.h"
#include "select_dev.cuh"
#include "tc_ptx.cuh"

struct sense_ivf {
  int64_t n;
  int32_t v;
  int32_t nlist;
  int32_t pq_m;  // 0: flat
  int32_t dsub;
  int64_t max_list;
  int device;
  float* centroids;  // [nlist, v]
  float* codebooks;  // [pq_m, 256, dsub] or null
  int64_t* offsets;  // [nlist + 1]
  int32_t* ids;      // [n] key index of each list slot
  float* vectors;    // flat: [n, v] in list order
  uint8_t* codes;    // pq: [n, pq_m] in list order
};

namespace sense {
namespace {

constexpr int kIdBlock = 4096;   // ids per block of the stable counting sort
constexpr int kMaxList = 16384;  // nlist limit (per-block histogram in shared memory)
constexpr float kFix = 2147483648.0f;  // 2^31

enum AssignMode { ARGMAX_IP = 0, ARGMIN_L2 = 1, ALL_IP = 2 };

// ---------------------------------------------------------------------------
// projection
// ---------------------------------------------------------------------------

__device__ __forceinline__ float madd(float acc, float a, float b) {
  return __fadd_rn(acc, __fmul_rn(a, b));
}

__device__ __forceinline__ float butterfly(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}

// Four bf16 columns j..j+3 of a row, centred (x - mu, rounded to fp32).
__device__ __forceinline__ float4 load_x4(const uint16_t* xr, const float* mu, int j) {
  const uint2 w = *reinterpret_cast<const uint2*>(xr + j);
  float4 x = make_float4(bf_lo(w.x), bf_hi(w.x), bf_lo(w.y), bf_hi(w.y));
  if (mu) {
    const float4 m = *reinterpret_cast<const float4*>(mu + j);
    x = make_float4(__fsub_rn(x.x, m.x), __fsub_rn(x.y, m.y), __fsub_rn(x.z, m.z),
                    __fsub_rn(x.w, m.w));
  }
  return x;
}

constexpr long long kBulkWaitCycles = 4000000000LL;

// Block (output group of opb <= 8, row): the row of x (bf16), the mean and
// the W rows of the block's outputs are brought in by one bulk copy each on
// one mbarrier, so the block pays a single round trip; warp w < opb then
// computes output opb * blockIdx.x + w from shared memory in the order of
// project_rows_kernel (lane l: its 4-column groups ascending; butterfly).
// NORM: the blocks of a row are one cluster (gridDim.x <= 16); block 0
// gathers the v outputs through distributed shared memory and writes the
// row divided by its L2 norm, in the order of normalize_rows_kernel.  With
// s_row (a fused caller) every block does the same into its own s_row[v]
// (block 0 still writes the row) and the function returns without the
// closing cluster barrier: the caller must pass one before it exits, since
// other blocks read this block's outputs.  A
// copy that never lands (bounded wait) sets SENSE_DEVST_TIMEOUT; the row is
// then left unwritten.
template <bool NORM>
__device__ __forceinline__ void project_bulk_block(const uint16_t* __restrict__ x, int d,
                                                   const float* __restrict__ w, int v,
                                                   const float* __restrict__ mu,
                                                   float* __restrict__ out, uint32_t* status,
                                                   int opb = 8, float* s_row = nullptr) {
  extern __shared__ __align__(128) uint8_t smb[];
  __shared__ __align__(8) uint64_t bar;
  __shared__ float s_out[8];
  __shared__ int s_fail;
  uint16_t* sxb = reinterpret_cast<uint16_t*>(smb);                   // [d]
  float* smu = reinterpret_cast<float*>(smb + (size_t)d * 2);         // [d] when mu
  float* sw = smu + (mu ? d : 0);                                     // [opb][d]
  const int64_t row = blockIdx.y;
  const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nw = min(opb, v - (int)blockIdx.x * opb);  // outputs of this block
  const int o = wid < nw ? (int)blockIdx.x * opb + wid : v;
  const uint32_t b = ptx::smem_u32(&bar);
  if (threadIdx.x == 0) {
    ptx::mbar_init(b, 1);
    ptx::fence_barrier_init();
    s_fail = 0;
    const uint32_t bytes = (uint32_t)d * 2u + (mu ? (uint32_t)d * 4u : 0u) + (uint32_t)nw * d * 4u;
    ptx::mbar_arrive_expect_tx(b, bytes);
    const uint64_t pol = ptx::policy_evict_first();
    ptx::bulk_load(ptx::smem_u32(sxb), x + row * d, (uint32_t)d * 2u, b, pol);
    if (mu) ptx::bulk_load(ptx::smem_u32(smu), mu, (uint32_t)d * 4u, b, pol);
    for (int k = 0; k < nw; ++k)
      ptx::bulk_load(ptx::smem_u32(sw + (size_t)k * d), w + (int64_t)(blockIdx.x * opb + k) * d,
                     (uint32_t)d * 4u, b, pol);
  }
  __syncthreads();
  bool got = ptx::mbar_try_wait(b, 0);
  if (!got) {
    const long long t0 = clock64();
    while (!(got = ptx::mbar_try_wait(b, 0)) && clock64() - t0 <= kBulkWaitCycles) {
    }
  }
  if (!got) s_fail = 1;
  __syncthreads();
  const bool fail = s_fail != 0;
  if (fail && threadIdx.x == 0) raise_status(status, SENSE_DEVST_TIMEOUT);
  float acc = 0.0f;
  if (!fail && o < v) {
    const float* wr = sw + (size_t)wid * d;
    for (int j0 = 4 * lane; j0 < d; j0 += 128) {
      const uint2 xw = *reinterpret_cast<const uint2*>(sxb + j0);
      float4 xv = make_float4(bf_lo(xw.x), bf_hi(xw.x), bf_lo(xw.y), bf_hi(xw.y));
      if (mu) {
        const float4 m = *reinterpret_cast<const float4*>(smu + j0);
        xv = make_float4(__fsub_rn(xv.x, m.x), __fsub_rn(xv.y, m.y), __fsub_rn(xv.z, m.z),
                         __fsub_rn(xv.w, m.w));
      }
      const float4 wv = *reinterpret_cast<const float4*>(wr + j0);
      acc = madd(acc, xv.x, wv.x);
      acc = madd(acc, xv.y, wv.y);
      acc = madd(acc, xv.z, wv.z);
      acc = madd(acc, xv.w, wv.w);
    }
    acc = butterfly(acc);
  }
  if constexpr (!NORM) {
    if (!fail && o < v && lane == 0) out[row * v + o] = acc;
  } else {
    namespace cg = cooperative_groups;
    cg::cluster_group cl = cg::this_cluster();
    if (lane == 0) s_out[wid] = acc;
    cl.sync();  // every block's outputs and failure flag are written
    if ((s_row || blockIdx.x == 0) && wid == 0) {
      bool any_fail = false;
      for (unsigned r = 0; r < gridDim.x; ++r) any_fail |= *cl.map_shared_rank(&s_fail, r) != 0;
      if (!any_fail) {
        float part[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int oo = 32 * t + lane;
          part[t] = (oo < v) ? *cl.map_shared_rank(&s_out[oo % opb], (unsigned)(oo / opb)) : 0.0f;
        }
        float ss = 0.0f;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          for (int l = 0; l < 32 && 32 * t + l < v; ++l) {
            const float e = __shfl_sync(0xffffffffu, part[t], l);
            ss = madd(ss, e, e);
          }
        }
        const float nrm = __fsqrt_rn(ss);
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          if (32 * t + lane < v) {
            const float y = nrm > 0.0f ? __fdiv_rn(part[t], nrm) : 0.0f;
            if (blockIdx.x == 0) out[row * v + 32 * t + lane] = y;
            if (s_row) s_row[32 * t + lane] = y;
          }
        }
      } else if (s_row) {
        for (int t = lane; t < v; t += 32) s_row[t] = 0.0f;
      }
    }
    if (s_row) {
      __syncthreads();  // s_row is complete
      return;
    }
    cl.sync();  // the other blocks' shared memory stays alive until it is read
  }
}

template <bool NORM>
__global__ void __launch_bounds__(256)
project_bulk_kernel(const uint16_t* __restrict__ x, int d, const float* __restrict__ w, int v,
                    const float* __restrict__ mu, float* __restrict__ out, uint32_t* status) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  project_bulk_block<NORM>(x, d, w, v, mu, out, status);
}

size_t project_bulk_smem(int d, bool mean, int opb = 8) {
  return (size_t)d * 2 + (mean ? (size_t)d * 4 : 0) + (size_t)opb * 4 * d;
}
constexpr size_t kProjectBulkMax = 200 * 1024;

// Block (output group, row): the centred row is staged in shared memory once;
// warp w computes output 8 * blockIdx.x + w, streaming its row of W.
__global__ void __launch_bounds__(256)
project_rows_kernel(const uint16_t* __restrict__ x, int64_t n, int d,
                    const float* __restrict__ w, int v, const float* __restrict__ mu,
                    float* __restrict__ out) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  extern __shared__ __align__(16) float sx[];  // [d]
  const int64_t row = blockIdx.y;
  const int lane = threadIdx.x & 31;
  const uint16_t* xr = x + row * d;
  for (int j = 4 * threadIdx.x; j < d; j += 4 * blockDim.x)
    *reinterpret_cast<float4*>(sx + j) = load_x4(xr, mu, j);
  __syncthreads();
  const int o = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (o >= v) return;  // warp-uniform
  const float* wr = w + (int64_t)o * d;
  float acc = 0.0f;
  // full rounds of 8 column groups per lane (W loads issued together, then
  // consumed in ascending order), then the remaining groups one by one
  constexpr int U = 8;
  int j0 = 4 * lane;
  for (; j0 + 128 * (U - 1) < d; j0 += 128 * U) {
    float4 wv[U];
#pragma unroll
    for (int u = 0; u < U; ++u) wv[u] = *reinterpret_cast<const float4*>(wr + j0 + 128 * u);
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const float4 xv = *reinterpret_cast<const float4*>(sx + j0 + 128 * u);
      acc = madd(acc, xv.x, wv[u].x);
      acc = madd(acc, xv.y, wv[u].y);
      acc = madd(acc, xv.z, wv[u].z);
      acc = madd(acc, xv.w, wv[u].w);
    }
  }
  for (; j0 < d; j0 += 128) {
    const float4 xv = *reinterpret_cast<const float4*>(sx + j0);
    const float4 wv = *reinterpret_cast<const float4*>(wr + j0);
    acc = madd(acc, xv.x, wv.x);
    acc = madd(acc, xv.y, wv.y);
    acc = madd(acc, xv.z, wv.z);
    acc = madd(acc, xv.w, wv.w);
  }
  acc = butterfly(acc);
  if (lane == 0) out[row * v + o] = acc;
}

// Block: 16 rows x 32 outputs, 16 warps.  Warp w takes rows 4*(w & 3) .. +3
// and outputs 8*(w >> 2) .. +7 of the block's 32; lane l keeps the 32
// partial sums of its column groups.  Columns are staged 128 at a time.
constexpr int kPtRows = 16, kPtOuts = 32, kPtCols = 128;

__global__ void __launch_bounds__(512)
project_tile_kernel(const uint16_t* __restrict__ x, int64_t n, int d,
                    const float* __restrict__ w, int v, const float* __restrict__ mu,
                    float* __restrict__ out) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  __shared__ __align__(16) float xs[kPtRows][kPtCols];
  __shared__ __align__(16) float ws[kPtOuts][kPtCols];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t row0 = (int64_t)blockIdx.x * kPtRows;
  const int out0 = blockIdx.y * kPtOuts;
  const int rg = 4 * (warp & 3), og = 8 * (warp >> 2);
  float acc[4][8];
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int o = 0; o < 8; ++o) acc[r][o] = 0.0f;
  for (int c0 = 0; c0 < d; c0 += kPtCols) {
    __syncthreads();
    // stage x: 16 rows x 128 columns as 4-column groups (512 groups)
    {
      const int r = threadIdx.x >> 5, g = threadIdx.x & 31;
      const int64_t row = row0 + r;
      float4 xv = make_float4(0.f, 0.f, 0.f, 0.f);
      if (row < n && c0 + 4 * g < d) xv = load_x4(x + row * d, mu, c0 + 4 * g);
      *reinterpret_cast<float4*>(&xs[r][4 * g]) = xv;
    }
    // stage w: 32 outputs x 128 columns (1024 float4, 2 per thread)
    for (int e = threadIdx.x; e < kPtOuts * 32; e += blockDim.x) {
      const int o = e >> 5, g = e & 31;
      float4 wv = make_float4(0.f, 0.f, 0.f, 0.f);
      if (out0 + o < v && c0 + 4 * g < d)
        wv = *reinterpret_cast<const float4*>(w + (int64_t)(out0 + o) * d + c0 + 4 * g);
      *reinterpret_cast<float4*>(&ws[o][4 * g]) = wv;
    }
    __syncthreads();
    if (c0 + 4 * lane < d) {
      float4 xv[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) xv[r] = *reinterpret_cast<const float4*>(&xs[rg + r][4 * lane]);
#pragma unroll
      for (int o = 0; o < 8; ++o) {
        const float4 wv = *reinterpret_cast<const float4*>(&ws[og + o][4 * lane]);
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          float a = acc[r][o];
          a = madd(a, xv[r].x, wv.x);
          a = madd(a, xv[r].y, wv.y);
          a = madd(a, xv[r].z, wv.z);
          a = madd(a, xv[r].w, wv.w);
          acc[r][o] = a;
        }
      }
    }
  }
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int o = 0; o < 8; ++o) acc[r][o] = butterfly(acc[r][o]);
  // every lane holds the 32 sums; lane l writes (r, o) = (l / 8, l % 8)
#pragma unroll
  for (int r = 0; r < 4; ++r) {
#pragma unroll
    for (int o = 0; o < 8; ++o) {
      if (lane == 8 * r + o) {
        const int64_t row = row0 + rg + r;
        const int oo = out0 + og + o;
        if (row < n && oo < v) out[row * v + oo] = acc[r][o];
      }
    }
  }
}

// One warp per row (v <= 128): the lanes load the row, every lane forms the
// sum of squares in index order from shuffled values, then scales its part.
__global__ void __launch_bounds__(256)
normalize_rows_kernel(float* __restrict__ y, int64_t n, int v) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  const int64_t i = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (i >= n) return;  // warp-uniform
  float* r = y + i * v;
  float part[4];
#pragma unroll
  for (int t = 0; t < 4; ++t) part[t] = (32 * t + lane < v) ? r[32 * t + lane] : 0.0f;
  float s = 0.0f;
#pragma unroll
  for (int t = 0; t < 4; ++t) {
    for (int l = 0; l < 32 && 32 * t + l < v; ++l) {
      const float e = __shfl_sync(0xffffffffu, part[t], l);
      s = madd(s, e, e);
    }
  }
  const float nrm = __fsqrt_rn(s);
#pragma unroll
  for (int t = 0; t < 4; ++t)
    if (32 * t + lane < v) r[32 * t + lane] = nrm > 0.0f ? __fdiv_rn(part[t], nrm) : 0.0f;
}

// ---------------------------------------------------------------------------
// assignment / coarse scores
// ---------------------------------------------------------------------------

// One thread per row of x ([n, D], row stride ld floats); the rows of c
// ([k, D], contiguous) are staged in shared memory tiles.
//  ARGMAX_IP: out_assign[i] = arg max_c <x_i, c> (first maximum)
//  ARGMIN_L2: out_assign[i] = arg min_c ||x_i - c||^2 (first minimum)
//  ALL_IP:    x = cells, c = queries: pool[c * n + i] = key(<x_i, c>, i)
template <int D, int MODE, bool VEC>
__device__ __forceinline__ void assign_block(const float* __restrict__ x, int64_t n, int ld,
                                             const float* __restrict__ c, int k,
                                             int32_t* __restrict__ out_assign,
                                             uint64_t* __restrict__ pool, int block) {
  constexpr int kTile = (D <= 16) ? 256 : (8192 / D);
  __shared__ __align__(16) float cs[kTile * D];
  const int64_t i = (int64_t)block * blockDim.x + threadIdx.x;
  const bool live = i < n;
  float xr[D];
  if (VEC) {  // 16-byte row loads (x 16-byte aligned, ld % 4 == 0)
#pragma unroll
    for (int j = 0; j < D; j += 4) {
      float4 t = make_float4(0.f, 0.f, 0.f, 0.f);
      if (live) t = *reinterpret_cast<const float4*>(x + i * ld + j);
      xr[j] = t.x;
      xr[j + 1] = t.y;
      xr[j + 2] = t.z;
      xr[j + 3] = t.w;
    }
  } else {
#pragma unroll
    for (int j = 0; j < D; ++j) xr[j] = live ? x[i * ld + j] : 0.0f;
  }
  float best = (MODE == ARGMIN_L2) ? __int_as_float(0x7f800000) : -__int_as_float(0x7f800000);
  int arg = 0;
  for (int t0 = 0; t0 < k; t0 += kTile) {
    const int tn = min(kTile, k - t0);
    __syncthreads();
    for (int e = threadIdx.x; e < tn * D; e += blockDim.x) cs[e] = c[(int64_t)t0 * D + e];
    __syncthreads();
    if (!live) continue;
    for (int t = 0; t < tn; ++t) {
      const float* cr = cs + t * D;
      float s = 0.0f;
      if (MODE == ARGMIN_L2) {
#pragma unroll
        for (int j = 0; j < D; ++j) {
          const float u = __fsub_rn(xr[j], cr[j]);
          s = madd(s, u, u);
        }
        if (s < best || (t0 + t == 0)) {
          best = s;
          arg = t0 + t;
        }
      } else {
#pragma unroll
        for (int j = 0; j < D; ++j) s = madd(s, xr[j], cr[j]);
        if (MODE == ALL_IP) {
          pool[(int64_t)(t0 + t) * n + i] = cand_key(s, (uint32_t)i);
        } else if (s > best || (t0 + t == 0)) {
          best = s;
          arg = t0 + t;
        }
      }
    }
  }
  if (MODE != ALL_IP && live) out_assign[i] = arg;
}

template <int D, int MODE, bool VEC>
__global__ void __launch_bounds__(128)
assign_kernel(const float* __restrict__ x, int64_t n, int ld, const float* __restrict__ c,
              int k, int32_t* __restrict__ out_assign, uint64_t* __restrict__ pool) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  assign_block<D, MODE, VEC>(x, n, ld, c, k, out_assign, pool, blockIdx.x);
}

// The query-side work of an IVF-PQ search in one launch: blocks [0, nbc)
// write the coarse keys of 128 cells each for every query (the ALL_IP
// assignment above), the following pq_m x q blocks the lookup table
// LUT[qi][m][b] = <q_m, B_m[b]> of one sub-quantizer and query (fp32 sums
// over the sub-vector's coordinates in order).
template <int D>
__global__ void __launch_bounds__(128)
coarse_lut_kernel(const float* __restrict__ cells, int64_t nlist, const float* __restrict__ queries,
                  int q, uint64_t* __restrict__ coarse, const float* __restrict__ cb, int pq_m,
                  int dsub, float* __restrict__ lut, int nbc) {
  pdl_wait();  // the projected queries are complete
  pdl_launch_dependents();
  if ((int)blockIdx.x < nbc) {
    assign_block<D, ALL_IP, true>(cells, nlist, D, queries, q, nullptr, coarse, blockIdx.x);
    return;
  }
  __shared__ float sq[128];
  const int b = (int)blockIdx.x - nbc;
  const int m = b % pq_m, qi = b / pq_m;
  for (int j = threadIdx.x; j < dsub; j += blockDim.x) sq[j] = queries[(int64_t)qi * D + m * dsub + j];
  __syncthreads();
  for (int w = threadIdx.x; w < 256; w += blockDim.x) {
    const int e = m * 256 + w;
    const float* bb = cb + (int64_t)e * dsub;
    float s = 0.0f;
    for (int j = 0; j < dsub; ++j) s = madd(s, sq[j], bb[j]);
    lut[(int64_t)qi * pq_m * 256 + e] = s;
  }
}

// The query side of an approximate search in one launch, per query row:
// the normalised projection (project_bulk_kernel<true>: the row's blocks
// form one cluster, block 0 writes the unit row), then, after the cluster
// barrier that makes that row visible, the cluster's C blocks compute the
// coarse keys of every cell (tiles of 256 cells, tile b taken by cluster
// block b mod C; the ALL_IP arithmetic) into block 0's shared memory and
// write the PQ lookup tables (sub-quantizer m by cluster block m mod C),
// with the arithmetic of coarse_lut_kernel.  It also empties the row's candidate
// pool for the list scan (counts[row] = 0).  After a second cluster barrier
// block 0 selects the row's nprobe best cells from the coarse keys (the
// block merge of merge_kernel, in the projection's shared memory).
template <int D>
__global__ void __launch_bounds__(256)
project_coarse_kernel(const uint16_t* __restrict__ x, int d, const float* __restrict__ w,
                      const float* __restrict__ mu, float* __restrict__ out,
                      const float* __restrict__ cells, int64_t nlist,
                      const float* __restrict__ cb, int pq_m, int dsub, float* __restrict__ lut,
                      uint32_t* __restrict__ counts, int nprobe, float* __restrict__ pscore,
                      int32_t* __restrict__ pcell, int keys_off, int opb, uint32_t* status) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  __shared__ float sqr[D];  // the normalised row, formed by every block
  // the closing cluster barrier is the one before the cell selection below
  project_bulk_block<true>(x, d, w, D, mu, out, status, opb, sqr);
  namespace cg = cooperative_groups;
  cg::cluster_group cl = cg::this_cluster();
  extern __shared__ __align__(128) uint8_t smd[];
  const int64_t row = blockIdx.y;
  if (blockIdx.x == 0 && threadIdx.x == 0) counts[row] = 0u;  // the list scan's pool is empty
  const int C = (int)gridDim.x, r = (int)blockIdx.x;
  // coarse keys: tiles of 256 cells staged in shared memory by coalesced
  // loads (row stride D + 1: conflict-free reads), each thread one cell's
  // in-order dot product (the ALL_IP arithmetic), the key stored straight
  // into block 0's shared memory for the cell selection
  constexpr int kTileCells = 256;
  float* tile = reinterpret_cast<float*>(smd);  // [kTileCells][D + 1]
  uint64_t* keys0 = cl.map_shared_rank(reinterpret_cast<uint64_t*>(smd + keys_off), 0);
  const int ntile = (int)((nlist + kTileCells - 1) / kTileCells);
  for (int b = r; b < ntile; b += C) {
    const int64_t c0 = (int64_t)b * kTileCells;
    const int rows = (int)min((int64_t)kTileCells, nlist - c0);
    __syncthreads();  // the previous tile (and sqr) are complete / used
    const float4* src4 = reinterpret_cast<const float4*>(cells + c0 * D);
    const int n4 = rows * (D / 4);
    for (int e0 = threadIdx.x; e0 < n4; e0 += 16 * blockDim.x) {  // sixteen loads in flight
      float4 v[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const int e = e0 + u * blockDim.x;
        v[u] = e < n4 ? __ldg(src4 + e) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const int e = e0 + u * blockDim.x;
        if (e < n4) {
          float* dst = tile + (e / (D / 4)) * (D + 1) + 4 * (e % (D / 4));
          dst[0] = v[u].x;
          dst[1] = v[u].y;
          dst[2] = v[u].z;
          dst[3] = v[u].w;
        }
      }
    }
    __syncthreads();
    for (int t = threadIdx.x; t < rows; t += blockDim.x) {
      const float* xr = tile + t * (D + 1);
      float sc = 0.0f;
#pragma unroll 8
      for (int j = 0; j < D; ++j) sc = madd(sc, xr[j], sqr[j]);
      keys0[c0 + t] = cand_key(sc, (uint32_t)(c0 + t));
    }
  }
  __shared__ float sq[128];
  for (int m = r; m < pq_m; m += C) {
    __syncthreads();
    for (int j = threadIdx.x; j < dsub; j += blockDim.x) sq[j] = sqr[m * dsub + j];
    __syncthreads();
    for (int cw = threadIdx.x; cw < 256; cw += blockDim.x) {
      const int e = m * 256 + cw;
      const float* bb = cb + (int64_t)e * dsub;
      float s = 0.0f;
      for (int j = 0; j < dsub; ++j) s = madd(s, sq[j], bb[j]);
      lut[row * pq_m * 256 + e] = s;
    }
  }
  cl.sync();  // every block's coarse keys are in block 0's shared memory
  if (r == 0)
    merge_pool_block(nullptr, nullptr, nlist, nprobe, pscore, pcell, status, 0, (int)row,
                     reinterpret_cast<uint64_t*>(smd + keys_off), (int)nlist, true);
}

sense_status launch_coarse_lut(const sense_ivf* ix, const float* queries, int q, uint64_t* coarse,
                               float* lut, cudaStream_t s) {
  const int nbc = (ix->nlist + 127) / 128;
  const dim3 grid((unsigned)(nbc + ix->pq_m * q));
  cudaError_t e = cudaSuccess;
#define SENSE_COARSE_LUT_CASE(DD)                                                            \
  case DD:                                                                                  \
    e = launch_pdl(coarse_lut_kernel<DD>, grid, dim3(128), 0, s, (const float*)ix->centroids,  \
                   (int64_t)ix->nlist, queries, q, coarse, (const float*)ix->codebooks,       \
                   ix->pq_m, ix->dsub, lut, nbc);                                             \
    break;
  switch (ix->v) {
    SENSE_COARSE_LUT_CASE(4)
    SENSE_COARSE_LUT_CASE(8)
    SENSE_COARSE_LUT_CASE(16)
    SENSE_COARSE_LUT_CASE(32)
    SENSE_COARSE_LUT_CASE(64)
    SENSE_COARSE_LUT_CASE(128)
    default:
      return fail(SENSE_ERR_UNSUPPORTED, "dimension %d not in {4, 8, 16, 32, 64, 128}", ix->v);
  }
#undef SENSE_COARSE_LUT_CASE
  return cuda_check(e, "launch coarse + lut");
}

constexpr size_t kProjectCoarseMax = 200 * 1024;  // + ~20 KB static (<= 227 KB)

using ProjectCoarseFn = void (*)(const uint16_t*, int, const float*, const float*, float*,
                                 const float*, int64_t, const float*, int, int, float*, uint32_t*,
                                 int, float*, int32_t*, int, int, uint32_t*);

// Whether clusters of 16 blocks of `smem` bytes can run (non-portable size;
// the occupancy query's answer is cached per device and size).
bool cluster16_ok(ProjectCoarseFn kern, size_t smem) {
  constexpr int kMaxDev = 64;
  static std::mutex mu;
  static size_t asked[kMaxDev] = {};
  static bool answer[kMaxDev] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) {
    (void)cudaGetLastError();
    return false;
  }
  std::lock_guard<std::mutex> lk(mu);
  if (asked[dev] == smem) return answer[dev];
  bool ok = cudaFuncSetAttribute(reinterpret_cast<const void*>(kern),
                                 cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess &&
            func_smem(reinterpret_cast<const void*>(kern), (int)smem) == cudaSuccess;
  if (ok) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(16, 1);
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 16;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int nclusters = 0;
    ok = cudaOccupancyMaxActiveClusters(&nclusters, kern, &cfg) == cudaSuccess && nclusters >= 1;
  }
  if (!ok) (void)cudaGetLastError();  // the failed query only means "not 16"
  asked[dev] = smem;
  answer[dev] = ok;
  return ok;
}

// Launches project_coarse_kernel when the row's projection blocks fit one
// cluster and its shared memory; *done = false (nothing launched) otherwise.
sense_status launch_project_coarse(const uint16_t* x, int n, int d, const float* basis,
                                   const float* mean, float* out, const sense_ivf* ix, float* lut,
                                   uint32_t* counts, int nprobe, float* pscore, int32_t* pcell,
                                   cudaStream_t s, bool* done) {
  *done = false;
  const int v = ix->v;
  const bool vdim = v == 4 || v == 8 || v == 16 || v == 32 || v == 64;
  if (!vdim || n > 64) return SENSE_OK;
  ProjectCoarseFn kern = nullptr;
  switch (v) {
    case 4: kern = project_coarse_kernel<4>; break;
    case 8: kern = project_coarse_kernel<8>; break;
    case 16: kern = project_coarse_kernel<16>; break;
    case 32: kern = project_coarse_kernel<32>; break;
    default: kern = project_coarse_kernel<64>; break;
  }
  // the projection's shared memory is reused for the cell tiles; the row's
  // coarse keys follow it (block 0's copy is the one used).  Four outputs
  // per block (16 blocks at v = 64: half the W rows per block and one cell
  // tile each) when a cluster of that size can run, else eight.
  size_t keys_off = 0, smem = 0;
  int opb = 4;
  auto size_for = [&](int ob) {
    keys_off = (std::max(project_bulk_smem(d, mean != nullptr, ob), (size_t)256 * (v + 1) * 4) + 127) &
               ~(size_t)127;
    smem = keys_off + (size_t)ix->nlist * 8;
  };
  size_for(opb);
  if ((v + opb - 1) / opb > 8 && (smem > kProjectCoarseMax || !cluster16_ok(kern, smem))) {
    opb = 8;
    size_for(opb);
  }
  if (smem > kProjectCoarseMax) return SENSE_OK;
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  sense_status st = cuda_check(func_smem(reinterpret_cast<const void*>(kern), (int)smem),
                               "cudaFuncSetAttribute(project_coarse)");
  if (st != SENSE_OK) return st;
  const int groups = (v + opb - 1) / opb;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)groups, (unsigned)n);
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)groups;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  LaunchScope ls(K_PROJECT, s);
  st = cuda_check(cudaLaunchKernelEx(&cfg, kern, x, d, basis, mean, out,
                                     (const float*)ix->centroids, (int64_t)ix->nlist,
                                     (const float*)ix->codebooks, ix->pq_m, ix->dsub, lut, counts,
                                     nprobe, pscore, pcell, (int)keys_off, opb, status),
                  "launch project + coarse");
  if (st == SENSE_OK) *done = true;
  return st;
}

template <int MODE>
sense_status launch_assign_mode(const float* x, int64_t n, int dim, int ld, const float* c, int k,
                                int32_t* out_assign, uint64_t* pool, cudaStream_t s) {
  const dim3 grid((unsigned)((n + 127) / 128));
  const bool vec = (reinterpret_cast<uintptr_t>(x) % 16 == 0) && (ld % 4 == 0);
  cudaError_t e = cudaSuccess;
#define SENSE_ASSIGN_CASE(DD)                                                               \
  case DD:                                                                                  \
    if (vec)                                                                                \
      e = launch_pdl(assign_kernel<DD, MODE, true>, grid, dim3(128), 0, s, x, n, ld, c, k,        \
                     out_assign, pool);                                                         \
    else                                                                                    \
      e = launch_pdl(assign_kernel<DD, MODE, false>, grid, dim3(128), 0, s, x, n, ld, c, k,       \
                     out_assign, pool);                                                         \
    break;
  switch (dim) {
    SENSE_ASSIGN_CASE(4)
    SENSE_ASSIGN_CASE(8)
    SENSE_ASSIGN_CASE(16)
    SENSE_ASSIGN_CASE(32)
    SENSE_ASSIGN_CASE(64)
    SENSE_ASSIGN_CASE(128)
    default:
      return fail(SENSE_ERR_UNSUPPORTED, "dimension %d not in {4, 8, 16, 32, 64, 128}", dim);
  }
#undef SENSE_ASSIGN_CASE
  return cuda_check(e, "launch assign");
}

// ---------------------------------------------------------------------------
// k-means update
// ---------------------------------------------------------------------------

__global__ void kmeans_accum_kernel(const float* __restrict__ x, int64_t n, int dim, int ld,
                                    const int32_t* __restrict__ assign,
                                    unsigned long long* __restrict__ sums,
                                    unsigned* __restrict__ cnt) {
  const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= n * dim) return;
  const int64_t i = e / dim;
  const int j = (int)(e - i * dim);
  const int a = assign[i];
  const long long f = __float2ll_rn(__fmul_rn(x[i * ld + j], kFix));  // exact scaling
  atomicAdd(&sums[(int64_t)a * dim + j], (unsigned long long)f);
  if (j == 0) atomicAdd(&cnt[a], 1u);
}

// One thread per centroid: member mean (previous centroid if empty), then
// unit norm for spherical k-means; clears the sums for the next round.
__global__ void kmeans_finish_kernel(float* __restrict__ c, int k, int dim,
                                     unsigned long long* __restrict__ sums,
                                     unsigned* __restrict__ cnt, int spherical) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= k) return;
  float* cr = c + (int64_t)t * dim;
  const unsigned m = cnt[t];
  for (int j = 0; j < dim; ++j) {
    unsigned long long* sp = &sums[(int64_t)t * dim + j];
    if (m > 0) {
      const double mean = __ddiv_rn(__ll2double_rn((long long)*sp), (double)m);
      cr[j] = __double2float_rn(mean * (1.0 / 2147483648.0));
    }
    *sp = 0ull;
  }
  cnt[t] = 0u;
  if (spherical) {
    float s = 0.0f;
    for (int j = 0; j < dim; ++j) s = madd(s, cr[j], cr[j]);
    const float nrm = __fsqrt_rn(s);
    for (int j = 0; j < dim; ++j) cr[j] = nrm > 0.0f ? __fdiv_rn(cr[j], nrm) : 0.0f;
  }
}

// Unit norm of every centroid (spherical k-means starts from unit seeds).
__global__ void normalize_centroids_kernel(float* __restrict__ c, int k, int dim) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= k) return;
  float* cr = c + (int64_t)t * dim;
  float s = 0.0f;
  for (int j = 0; j < dim; ++j) s = madd(s, cr[j], cr[j]);
  const float nrm = __fsqrt_rn(s);
  for (int j = 0; j < dim; ++j) cr[j] = nrm > 0.0f ? __fdiv_rn(cr[j], nrm) : 0.0f;
}

// ---------------------------------------------------------------------------
// inverted lists: stable counting sort of the cells
// ---------------------------------------------------------------------------

__global__ void cell_hist_kernel(const int32_t* __restrict__ cell, int64_t n, int nlist,
                                 unsigned* __restrict__ hist) {
  extern __shared__ unsigned sh[];
  for (int c = threadIdx.x; c < nlist; c += blockDim.x) sh[c] = 0u;
  __syncthreads();
  const int64_t lo = (int64_t)blockIdx.x * kIdBlock;
  const int64_t hi = min(n, lo + kIdBlock);
  for (int64_t i = lo + threadIdx.x; i < hi; i += blockDim.x) atomicAdd(&sh[cell[i]], 1u);
  __syncthreads();
  unsigned* row = hist + (int64_t)blockIdx.x * nlist;
  for (int c = threadIdx.x; c < nlist; c += blockDim.x) row[c] = sh[c];
}

// One thread per cell: total over the id blocks, and each block's base
// (count of this cell's members in earlier blocks).
__global__ void cell_totals_kernel(const unsigned* __restrict__ hist, int nb, int nlist,
                                   unsigned* __restrict__ base, int64_t* __restrict__ totals) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= nlist) return;
  unsigned run = 0;
  for (int b = 0; b < nb; ++b) {
    base[(int64_t)b * nlist + c] = run;
    run += hist[(int64_t)b * nlist + c];
  }
  totals[c] = run;
}

// One block: offsets[c] = sum of totals[0..c), offsets[nlist] = n (in place
// over totals[0..nlist] -> offsets), and the longest list.
__global__ void __launch_bounds__(1024)
cell_offsets_kernel(int64_t* __restrict__ off, int nlist, int64_t* __restrict__ max_list) {
  __shared__ int64_t part[1024];
  __shared__ int64_t mx[1024];
  const int per = (nlist + blockDim.x - 1) / blockDim.x;
  const int lo = threadIdx.x * per, hi = min(nlist, lo + per);
  int64_t s = 0, m = 0;
  for (int c = lo; c < hi; ++c) {
    s += off[c];
    m = max(m, off[c]);
  }
  part[threadIdx.x] = s;
  mx[threadIdx.x] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    int64_t run = 0, mm = 0;
    for (int t = 0; t < (int)blockDim.x; ++t) {
      const int64_t v = part[t];
      part[t] = run;
      run += v;
      mm = max(mm, mx[t]);
    }
    off[nlist] = run;
    *max_list = mm;
  }
  __syncthreads();
  int64_t run = part[threadIdx.x];
  for (int c = lo; c < hi; ++c) {
    const int64_t v = off[c];
    off[c] = run;
    run += v;
  }
}

// One warp per id block: walks the ids in ascending order, 32 at a time, and
// gives each the next slot of its cell (stable).
__global__ void __launch_bounds__(32)
cell_place_kernel(const int32_t* __restrict__ cell, int64_t n, int nlist,
                  const int64_t* __restrict__ off, const unsigned* __restrict__ base,
                  int32_t* __restrict__ pos, int32_t* __restrict__ ids) {
  extern __shared__ int64_t next[];
  const int lane = threadIdx.x;
  for (int c = lane; c < nlist; c += 32) next[c] = off[c] + base[(int64_t)blockIdx.x * nlist + c];
  __syncwarp();
  const int64_t lo = (int64_t)blockIdx.x * kIdBlock;
  const int64_t hi = min(n, lo + kIdBlock);
  for (int64_t i0 = lo; i0 < hi; i0 += 32) {
    const int64_t i = i0 + lane;
    const bool live = i < hi;
    const unsigned act = __ballot_sync(0xffffffffu, live);
    if (live) {
      const int c = cell[i];
      const unsigned peers = __match_any_sync(act, c);
      const int rank = __popc(peers & ((1u << lane) - 1u));
      const int64_t p = next[c] + rank;
      pos[i] = (int32_t)p;
      ids[p] = (int32_t)i;
      __syncwarp(act);
      if (rank == 0) next[c] += __popc(peers);
    }
    __syncwarp();
  }
}

// Flat lists: one warp per vector copies it to its slot.
__global__ void scatter_vectors_kernel(const float* __restrict__ x, int64_t n, int v,
                                       const int32_t* __restrict__ pos, float* __restrict__ out) {
  const int64_t i = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (i >= n) return;
  const float* src = x + i * v;
  float* dst = out + (int64_t)pos[i] * v;
  for (int j = lane; j < v; j += 32) dst[j] = src[j];
}

// PQ codes: a block covers 32 vectors (lanes) x all sub-quantizers (warps
// stride over them); the codebooks sit in shared memory.  Residual
// r = x - c_cell, code_m = arg min_b ||r_m - B_m[b]||^2 (first minimum).
__global__ void __launch_bounds__(256)
pq_encode_kernel(const float* __restrict__ x, int64_t n, int v, const float* __restrict__ cent,
                 const int32_t* __restrict__ cell, const float* __restrict__ cb, int pq_m,
                 int dsub, const int32_t* __restrict__ pos, uint8_t* __restrict__ codes) {
  extern __shared__ float scb[];  // [pq_m][256][dsub]
  const int total = pq_m * 256 * dsub;
  for (int e = threadIdx.x; e < total; e += blockDim.x) scb[e] = cb[e];
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t i = (int64_t)blockIdx.x * 32 + lane;
  if (i >= n) return;
  const float* xr = x + i * v;
  const float* cr = cent + (int64_t)cell[i] * v;
  uint8_t* out = codes + (int64_t)pos[i] * pq_m;
  float r[16];
  for (int m = warp; m < pq_m; m += blockDim.x >> 5) {
    for (int j = 0; j < dsub; ++j) r[j] = __fsub_rn(xr[m * dsub + j], cr[m * dsub + j]);
    const float* bm = scb + m * 256 * dsub;
    float best = 0.0f;
    int arg = 0;
    for (int b = 0; b < 256; ++b) {
      float s = 0.0f;
      for (int j = 0; j < dsub; ++j) {
        const float u = __fsub_rn(r[j], bm[b * dsub + j]);
        s = madd(s, u, u);
      }
      if (b == 0 || s < best) {
        best = s;
        arg = b;
      }
    }
    out[m] = (uint8_t)arg;
  }
}

// Residuals r = x - c_cell (for training PQ codebooks).
__global__ void residual_kernel(const float* __restrict__ x, int64_t n, int v,
                                const float* __restrict__ cent, const int32_t* __restrict__ cell,
                                float* __restrict__ out) {
  const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= n * v) return;
  const int64_t i = e / v;
  const int j = (int)(e - i * v);
  out[e] = __fsub_rn(x[e], cent[(int64_t)cell[i] * v + j]);
}

// ---------------------------------------------------------------------------
// search: lookup tables and list scan
// ---------------------------------------------------------------------------

// PQ lookup table of each query: lut[qi][m][b] = <q_m, B_m[b]> (dsub terms in
// index order).  One block per (sub-quantizer m, query), one thread per
// codeword b: every codeword row is loaded at once (one round trip).
constexpr int kScanThreads = 256;
// Flat lists are staged in chunks of kScanThreads x flat_rows_per_thread(v)
// vectors with a padded row stride of v + 4 floats (16-byte reads of 8
// consecutive threads hit distinct bank groups).  One row per thread keeps
// a block at <= 135 KB of shared memory (70 KB at v = 64, three blocks per
// SM); long lists are split across blocks instead.
__host__ __device__ constexpr int flat_rows_per_thread(int) { return 1; }

// 16-byte asynchronous global -> shared copy through L2 (cp.async.cg);
// cp_async_wait() completes the thread's copies.
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(ptx::smem_u32(dst)), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_all;" ::: "memory");
}

// One block per (probe p, query qi, list part z): part z of a list takes
// its chunks z, z + gridDim.z, ... (a flat chunk is kScanThreads x
// flat_rows_per_thread(v) entries, a PQ chunk kScanThreads), so that a long
// list is not scanned by one block alone.  Flat: the chunk's vectors are
// staged and each thread scores its rows (<q, x> in index order).  PQ: the block stages the query's lookup
// table in shared memory (copies issued before the probe's cell is read,
// which they do not depend on); each thread reads its code row (16 codes
// per 16-byte load when pq_m % 16 == 0) and sums
// coarse + LUT[0][c_0] + ... + LUT[pq_m-1][c_{pq_m-1}] in that order.
// Candidates go to the query's pool (warp-aggregated append).
__global__ void __launch_bounds__(kScanThreads)
ivf_scan_kernel(const sense_ivf ix, const float* __restrict__ queries,
                const float* __restrict__ lut, int nprobe,
                const float* __restrict__ probe_score, const int32_t* __restrict__ probe_cell,
                uint64_t* __restrict__ pool, uint32_t* __restrict__ counts, int64_t pool_cap,
                uint32_t* status) {
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  extern __shared__ __align__(16) float sm[];
  const int p = blockIdx.x, qi = blockIdx.y;
  const int v = ix.v;
  float* sq = sm;                  // [v]
  float* stage = sm + 128;         // flat: staged vectors [rows][v + 4]; pq: LUT [pq_m][256]
  const float* q = queries + (int64_t)qi * v;
  if (ix.pq_m > 0) {  // the lookup table goes to shared memory while the cell is read
    const float4* src = reinterpret_cast<const float4*>(lut + (int64_t)qi * ix.pq_m * 256);
    for (int e = threadIdx.x; e < ix.pq_m * 64; e += blockDim.x)
      cp_async16(reinterpret_cast<float4*>(stage) + e, src + e);
  } else {
    for (int j = threadIdx.x; j < v; j += blockDim.x) sq[j] = q[j];
  }
  const int cell = probe_cell[(int64_t)qi * nprobe + p];
  const float coarse = probe_score[(int64_t)qi * nprobe + p];
  if (cell < 0 || cell >= ix.nlist) {
    cp_async_wait();
    if (threadIdx.x == 0) raise_status(status, SENSE_DEVST_INTERNAL);
    return;
  }
  const int64_t lo = ix.offsets[cell], hi = ix.offsets[cell + 1];
  cp_async_wait();
  __syncthreads();
  uint64_t* dst = pool + (int64_t)qi * pool_cap;
  if (ix.pq_m > 0) {
    const bool wide = (ix.pq_m & 15) == 0;
    for (int64_t s0 = lo + (int64_t)blockIdx.z * blockDim.x; s0 < hi;
         s0 += (int64_t)gridDim.z * blockDim.x) {
      const int64_t slot = s0 + threadIdx.x;
      const bool live = slot < hi;
      float s = coarse;
      if (live) {
        const uint8_t* cr = ix.codes + slot * ix.pq_m;
        if (wide) {
          for (int m0 = 0; m0 < ix.pq_m; m0 += 16) {
            const uint4 w4 = __ldg(reinterpret_cast<const uint4*>(cr + m0));
            const uint32_t w[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
            for (int b = 0; b < 16; ++b) {
              const uint32_t c = (w[b >> 2] >> (8 * (b & 3))) & 255u;
              s = __fadd_rn(s, stage[((m0 + b) << 8) + c]);
            }
          }
        } else {
          for (int m = 0; m < ix.pq_m; ++m) s = __fadd_rn(s, stage[(m << 8) + cr[m]]);
        }
      }
      const uint32_t at = warp_append(&counts[qi], live);
      if (live) {
        if ((int64_t)at < pool_cap) dst[at] = cand_key(s, (uint32_t)ix.ids[slot]);
        else raise_status(status, SENSE_DEVST_INTERNAL);
      }
    }
  } else {
    // one chunk of vectors is copied with every 16-byte copy in flight at
    // once, then each thread scores its rows (<q, x> in index order)
    const int vq = v >> 2, fs = v + 4;
    const int64_t chunk = (int64_t)blockDim.x * flat_rows_per_thread(v);
    for (int64_t c0 = lo + blockIdx.z * chunk; c0 < hi; c0 += gridDim.z * chunk) {
      const int rows = (int)min(chunk, hi - c0);
      __syncthreads();  // the previous chunk's rows are read
      const float4* src = reinterpret_cast<const float4*>(ix.vectors + c0 * v);
      for (int e = threadIdx.x; e < rows * vq; e += blockDim.x) {
        const int r = e / vq, g = e - r * vq;
        cp_async16(stage + r * fs + 4 * g, src + e);
      }
      cp_async_wait();
      __syncthreads();
      for (int r0 = 0; r0 < rows; r0 += blockDim.x) {
        const int r = r0 + threadIdx.x;
        const bool live = r < rows;
        float s = 0.0f;
        if (live) {
          const float* xr = stage + r * fs;
          for (int g = 0; g < vq; ++g) {
            const float4 xv = *reinterpret_cast<const float4*>(xr + 4 * g);
            s = madd(s, sq[4 * g], xv.x);
            s = madd(s, sq[4 * g + 1], xv.y);
            s = madd(s, sq[4 * g + 2], xv.z);
            s = madd(s, sq[4 * g + 3], xv.w);
          }
        }
        const uint32_t at = warp_append(&counts[qi], live);
        if (live) {
          const int64_t slot = c0 + r;
          if ((int64_t)at < pool_cap) dst[at] = cand_key(s, (uint32_t)ix.ids[slot]);
          else raise_status(status, SENSE_DEVST_INTERNAL);
        }
      }
    }
  }
}

// Parts per probed list: enough that the longest list is one chunk per
// block, at most 8, and fewer when the probes alone fill the GPU.
int scan_parts(const sense_ivf* ix, int q, int nprobe) {
  const int64_t chunk = (int64_t)kScanThreads * (ix->pq_m > 0 ? 1 : flat_rows_per_thread(ix->v));
  int parts = (int)std::min<int64_t>(8, std::max<int64_t>(1, (ix->max_list + chunk - 1) / chunk));
  const int64_t blocks = (int64_t)nprobe * q;
  const int64_t budget = 4LL * sm_count();
  if (blocks * parts > budget) parts = (int)std::max<int64_t>(1, budget / blocks);
  return parts;
}

size_t scan_smem_bytes(const sense_ivf* ix) {
  const size_t stage = ix->pq_m > 0 ? (size_t)ix->pq_m * 256
                                     : (size_t)kScanThreads * flat_rows_per_thread(ix->v) * (ix->v + 4);
  return (128 + stage) * sizeof(float);
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

struct SearchPlan {
  size_t off_coarse, off_pscore, off_pcell, off_counts, off_lut, off_pool, total;
  int64_t pool_cap;
};

SearchPlan search_plan(const sense_ivf* ix, int q, int nprobe) {
  SearchPlan p{};
  size_t o = 0;
  p.off_coarse = o;
  o = align256(o + (size_t)q * ix->nlist * 8);
  p.off_pscore = o;
  o = align256(o + (size_t)q * nprobe * 4);
  p.off_pcell = o;
  o = align256(o + (size_t)q * nprobe * 4);
  p.off_counts = o;
  o = align256(o + (size_t)q * 4);
  p.off_lut = o;
  o = align256(o + (size_t)q * ix->pq_m * 256 * 4);
  p.pool_cap = std::max<int64_t>(1, (int64_t)nprobe * ix->max_list);
  p.off_pool = o;
  o = align256(o + (size_t)q * p.pool_cap * 8);
  p.total = o;
  return p;
}

int current_device() {
  int dev = 0;
  cudaGetDevice(&dev);
  return dev;
}

bool aligned(const void* ptr, size_t a) { return (reinterpret_cast<uintptr_t>(ptr) % a) == 0; }

bool dim_ok(int dim) {
  return dim == 4 || dim == 8 || dim == 16 || dim == 32 || dim == 64 || dim == 128;
}

void free_ivf(sense_ivf* ix) {
  if (!ix) return;
  cudaFree(ix->centroids);
  cudaFree(ix->codebooks);
  cudaFree(ix->offsets);
  cudaFree(ix->ids);
  cudaFree(ix->vectors);
  cudaFree(ix->codes);
  delete ix;
}

}  // namespace
}  // namespace sense

using namespace sense;

extern "C" {

sense_status sense_project(const uint16_t* x, int64_t n, int32_t d, const float* basis, int32_t v,
                           const float* mean, uint32_t flags, float* out, sense_stream_t stream) {
  if (!x || !basis || !out) return fail(SENSE_ERR_INVALID_ARG, "x, basis and out must be non-NULL");
  if (n < 1) return fail(SENSE_ERR_INVALID_ARG, "n=%lld must be >= 1", (long long)n);
  if (d < 8 || d % 8) return fail(SENSE_ERR_INVALID_ARG, "d=%d must be a positive multiple of 8", d);
  if (v < 1 || v > SENSE_MAX_PROJ_DIM)
    return fail(SENSE_ERR_INVALID_ARG, "v=%d outside [1, %d]", v, SENSE_MAX_PROJ_DIM);
  if (flags & ~SENSE_PROJECT_NORMALIZE) return fail(SENSE_ERR_INVALID_ARG, "unknown flags 0x%x", flags);
  if (!aligned(x, 16) || !aligned(basis, 16) || (mean && !aligned(mean, 16)) || !aligned(out, 4))
    return fail(SENSE_ERR_INVALID_ARG, "x, basis and mean must be 16-byte aligned");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int groups = (v + 7) / 8;
  const size_t bulk_smem = project_bulk_smem(d, mean != nullptr);
  if (n <= 64 && bulk_smem <= kProjectBulkMax) {
    // one query batch: bulk copies, normalisation fused when a row's blocks fit a cluster
    uint32_t* status = device_status_word();
    if (!status) return SENSE_ERR_OOM;
    const bool fuse = (flags & SENSE_PROJECT_NORMALIZE) && groups <= 8;
    void (*kern)(const uint16_t*, int, const float*, int, const float*, float*, uint32_t*) =
        fuse ? project_bulk_kernel<true> : project_bulk_kernel<false>;
    sense_status st = cuda_check(
        func_smem(reinterpret_cast<const void*>(kern), (int)bulk_smem),
        "cudaFuncSetAttribute(project_bulk)");
    if (st != SENSE_OK) return st;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)groups, (unsigned)n);
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = bulk_smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = fuse ? (unsigned)groups : 1u;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    {
      LaunchScope ls(K_PROJECT, s);
      st = cuda_check(cudaLaunchKernelEx(&cfg, kern, x, (int)d, basis, (int)v, mean, out, status),
                      "launch project_bulk");
      if (st != SENSE_OK) return st;
    }
    if (fuse || !(flags & SENSE_PROJECT_NORMALIZE)) return SENSE_OK;
    LaunchScope ls(K_PROJECT, s);
    return cuda_check(launch_pdl(normalize_rows_kernel, dim3((unsigned)((n * 32 + 255) / 256)),
                                 dim3(256), 0, s, out, n, v),
                      "launch normalize rows");
  }
  {
    LaunchScope ls(K_PROJECT, s);
    cudaError_t e = cudaSuccess;
    if (n * v <= 16384 && n <= 65535 && d <= 12288) {
      const dim3 grid((unsigned)((v + 7) / 8), (unsigned)n);
      e = launch_pdl(project_rows_kernel, grid, dim3(256), (size_t)d * 4, s, x, n, d, basis, v,
                     mean, out);
    } else {
      const dim3 grid((unsigned)((n + kPtRows - 1) / kPtRows), (unsigned)((v + kPtOuts - 1) / kPtOuts));
      e = launch_pdl(project_tile_kernel, grid, dim3(512), 0, s, x, n, d, basis, v, mean, out);
    }
    sense_status st = cuda_check(e, "launch project");
    if (st != SENSE_OK) return st;
  }
  if (flags & SENSE_PROJECT_NORMALIZE) {
    LaunchScope ls(K_PROJECT, s);
    return cuda_check(launch_pdl(normalize_rows_kernel, dim3((unsigned)((n * 32 + 255) / 256)),
                                 dim3(256), 0, s, out, n, v),
                      "launch normalize rows");
  }
  return SENSE_OK;
}

size_t sense_kmeans_workspace_bytes(int64_t n, int32_t dim, int32_t k) {
  if (n < 1 || dim < 1 || k < 1) return 0;
  return align256((size_t)n * 4) + align256((size_t)k * dim * 8) + align256((size_t)k * 4);
}

sense_status sense_kmeans(const float* x, int64_t n, int32_t dim, int32_t ld, int32_t k,
                          int32_t iters, uint32_t flags, const float* init, float* centroids,
                          int32_t* out_assign, void* workspace, size_t workspace_bytes,
                          sense_stream_t stream) {
  if (!x || !init || !centroids || !workspace)
    return fail(SENSE_ERR_INVALID_ARG, "x, init, centroids and workspace must be non-NULL");
  if (n < 1 || n > INT32_MAX) return fail(SENSE_ERR_INVALID_ARG, "n=%lld outside [1, 2^31)", (long long)n);
  if (!dim_ok(dim)) return fail(SENSE_ERR_INVALID_ARG, "dim=%d not in {4, 8, 16, 32, 64, 128}", dim);
  if (ld < dim) return fail(SENSE_ERR_INVALID_ARG, "ld=%d < dim=%d", ld, dim);
  if (k < 1 || k > 65536) return fail(SENSE_ERR_INVALID_ARG, "k=%d outside [1, 65536]", k);
  if (iters < 0) return fail(SENSE_ERR_INVALID_ARG, "iters=%d must be >= 0", iters);
  if (flags & ~SENSE_KMEANS_SPHERICAL) return fail(SENSE_ERR_INVALID_ARG, "unknown flags 0x%x", flags);
  if (workspace_bytes < sense_kmeans_workspace_bytes(n, dim, k))
    return fail(SENSE_ERR_INVALID_ARG, "workspace of %zu bytes < %zu", workspace_bytes,
                sense_kmeans_workspace_bytes(n, dim, k));
  if (!aligned(workspace, 256)) return fail(SENSE_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  char* ws = static_cast<char*>(workspace);
  int32_t* assign = reinterpret_cast<int32_t*>(ws);
  auto* sums = reinterpret_cast<unsigned long long*>(ws + align256((size_t)n * 4));
  auto* cnt = reinterpret_cast<unsigned*>(ws + align256((size_t)n * 4) + align256((size_t)k * dim * 8));
  const bool sph = (flags & SENSE_KMEANS_SPHERICAL) != 0;
  sense_status st = cuda_check(cudaMemcpyAsync(centroids, init, (size_t)k * dim * 4,
                                               cudaMemcpyDeviceToDevice, s), "copy init");
  if (st != SENSE_OK) return st;
  st = cuda_check(cudaMemsetAsync(sums, 0, (size_t)k * dim * 8, s), "clear sums");
  if (st != SENSE_OK) return st;
  st = cuda_check(cudaMemsetAsync(cnt, 0, (size_t)k * 4, s), "clear counts");
  if (st != SENSE_OK) return st;
  LaunchScope ls(K_KMEANS, s);
  if (sph) normalize_centroids_kernel<<<(k + 127) / 128, 128, 0, s>>>(centroids, k, dim);
  for (int it = 0; it < iters; ++it) {
    st = sph ? launch_assign_mode<ARGMAX_IP>(x, n, dim, ld, centroids, k, assign, nullptr, s)
             : launch_assign_mode<ARGMIN_L2>(x, n, dim, ld, centroids, k, assign, nullptr, s);
    if (st != SENSE_OK) return st;
    const int64_t e = n * dim;
    kmeans_accum_kernel<<<(unsigned)((e + 255) / 256), 256, 0, s>>>(x, n, dim, ld, assign, sums, cnt);
    kmeans_finish_kernel<<<(k + 127) / 128, 128, 0, s>>>(centroids, k, dim, sums, cnt, sph ? 1 : 0);
  }
  if (out_assign && iters > 0) {
    st = cuda_check(cudaMemcpyAsync(out_assign, assign, (size_t)n * 4, cudaMemcpyDeviceToDevice, s),
                    "copy assignment");
    if (st != SENSE_OK) return st;
  }
  return cuda_check(cudaGetLastError(), "launch kmeans");
}

sense_status sense_ivf_residuals(const float* vecs, int64_t n, int32_t v, const float* centroids,
                                 int32_t nlist, int32_t* out_cell, float* out_residuals,
                                 sense_stream_t stream) {
  if (!vecs || !centroids || !out_cell || !out_residuals)
    return fail(SENSE_ERR_INVALID_ARG, "arrays must be non-NULL");
  if (n < 1 || n > INT32_MAX) return fail(SENSE_ERR_INVALID_ARG, "n=%lld outside [1, 2^31)", (long long)n);
  if (!dim_ok(v) || v < 16) return fail(SENSE_ERR_INVALID_ARG, "v=%d not in {16, 32, 64, 128}", v);
  if (nlist < 1 || nlist > kMaxList) return fail(SENSE_ERR_INVALID_ARG, "nlist=%d outside [1, %d]", nlist, kMaxList);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  LaunchScope ls(K_IVF_BUILD, s);
  sense_status st = launch_assign_mode<ARGMAX_IP>(vecs, n, v, v, centroids, nlist, out_cell, nullptr, s);
  if (st != SENSE_OK) return st;
  residual_kernel<<<(unsigned)((n * v + 255) / 256), 256, 0, s>>>(vecs, n, v, centroids, out_cell,
                                                                  out_residuals);
  return cuda_check(cudaGetLastError(), "launch residuals");
}

sense_status sense_ivf_build(const float* vecs, int64_t n, int32_t v, const float* centroids,
                             int32_t nlist, const float* codebooks, int32_t pq_m,
                             sense_stream_t stream, sense_ivf** out) {
  if (!out) return fail(SENSE_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (!vecs || !centroids) return fail(SENSE_ERR_INVALID_ARG, "vecs and centroids must be non-NULL");
  if (n < 1 || n > INT32_MAX) return fail(SENSE_ERR_INVALID_ARG, "n=%lld outside [1, 2^31)", (long long)n);
  if (!dim_ok(v) || v < 16) return fail(SENSE_ERR_INVALID_ARG, "v=%d not in {16, 32, 64, 128}", v);
  if (nlist < 1 || nlist > kMaxList) return fail(SENSE_ERR_INVALID_ARG, "nlist=%d outside [1, %d]", nlist, kMaxList);
  if (codebooks) {
    if (pq_m < 1 || v % pq_m || v / pq_m > 16)
      return fail(SENSE_ERR_INVALID_ARG, "pq_m=%d must divide v=%d with v/pq_m <= 16", pq_m, v);
  } else if (pq_m != 0) {
    return fail(SENSE_ERR_INVALID_ARG, "pq_m=%d needs codebooks", pq_m);
  }
  if (!aligned(vecs, 16) || !aligned(centroids, 16)) return fail(SENSE_ERR_INVALID_ARG, "vecs and centroids must be 16-byte aligned");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  auto* ix = new sense_ivf{};
  ix->n = n;
  ix->v = v;
  ix->nlist = nlist;
  ix->pq_m = codebooks ? pq_m : 0;
  ix->dsub = codebooks ? v / pq_m : 0;
  ix->device = current_device();
  const int nb = (int)((n + kIdBlock - 1) / kIdBlock);
  int32_t* cell = nullptr;
  int32_t* pos = nullptr;
  unsigned* hist = nullptr;
  unsigned* base = nullptr;
  int64_t* dmax = nullptr;
  auto cleanup = [&](sense_status st) {
    cudaFree(cell);
    cudaFree(pos);
    cudaFree(hist);
    cudaFree(base);
    cudaFree(dmax);
    if (st != SENSE_OK) free_ivf(ix);
    return st;
  };
  auto alloc = [&](void** p, size_t bytes) {
    return cudaMalloc(p, bytes) == cudaSuccess;
  };
  bool ok = alloc((void**)&ix->centroids, (size_t)nlist * v * 4) &&
            alloc((void**)&ix->offsets, (size_t)(nlist + 1) * 8) &&
            alloc((void**)&ix->ids, (size_t)n * 4) && alloc((void**)&cell, (size_t)n * 4) &&
            alloc((void**)&pos, (size_t)n * 4) && alloc((void**)&hist, (size_t)nb * nlist * 4) &&
            alloc((void**)&base, (size_t)nb * nlist * 4) && alloc((void**)&dmax, 8);
  if (ok && codebooks)
    ok = alloc((void**)&ix->codebooks, (size_t)pq_m * 256 * ix->dsub * 4) &&
         alloc((void**)&ix->codes, (size_t)n * pq_m);
  if (ok && !codebooks) ok = alloc((void**)&ix->vectors, (size_t)n * v * 4);
  if (!ok) {
    cudaGetLastError();
    return cleanup(fail(SENSE_ERR_OOM, "index allocation failed"));
  }
  sense_status st = cuda_check(cudaMemcpyAsync(ix->centroids, centroids, (size_t)nlist * v * 4,
                                               cudaMemcpyDeviceToDevice, s), "copy centroids");
  if (st == SENSE_OK && codebooks)
    st = cuda_check(cudaMemcpyAsync(ix->codebooks, codebooks, (size_t)pq_m * 256 * ix->dsub * 4,
                                    cudaMemcpyDeviceToDevice, s), "copy codebooks");
  if (st != SENSE_OK) return cleanup(st);
  {
    LaunchScope ls(K_IVF_BUILD, s);
    st = launch_assign_mode<ARGMAX_IP>(vecs, n, v, v, ix->centroids, nlist, cell, nullptr, s);
    if (st != SENSE_OK) return cleanup(st);
    const size_t hsm = (size_t)nlist * 4;
    if (hsm > 48 * 1024) {
      st = cuda_check(func_smem(reinterpret_cast<const void*>(cell_hist_kernel), (int)hsm), "smem attribute");
      if (st != SENSE_OK) return cleanup(st);
    }
    cell_hist_kernel<<<nb, 256, hsm, s>>>(cell, n, nlist, hist);
    cell_totals_kernel<<<(nlist + 127) / 128, 128, 0, s>>>(hist, nb, nlist, base, ix->offsets);
    cell_offsets_kernel<<<1, 1024, 0, s>>>(ix->offsets, nlist, dmax);
    const size_t psm = (size_t)nlist * 8;
    if (psm > 48 * 1024) {
      st = cuda_check(func_smem(reinterpret_cast<const void*>(cell_place_kernel), (int)psm), "smem attribute");
      if (st != SENSE_OK) return cleanup(st);
    }
    cell_place_kernel<<<nb, 32, psm, s>>>(cell, n, nlist, ix->offsets, base, pos, ix->ids);
    if (codebooks) {
      const size_t csm = (size_t)pq_m * 256 * ix->dsub * 4;
      if (csm > 48 * 1024) {
        st = cuda_check(func_smem(reinterpret_cast<const void*>(pq_encode_kernel), (int)csm), "smem attribute");
        if (st != SENSE_OK) return cleanup(st);
      }
      pq_encode_kernel<<<(unsigned)((n + 31) / 32), 256, csm, s>>>(vecs, n, v, ix->centroids, cell,
                                                                  ix->codebooks, pq_m, ix->dsub, pos,
                                                                  ix->codes);
    } else {
      scatter_vectors_kernel<<<(unsigned)((n * 32 + 255) / 256), 256, 0, s>>>(vecs, n, v, pos,
                                                                            ix->vectors);
    }
    st = cuda_check(cudaGetLastError(), "launch ivf build");
    if (st != SENSE_OK) return cleanup(st);
  }
  st = cuda_check(cudaMemcpyAsync(&ix->max_list, dmax, 8, cudaMemcpyDeviceToHost, s), "read max list");
  if (st == SENSE_OK) st = cuda_check(cudaStreamSynchronize(s), "ivf build");
  if (st != SENSE_OK) return cleanup(st);
  *out = ix;
  return cleanup(SENSE_OK);
}

sense_status sense_ivf_destroy(sense_ivf* ix) {
  free_ivf(ix);
  return SENSE_OK;
}

sense_status sense_ivf_arrays(const sense_ivf* ix, int64_t* out_info, const int64_t** out_offsets,
                              const int32_t** out_ids, const void** out_payload) {
  if (!ix) return fail(SENSE_ERR_INVALID_ARG, "ix is NULL");
  if (out_info) {
    out_info[0] = ix->n;
    out_info[1] = ix->v;
    out_info[2] = ix->nlist;
    out_info[3] = ix->pq_m;
    out_info[4] = ix->max_list;
  }
  if (out_offsets) *out_offsets = ix->offsets;
  if (out_ids) *out_ids = ix->ids;
  if (out_payload) *out_payload = ix->pq_m ? (const void*)ix->codes : (const void*)ix->vectors;
  return SENSE_OK;
}

size_t sense_ivf_search_workspace_bytes(const sense_ivf* ix, int32_t q, int32_t k, int32_t nprobe) {
  if (!ix || q < 1 || k < 1 || nprobe < 1) return 0;
  return search_plan(ix, q, nprobe).total;
}

}  // extern "C"

namespace {
// Validation, coarse scores, probe selection, PQ tables and the list scan of
// a search: each query's scanned candidates are left in the workspace's
// pool (`*pool`, `*counts`, `*pool_cap` keys per query).
sense_status ivf_scan_pool(const sense_ivf* ix, const float* queries, int32_t q, int32_t k,
                           int32_t nprobe, int32_t* out_probes, void* workspace,
                           size_t workspace_bytes, cudaStream_t s, uint64_t** pool_out,
                           uint32_t** counts_out, int64_t* pool_cap_out, uint32_t** status_out,
                           bool coarse_done = false) {
  if (!ix) return fail(SENSE_ERR_INVALID_ARG, "ix is NULL");
  if (!queries || !workspace)
    return fail(SENSE_ERR_INVALID_ARG, "queries, outputs and workspace must be non-NULL");
  if (q < 1 || q > 65535) return fail(SENSE_ERR_INVALID_ARG, "q=%d outside [1, 65535]", q);
  if (k < 1 || k > SENSE_MAX_K) return fail(SENSE_ERR_INVALID_ARG, "k=%d outside [1, %d]", k, SENSE_MAX_K);
  if (nprobe < 1 || nprobe > ix->nlist || nprobe > SENSE_MAX_K)
    return fail(SENSE_ERR_INVALID_ARG, "nprobe=%d outside [1, min(nlist=%d, %d)]", nprobe, ix->nlist,
                SENSE_MAX_K);
  if (!aligned(queries, 16)) return fail(SENSE_ERR_INVALID_ARG, "queries must be 16-byte aligned");
  if (!aligned(workspace, 256)) return fail(SENSE_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  const SearchPlan p = search_plan(ix, q, nprobe);
  if (workspace_bytes < p.total)
    return fail(SENSE_ERR_INVALID_ARG, "workspace of %zu bytes < %zu", workspace_bytes, p.total);
  if (current_device() != ix->device) return fail(SENSE_ERR_INVALID_ARG, "index lives on device %d", ix->device);
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  char* ws = static_cast<char*>(workspace);
  auto* coarse = reinterpret_cast<uint64_t*>(ws + p.off_coarse);
  auto* pscore = reinterpret_cast<float*>(ws + p.off_pscore);
  auto* pcell = out_probes ? out_probes : reinterpret_cast<int32_t*>(ws + p.off_pcell);
  auto* counts = reinterpret_cast<uint32_t*>(ws + p.off_counts);
  auto* pool = reinterpret_cast<uint64_t*>(ws + p.off_pool);
  auto* lut = reinterpret_cast<float*>(ws + p.off_lut);
  sense_status st = SENSE_OK;
  if (coarse_done) {  // coarse keys, tables and empty pools written by project_coarse_kernel
  } else {
    st = cuda_check(cudaMemsetAsync(counts, 0, (size_t)q * 4, s), "clear counts");
    if (st != SENSE_OK) return st;
  }
  if (coarse_done) {
  } else if (ix->pq_m > 0) {  // coarse keys and lookup tables in one launch
    LaunchScope ls(K_IVF_COARSE, s);
    st = launch_coarse_lut(ix, queries, q, coarse, lut, s);
    if (st != SENSE_OK) return st;
  } else {
    LaunchScope ls(K_IVF_COARSE, s);
    // cells as rows, queries staged: pool row qi holds key(<q_qi, c>, c)
    st = launch_assign_mode<ALL_IP>(ix->centroids, ix->nlist, ix->v, ix->v, queries, q, nullptr,
                                    coarse, s);
    if (st != SENSE_OK) return st;
  }
  if (!coarse_done) {  // else the best cells were selected with the coarse keys
    st = launch_merge(coarse, nullptr, ix->nlist, q, nprobe, pscore, pcell, status, s);
    if (st != SENSE_OK) return st;
  }
  {
    const size_t smem = scan_smem_bytes(ix);
    st = cuda_check(func_smem(reinterpret_cast<const void*>(ivf_scan_kernel), (int)smem), "smem attribute");
    if (st != SENSE_OK) return st;
    LaunchScope ls(K_IVF_SCAN, s);
    st = cuda_check(launch_pdl(ivf_scan_kernel, dim3(nprobe, q, scan_parts(ix, q, nprobe)),
                               dim3(kScanThreads), smem, s, *ix,
                               queries, (const float*)lut, nprobe, (const float*)pscore,
                               (const int32_t*)pcell, pool, counts, p.pool_cap, status),
                    "launch ivf scan");
    if (st != SENSE_OK) return st;
  }
  *pool_out = pool;
  *counts_out = counts;
  *pool_cap_out = p.pool_cap;
  *status_out = status;
  return SENSE_OK;
}
}  // namespace

extern "C" {

sense_status sense_ivf_search(const sense_ivf* ix, const float* queries, int32_t q, int32_t k,
                              int32_t nprobe, float* out_scores, int32_t* out_idx,
                              int32_t* out_probes, void* workspace, size_t workspace_bytes,
                              sense_stream_t stream) {
  if (!ix) return fail(SENSE_ERR_INVALID_ARG, "ix is NULL");
  if (!queries || !out_scores || !out_idx || !workspace)
    return fail(SENSE_ERR_INVALID_ARG, "queries, outputs and workspace must be non-NULL");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  uint64_t* pool = nullptr;
  uint32_t* counts = nullptr;
  uint32_t* status = nullptr;
  int64_t pool_cap = 0;
  sense_status st = ivf_scan_pool(ix, queries, q, k, nprobe, out_probes, workspace,
                                  workspace_bytes, s, &pool, &counts, &pool_cap, &status);
  if (st != SENSE_OK) return st;
  return launch_merge_short(pool, counts, pool_cap, q, k, out_scores, out_idx, status, s);
}

size_t sense_ann_draft_workspace_bytes(const sense_ivf* ix, int32_t q, int32_t k, int32_t nprobe,
                                       int32_t rerank) {
  if (!ix || q < 1 || k < 1 || nprobe < 1 || rerank < 0) return 0;
  const int kk = std::max(k, rerank);
  size_t b = align256((size_t)q * ix->v * 4);
  if (rerank > 0) b += 2 * align256((size_t)q * kk * 4);
  return b + sense_ivf_search_workspace_bytes(ix, q, kk, nprobe);
}

}  // extern "C"

namespace {
// sense_ann_draft (draft = true) and sense_ann_search (draft = false: the
// step ends with the top k, the span and tree outputs are unused).
sense_status ann_step(bool draft, const sense_ivf* ix, const sense_datastore* ds,
                      const uint16_t* queries, int32_t q, const float* basis, const float* mean,
                      int32_t k, int32_t nprobe, int32_t rerank, int32_t node_cap,
                      uint32_t flags, void* workspace, size_t workspace_bytes, float* out_scores,
                      int32_t* out_idx, int32_t* out_spans, int32_t* out_num_nodes,
                      int32_t* out_tokens, int32_t* out_parent, int32_t* out_depth,
                      int32_t* out_gamma, uint32_t* out_mask_bits, sense_stream_t stream) {
  if (!ix || !ds) return fail(SENSE_ERR_INVALID_ARG, "index and datastore must be non-NULL");
  if (!queries || !basis || !workspace || !out_scores || !out_idx ||
      (draft && (!out_spans || !out_num_nodes || !out_tokens || !out_parent || !out_depth ||
                 !out_gamma)))
    return fail(SENSE_ERR_INVALID_ARG, "queries, basis, workspace and outputs must be non-NULL");
  if (ds->device != current_device() || ix->device != current_device())
    return fail(SENSE_ERR_INVALID_ARG, "index and datastore must live on the current device");
  if (q < 1 || q > 65535) return fail(SENSE_ERR_INVALID_ARG, "q=%d outside [1, 65535]", q);
  if (k < 1 || k > SENSE_MAX_K) return fail(SENSE_ERR_INVALID_ARG, "k=%d outside [1, %d]", k, SENSE_MAX_K);
  if (rerank < 0 || (rerank > 0 && (rerank < k || rerank > SENSE_MAX_RESCORE)))
    return fail(SENSE_ERR_INVALID_ARG, "rerank=%d must be 0 or in [k=%d, %d]", rerank, k,
                SENSE_MAX_RESCORE);
  const int m = ds->m;
  if (draft && (int64_t)k * m > SENSE_MAX_TREE_TOKENS)
    return fail(SENSE_ERR_INVALID_ARG, "k*m=%d exceeds %d", k * m, SENSE_MAX_TREE_TOKENS);
  if (node_cap < 0) return fail(SENSE_ERR_INVALID_ARG, "node_cap=%d must be >= 0", node_cap);
  if (flags & ~SENSE_TREE_MASK_BITS) return fail(SENSE_ERR_INVALID_ARG, "unknown tree flags 0x%x", flags);
  const bool bits = (flags & SENSE_TREE_MASK_BITS) != 0;
  if (draft && bits && !out_mask_bits)
    return fail(SENSE_ERR_INVALID_ARG, "SENSE_TREE_MASK_BITS needs out_mask_bits");
  if (!aligned(workspace, 256) || (draft && !aligned(out_spans, 16)))
    return fail(SENSE_ERR_INVALID_ARG, "workspace must be 256-byte and out_spans 16-byte aligned");
  const size_t need = sense_ann_draft_workspace_bytes(ix, q, k, nprobe, rerank);
  if (workspace_bytes < need)
    return fail(SENSE_ERR_INVALID_ARG, "workspace of %zu bytes < %zu", workspace_bytes, need);
  const int kk = std::max(k, rerank);
  char* ws = static_cast<char*>(workspace);
  float* qproj = reinterpret_cast<float*>(ws);
  ws += align256((size_t)q * ix->v * 4);
  float* cand_s = nullptr;
  int32_t* cand_i = nullptr;
  if (rerank > 0) {
    cand_s = reinterpret_cast<float*>(ws);
    ws += align256((size_t)q * kk * 4);
    cand_i = reinterpret_cast<int32_t*>(ws);
    ws += align256((size_t)q * kk * 4);
  }
  const size_t ivf_bytes = sense_ivf_search_workspace_bytes(ix, q, kk, nprobe);
  const int cap = node_cap > 0 ? node_cap : k * m;
  const bool fused = draft && draft_fused_fits(k, m);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (!aligned(queries, 16) || !aligned(basis, 16) || (mean && !aligned(mean, 16)))
    return fail(SENSE_ERR_INVALID_ARG, "queries, basis and mean must be 16-byte aligned");
  // query construction (Alg. 2: k = L2Norm(PCA(h))) with the coarse keys and
  // lookup tables in the same launch when it fits, search, optional exact
  // re-scoring (Eq. 8), gather and trie
  const SearchPlan plan = search_plan(ix, q, nprobe);
  bool coarse_done = false;
  sense_status st = launch_project_coarse(
      queries, q, ds->d, basis, mean, qproj, ix, reinterpret_cast<float*>(ws + plan.off_lut),
      reinterpret_cast<uint32_t*>(ws + plan.off_counts),
      nprobe, reinterpret_cast<float*>(ws + plan.off_pscore),
      reinterpret_cast<int32_t*>(ws + plan.off_pcell), s, &coarse_done);
  if (st != SENSE_OK) return st;
  if (!coarse_done) {
    st = sense_project(queries, q, ds->d, basis, ix->v, mean, SENSE_PROJECT_NORMALIZE, qproj,
                       stream);
    if (st != SENSE_OK) return st;
  }
  uint64_t* pool = nullptr;
  uint32_t* counts = nullptr;
  uint32_t* status = nullptr;
  int64_t pool_cap = 0;
  st = ivf_scan_pool(ix, qproj, q, rerank > 0 ? rerank : k, nprobe, nullptr, ws, ivf_bytes, s,
                     &pool, &counts, &pool_cap, &status, coarse_done);
  if (st != SENSE_OK) return st;
  if (rerank == 0 && fused)  // pool merge, gather and trie in one kernel per query
    return launch_pool_draft(pool, counts, pool_cap, q, k, out_scores, out_idx, ds->spans, ds->n,
                             m, out_spans, cap, bits ? 1 : 0, out_num_nodes, out_tokens,
                             out_parent, out_depth, out_gamma, out_mask_bits, status, s);
  if (rerank > 0) {
    st = launch_merge_short(pool, counts, pool_cap, q, rerank, cand_s, cand_i, status, s);
    if (st != SENSE_OK) return st;
    st = sense_rescore_topk(ds, queries, q, cand_i, rerank, k, out_scores, out_idx, stream);
  } else {
    st = launch_merge_short(pool, counts, pool_cap, q, k, out_scores, out_idx, status, s);
  }
  if (st != SENSE_OK || !draft) return st;
  if (fused)  // gather and trie in one kernel per query
    return launch_span_draft(out_idx, q, k, ds->spans, ds->n, m, out_spans, cap, bits ? 1 : 0,
                             out_num_nodes, out_tokens, out_parent, out_depth, out_gamma,
                             out_mask_bits, status, s);
  st = launch_gather(ds->spans, ds->n, m, out_idx, q, k, nullptr, k, 0, out_spans, status, stream);
  if (st != SENSE_OK) return st;
  return launch_tree(out_spans, q, k, m, cap, bits ? 1 : 0, out_num_nodes, out_tokens, out_parent,
                     out_depth, out_gamma, out_mask_bits, status, stream);
}
}  // namespace

extern "C" {

sense_status sense_ann_draft(const sense_ivf* ix, const sense_datastore* ds, const uint16_t* queries,
                             int32_t q, const float* basis, const float* mean, int32_t k,
                             int32_t nprobe, int32_t rerank, int32_t node_cap, uint32_t flags,
                             void* workspace, size_t workspace_bytes, float* out_scores,
                             int32_t* out_idx, int32_t* out_spans, int32_t* out_num_nodes,
                             int32_t* out_tokens, int32_t* out_parent, int32_t* out_depth,
                             int32_t* out_gamma, uint32_t* out_mask_bits, sense_stream_t stream) {
  return ann_step(true, ix, ds, queries, q, basis, mean, k, nprobe, rerank, node_cap, flags,
                  workspace, workspace_bytes, out_scores, out_idx, out_spans, out_num_nodes,
                  out_tokens, out_parent, out_depth, out_gamma, out_mask_bits, stream);
}

sense_status sense_ann_search(const sense_ivf* ix, const sense_datastore* ds,
                              const uint16_t* queries, int32_t q, const float* basis,
                              const float* mean, int32_t k, int32_t nprobe, int32_t rerank,
                              void* workspace, size_t workspace_bytes, float* out_scores,
                              int32_t* out_idx, sense_stream_t stream) {
  return ann_step(false, ix, ds, queries, q, basis, mean, k, nprobe, rerank, 0, 0, workspace,
                  workspace_bytes, out_scores, out_idx, nullptr, nullptr, nullptr, nullptr,
                  nullptr, nullptr, nullptr, stream);
}

}  // extern "C"
