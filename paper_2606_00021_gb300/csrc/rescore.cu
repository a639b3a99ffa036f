// Exact re-scoring of an approximate shortlist (Sec. 3.2.2 Eq. 8).
//
// The approximate search returns N' candidates D_ret scored in the projected
// space; Eq. 8 ranks them by sim(h, k_i), the similarity of the full hidden
// state to each candidate's key, and keeps the top N.  This kernel computes
// that similarity exactly over the stored bf16 keys (fp32 accumulation, the
// same arithmetic as the exact scan) and selects the top k of the shortlist
// in the order (score desc, key index asc).
//
// A query's shortlist is a gather of N' scattered key rows (4 MB for 512
// rows of 4096 dims), paced by how many bytes are in flight, so one query is
// spread over a cluster of C CTAs (16 where the device schedules clusters
// that wide, else 8) and each CTA keeps 24 rows in flight:
//  1. CTA r takes the candidates [r * per, (r + 1) * per), per =
//     ceil(N' / C); warp w of the CTA takes every 8th of them.  Lane 0 of
//     the warp streams its candidates' rows through a 3-stage ring of
//     8 KB shared-memory stages with 1-D bulk copies (cp.async.bulk,
//     completion on an mbarrier, every wait bounded); a row longer than a
//     stage takes several stages.  Lane l holds its query chunks in
//     registers and accumulates chunks l, l + 64, ... and l + 32, l + 96,
//     ... of 8 bf16 in two fp32 sums (each in increasing order), added
//     before a butterfly sums the lanes.
//  2. Warp 0 sorts the CTA's candidate keys (score code, inverted index)
//     in registers with a bitonic network.
//  3. Each CTA stores its sorted list into every CTA of the cluster through
//     distributed shared memory; after one cluster barrier the rank of each
//     of its own keys is its position in its list plus, per other list, a
//     binary-search count of the keys ahead of it; keys ranked below k are
//     written in place.
// Slots with index -1 (fewer candidates than N') are empty; an index
// outside [0, n) is empty too and sets SENSE_DEVST_BAD_INDEX.  A copy that
// never lands sets SENSE_DEVST_TIMEOUT and drops the warp's later
// candidates.
#include <cooperative_groups.h>
#include <cuda_bf16.h>

#include <cstdlib>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "launch.h"
#include "tc_ptx.cuh"

namespace sense {
namespace {

namespace cg = cooperative_groups;

constexpr int kRsThreads = 256;                  // 8 warps
constexpr int kRsWarps = kRsThreads / 32;
constexpr int kRsStage = 8192;                   // bytes per ring stage
constexpr int kRsChunks = kRsStage / 16;         // 16-byte chunks per stage
constexpr int kRsLaneChunks = kRsChunks / 32;
constexpr int kRsDepth = 3;                      // stages per warp ring
constexpr int kRsListMax = 128;                  // candidates per CTA (N' / C)
constexpr int kRsWarpMax = kRsListMax / kRsWarps;
constexpr long long kRsWaitCycles = 4000000000LL;

constexpr size_t kRsRingBytes = (size_t)kRsWarps * kRsDepth * kRsStage;
constexpr size_t kRsSmemBytes = kRsRingBytes + sizeof(uint64_t) * kRsWarps * kRsDepth +
                                sizeof(uint64_t) * (kRsListMax + SENSE_MAX_RESCORE) +
                                sizeof(int32_t) * kRsWarps * kRsWarpMax;

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

// Bounded wait on an mbarrier phase; false after ~2 s.
__device__ __forceinline__ bool rs_wait(uint32_t bar, uint32_t parity) {
  if (ptx::mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!ptx::mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > kRsWaitCycles) return false;
  }
  return true;
}

// Bitonic sort, descending, of the 32 * KPL keys a warp holds (element
// lane + 32 r in x[r]).
template <int KPL>
__device__ __forceinline__ void warp_sort_desc(uint64_t (&x)[KPL]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int size = 2; size <= 32 * KPL; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      if (stride >= 32) {  // partner in register r ^ (stride / 32) of the same lane
        const int rs = stride >> 5;
#pragma unroll
        for (int r = 0; r < KPL; ++r) {
          if (r & rs) continue;
          const bool desc = (((lane + 32 * r) & size) == 0);
          const uint64_t a = x[r], b = x[r | rs];
          const uint64_t hi = a > b ? a : b, lo = a > b ? b : a;
          x[r] = desc ? hi : lo;
          x[r | rs] = desc ? lo : hi;
        }
      } else {
        const bool lower = (lane & stride) == 0;
#pragma unroll
        for (int r = 0; r < KPL; ++r) {
          const uint64_t p = __shfl_xor_sync(0xffffffffu, x[r], stride);
          const bool desc = (((lane + 32 * r) & size) == 0);
          const bool keep_max = (lower == desc);
          x[r] = keep_max ? (x[r] > p ? x[r] : p) : (x[r] < p ? x[r] : p);
        }
      }
    }
  }
}

// Split cluster barrier: every thread arrives (relaxed, nothing to
// publish) and later waits; between the two the CTA runs its own work.
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
}

template <int KPL>
__global__ void __launch_bounds__(kRsThreads, 1)
rescore_kernel(const uint16_t* __restrict__ keys, int64_t n, int d,
               const uint16_t* __restrict__ queries, const int32_t* __restrict__ cand,
               int n_cand, int k, float* __restrict__ out_scores,
               int32_t* __restrict__ out_idx, uint32_t* status) {
  constexpr int L = 32 * KPL;  // sorted-list length per CTA (padded with empty keys)
  pdl_wait();  // inputs written by the kernels before this one
  pdl_launch_dependents();
  cg::cluster_group cl = cg::this_cluster();
  extern __shared__ __align__(128) unsigned char rs_smem[];
  uint4* ring = reinterpret_cast<uint4*>(rs_smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(rs_smem + kRsRingBytes);
  uint64_t* s_list = bars + kRsWarps * kRsDepth;  // this CTA's keys, then sorted
  uint64_t* s_all = s_list + kRsListMax;          // the cluster's sorted lists
  int32_t* s_cidx = reinterpret_cast<int32_t*>(s_all + SENSE_MAX_RESCORE);
  __shared__ unsigned s_total;

  const int C = (int)cl.num_blocks();
  const int r = (int)cl.block_rank();
  const int qi = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int per = (n_cand + C - 1) / C;  // <= L (chosen by the host)
  const int lo = min(r * per, n_cand);
  const int cnt = min(per, n_cand - lo);
  if (threadIdx.x == 0) {
    for (int b = 0; b < kRsWarps * kRsDepth; ++b) ptx::mbar_init(ptx::smem_u32(bars + b), 1);
    ptx::fence_barrier_init();
    s_total = 0u;
  }
  for (int i = threadIdx.x; i < kRsListMax; i += blockDim.x) s_list[i] = 0ull;
  cluster_arrive_relaxed();  // waited for before the first remote store
  __syncthreads();

  // 1. score the warp's candidates
  const int nwc = cnt > warp ? (cnt - warp + kRsWarps - 1) / kRsWarps : 0;  // <= kRsWarpMax
  int32_t my = -1;  // lane j: key index of the warp's j-th candidate, -1 if empty
  if (lane < nwc) {
    const int32_t idx = cand[(int64_t)qi * n_cand + lo + warp + kRsWarps * lane];
    if ((int64_t)idx >= n) raise_status(status, SENSE_DEVST_BAD_INDEX);
    else my = idx;  // -1 (or any negative) stays empty
  }
  if (my < -1) my = -1;
  const unsigned valid = __ballot_sync(0xffffffffu, my >= 0);
  const int nv = __popc(valid);
  int32_t* wcidx = s_cidx + warp * kRsWarpMax;
  if (my >= 0) wcidx[__popc(valid & ((1u << lane) - 1u))] = my;
  __syncwarp();
  const int rowb = 2 * d;
  const int spr = (rowb + kRsStage - 1) / kRsStage;  // stages per row
  const int total = nv * spr;
  uint64_t* wbars = bars + warp * kRsDepth;
  uint4* wring = ring + (size_t)warp * kRsDepth * kRsChunks;
  const uint64_t pol = ptx::policy_evict_first();
  auto issue = [&](int g) {  // lane 0: stage g of the warp's stream
    const int v = g / spr, piece = g - v * spr;
    const int off = piece * kRsStage;
    const int bytes = min(kRsStage, rowb - off);
    const uint32_t bar = ptx::smem_u32(wbars + g % kRsDepth);
    ptx::mbar_arrive_expect_tx(bar, (uint32_t)bytes);
    ptx::bulk_load(ptx::smem_u32(wring + (size_t)(g % kRsDepth) * kRsChunks),
                   reinterpret_cast<const char*>(keys + (int64_t)wcidx[v] * d) + off,
                   (uint32_t)bytes, bar, pol);
  };
  if (lane == 0)
    for (int g = 0; g < min(kRsDepth, total); ++g) issue(g);
  // the query chunks a lane multiplies: loaded once when a row is one
  // stage, else with each stage, always all before the products
  const uint4* qrow4 = reinterpret_cast<const uint4*>(queries + (int64_t)qi * d);
  uint4 qv[kRsLaneChunks];
  auto load_q = [&](int piece, int nc) {
#pragma unroll
    for (int u = 0; u < kRsLaneChunks; ++u) {
      const int j = lane + 32 * u;
      qv[u] = j < nc ? __ldg(qrow4 + piece * kRsChunks + j) : make_uint4(0u, 0u, 0u, 0u);
    }
  };
  if (spr == 1) load_q(0, rowb >> 4);
  float acc0 = 0.0f, acc1 = 0.0f;  // even and odd chunks of the lane
  for (int g = 0; g < total; ++g) {
    const bool got = rs_wait(ptx::smem_u32(wbars + g % kRsDepth), (uint32_t)(g / kRsDepth) & 1u);
    if (!__all_sync(0xffffffffu, got)) {
      if (lane == 0) {  // let the copies in flight land before giving up
        for (int j = g; j < min(total, g + kRsDepth); ++j)
          rs_wait(ptx::smem_u32(wbars + j % kRsDepth), (uint32_t)(j / kRsDepth) & 1u);
        raise_status(status, SENSE_DEVST_TIMEOUT);
      }
      break;
    }
    const int v = g / spr, piece = g - v * spr;
    const int nc = min(kRsChunks, (rowb - piece * kRsStage) >> 4);
    const uint4* st = wring + (size_t)(g % kRsDepth) * kRsChunks;
    if (spr > 1) load_q(piece, nc);
#pragma unroll
    for (int u = 0; u < kRsLaneChunks; u += 2) {
      const int j = lane + 32 * u;
      if (j < nc) acc0 = dot8(st[j], qv[u], acc0);
      if (j + 32 < nc) acc1 = dot8(st[j + 32], qv[u + 1], acc1);
    }
    __syncwarp();  // every lane has read the stage: its buffer takes stage g + depth
    if (lane == 0 && g + kRsDepth < total) {
      ptx::fence_proxy_async_smem();
      issue(g + kRsDepth);
    }
    if (piece == spr - 1) {
      float acc = acc0 + acc1;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
      if (lane == 0) s_list[warp + kRsWarps * v] = cand_key(acc, (uint32_t)wcidx[v]);
      acc0 = 0.0f;
      acc1 = 0.0f;
    }
  }
  __syncthreads();

  // 2. sort this CTA's keys and store the sorted list into every CTA's
  //    copy of the cluster's lists (row r of s_all)
  if (warp == 0) {
    uint64_t x[KPL];
#pragma unroll
    for (int i = 0; i < KPL; ++i) x[i] = s_list[lane + 32 * i];
    warp_sort_desc<KPL>(x);
#pragma unroll
    for (int i = 0; i < KPL; ++i) s_list[lane + 32 * i] = x[i];
  }
  cluster_wait();  // every CTA of the cluster is running
  __syncthreads();
  for (int t = threadIdx.x; t < C * L; t += blockDim.x)
    *cl.map_shared_rank(s_all + r * L + (t % L), (unsigned)(t / L)) = s_list[t % L];
  cl.sync();  // the lists are complete; no remote access after this

  // 3. rank this CTA's keys among the cluster's lists
  for (int t = threadIdx.x; t < C * L; t += blockDim.x) {  // C * L: a multiple of blockDim
    const unsigned nz = __ballot_sync(0xffffffffu, s_all[t] != 0ull);
    if (lane == 0) atomicAdd(&s_total, (unsigned)__popc(nz));
  }
  float* os = out_scores + (int64_t)qi * k;
  int32_t* oi = out_idx + (int64_t)qi * k;
  for (int t0 = 0; t0 < L * C; t0 += blockDim.x) {  // L * C is a multiple of blockDim
    const int t = t0 + threadIdx.x;
    const int p = t / C, b = t - p * C;
    const uint64_t x = s_all[r * L + p];
    int ahead = 0;  // keys of list b ahead of x: larger, or equal in an earlier list
    if (x != 0ull && b != r) {
      const uint64_t* lb = s_all + b * L;
      int a = 0, e = L;
      while (a < e) {
        const int mid = (a + e) >> 1;
        const uint64_t y = lb[mid];
        if (y > x || (y == x && b < r)) a = mid + 1;
        else e = mid;
      }
      ahead = a;
    }
    for (int off = C >> 1; off > 0; off >>= 1) ahead += __shfl_xor_sync(0xffffffffu, ahead, off);
    if (b == 0 && x != 0ull) {
      const int rank = p + ahead;
      if (rank < k) {
        os[rank] = code_score((uint32_t)(x >> 32));
        oi[rank] = (int32_t)cand_index(x);
      }
    }
  }
  __syncthreads();  // s_total complete
  if (r == 0) {  // fewer valid candidates than k: -inf, -1
    const float NEG = -__int_as_float(0x7f800000);
    for (int t = (int)s_total + threadIdx.x; t < k; t += blockDim.x) {
      os[t] = NEG;
      oi[t] = -1;
    }
  }
}

using RescoreFn = void (*)(const uint16_t*, int64_t, int, const uint16_t*, const int32_t*, int, int,
                           float*, int32_t*, uint32_t*);
constexpr int kMaxDev = 64;

// Cluster width per device: 16 when a cluster of 16 of these CTAs can be
// resident, else 8 (the portable size); SENSE_RESCORE_CLUSTER=8 in the
// environment selects 8 regardless.  Attributes are set once.
sense_status rescore_setup(int dev, int* width) {
  static std::mutex mu;
  static int widths[kMaxDev] = {0};
  std::lock_guard<std::mutex> lk(mu);
  if (dev >= 0 && dev < kMaxDev && widths[dev] > 0) {
    *width = widths[dev];
    return SENSE_OK;
  }
  const RescoreFn fns[3] = {rescore_kernel<1>, rescore_kernel<2>, rescore_kernel<4>};
  for (RescoreFn f : fns) {
    sense_status st = cuda_check(cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      (int)kRsSmemBytes),
                                 "rescore shared-memory attribute");
    if (st != SENSE_OK) return st;
    st = cuda_check(cudaFuncSetAttribute(f, cudaFuncAttributeNonPortableClusterSizeAllowed, 1),
                    "rescore cluster attribute");
    if (st != SENSE_OK) return st;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(16, 1);
  cfg.blockDim = dim3(kRsThreads);
  cfg.dynamicSmemBytes = kRsSmemBytes;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 16;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int nclusters = 0;
  int w = 8;
  const char* force = std::getenv("SENSE_RESCORE_CLUSTER");
  const bool portable = force && std::strcmp(force, "8") == 0;
  if (!portable) {
    if (cudaOccupancyMaxActiveClusters(&nclusters, fns[2], &cfg) == cudaSuccess && nclusters >= 1)
      w = 16;
    else
      (void)cudaGetLastError();  // the query's failure only means "not 16"
  }
  if (dev >= 0 && dev < kMaxDev) widths[dev] = w;
  *width = w;
  return SENSE_OK;
}

}  // namespace

sense_status launch_rescore(const uint16_t* keys, int64_t n, int d, const uint16_t* queries, int q,
                            const int32_t* cand, int n_cand, int k, float* out_scores,
                            int32_t* out_idx, uint32_t* status, cudaStream_t s) {
  int C = 8, dev = 0;
  sense_status st = cuda_check(cudaGetDevice(&dev), "cudaGetDevice");
  if (st != SENSE_OK) return st;
  st = rescore_setup(dev, &C);
  if (st != SENSE_OK) return st;
  const int per = (n_cand + C - 1) / C;  // <= SENSE_MAX_RESCORE / 8 = kRsListMax
  const RescoreFn fn = per <= 32 ? rescore_kernel<1> : per <= 64 ? rescore_kernel<2> : rescore_kernel<4>;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)C, (unsigned)q);
  cfg.blockDim = dim3(kRsThreads);
  cfg.dynamicSmemBytes = kRsSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  LaunchScope ls(K_RESCORE, s);
  return cuda_check(cudaLaunchKernelEx(&cfg, fn, keys, n, d, queries, cand, n_cand, k, out_scores,
                                       out_idx, status),
                    "launch rescore");
}

}  // namespace sense
