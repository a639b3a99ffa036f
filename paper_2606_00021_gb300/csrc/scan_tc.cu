// Key scoring for batched queries (8 < q <= 128 per pass) on tcgen05 tensor
// cores, fused with the candidate filter of the top-k.
//
// Sec. 3.2.2 (Eq. 7, Eq. 8 sim) scores every key against every query of the
// batch: S = K Q^T, a real matrix product once q reaches 16.  It stays
// bound by the single read of the n x d x 2-byte key matrix (q flop per key
// byte, far below the bf16 tensor ridge), so the tensor cores are there to
// keep the arithmetic hidden under the stream:
//  - persistent grid, one CTA per SM; a work unit is 256 key rows (two
//    128-row tiles of the scan's tile set);
//  - warp 0 (one lane) streams, per 64-column slice of d, both 128 x 64 key
//    tiles and the padded nq x 64 query tile with 2-D TMA loads (128-byte
//    swizzle, keys marked evict-first in L2) into a multi-stage ring, two
//    consecutive slices per stage up to 32 queries;
//  - warp 1 (one lane) issues tcgen05.mma kind::f16 (M = 128 keys,
//    N = nq queries, K = 16) into fp32 TMEM accumulators: two tiles x two
//    buffers, so the epilogue of one unit overlaps the MMAs of the next;
//  - warps 2-5 read the accumulators with tcgen05.ld (one key row per
//    thread, 16 queries per load) and apply the same filter as the GEMV
//    scan: store every candidate key (sample tiles) or append the ones at or
//    above the query's threshold to its pool.
// Every mbarrier wait gives up after ~2 s of clock64 time: it sets
// SENSE_DEVST_TIMEOUT and an abort flag that releases the other roles; the
// producer then waits (bounded) for its copies in flight, the MMA thread for
// its MMAs, and the CTA frees its TMEM before returning.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "launch.h"
#include "tc_ptx.cuh"

namespace sense {
namespace {

constexpr int kThreads = 192;
constexpr int kBlockK = 64;                    // bf16 columns per stage (128 bytes)
constexpr int kTileBytes = 128 * kBlockK * 2;  // one 128 x 64 key tile
constexpr long long kWaitCycles = 4000000000LL;

struct TcArgs {
  int64_t n;
  int d;
  int qg;      // real queries in this group
  int nq;      // padded to a multiple of 16
  int64_t n_half;  // 128-row work tiles
  int64_t n_work;  // n_half * 128
  int kc;      // 64-column slices of d
  int cps;     // slices per ring stage
  int stages;
  uint32_t tmem_cols;
  const uint64_t* thresh;
  uint64_t* out;
  uint32_t* counts;
  int64_t pool_cap;
  uint32_t* status;
};

template <int MODE>
__device__ __forceinline__ int64_t key_tile(int64_t h) {
  if (MODE == SCAN_SAMPLE) return h * kSampleStride;
  if (MODE == SCAN_REST) return h + h / (kSampleStride - 1) + 1;
  return h;
}

struct Shared {
  uint32_t tmem_base;
  int abort;
};

// Bounded wait: false if the abort flag is raised or the wait times out.
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int* abort,
                                         uint32_t* status, long long limit = kWaitCycles) {
  if (ptx::mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (ptx::mbar_try_wait(bar, parity)) return true;
    if (*abort) return false;
    if (clock64() - t0 > limit) {
      *abort = 1;
      raise_status(status, SENSE_DEVST_TIMEOUT);
      return false;
    }
  }
}
// Bounded wait that ignores the abort flag (draining after an abort).
__device__ __forceinline__ void drain_bar(uint32_t bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!ptx::mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > kWaitCycles) return;
  }
}

template <int MODE>
__global__ void __launch_bounds__(kThreads, 1)
scan_tc_kernel(const __grid_constant__ CUtensorMap tm_keys,
               const __grid_constant__ CUtensorMap tm_q, const TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int S = a.stages;
  const int cps = a.cps;
  // a stage holds cps consecutive 64-column slices: slice c of tile t at
  // (2 c + t) kTileBytes, then the query slices (nq x 64 each)
  const uint32_t q_off = (uint32_t)(2 * cps * kTileBytes);
  const uint32_t stage_bytes = (uint32_t)cps * (2 * kTileBytes + a.nq * kBlockK * 2);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)S * stage_bytes);
  // bars: full[S], empty[S], acc_full[2], acc_empty[2], mma_done
  Shared* sh = reinterpret_cast<Shared*>(bars + 2 * S + 5);
  uint64_t* s_thr = reinterpret_cast<uint64_t*>(sh + 1);
  volatile int* abort = &sh->abort;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  auto bar = [&](int i) { return ptx::smem_u32(bars + i); };
  const int FULL = 0, EMPTY = S, ACC_FULL = 2 * S, ACC_EMPTY = 2 * S + 2, MMA_DONE = 2 * S + 4;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      ptx::mbar_init(bar(FULL + s), 1);
      ptx::mbar_init(bar(EMPTY + s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(bar(ACC_FULL + b), 1);
      ptx::mbar_init(bar(ACC_EMPTY + b), 4);
    }
    ptx::mbar_init(bar(MMA_DONE), 1);
    sh->abort = 0;
    ptx::fence_barrier_init();
    ptx::prefetch_tensormap(&tm_keys);
    ptx::prefetch_tensormap(&tm_q);
  }
  if (warp == 1) ptx::tmem_alloc(ptx::smem_u32(&sh->tmem_base), a.tmem_cols);
  for (int i = threadIdx.x; i < a.qg; i += blockDim.x) s_thr[i] = a.thresh ? a.thresh[i] : 0ull;
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = sh->tmem_base;
  const int64_t n_units = (a.n_half + 1) / 2;
  const int64_t dummy_tile = (a.n + 127) / 128 + 1;  // wholly out of range: zero-filled

  if (warp == 0 && lane == 0) {
    // ------------------------------------------------ TMA producer
    const uint64_t pol_keys = ptx::policy_evict_first();
    const uint64_t pol_q = ptx::policy_evict_last();
    int s = 0;
    uint32_t ph = 0;
    int64_t issued = 0;
    bool ok = true;
    for (int64_t u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
      const int64_t t0 = key_tile<MODE>(2 * u);
      const int64_t t1 = (2 * u + 1 < a.n_half) ? key_tile<MODE>(2 * u + 1) : dummy_tile;
      for (int kc = 0; kc < a.kc; kc += cps) {
        if (!wait_bar(bar(EMPTY + s), ph ^ 1u, abort, a.status)) {
          ok = false;
          break;
        }
        uint8_t* st = smem + (size_t)s * stage_bytes;
        // slices past d (the last stage when kc % cps != 0) are zero-filled
        // and still count their full box bytes
        ptx::mbar_arrive_expect_tx(bar(FULL + s), stage_bytes);
        for (int c = 0; c < cps; ++c) {
          const int col = (kc + c) * kBlockK;
          ptx::tma_load_2d(ptx::smem_u32(st + (2 * c) * kTileBytes), &tm_keys, bar(FULL + s), col,
                           (int32_t)(t0 * 128), pol_keys);
          ptx::tma_load_2d(ptx::smem_u32(st + (2 * c + 1) * kTileBytes), &tm_keys, bar(FULL + s),
                           col, (int32_t)(t1 * 128), pol_keys);
        }
        for (int c = 0; c < cps; ++c)
          ptx::tma_load_2d(ptx::smem_u32(st + q_off + c * a.nq * kBlockK * 2), &tm_q, bar(FULL + s),
                           (kc + c) * kBlockK, 0, pol_q);
        ++issued;
        if (++s == S) {
          s = 0;
          ph ^= 1u;
        }
      }
    }
    if (!ok) {
      // Wait for the copies that may still be in flight (the last S issued).
      int ds = s;
      uint32_t dph = ph;
      for (int64_t i = 0; i < issued && i < S; ++i) {
        if (--ds < 0) {
          ds = S - 1;
          dph ^= 1u;
        }
        drain_bar(bar(FULL + ds), dph);
      }
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------ MMA issuer
    const uint32_t idesc = ptx::idesc_bf16_f32(128, a.nq);
    int s = 0;
    uint32_t ph = 0;
    int64_t local = 0;
    bool ok = true;
    for (int64_t u = blockIdx.x; u < n_units && ok; u += gridDim.x, ++local) {
      const int b = (int)(local & 1);
      const uint32_t aph = (uint32_t)((local >> 1) & 1);
      if (!wait_bar(bar(ACC_EMPTY + b), aph ^ 1u, abort, a.status)) break;
      ptx::tc_fence_after();
      const uint32_t d0 = tmem + (uint32_t)((2 * b) * a.nq);
      const uint32_t d1 = tmem + (uint32_t)((2 * b + 1) * a.nq);
      for (int kc = 0; kc < a.kc; kc += cps) {
        if (!wait_bar(bar(FULL + s), ph, abort, a.status)) {
          ok = false;
          break;
        }
        ptx::tc_fence_after();
        const uint32_t st = ptx::smem_u32(smem + (size_t)s * stage_bytes);
        for (int c = 0; c < cps; ++c) {
          const uint32_t ta = st + (uint32_t)(2 * c) * kTileBytes;
          const uint32_t qa = st + q_off + (uint32_t)(c * a.nq * kBlockK * 2);
#pragma unroll
          for (int kk = 0; kk < kBlockK / 16; ++kk) {
            const uint64_t db = ptx::desc_sw128(qa + kk * 32);
            const uint32_t acc = (kc | c | kk) != 0;
            ptx::mma_bf16(d0, ptx::desc_sw128(ta + kk * 32), db, idesc, acc);
            ptx::mma_bf16(d1, ptx::desc_sw128(ta + kTileBytes + kk * 32), db, idesc, acc);
          }
        }
        ptx::mma_commit(bar(EMPTY + s));
        if (++s == S) {
          s = 0;
          ph ^= 1u;
        }
      }
      if (ok) ptx::mma_commit(bar(ACC_FULL + b));
    }
    ptx::mma_commit(bar(MMA_DONE));
    drain_bar(bar(MMA_DONE), 0);
  } else if (warp >= 2) {
    // ------------------------------------------------ epilogue
    const int q4 = warp & 3;  // TMEM lane quarter this warp may access
    const int r_in = q4 * 32 + lane;
    int64_t local = 0;
    for (int64_t u = blockIdx.x; u < n_units; u += gridDim.x, ++local) {
      const int b = (int)(local & 1);
      const uint32_t aph = (uint32_t)((local >> 1) & 1);
      if (!wait_bar(bar(ACC_FULL + b), aph, abort, a.status)) break;
      ptx::tc_fence_after();
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
        const int64_t half = 2 * u + h;
        if (half >= a.n_half) continue;
        const int64_t row = key_tile<MODE>(half) * 128 + r_in;
        const int64_t w = half * 128 + r_in;
        const uint32_t col0 = (uint32_t)((2 * b + h) * a.nq);
        for (int c0 = 0; c0 < a.nq; c0 += 16) {
          uint32_t r[16];
          ptx::tmem_ld16(tmem + ((uint32_t)(q4 * 32) << 16) + col0 + c0, r);
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int qi = c0 + j;
            if (qi >= a.qg) break;
            const float score = __uint_as_float(r[j]);
            if (MODE == SCAN_SAMPLE) {
              a.out[(int64_t)qi * a.n_work + w] = (row < a.n) ? cand_key(score, (uint32_t)row) : 0ull;
            } else if (row < a.n) {
              const uint64_t c = cand_key(score, (uint32_t)row);
              if (c >= s_thr[qi]) {
                const uint32_t pos = atomicAdd(&a.counts[qi], 1u);
                if ((int64_t)pos < a.pool_cap) a.out[(int64_t)qi * a.pool_cap + pos] = c;
                else raise_status(a.status, SENSE_DEVST_INTERNAL);
              }
            }
          }
        }
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(bar(ACC_EMPTY + b));
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, a.tmem_cols);
  }
}

// One block waits, through the same bounded wait as the scan's pipeline,
// on a barrier nothing arrives on: the wait gives up after `limit` cycles
// and reports SENSE_DEVST_TIMEOUT.
__global__ void selftest_wait_kernel(long long limit, uint32_t* status) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort;
  if (threadIdx.x == 0) {
    ptx::mbar_init(ptx::smem_u32(&bar), 1);
    abort = 0;
    ptx::fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) wait_bar(ptx::smem_u32(&bar), 0, &abort, status, limit);
}

__global__ void pad_queries_kernel(const uint16_t* __restrict__ src, int qg, int d,
                                   uint16_t* __restrict__ dst, int nq) {
  const int64_t total = (int64_t)nq * d;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / d;
    dst[i] = (r < qg) ? src[i] : (uint16_t)0;
  }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::mutex g_encode_mu;

sense_status get_encode(PFN_cuTensorMapEncodeTiled_v12000* fn) {
  std::lock_guard<std::mutex> lk(g_encode_mu);
  if (!g_encode) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                                     cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !p)
      return fail(SENSE_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  *fn = g_encode;
  return SENSE_OK;
}

}  // namespace

sense_status tensor_map_encoder(void** fn) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = nullptr;
  sense_status st = get_encode(&enc);
  *fn = reinterpret_cast<void*>(enc);
  return st;
}

namespace {

sense_status make_map(CUtensorMap* m, const void* base, int64_t rows, int d, int box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = nullptr;
  sense_status st = get_encode(&enc);
  if (st != SENSE_OK) return st;
  const cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kBlockK, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(SENSE_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return SENSE_OK;
}

// 64-column slices per ring stage: consecutive slices of a key row go out
// in one stage, so each row is requested cps x 128 contiguous bytes at a
// time.  Two slices keep three stages (192 KB of keys) in flight up to 32
// queries; past that they would cut the ring to two stages.
int slices_per_stage(int nq) { return nq <= 32 ? 2 : 1; }

int stages_for(int nq, int cps) {
  const int stage = cps * (2 * kTileBytes + nq * kBlockK * 2);
  const int budget = 227 * 1024 - 1024 - 512 - 8 * 128;
  int s = budget / stage;
  return s > 8 ? 8 : s;
}

}  // namespace

size_t scan_tc_smem_bytes(int d, int nq) {
  (void)d;
  const int cps = slices_per_stage(nq);
  const int S = stages_for(nq, cps);
  const size_t stage = (size_t)cps * (2 * kTileBytes + (size_t)nq * kBlockK * 2);
  return 1024 + S * stage + (2 * S + 5) * 8 + sizeof(Shared) + 8 * 128;
}

sense_status launch_selftest_wait(long long limit, uint32_t* status, cudaStream_t s) {
  selftest_wait_kernel<<<1, 32, 0, s>>>(limit, status);
  return cuda_check(cudaGetLastError(), "launch selftest_wait");
}

sense_status launch_pad_queries(const uint16_t* src, int qg, int d, uint16_t* dst, int nq,
                                cudaStream_t s) {
  LaunchScope ls(K_PAD_QUERIES, s);
  pad_queries_kernel<<<64, 256, 0, s>>>(src, qg, d, dst, nq);
  return cuda_check(cudaGetLastError(), "launch pad_queries");
}

sense_status launch_scan_tc(const uint16_t* keys, int64_t n, int d, const uint16_t* qpad, int qg,
                            int nq, int mode, int64_t n_half, const uint64_t* thresh,
                            uint64_t* out, uint32_t* counts, int64_t pool_cap, uint32_t* status,
                            cudaStream_t s) {
  if (nq < 16 || nq > 128 || (nq % 16) != 0 || qg > nq)
    return fail(SENSE_ERR_UNSUPPORTED, "tensor-core scan needs 16 <= nq <= 128, nq %% 16 == 0");
  alignas(64) CUtensorMap tm_keys;
  alignas(64) CUtensorMap tm_q;
  sense_status st = make_map(&tm_keys, keys, n, d, 128);
  if (st != SENSE_OK) return st;
  st = make_map(&tm_q, qpad, nq, d, nq);
  if (st != SENSE_OK) return st;
  TcArgs a{};
  a.n = n;
  a.d = d;
  a.qg = qg;
  a.nq = nq;
  a.n_half = n_half;
  a.n_work = n_half * 128;
  a.kc = (d + kBlockK - 1) / kBlockK;
  a.cps = slices_per_stage(nq);
  a.stages = stages_for(nq, a.cps);
  if (a.stages < 2) {
    a.cps = 1;
    a.stages = stages_for(nq, 1);
  }
  uint32_t cols = 32;
  while (cols < (uint32_t)(4 * nq)) cols <<= 1;
  a.tmem_cols = cols;
  a.thresh = thresh;
  a.out = out;
  a.counts = counts;
  a.pool_cap = pool_cap;
  a.status = status;
  const size_t smem = scan_tc_smem_bytes(d, nq);
  const int64_t units = (n_half + 1) / 2;
  int64_t grid = sm_count();
  if (grid > units) grid = units;
  if (grid < 1) grid = 1;
  auto run = [&](auto kern) -> sense_status {
    cudaError_t e = func_smem(reinterpret_cast<const void*>(kern), (int)smem);
    if (e != cudaSuccess) return cuda_check(e, "cudaFuncSetAttribute(scan_tc)");
    LaunchScope ls(K_SCAN_TC, s);
    kern<<<(unsigned)grid, kThreads, smem, s>>>(tm_keys, tm_q, a);
    return cuda_check(cudaGetLastError(), "launch scan_tc");
  };
  switch (mode) {
    case SCAN_SAMPLE: return run(scan_tc_kernel<SCAN_SAMPLE>);
    case SCAN_REST: return run(scan_tc_kernel<SCAN_REST>);
    default: return run(scan_tc_kernel<SCAN_ALL>);
  }
}

}  // namespace sense
