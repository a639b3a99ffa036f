// Tree-masked attention of the draft tokens over a static KV cache, on
// tcgen05 tensor cores (the attention of Alg. 1's verify forward,
// Forward(T, M_full, K), under the mask M_full of App. C.6 Eq. 20).
//
// For one head, the L <= 128 draft tokens attend to the n = m + L cache
// positions: position j is visible to token i if j < m (committed tokens)
// or if m <= j < m + L and node j - m is an ancestor of i or i itself
// (Alg. 3's mask, given as ancestor bit rows).  O = softmax(scale Q K^T +
// M_full) V.
//
// Design (flash-attention over 64-key blocks; one CTA per (head, key split)):
//  - warp 0 (one lane) loads Q [128 x 128] once and, per block, the K tile
//    [64 keys x 128] and the V^T tile [128 x 64 keys] with 3-D TMA loads
//    (128-byte swizzle; keys past n are zero-filled) into a 4-stage ring;
//  - warp 1 (one lane) issues S = Q K^T into one of two fp32 TMEM buffers
//    (M = 128 tokens, N = 64 keys, K = 128), then O += P V into a third
//    TMEM buffer once the softmax warps have written P (two P buffers, so
//    the softmax of block j overlaps the product of block j - 1);
//  - warps 2-9 own half a token row each (two warps per TMEM lane quarter,
//    32 of a block's 64 keys and 64 of O's 128 dims each; the pair exchanges
//    row maxima and sums
//    through shared memory): they read S with tcgen05.ld, apply
//    the scale and the mask (blocks wholly inside the committed prefix need
//    none), keep a running reference maximum (log2 domain; O and the row sum
//    are rescaled only when the block maximum exceeds the reference by more
//    than 2^8, and only then wait for the previous product), write
//    P = 2^(s - ref) (ex2.approx) as bf16 into shared memory in the
//    128-byte-swizzled K-major layout the MMA reads, and sum the bf16
//    values of P into the row sum;
//  - each split keeps its unnormalised O, reference maximum and row sum;
//    with at most 8 splits per head the splits are one cluster and merge
//    in place (each CTA combines every splits-th row from the others'
//    shared memory, rescaled to a common maximum, and divides), else they
//    go to global memory for a combine kernel.
// The key range is split so that heads x splits fill the SMs: the cache
// (2 x n x 128 x 2 bytes per head) is streamed once.
// Every mbarrier wait gives up after ~2 s of clock64 time: it sets
// SENSE_DEVST_TIMEOUT and an abort flag that releases the other roles; the
// producer then waits (bounded) for its copies in flight, the MMA thread for
// its MMAs, and the CTA frees its TMEM before returning.
#include <cooperative_groups.h>
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include <algorithm>

#include "common.cuh"
#include "launch.h"
#include "tc_ptx.cuh"

namespace sense {
namespace {

constexpr int kSoftWarps = 8;                 // two per TMEM lane quarter
constexpr int kAttnThreads = (2 + kSoftWarps) * 32;
constexpr int kHd = 128;                  // head dimension
constexpr int kBN = 64;                   // keys per block (64 or 128)
constexpr int kKS = kBN / 64;             // 64-key slabs per block
constexpr int kSlab = 128 * 64 * 2;       // 128 rows x 64 bf16 (one 128-byte swizzle slab)
constexpr int kKSlab = kBN * 64 * 2;      // kBN keys x 64 dims
constexpr int kQBytes = 2 * kSlab;        // Q: 128 tokens x 128 dims
constexpr int kPBytes = kKS * kSlab;      // P: 128 tokens x kBN keys
constexpr int kKBytes = 2 * kKSlab;       // K tile: kBN keys x 128 dims
constexpr int kVBytes = kKS * kSlab;      // V^T tile: 128 dims x kBN keys
constexpr int kStages = (kBN == 64) ? 4 : 2;
constexpr int kStageBytes = kKBytes + kVBytes;
constexpr long long kWaitCycles = 4000000000LL;
constexpr float kRescale = 8.0f;          // log2 growth that triggers a rescale of O

struct AttnArgs {
  int L, m, n, nb, splits, bps;
  float scale_log2;
  const uint32_t* mask;
  int mask_words;
  float* part_o;   // [H, splits, 128, 128]
  float* part_ml;  // [H, splits, 128, 2]: reference maximum (log2), row sum
  float* out;      // [H, L, 128] (fused combine)
  int fused;       // the splits of a head form a cluster and combine in place
  uint32_t* status;
};

struct AttnShared {
  uint32_t tmem_base;
  int abort;
};

__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int* abort,
                                         uint32_t* status) {
  if (ptx::mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (ptx::mbar_try_wait(bar, parity)) return true;
    if (*abort) return false;
    if (clock64() - t0 > kWaitCycles) {
      *abort = 1;
      raise_status(status, SENSE_DEVST_TIMEOUT);
      return false;
    }
  }
}
__device__ __forceinline__ void drain_bar(uint32_t bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!ptx::mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > kWaitCycles) return;
  }
}

// Bit t (0 <= t < 128) of the four mask words, without indexing a register array.
__device__ __forceinline__ bool tree_bit(uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3, int t) {
  const uint32_t w = t < 64 ? (t < 32 ? w0 : w1) : (t < 96 ? w2 : w3);
  return (w >> (t & 31)) & 1u;
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Two floats rounded to bf16 (nearest even) in one conversion: a in the low
// half, b in the high half.
__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// The head's splits (one cluster) merge their partials: row r is done by
// CTA r % splits, one warp per row, reading every split's statistics and rows
// through distributed shared memory, in the order of
// tree_attn_combine_kernel.  `so` is this CTA's partial O [128][128] f32
// followed by its statistics [128][2].
__device__ __forceinline__ void cluster_merge(const float* so, const AttnArgs& a, int h, int sp,
                                              int warp, int lane, int nwarps) {
  namespace cg = cooperative_groups;
  cg::cluster_group cl = cg::this_cluster();
  cl.sync();
  const int nsp = a.splits;
  const float* sml = so + 128 * kHd;
  const float NEG = -__int_as_float(0x7f800000);
  for (int r = sp + nsp * warp; r < a.L; r += nsp * nwarps) {
    float ref_s = NEG, l_s = 0.0f;
    if (lane < nsp) {
      const float* m = cl.map_shared_rank(sml, (unsigned)lane) + 2 * r;
      ref_s = m[0];
      l_s = m[1];
    }
    float mx = (lane < nsp && l_s > 0.0f) ? ref_s : NEG;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    float f = 0.0f, l = 0.0f;
    if (lane < nsp) {
      l = l_s;
      if (l > 0.0f) f = exp2f(ref_s - mx);
      else l = 0.0f;
    }
    float fl = f * l;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) fl += __shfl_xor_sync(0xffffffffu, fl, off);
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int t = 0; t < nsp; ++t) {
      const float ft = __shfl_sync(0xffffffffu, f, t);
      if (ft == 0.0f) continue;  // warp-uniform
      const float4 o =
          *reinterpret_cast<const float4*>(cl.map_shared_rank(so, (unsigned)t) + r * kHd + 4 * lane);
      acc.x += ft * o.x;
      acc.y += ft * o.y;
      acc.z += ft * o.z;
      acc.w += ft * o.w;
    }
    const float inv = fl > 0.0f ? 1.0f / fl : 0.0f;
    *reinterpret_cast<float4*>(a.out + ((int64_t)h * a.L + r) * kHd + 4 * lane) =
        make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
  }
  cl.sync();  // the other CTAs' shared memory stays alive until it is read
}

__global__ void __launch_bounds__(kAttnThreads, 1)
tree_attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                 const __grid_constant__ CUtensorMap tm_vt, const AttnArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* s_q = smem;                       // Q tile
  uint8_t* s_p = smem + kQBytes;             // two P tiles
  uint8_t* s_kv = s_p + 2 * kPBytes;         // stages: K tile, V^T tile
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_kv + kStages * kStageBytes);
  // bars: q_full, kv_full[S], kv_empty[S], s_full[2], s_empty[2], p_full[2],
  // p_empty[2], o_done, mma_done
  const int Q_FULL = 0, KV_FULL = 1, KV_EMPTY = 1 + kStages, S_FULL = 1 + 2 * kStages,
            S_EMPTY = 3 + 2 * kStages, P_FULL = 5 + 2 * kStages, P_EMPTY = 7 + 2 * kStages,
            O_DONE = 9 + 2 * kStages, MMA_DONE = 10 + 2 * kStages, NBARS = 11 + 2 * kStages;
  AttnShared* sh = reinterpret_cast<AttnShared*>(bars + NBARS);
  volatile int* abort = &sh->abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x, sp = blockIdx.y;
  const int j0 = sp * a.bps;
  const int j1 = min(a.nb, j0 + a.bps);
  const int nbl = max(0, j1 - j0);
  auto bar = [&](int i) { return ptx::smem_u32(bars + i); };

  if (threadIdx.x == 0) {
    ptx::mbar_init(bar(Q_FULL), 1);
    for (int s = 0; s < kStages; ++s) {
      ptx::mbar_init(bar(KV_FULL + s), 1);
      ptx::mbar_init(bar(KV_EMPTY + s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(bar(S_FULL + b), 1);
      ptx::mbar_init(bar(S_EMPTY + b), kSoftWarps);
      ptx::mbar_init(bar(P_FULL + b), kSoftWarps);
      ptx::mbar_init(bar(P_EMPTY + b), 1);
    }
    ptx::mbar_init(bar(O_DONE), 1);
    ptx::mbar_init(bar(MMA_DONE), 1);
    sh->abort = 0;
    ptx::fence_barrier_init();
    ptx::prefetch_tensormap(&tm_q);
    ptx::prefetch_tensormap(&tm_k);
    ptx::prefetch_tensormap(&tm_vt);
  }
  constexpr uint32_t kTmemCols = (2 * kBN + kHd <= 256) ? 256 : 512;
  if (warp == 1) ptx::tmem_alloc(ptx::smem_u32(&sh->tmem_base), kTmemCols);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = sh->tmem_base;  // S buffers at columns 0 and kBN, O at 2 kBN

  if (warp == 0 && lane == 0 && nbl > 0) {
    // ------------------------------------------------ TMA producer
    const uint64_t pol_stream = ptx::policy_evict_first();
    const uint64_t pol_keep = ptx::policy_evict_last();
    ptx::mbar_arrive_expect_tx(bar(Q_FULL), kQBytes);
    ptx::tma_load_3d(ptx::smem_u32(s_q), &tm_q, bar(Q_FULL), 0, 0, h, pol_keep);
    ptx::tma_load_3d(ptx::smem_u32(s_q + kSlab), &tm_q, bar(Q_FULL), 64, 0, h, pol_keep);
    int issued = 0;
    bool ok = true;
    for (int jj = 0; jj < nbl && ok; ++jj) {
      const int s = jj % kStages;
      const uint32_t ph = (uint32_t)((jj / kStages) & 1);
      if (!wait_bar(bar(KV_EMPTY + s), ph ^ 1u, abort, a.status)) {
        ok = false;
        break;
      }
      uint8_t* st = s_kv + s * kStageBytes;
      const int key0 = (j0 + jj) * kBN;
      ptx::mbar_arrive_expect_tx(bar(KV_FULL + s), kStageBytes);
      ptx::tma_load_3d(ptx::smem_u32(st), &tm_k, bar(KV_FULL + s), 0, key0, h, pol_stream);
      ptx::tma_load_3d(ptx::smem_u32(st + kKSlab), &tm_k, bar(KV_FULL + s), 64, key0, h, pol_stream);
#pragma unroll
      for (int i = 0; i < kKS; ++i)
        ptx::tma_load_3d(ptx::smem_u32(st + kKBytes + i * kSlab), &tm_vt, bar(KV_FULL + s),
                         key0 + 64 * i, 0, h, pol_stream);
      ++issued;
    }
    drain_bar(bar(Q_FULL), 0);
    if (!ok) {  // wait (bounded) for the copies that may still be in flight
      for (int jj = max(0, issued - kStages); jj < issued; ++jj)
        drain_bar(bar(KV_FULL + jj % kStages), (uint32_t)((jj / kStages) & 1));
    }
  } else if (warp == 1 && lane == 0 && nbl > 0) {
    // ------------------------------------------------ MMA issuer
    const uint32_t idesc_s = ptx::idesc_bf16_f32(128, kBN);   // S = Q K^T
    const uint32_t idesc_o = ptx::idesc_bf16_f32(128, kHd);   // O += P V
    const uint32_t q_addr = ptx::smem_u32(s_q), p_addr = ptx::smem_u32(s_p);
    bool ok = wait_bar(bar(Q_FULL), 0, abort, a.status);
    auto pv = [&](int i) -> bool {
      const int pb = i & 1;
      if (!wait_bar(bar(P_FULL + pb), (uint32_t)((i >> 1) & 1), abort, a.status)) return false;
      ptx::tc_fence_after();
      const uint32_t vt = ptx::smem_u32(s_kv + (i % kStages) * kStageBytes + kKBytes);
      const uint32_t pa = p_addr + pb * kPBytes;
#pragma unroll
      for (int ks = 0; ks < kKS; ++ks)
#pragma unroll
        for (int t = 0; t < 4; ++t)
          ptx::mma_bf16(tmem + 2 * kBN, ptx::desc_sw128(pa + ks * kSlab + t * 32),
                        ptx::desc_sw128(vt + ks * kSlab + t * 32), idesc_o,
                        (i > 0 || ks > 0 || t > 0) ? 1u : 0u);
      ptx::mma_commit(bar(O_DONE));
      ptx::mma_commit(bar(P_EMPTY + pb));
      ptx::mma_commit(bar(KV_EMPTY + i % kStages));
      return true;
    };
    for (int jj = 0; jj < nbl && ok; ++jj) {
      const int s = jj % kStages, b = jj & 1;
      if (!wait_bar(bar(KV_FULL + s), (uint32_t)((jj / kStages) & 1), abort, a.status) ||
          !wait_bar(bar(S_EMPTY + b), (uint32_t)(((jj >> 1) & 1) ^ 1), abort, a.status)) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
      const uint32_t kt = ptx::smem_u32(s_kv + s * kStageBytes);
#pragma unroll
      for (int kc = 0; kc < 2; ++kc)
#pragma unroll
        for (int t = 0; t < 4; ++t)
          ptx::mma_bf16(tmem + kBN * b, ptx::desc_sw128(q_addr + kc * kSlab + t * 32),
                        ptx::desc_sw128(kt + kc * kKSlab + t * 32), idesc_s,
                        (kc > 0 || t > 0) ? 1u : 0u);
      ptx::mma_commit(bar(S_FULL + b));
      if (jj > 0 && !pv(jj - 1)) ok = false;
    }
    if (ok) pv(nbl - 1);
    ptx::mma_commit(bar(MMA_DONE));
    drain_bar(bar(MMA_DONE), 0);
  } else if (warp >= 2) {
    // ------------------------------------------------ softmax / epilogue
    // Warps w and w + 4 share TMEM lane quarter w & 3 (rows q4 * 32 + lane);
    // `half` selects the 32 of a block's 64 keys and the 64 of O's 128 dims
    // this thread owns.  The pair exchanges row maxima (and at the end row sums)
    // through its own rows of the free P buffer, synchronised by a 64-thread
    // named barrier.
    constexpr int kCols = kBN / 2;
    const int q4 = warp & 3;
    const int half = (warp - 2) >> 2;
    const int r = q4 * 32 + lane;
    const int c0 = half * kCols;
    const uint32_t pair_bar = 1 + q4;
    auto pair_sync = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(pair_bar) : "memory"); };
    const uint32_t lane_base = tmem + ((uint32_t)(q4 * 32) << 16);
    uint32_t mw0 = 0u, mw1 = 0u, mw2 = 0u, mw3 = 0u;
    if (r < a.L) {
      const uint32_t* mr = a.mask + (int64_t)r * a.mask_words;
      mw0 = mr[0];
      if (a.mask_words > 1) mw1 = mr[1];
      if (a.mask_words > 2) mw2 = mr[2];
      if (a.mask_words > 3) mw3 = mr[3];
    }
    const float NEG = -__int_as_float(0x7f800000);
    float ref = NEG, rowsum = 0.0f;
    // `ok` is kept warp-uniform and no thread leaves the loop early: every
    // iteration executes both pair barriers, so a failed (aborted) wait in
    // one warp can never leave its partner blocked in bar.sync.
    bool ok = true;
    const int sw = r & 7;
    constexpr int kChunksT = kCols / 8;  // 16-byte chunks of a P row per thread
    // logical chunk g (8 keys) of this row in a P tile: slab g / 8, swizzled
    // position (g % 8) ^ (row % 8) inside the row's 128 bytes
    auto pchunk = [&](uint8_t* tile, int g) {
      return tile + (g >> 3) * kSlab + r * 128 + ((((g & 7) ^ sw)) << 4);
    };
    for (int jj = 0; jj < nbl; ++jj) {
      const int b = jj & 1;
      ok = __all_sync(0xffffffffu,
                      ok && wait_bar(bar(S_FULL + b), (uint32_t)((jj >> 1) & 1), abort, a.status));
      float sv[kCols];
      float pmax = NEG;
      if (ok) {
        ptx::tc_fence_after();
        {
          uint32_t rr[kCols / 16][16];
#pragma unroll
          for (int c = 0; c < kCols / 16; ++c)
            ptx::tmem_ld16_nowait(lane_base + kBN * b + c0 + 16 * c, rr[c]);
          ptx::tmem_ld_wait();
#pragma unroll
          for (int c = 0; c < kCols / 16; ++c)
#pragma unroll
            for (int e = 0; e < 16; ++e) sv[16 * c + e] = __uint_as_float(rr[c][e]);
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(bar(S_EMPTY + b));
        // scale (log2 domain) and mask; blocks inside the prefix are all visible
        const int key0 = (j0 + jj) * kBN + c0;
        float bm[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) bm[e] = NEG;
        if (key0 + kCols <= a.m) {
#pragma unroll
          for (int c = 0; c < kCols; ++c) {
            sv[c] *= a.scale_log2;
            bm[c & 7] = fmaxf(bm[c & 7], sv[c]);
          }
        } else {
#pragma unroll
          for (int c = 0; c < kCols; ++c) {
            const int col = key0 + c;
            bool vis = col < a.m;
            if (!vis && r < a.L && col < a.m + a.L) vis = tree_bit(mw0, mw1, mw2, mw3, col - a.m);
            sv[c] = vis ? sv[c] * a.scale_log2 : NEG;
            bm[c & 7] = fmaxf(bm[c & 7], sv[c]);
          }
        }
        pmax = fmaxf(fmaxf(fmaxf(bm[0], bm[1]), fmaxf(bm[2], bm[3])),
                     fmaxf(fmaxf(bm[4], bm[5]), fmaxf(bm[6], bm[7])));
      }
      // P buffer b is free once the product of block jj - 2 is done
      ok = __all_sync(0xffffffffu, ok && wait_bar(bar(P_EMPTY + b),
                                                 (uint32_t)(((jj >> 1) & 1) ^ 1), abort, a.status));
      // exchange through this row of P buffer b: each thread's first 16-byte
      // chunk (bytes only this pair touches; written over by P below)
      uint8_t* ptile = s_p + b * kPBytes;
      if (ok) *reinterpret_cast<float*>(pchunk(ptile, kChunksT * half)) = pmax;
      pair_sync();
      const float other = *reinterpret_cast<const float*>(pchunk(ptile, kChunksT * (1 - half)));
      pair_sync();
      if (!ok) continue;
      const float bmax = fmaxf(pmax, other);
      float factor = 1.0f;
      bool rescale = false;
      if (ref == NEG) {
        ref = bmax;  // O is still zero for this row: nothing to rescale
      } else if (bmax > ref + kRescale) {
        factor = ex2(ref - bmax);
        ref = bmax;
        rescale = true;
      }
      // O must hold the product of block jj - 1 before it is scaled
      const bool any_rescale = __any_sync(0xffffffffu, rescale);
      if (any_rescale) {
        ok = __all_sync(0xffffffffu,
                        wait_bar(bar(O_DONE), (uint32_t)((jj - 1) & 1), abort, a.status));
        if (!ok) continue;
        ptx::tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < kHd / 2 / 16; ++c) {
          uint32_t rr[16];
          const uint32_t ta = lane_base + 2 * kBN + half * (kHd / 2) + 16 * c;
          ptx::tmem_ld16(ta, rr);
#pragma unroll
          for (int e = 0; e < 16; ++e) rr[e] = __float_as_uint(__uint_as_float(rr[e]) * factor);
          ptx::tmem_st16(ta, rr);
        }
        rowsum *= factor;
      }
      // P = 2^(s - ref) as bf16 into this thread's chunks of the swizzled row

      float ps[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int g = 0; g < kCols / 8; ++g) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 8; e += 2) {
          const float x0 = sv[8 * g + e], x1 = sv[8 * g + e + 1];
          const float p0 = (x0 == NEG || ref == NEG) ? 0.0f : ex2(x0 - ref);
          const float p1 = (x1 == NEG || ref == NEG) ? 0.0f : ex2(x1 - ref);
          const uint32_t pk = pack_bf16(p0, p1);  // one paired conversion
          w[e >> 1] = pk;
          ps[e] += __uint_as_float(pk << 16);          // the rounded values
          ps[e + 1] += __uint_as_float(pk & 0xffff0000u);
        }
        *reinterpret_cast<uint4*>(pchunk(ptile, kChunksT * half + g)) =
            make_uint4(w[0], w[1], w[2], w[3]);
      }
      rowsum += ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
      ptx::fence_proxy_async_smem();
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(bar(P_FULL + b));
    }
    // partial output of this split: each thread its 64 dims, row sums
    // combined; into global memory, or (fused) into this CTA's shared memory
    // where the K/V stages were (every load has landed, every product is
    // done once MMA_DONE has completed)
    const int64_t pbase = ((int64_t)h * a.splits + sp) * 128 + r;
    float* so = reinterpret_cast<float*>(s_kv);  // fused: [128][128] partial O
    float* sml = so + 128 * kHd;                  // fused: [128][2] statistics
    float* po = a.fused ? so + r * kHd + half * (kHd / 2)
                        : a.part_o + pbase * kHd + half * (kHd / 2);
    float* pml = a.fused ? sml + 2 * r : a.part_ml + pbase * 2;
    const bool done =
        __all_sync(0xffffffffu, ok && nbl > 0 && wait_bar(bar(MMA_DONE), 0, abort, a.status));
    if (done && q4 * 32 < a.L) {  // rows past L are padding: not written
      ptx::tc_fence_after();
      uint32_t rr[kHd / 2 / 16][16];
#pragma unroll
      for (int c = 0; c < kHd / 2 / 16; ++c)
        ptx::tmem_ld16_nowait(lane_base + 2 * kBN + half * (kHd / 2) + 16 * c, rr[c]);
      ptx::tmem_ld_wait();
      if (r < a.L) {
#pragma unroll
        for (int c = 0; c < kHd / 2 / 16; ++c)
#pragma unroll
          for (int e = 0; e < 16; e += 4)
            *reinterpret_cast<float4*>(po + 16 * c + e) =
                make_float4(__uint_as_float(rr[c][e]), __uint_as_float(rr[c][e + 1]),
                            __uint_as_float(rr[c][e + 2]), __uint_as_float(rr[c][e + 3]));
      }
    }
    // every product is done (or the CTA aborted): P buffer 0 is free; the row
    // sums meet in this row's words of it
    *reinterpret_cast<float*>(pchunk(s_p, kChunksT * half)) = rowsum;
    pair_sync();
    if (half == 0) {
      pml[0] = done ? ref : NEG;
      pml[1] = done ? rowsum + *reinterpret_cast<const float*>(pchunk(s_p, kChunksT)) : 0.0f;
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, kTmemCols);
  }
  if (a.fused)
    cluster_merge(reinterpret_cast<const float*>(s_kv), a, h, sp, warp, lane, kAttnThreads / 32);
}

// ---------------------------------------------------------------------------
// Transposed products for trees of at most 64 nodes.
//
// With L <= 64 draft tokens, half of the M = 128 rows of S = Q K^T and of
// O = P V are padding, and an MMA of M <= 128 costs about N cycles per K = 16
// step whatever M is.  This kernel computes both products transposed, with
// the 64 token columns as N:
//   S^T = K Q^T   (M = 128 keys of a block, N = 64 tokens, K = 128 dims)
//   O^T += V^T P^T (M = 128 dims, N = 64 tokens, K = 128 keys)
// which halves the tensor time per key and, with 128-key blocks, halves the
// exponentials per key (no padding rows).  In TMEM a softmax thread now owns
// one key (a lane) and 16 token columns; 16 softmax warps cover the 128
// keys x 64 tokens of a block.  The row statistics need cross-thread
// reductions, but only when the lazy-rescale test fires:
//  - the four warps that share 16 tokens (one per TMEM lane quarter) keep
//    the tokens' reference maxima in shared memory;
//  - per block, each thread tests whether any visible score exceeds its
//    token's reference by more than 2^8 (log2 domain); one barrier-reduction
//    over the four warps decides for them;
//  - only then (always on the first block) the block maxima per token are
//    reduced (a transposing shuffle reduction per warp, the four lane
//    quarters through shared memory), the references raised, and the row
//    sums and O^T columns of those tokens rescaled;
//  - P = 2^(s - ref_t) is rounded to bf16 and written to P[token][key] in the
//    swizzled K-major layout the product reads; each thread adds its rounded
//    values into per-token partial row sums, reduced across keys once at
//    the end.
// The MMA thread issues the scores of a block as soon as its K tile and one
// of three S^T buffers are free, ahead of the value products, so the softmax
// warps never wait behind a product.  K and V^T tiles have separate rings
// (3 and 2 stages of 32 KB), so keys can be loaded ahead while the products
// of earlier blocks still hold their V^T tiles.  The split partials and
// their merge are those of tree_attn_kernel.
constexpr int kTB = 128;                  // keys per block
constexpr int kTN = 64;                   // token columns (N of both products)
constexpr int kTSoftWarps = 16;           // four per TMEM lane quarter
constexpr int kTTok = kTN / 4;            // token columns per softmax thread
constexpr int kTThreads = (2 + kTSoftWarps) * 32;
constexpr int kTSlabQ = kTN * 128;        // 64 rows x 64 bf16 (one swizzle slab)
constexpr int kTQBytes = 2 * kTSlabQ;     // Q: 64 tokens x 128 dims
constexpr int kTPBytes = 2 * kTSlabQ;     // P: 64 tokens x 128 keys
constexpr int kTSlab = 128 * 128;         // 128 rows x 64 bf16
constexpr int kTKBytes = 2 * kTSlab;      // K tile: 128 keys x 128 dims
constexpr int kTVBytes = 2 * kTSlab;      // V^T tile: 128 dims x 128 keys
constexpr int kTKStages = 3;
constexpr int kTVStages = 2;
constexpr int kTSBufs = 3;                // S^T buffers in TMEM
constexpr int kTOCol = kTSBufs * kTN;     // TMEM column of O^T
constexpr int kTNBars = 1 + 2 * kTKStages + 2 * kTVStages + 2 * kTSBufs + 4 + 2;

struct AttnTShared {
  uint32_t tmem_base;
  int abort;
  uint32_t maskT[kTN][2];   // tree key j: bit t of word t / 32 set iff node j is visible to token t
  float4 qmax[kTN];         // per token: block maxima of the four lane quarters
  float4 qsum[kTN];         // per token: row sums of the four lane quarters
  float ref[kTN];           // per token: reference maximum (log2 domain)
  float factor[kTN];        // per token: rescale factor of the last raise
};

size_t attn_t_smem_bytes() {
  return 1024 + kTQBytes + 2 * kTPBytes + kTKStages * kTKBytes + kTVStages * kTVBytes +
         kTNBars * 8 + 16 + sizeof(AttnTShared);
}

__device__ __forceinline__ void soft_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kTSoftWarps * 32) : "memory");
}

// The four warps of token group `tg` (one per lane quarter) share the
// reference maxima of their 16 tokens: a barrier over them (ids 3..6) that
// also returns whether any of their threads passed `p`, and a plain one
// (ids 7..10).
__device__ __forceinline__ bool group_any(int tg, bool p) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\t"
      "setp.ne.u32 pi, %1, 0;\n\t"
      "bar.red.or.pred po, %2, 128, pi;\n\t"
      "selp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)p), "r"(3 + tg)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ void group_sync(int tg) {
  asm volatile("bar.sync %0, 128;" ::"r"(7 + tg) : "memory");
}

// Lane i (and lane i ^ 16) ends up with op over the warp's 32 lanes of
// v[i % 16] (each lane passes 16 values indexed by token).  Four exchange
// rounds: in round `off` a lane keeps the half of its remaining values
// selected by its bit `off` and receives the partner's copy of that half;
// a last exchange combines the two half-warps.
template <bool kMax>
__device__ __forceinline__ float transpose_reduce(float (&v)[kTTok], int lane) {
#pragma unroll
  for (int off = kTTok / 2; off > 0; off >>= 1) {
    const bool upper = (lane & off) != 0;
#pragma unroll
    for (int i = 0; i < off; ++i) {
      const float keep = upper ? v[i + off] : v[i];
      const float send = upper ? v[i] : v[i + off];
      const float got = __shfl_xor_sync(0xffffffffu, send, off);
      v[i] = kMax ? fmaxf(keep, got) : keep + got;
    }
  }
  const float other = __shfl_xor_sync(0xffffffffu, v[0], 16);
  return kMax ? fmaxf(v[0], other) : v[0] + other;
}

__global__ void __launch_bounds__(kTThreads, 1)
tree_attn_t_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                   const __grid_constant__ CUtensorMap tm_vt, const AttnArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* s_q = smem;                          // Q tile (B of S^T)
  uint8_t* s_p = s_q + kTQBytes;                // two P tiles (B of O^T)
  uint8_t* s_k = s_p + 2 * kTPBytes;            // K ring (A of S^T)
  uint8_t* s_v = s_k + kTKStages * kTKBytes;    // V^T ring (A of O^T)
  uint64_t* bars = reinterpret_cast<uint64_t*>(s_v + kTVStages * kTVBytes);
  const int Q_FULL = 0, K_FULL = 1, K_EMPTY = 1 + kTKStages, V_FULL = 1 + 2 * kTKStages,
            V_EMPTY = V_FULL + kTVStages, S_FULL = V_EMPTY + kTVStages, S_EMPTY = S_FULL + kTSBufs,
            P_FULL = S_EMPTY + kTSBufs, P_EMPTY = P_FULL + 2, O_DONE = P_EMPTY + 2,
            MMA_DONE = O_DONE + 1;
  AttnTShared* sh = reinterpret_cast<AttnTShared*>(
      (reinterpret_cast<uintptr_t>(bars + kTNBars) + 15) & ~static_cast<uintptr_t>(15));
  volatile int* abort = &sh->abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x, sp = blockIdx.y;
  const int j0 = sp * a.bps;
  const int j1 = min(a.nb, j0 + a.bps);
  const int nbl = max(0, j1 - j0);
  auto bar = [&](int i) { return ptx::smem_u32(bars + i); };

  if (threadIdx.x == 0) {
    ptx::mbar_init(bar(Q_FULL), 1);
    for (int s = 0; s < kTKStages; ++s) {
      ptx::mbar_init(bar(K_FULL + s), 1);
      ptx::mbar_init(bar(K_EMPTY + s), 1);
    }
    for (int s = 0; s < kTVStages; ++s) {
      ptx::mbar_init(bar(V_FULL + s), 1);
      ptx::mbar_init(bar(V_EMPTY + s), 1);
    }
    for (int b = 0; b < kTSBufs; ++b) {
      ptx::mbar_init(bar(S_FULL + b), 1);
      ptx::mbar_init(bar(S_EMPTY + b), kTSoftWarps);
    }
    for (int b = 0; b < 2; ++b) {
      ptx::mbar_init(bar(P_FULL + b), kTSoftWarps);
      ptx::mbar_init(bar(P_EMPTY + b), 1);
    }
    ptx::mbar_init(bar(O_DONE), 1);
    ptx::mbar_init(bar(MMA_DONE), 1);
    sh->abort = 0;
    ptx::fence_barrier_init();
    if (nbl > 0 && (j0 + 1) * kTB <= a.m) {
      // the first K and V^T tiles go out before the block barrier when they
      // hold committed keys only (nothing launched before this kernel
      // writes those); Q waits for the dependency below
      const uint64_t pol_stream = ptx::policy_evict_first();
      const int key0 = j0 * kTB;
      ptx::mbar_arrive_expect_tx(bar(K_FULL), kTKBytes);
      ptx::tma_load_3d(ptx::smem_u32(s_k), &tm_k, bar(K_FULL), 0, key0, h, pol_stream);
      ptx::tma_load_3d(ptx::smem_u32(s_k + kTSlab), &tm_k, bar(K_FULL), 64, key0, h, pol_stream);
      ptx::mbar_arrive_expect_tx(bar(V_FULL), kTVBytes);
      ptx::tma_load_3d(ptx::smem_u32(s_v), &tm_vt, bar(V_FULL), key0, 0, h, pol_stream);
      ptx::tma_load_3d(ptx::smem_u32(s_v + kTSlab), &tm_vt, bar(V_FULL), key0 + 64, 0, h,
                       pol_stream);
    }
  }
  if (warp == 1) ptx::tmem_alloc(ptx::smem_u32(&sh->tmem_base), 256);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  pdl_launch_dependents();
  const uint32_t tmem = sh->tmem_base;  // S^T buffers at columns kTN b (b < 3), O^T at kTOCol

  if (warp == 0 && lane == 0 && nbl > 0) {
    // ------------------------------------------------ TMA producer
    // K and V^T tiles are issued in block order as their ring slots free up;
    // the slot tests do not block (test_wait), so a late V^T slot does not
    // hold back the next K tile or the other way round.
    const uint64_t pol_stream = ptx::policy_evict_first();
    auto committed = [&](int j) { return (j0 + j + 1) * kTB <= a.m; };
    auto issue_k = [&](int j) {
      const int s = j % kTKStages;
      uint8_t* st = s_k + s * kTKBytes;
      const int key0 = (j0 + j) * kTB;
      ptx::mbar_arrive_expect_tx(bar(K_FULL + s), kTKBytes);
      ptx::tma_load_3d(ptx::smem_u32(st), &tm_k, bar(K_FULL + s), 0, key0, h, pol_stream);
      ptx::tma_load_3d(ptx::smem_u32(st + kTSlab), &tm_k, bar(K_FULL + s), 64, key0, h,
                       pol_stream);
    };
    auto issue_v = [&](int j) {
      const int s = j % kTVStages;
      uint8_t* st = s_v + s * kTVBytes;
      const int key0 = (j0 + j) * kTB;
      ptx::mbar_arrive_expect_tx(bar(V_FULL + s), kTVBytes);
      ptx::tma_load_3d(ptx::smem_u32(st), &tm_vt, bar(V_FULL + s), key0, 0, h, pol_stream);
      ptx::tma_load_3d(ptx::smem_u32(st + kTSlab), &tm_vt, bar(V_FULL + s), key0 + 64, 0, h,
                       pol_stream);
    };
    // block 0's tiles went out with the barriers when committed; the other
    // free ring slots take further committed blocks before the dependency
    // wait, everything else (Q, draft keys) after it
    int jk = committed(0) ? 1 : 0, jv = jk;
    for (; jk < min(nbl, kTKStages) && committed(jk); ++jk) issue_k(jk);
    for (; jv < min(nbl, kTVStages) && jv < jk; ++jv) issue_v(jv);
    pdl_wait();  // Q, the tree's keys and the mask are written
    ptx::mbar_arrive_expect_tx(bar(Q_FULL), kTQBytes);
    {
      const uint64_t pol_keep = ptx::policy_evict_last();
      ptx::tma_load_3d(ptx::smem_u32(s_q), &tm_q, bar(Q_FULL), 0, 0, h, pol_keep);
      ptx::tma_load_3d(ptx::smem_u32(s_q + kTSlabQ), &tm_q, bar(Q_FULL), 64, 0, h, pol_keep);
    }
    long long t0 = clock64();
    while ((jk < nbl || jv < nbl) && !*abort) {
      bool moved = false;
      if (jk < nbl && ptx::mbar_test_wait(bar(K_EMPTY + jk % kTKStages),
                                          (uint32_t)(((jk / kTKStages) & 1) ^ 1))) {
        issue_k(jk);
        ++jk;
        moved = true;
      }
      if (jv < nbl && jv < jk &&
          ptx::mbar_test_wait(bar(V_EMPTY + jv % kTVStages), (uint32_t)(((jv / kTVStages) & 1) ^ 1))) {
        issue_v(jv);
        ++jv;
        moved = true;
      }
      if (moved) {
        t0 = clock64();
      } else if (clock64() - t0 > kWaitCycles) {
        *abort = 1;
        raise_status(a.status, SENSE_DEVST_TIMEOUT);
      }
    }
    drain_bar(bar(Q_FULL), 0);
    if (*abort) {  // wait (bounded) for the copies that may still be in flight
      for (int j = max(0, jk - kTKStages); j < jk; ++j)
        drain_bar(bar(K_FULL + j % kTKStages), (uint32_t)((j / kTKStages) & 1));
      for (int j = max(0, jv - kTVStages); j < jv; ++j)
        drain_bar(bar(V_FULL + j % kTVStages), (uint32_t)((j / kTVStages) & 1));
    }
  } else if (warp == 1 && lane == 0 && nbl > 0) {
    // ------------------------------------------------ MMA issuer
    // Score products run ahead of the value products as far as the three
    // S^T buffers allow (a block's scores are released as soon as the
    // softmax has read them), so the softmax never waits behind a value
    // product; the barrier tests do not block (test_wait).
    const uint32_t idesc = ptx::idesc_bf16_f32(128, kTN);
    const uint32_t q_addr = ptx::smem_u32(s_q), p_addr = ptx::smem_u32(s_p);
    bool ok = wait_bar(bar(Q_FULL), 0, abort, a.status);
    ptx::tc_fence_after();
    int js = 0, jp = 0;
    long long t0 = clock64();
    while (ok && jp < nbl) {
      bool moved = false;
      if (js < nbl && ptx::mbar_test_wait(bar(K_FULL + js % kTKStages), (uint32_t)((js / kTKStages) & 1)) &&
          ptx::mbar_test_wait(bar(S_EMPTY + js % kTSBufs), (uint32_t)(((js / kTSBufs) & 1) ^ 1))) {
        ptx::tc_fence_after();
        const uint32_t kt = ptx::smem_u32(s_k + (js % kTKStages) * kTKBytes);
        const uint32_t sd = tmem + kTN * (js % kTSBufs);
#pragma unroll
        for (int kc = 0; kc < 2; ++kc)
#pragma unroll
          for (int t = 0; t < 4; ++t)
            ptx::mma_bf16(sd, ptx::desc_sw128(kt + kc * kTSlab + t * 32),
                          ptx::desc_sw128(q_addr + kc * kTSlabQ + t * 32), idesc,
                          (kc > 0 || t > 0) ? 1u : 0u);
        ptx::mma_commit(bar(S_FULL + js % kTSBufs));
        ptx::mma_commit(bar(K_EMPTY + js % kTKStages));
        ++js;
        moved = true;
      }
      if (jp < js && ptx::mbar_test_wait(bar(P_FULL + (jp & 1)), (uint32_t)((jp >> 1) & 1)) &&
          ptx::mbar_test_wait(bar(V_FULL + jp % kTVStages), (uint32_t)((jp / kTVStages) & 1))) {
        ptx::tc_fence_after();
        const int pb = jp & 1, sv = jp % kTVStages;
        const uint32_t vt = ptx::smem_u32(s_v + sv * kTVBytes);
        const uint32_t pa = p_addr + pb * kTPBytes;
#pragma unroll
        for (int ks = 0; ks < 2; ++ks)
#pragma unroll
          for (int t = 0; t < 4; ++t)
            ptx::mma_bf16(tmem + kTOCol, ptx::desc_sw128(vt + ks * kTSlab + t * 32),
                          ptx::desc_sw128(pa + ks * kTSlabQ + t * 32), idesc,
                          (jp > 0 || ks > 0 || t > 0) ? 1u : 0u);
        ptx::mma_commit(bar(O_DONE));
        ptx::mma_commit(bar(P_EMPTY + pb));
        ptx::mma_commit(bar(V_EMPTY + sv));
        ++jp;
        moved = true;
      }
      if (moved) {
        t0 = clock64();
      } else if (*abort) {
        ok = false;
      } else if (clock64() - t0 > kWaitCycles) {
        *abort = 1;
        raise_status(a.status, SENSE_DEVST_TIMEOUT);
        ok = false;
      }
    }
    ptx::mma_commit(bar(MMA_DONE));
    drain_bar(bar(MMA_DONE), 0);
  } else if (warp >= 2) {
    pdl_wait();  // the mask and the outputs' previous readers are done
    // ------------------------------------------------ softmax / epilogue
    // Warp w owns TMEM lane quarter q4 = w & 3: keys 32 q4 + lane of a block
    // in S^T, dims 32 q4 + lane in O^T; `tg` = (w - 2) / 4 selects its 16
    // token columns.
    const int q4 = warp & 3;
    const int tg = (warp - 2) >> 2;
    const int tb = kTTok * tg;                // first token of this thread
    const uint32_t lane_base = tmem + ((uint32_t)(q4 * 32) << 16);
    const int kl = 32 * q4 + lane;            // this thread's key within a block
    const float NEG = -__int_as_float(0x7f800000);
    // transposed tree mask: warp w' = w - 2 ballots tokens 32 (w' & 1) + lane
    // for tree keys j in [8 (w' >> 1), +8)
    {
      const int wp = warp - 2;
      const int t = 32 * (wp & 1) + lane;
      uint32_t m0 = 0u, m1 = 0u;
      if (t < a.L) {
        const uint32_t* mr = a.mask + (int64_t)t * a.mask_words;
        m0 = mr[0];
        if (a.mask_words > 1) m1 = mr[1];
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int j = 8 * (wp >> 1) + i;
        const uint32_t bit = ((j < 32 ? m0 : m1) >> (j & 31)) & 1u;
        const uint32_t word = __ballot_sync(0xffffffffu, bit != 0u && j < a.L);
        if (lane == 0) sh->maskT[j][wp & 1] = word;
      }
    }
    if (warp < 4) sh->ref[32 * (warp - 2) + lane] = NEG;
    soft_sync();  // every warp's maskT words and the references are in place
    // tokens of this thread that exist (t < L)
    const uint32_t live = a.L >= tb + kTTok ? 0xffffu : (a.L <= tb ? 0u : ((1u << (a.L - tb)) - 1u));
    const int mshift = tb & 31;               // this thread's tokens in a maskT word
    float psum[kTTok];
#pragma unroll
    for (int u = 0; u < kTTok; ++u) psum[u] = 0.0f;
    const float4* ref4 = reinterpret_cast<const float4*>(sh->ref + tb);
    // P[token][key]: slab kl / 64, 16-byte chunk (kl % 64) / 8 swizzled by
    // token % 8 inside the token's 128-byte row, 2 bytes per key
    const int g = (kl & 63) >> 3;
    const uint32_t p_off = (uint32_t)((kl >> 6) * kTSlabQ + ((kl & 7) << 1));
    bool ok = true;
    for (int jj = 0; jj < nbl; ++jj) {
      const int b = jj & 1;                     // P buffer
      const int sb = jj % kTSBufs;              // S^T buffer
      const int key0 = (j0 + jj) * kTB;
      ok = __all_sync(0xffffffffu, ok && wait_bar(bar(S_FULL + sb), (uint32_t)((jj / kTSBufs) & 1),
                                                 abort, a.status));
      float x[kTTok];                         // log2-domain scores (-inf: not visible)
      bool exceed = false;
      if (ok) {
        ptx::tc_fence_after();
        uint32_t rr[kTTok];
        ptx::tmem_ld16(lane_base + kTN * sb + tb, rr);
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(bar(S_EMPTY + sb));
        const int key = key0 + kl;
#pragma unroll
        for (int u = 0; u < kTTok; ++u) x[u] = __uint_as_float(rr[u]) * a.scale_log2;
        if (!(key0 + kTB <= a.m && live == 0xffffu)) {  // not a block inside the prefix
          uint32_t vis = 0u;
          if (key < a.m) vis = live;
          else if (key < a.m + a.L) vis = (sh->maskT[key - a.m][tb >> 5] >> mshift) & 0xffffu;
#pragma unroll
          for (int u = 0; u < kTTok; ++u)
            if (!((vis >> u) & 1u)) x[u] = NEG;
        }
        // a visible score above its token's reference by more than 2^8 (the
        // first visible score of a token always is: its reference is -inf)
        float dmax = NEG;
#pragma unroll
        for (int u4 = 0; u4 < kTTok / 4; ++u4) {
          const float4 r4 = ref4[u4];
          dmax = fmaxf(dmax, fmaxf(fmaxf(x[4 * u4] - r4.x, x[4 * u4 + 1] - r4.y),
                                   fmaxf(x[4 * u4 + 2] - r4.z, x[4 * u4 + 3] - r4.w)));
        }
        exceed = dmax > kRescale;  // -inf - -inf = NaN compares false
      }
      // P buffer b is free once the product of block jj - 2 is done; after
      // this wait at most the product of block jj - 1 is still running, so
      // the O_DONE phase tested below is that product's
      ok = __all_sync(0xffffffffu, ok && wait_bar(bar(P_EMPTY + b),
                                                 (uint32_t)(((jj >> 1) & 1) ^ 1), abort, a.status));
      if (group_any(tg, ok && exceed)) {
        {
          float bm[kTTok];  // block maxima per token
#pragma unroll
          for (int u = 0; u < kTTok; ++u) bm[u] = x[u];
          const float wmax = transpose_reduce<true>(bm, lane);  // token tb + lane % 16
          if (lane < kTTok) reinterpret_cast<float*>(&sh->qmax[tb + lane])[q4] = wmax;
        }
        group_sync(tg);
        if (q4 == 0 && lane < kTTok) {  // one thread per token raises its reference
          const int t = tb + lane;
          const float4 qm = sh->qmax[t];
          const float m4 = fmaxf(fmaxf(qm.x, qm.y), fmaxf(qm.z, qm.w));
          const float r = sh->ref[t];
          float f = 1.0f;
          if (m4 > r + kRescale) {
            if (r != NEG) f = ex2(r - m4);
            sh->ref[t] = m4;
          }
          sh->factor[t] = f;
        }
        group_sync(tg);
        const float4* f4 = reinterpret_cast<const float4*>(sh->factor + tb);
        bool rescale = false;
#pragma unroll
        for (int u4 = 0; u4 < kTTok / 4; ++u4) {
          const float4 f = f4[u4];
          psum[4 * u4] *= f.x;
          psum[4 * u4 + 1] *= f.y;
          psum[4 * u4 + 2] *= f.z;
          psum[4 * u4 + 3] *= f.w;
          rescale |= (f.x != 1.0f) || (f.y != 1.0f) || (f.z != 1.0f) || (f.w != 1.0f);
        }
        // this warp's O^T columns (its tokens, its dims) must hold the
        // product of block jj - 1 before they are scaled
        if (__any_sync(0xffffffffu, rescale) && ok) {
          ok = __all_sync(0xffffffffu,
                          wait_bar(bar(O_DONE), (uint32_t)((jj - 1) & 1), abort, a.status));
          if (ok) {
            ptx::tc_fence_after();
            uint32_t rr[kTTok];
            const uint32_t ta = lane_base + kTOCol + tb;
            ptx::tmem_ld16(ta, rr);
#pragma unroll
            for (int u4 = 0; u4 < kTTok / 4; ++u4) {
              const float4 f = f4[u4];
              rr[4 * u4] = __float_as_uint(__uint_as_float(rr[4 * u4]) * f.x);
              rr[4 * u4 + 1] = __float_as_uint(__uint_as_float(rr[4 * u4 + 1]) * f.y);
              rr[4 * u4 + 2] = __float_as_uint(__uint_as_float(rr[4 * u4 + 2]) * f.z);
              rr[4 * u4 + 3] = __float_as_uint(__uint_as_float(rr[4 * u4 + 3]) * f.w);
            }
            ptx::tmem_st16(ta, rr);
          }
        }
      }
      if (!ok) continue;
      // P = 2^(x - ref) rounded to bf16 into P[token][this key]; every
      // visible x is at most ref + 2^8 here; invisible -> 0
      uint8_t* prow = s_p + b * kTPBytes + p_off + tb * 128;
#pragma unroll
      for (int u4 = 0; u4 < kTTok / 4; ++u4) {
        const float4 r4 = ref4[u4];
        const float rv[4] = {r4.x, r4.y, r4.z, r4.w};
#pragma unroll
        for (int e = 0; e < 4; e += 2) {
          const int u = 4 * u4 + e;
          const float p0 = x[u] == NEG ? 0.0f : ex2(x[u] - rv[e]);
          const float p1 = x[u + 1] == NEG ? 0.0f : ex2(x[u + 1] - rv[e + 1]);
          const uint32_t pk = pack_bf16(p0, p1);
          psum[u] += __uint_as_float(pk << 16);
          psum[u + 1] += __uint_as_float(pk & 0xffff0000u);
          *reinterpret_cast<uint16_t*>(prow + u * 128 + ((g ^ (u & 7)) << 4)) =
              (uint16_t)(pk & 0xffffu);
          *reinterpret_cast<uint16_t*>(prow + (u + 1) * 128 + ((g ^ ((u + 1) & 7)) << 4)) =
              (uint16_t)(pk >> 16);
        }
      }
      ptx::fence_proxy_async_smem();
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(bar(P_FULL + b));
    }
    // row sums: this warp's 32 keys, then the four lane quarters
    const float wsum = transpose_reduce<false>(psum, lane);  // token tb + lane % 16
    if (lane < kTTok) reinterpret_cast<float*>(&sh->qsum[tb + lane])[q4] = wsum;
    const bool done =
        __all_sync(0xffffffffu, ok && nbl > 0 && wait_bar(bar(MMA_DONE), 0, abort, a.status));
    group_sync(tg);
    // partial output of this split in row layout [token][dim]: into global
    // memory, or (fused) into this CTA's shared memory where the K ring was
    // (every load has landed, every product is done once MMA_DONE completed)
    float* so = reinterpret_cast<float*>(s_k);   // fused: [128][128] partial O
    float* sml = so + 128 * kHd;                  // fused: [128][2] statistics
    const int dim = 32 * q4 + lane;
    const int64_t pbase = ((int64_t)h * a.splits + sp) * 128;
    if (done && tb < a.L) {
      ptx::tc_fence_after();
      uint32_t rr[kTTok];
      ptx::tmem_ld16(lane_base + kTOCol + tb, rr);
#pragma unroll
      for (int u = 0; u < kTTok; ++u) {
        const int t = tb + u;
        if (t < a.L) {
          const float v = __uint_as_float(rr[u]);
          if (a.fused) so[t * kHd + dim] = v;
          else a.part_o[(pbase + t) * kHd + dim] = v;
        }
      }
    }
    if (q4 == 0 && lane < kTTok) {
      const int t = tb + lane;
      const float4 qs = sh->qsum[t];
      float* pml = a.fused ? sml + 2 * t : a.part_ml + (pbase + t) * 2;
      if (t < a.L) {
        pml[0] = done ? sh->ref[t] : NEG;
        pml[1] = done ? (qs.x + qs.y) + (qs.z + qs.w) : 0.0f;
      }
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 256);
  }
  if (a.fused)
    cluster_merge(reinterpret_cast<const float*>(s_k), a, h, sp, warp, lane, kTThreads / 32);
}

// out[h, r, :] = sum_s 2^(ref_s - M) O_s / sum_s 2^(ref_s - M) l_s, one warp
// per (head, row): lane s holds split s's statistics (32 splits at a time),
// the weights are shuffled to every lane, and each lane adds its 4 dims of
// every split with the loads issued together.
__global__ void __launch_bounds__(256)
tree_attn_combine_kernel(const float* __restrict__ part_o, const float* __restrict__ part_ml,
                         int heads, int splits, int L, float* __restrict__ out) {
  const int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (w >= (int64_t)heads * L) return;
  const int h = (int)(w / L), r = (int)(w - (int64_t)h * L);
  const float NEG = -__int_as_float(0x7f800000);
  const int64_t base = (int64_t)h * splits * 128 + r;  // partial of split s: base + s * 128
  float mx = NEG;
  for (int s0 = 0; s0 < splits; s0 += 32) {
    const int s = s0 + lane;
    if (s < splits && part_ml[(base + (int64_t)s * 128) * 2 + 1] > 0.0f)
      mx = fmaxf(mx, part_ml[(base + (int64_t)s * 128) * 2]);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  float den = 0.0f;
  for (int s0 = 0; s0 < splits; s0 += 32) {
    const int s = s0 + lane;
    float f = 0.0f, l = 0.0f;
    if (s < splits) {
      l = part_ml[(base + (int64_t)s * 128) * 2 + 1];
      if (l > 0.0f) f = exp2f(part_ml[(base + (int64_t)s * 128) * 2] - mx);
      else l = 0.0f;
    }
    float fl = f * l;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) fl += __shfl_xor_sync(0xffffffffu, fl, off);
    den += fl;
    const int n = min(32, splits - s0);
    for (int t = 0; t < n; ++t) {
      const float ft = __shfl_sync(0xffffffffu, f, t);
      if (ft == 0.0f) continue;  // warp-uniform
      const float4 o = *reinterpret_cast<const float4*>(
          part_o + (base + (int64_t)(s0 + t) * 128) * kHd + 4 * lane);
      acc.x += ft * o.x;
      acc.y += ft * o.y;
      acc.z += ft * o.z;
      acc.w += ft * o.w;
    }
  }
  const float inv = den > 0.0f ? 1.0f / den : 0.0f;
  *reinterpret_cast<float4*>(out + ((int64_t)h * L + r) * kHd + 4 * lane) =
      make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
}

sense_status make_map3(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                       uint64_t stride1, uint64_t stride2, uint32_t box_rows) {
  void* fn = nullptr;
  sense_status st = tensor_map_encoder(&fn);
  if (st != SENSE_OK) return st;
  auto enc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {stride1, stride2};
  const cuuint32_t box[3] = {64, box_rows, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(SENSE_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return SENSE_OK;
}

size_t attn_smem_bytes() {
  return 1024 + kQBytes + 2 * kPBytes + kStages * kStageBytes + (11 + 2 * kStages) * 8 +
         sizeof(AttnShared);
}

int attn_splits(int heads, int nb) {
  const int per = std::max(1, sm_count() / heads);
  return std::max(1, std::min(nb, per));
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Trees of at most 64 nodes: the transposed-product kernel over 128-key
// blocks (splits of a head merged in their cluster when <= 8, else by
// tree_attn_combine_kernel through the workspace).
sense_status launch_attn_t(const uint16_t* q, const uint16_t* k_cache, const uint16_t* vt_cache,
                           int heads, int L, int capacity, int prefix_len,
                           const uint32_t* mask_bits, int mask_words, float scale, float* out,
                           void* workspace, uint32_t* status, cudaStream_t s) {
  const int n = prefix_len + L;
  const int nb = (n + kTB - 1) / kTB;
  const int splits = attn_splits(heads, nb);
  alignas(64) CUtensorMap tm_q, tm_k, tm_vt;
  // Q [H, L, 128] in boxes of 64 rows (rows past L read as zero); K [H,
  // capacity, 128] seen up to n keys in boxes of 128 keys; V^T [H, 128,
  // capacity] up to n keys
  sense_status st =
      make_map3(&tm_q, q, kHd, L, heads, (uint64_t)kHd * 2, (uint64_t)L * kHd * 2, kTN);
  if (st == SENSE_OK)
    st = make_map3(&tm_k, k_cache, kHd, n, heads, (uint64_t)kHd * 2, (uint64_t)capacity * kHd * 2,
                   kTB);
  if (st == SENSE_OK)
    st = make_map3(&tm_vt, vt_cache, n, kHd, heads, (uint64_t)capacity * 2,
                   (uint64_t)kHd * capacity * 2, 128);
  if (st != SENSE_OK) return st;
  AttnArgs a{};
  a.L = L;
  a.m = prefix_len;
  a.n = n;
  a.nb = nb;
  a.splits = splits;
  a.bps = (nb + splits - 1) / splits;
  a.scale_log2 = scale * 1.4426950408889634f;
  a.mask = mask_bits;
  a.mask_words = mask_words;
  char* ws = static_cast<char*>(workspace);
  a.part_o = reinterpret_cast<float*>(ws);
  a.part_ml = reinterpret_cast<float*>(ws + align256((size_t)heads * splits * 128 * kHd * 4));
  a.status = status;
  a.out = out;
  a.fused = splits <= 8 ? 1 : 0;
  const size_t smem = attn_t_smem_bytes();
  st = cuda_check(func_smem(reinterpret_cast<const void*>(tree_attn_t_kernel), (int)smem),
                  "cudaFuncSetAttribute(tree_attn_t)");
  if (st != SENSE_OK) return st;
  {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)heads, (unsigned)splits);
    cfg.blockDim = dim3(kTThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = a.fused ? (unsigned)splits : 1u;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    LaunchScope ls(K_TREE_ATTN, s);
    st = cuda_check(cudaLaunchKernelEx(&cfg, tree_attn_t_kernel, tm_q, tm_k, tm_vt, a),
                    "launch tree attention (transposed)");
    if (st != SENSE_OK) return st;
  }
  if (a.fused) return SENSE_OK;
  LaunchScope ls(K_TREE_ATTN, s);
  const int64_t threads = (int64_t)heads * L * 32;
  tree_attn_combine_kernel<<<(unsigned)((threads + 255) / 256), 256, 0, s>>>(
      a.part_o, a.part_ml, heads, splits, L, out);
  return cuda_check(cudaGetLastError(), "launch tree attention combine");
}

}  // namespace
}  // namespace sense

using namespace sense;

extern "C" {

size_t sense_tree_attention_workspace_bytes(int32_t heads, int32_t L, int32_t prefix_len) {
  if (heads < 1 || L < 1 || prefix_len < 0) return 0;
  const int nb = (prefix_len + L + kBN - 1) / kBN;
  const int splits = attn_splits(heads, nb);
  return align256((size_t)heads * splits * 128 * kHd * 4) + align256((size_t)heads * splits * 128 * 8);
}

sense_status sense_tree_attention(const uint16_t* q, const uint16_t* k_cache,
                                  const uint16_t* vt_cache, int32_t heads, int32_t L,
                                  int32_t d_head, int32_t capacity, int32_t prefix_len,
                                  const uint32_t* mask_bits, int32_t mask_words, float scale,
                                  float* out, void* workspace, size_t workspace_bytes,
                                  sense_stream_t stream) {
  if (!q || !k_cache || !vt_cache || !mask_bits || !out || !workspace)
    return fail(SENSE_ERR_INVALID_ARG, "arrays and workspace must be non-NULL");
  if (d_head != kHd) return fail(SENSE_ERR_UNSUPPORTED, "d_head=%d: only 128 is implemented", d_head);
  if (heads < 1 || heads > 65535) return fail(SENSE_ERR_INVALID_ARG, "heads=%d outside [1, 65535]", heads);
  if (L < 1 || L > 128) return fail(SENSE_ERR_INVALID_ARG, "L=%d outside [1, 128]", L);
  if (capacity < 128 || capacity % 128)
    return fail(SENSE_ERR_INVALID_ARG, "capacity=%d must be a positive multiple of 128", capacity);
  if (prefix_len < 0 || (int64_t)prefix_len + L > capacity)
    return fail(SENSE_ERR_INVALID_ARG, "prefix_len=%d + L=%d exceeds capacity=%d", prefix_len, L, capacity);
  if (mask_words < (L + 31) / 32) return fail(SENSE_ERR_INVALID_ARG, "mask_words=%d < ceil(L/32)", mask_words);
  if (!(scale > 0.0f) || scale > 1e30f) return fail(SENSE_ERR_INVALID_ARG, "scale must be positive and finite");
  if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(vt_cache, 16) || !aligned(out, 16))
    return fail(SENSE_ERR_INVALID_ARG, "q, caches and out must be 16-byte aligned");
  if (!aligned(workspace, 256)) return fail(SENSE_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  if (workspace_bytes < sense_tree_attention_workspace_bytes(heads, L, prefix_len))
    return fail(SENSE_ERR_INVALID_ARG, "workspace of %zu bytes < %zu", workspace_bytes,
                sense_tree_attention_workspace_bytes(heads, L, prefix_len));
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int n = prefix_len + L;
  if (L <= kTN) return launch_attn_t(q, k_cache, vt_cache, heads, L, capacity, prefix_len, mask_bits,
                                     mask_words, scale, out, workspace, status, s);
  const int nb = (n + kBN - 1) / kBN;
  const int splits = attn_splits(heads, nb);
  alignas(64) CUtensorMap tm_q, tm_k, tm_vt;
  // Q [H, L, 128]; K [H, capacity, 128] seen up to n keys; V^T [H, 128, capacity] up to n keys
  sense_status st =
      make_map3(&tm_q, q, kHd, L, heads, (uint64_t)kHd * 2, (uint64_t)L * kHd * 2, 128);
  if (st == SENSE_OK)
    st = make_map3(&tm_k, k_cache, kHd, n, heads, (uint64_t)kHd * 2, (uint64_t)capacity * kHd * 2,
                   kBN);
  if (st == SENSE_OK)
    st = make_map3(&tm_vt, vt_cache, n, kHd, heads, (uint64_t)capacity * 2,
                   (uint64_t)kHd * capacity * 2, 128);
  if (st != SENSE_OK) return st;
  AttnArgs a{};
  a.L = L;
  a.m = prefix_len;
  a.n = n;
  a.nb = nb;
  a.splits = splits;
  a.bps = (nb + splits - 1) / splits;
  a.scale_log2 = scale * 1.4426950408889634f;
  a.mask = mask_bits;
  a.mask_words = mask_words;
  char* ws = static_cast<char*>(workspace);
  a.part_o = reinterpret_cast<float*>(ws);
  a.part_ml = reinterpret_cast<float*>(ws + align256((size_t)heads * splits * 128 * kHd * 4));
  a.status = status;
  const size_t smem = attn_smem_bytes();
  st = cuda_check(func_smem(reinterpret_cast<const void*>(tree_attn_kernel), (int)smem), "cudaFuncSetAttribute(tree_attn)");
  if (st != SENSE_OK) return st;
  // up to 8 splits per head: the splits form a cluster and combine in place
  a.out = out;
  a.fused = splits <= 8 ? 1 : 0;
  {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)heads, (unsigned)splits);
    cfg.blockDim = dim3(kAttnThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = a.fused ? (unsigned)splits : 1u;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    LaunchScope ls(K_TREE_ATTN, s);
    st = cuda_check(cudaLaunchKernelEx(&cfg, tree_attn_kernel, tm_q, tm_k, tm_vt, a),
                    "launch tree attention");
    if (st != SENSE_OK) return st;
  }
  if (a.fused) return SENSE_OK;
  LaunchScope ls(K_TREE_ATTN, s);
  const int64_t threads = (int64_t)heads * L * 32;
  tree_attn_combine_kernel<<<(unsigned)((threads + 255) / 256), 256, 0, s>>>(
      a.part_o, a.part_ml, heads, splits, L, out);
  return cuda_check(cudaGetLastError(), "launch tree attention combine");
}

}  // extern "C"
