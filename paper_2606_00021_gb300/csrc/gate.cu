// Soft-gated evaluation (Sec. 3.3, Eqs. 12-19; App. C.4 Alg. 4).
//
// Alg. 4 evaluates argmax, softmax entropy and top-k on every aligned row
// P_align[i, j].  Many (i, j) share a row: position j of candidate i is
// predicted by the row of node gamma[i, j-1] (the root row for j = 0), so the
// distinct rows are the root and the tree's inner nodes.  The gate therefore
// runs in two kernels:
//  1. gate_rows: a persistent grid of warps; each warp takes whole rows
//     (root or inner-node logits) from an atomic counter and streams a row
//     through its own 3-stage shared-memory ring with 1-D bulk copies
//     (cp.async.bulk, 4 KB per stage, completion on an mbarrier; every wait
//     is bounded by clock64 and a timeout sets SENSE_DEVST_TIMEOUT).  Each
//     lane keeps the running max, the sums exp(x - max) and (x - max)
//     exp(x - max) in packed fp32 pairs (entropy H = log Z - S / Z, with
//     ex2 in base-2 units), the index of its first maximum (found in the
//     stage that raised the maximum: lowest index among maxima) and a
//     top-kappa list under (logit desc, index asc).  A lower bound of the
//     row's kappa-th largest value, seeded from the lane maxima of the
//     first stage and refreshed from the lists after stages 1, 3, 7, 15, 31,
//     keeps list updates (warp-voted) off the common path.  All combining is
//     done with warp shuffles: no block barriers.  A node is an inner node
//     iff the next node in preorder is its child, so the test is O(1).
//     With at most one row per SM (a single query's tree) the same warp
//     pass runs as one block per row instead, its warps on consecutive
//     slices, merged in shared memory (gate_row_block_kernel).
//  2. gate_decide: one block per query evaluates B_em, B_ent, B_topk, the
//     lookahead B_con, G, the accepted prefix lengths L_i, i*, and writes
//     the accepted tokens, the next node, its argmax (streaming that row if
//     it is a leaf) and h_next.  When they fit, the query's Gamma, tokens,
//     parents and row statistics are first staged in shared memory with
//     independent loads, so that the block pays one round trip for them.
#include <cooperative_groups.h>
#include <float.h>

#include "common.cuh"
#include "launch.h"
#include "tc_ptx.cuh"

namespace sense {
namespace {

namespace cg = cooperative_groups;

constexpr int kRowThreads = 512;
constexpr int kWarps = kRowThreads / 32;
constexpr int kWStageF4 = 256;                     // float4 per warp stage (4 KB)
constexpr int kWStages = 3;                        // ring depth per warp
constexpr int kLaneF4 = kWStageF4 / 32;            // float4 per lane per stage
constexpr size_t kRingBytes = (size_t)kWarps * kWStages * kWStageF4 * 16;
constexpr size_t kRowSmemMax = 216 * 1024;  // dynamic shared memory of a row block (+ ~8 KB static)
constexpr int kStatsInts = 2 + SENSE_MAX_KAPPA;    // argmax, ent flag, top list
constexpr int kMaxSegs = 16;
constexpr long long kWaitCycles = 4000000000LL;

struct ArgMax {
  float v;
  int i;
};
__device__ __forceinline__ bool better(float va, int ia, float vb, int ib) {
  return va > vb || (va == vb && ia < ib);
}

template <int KM>
struct TopList {
  float v[KM];
  int i[KM];
  __device__ __forceinline__ void init() {
#pragma unroll
    for (int s = 0; s < KM; ++s) {
      v[s] = -FLT_MAX;
      i[s] = 0x7fffffff;
    }
  }
  // Elements arrive in increasing index order within a thread: a later
  // element only displaces strictly smaller values.
  __device__ __forceinline__ void push(float x, int ix) {
    if (x > v[KM - 1]) {
      v[KM - 1] = x;
      i[KM - 1] = ix;
#pragma unroll
      for (int s = KM - 1; s > 0; --s) {
        if (better(v[s], i[s], v[s - 1], i[s - 1])) {
          const float tv = v[s];
          v[s] = v[s - 1];
          v[s - 1] = tv;
          const int ti = i[s];
          i[s] = i[s - 1];
          i[s - 1] = ti;
        }
      }
    }
  }
};

// 2^x (one MUFU op; results below the normal range flush to 0).
__device__ __forceinline__ float exp2_ftz(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Two fp32 lanes in one 64-bit register: packed Blackwell FMA / ADD.
__device__ __forceinline__ uint64_t pk(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void upk(uint64_t r, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(r));
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

constexpr float kLog2e = 1.4426950408889634f;  // log2(e)

template <int KM>
struct RowAcc {
  float m = -FLT_MAX;       // running max (also the argmax value)
  uint64_t z = 0, s = 0;    // packed pairs: sum exp(x - m), sum ((x - m) log2 e) exp(x - m)
  int am = 0x7fffffff;      // index of this thread's first maximum
  float lb = -FLT_MAX;      // lower bound of the row's kappa-th largest value
  TopList<KM> tl;

  __device__ __forceinline__ void rescale(float cm) {
    if (m > -FLT_MAX) {
      const float d2 = (m - cm) * kLog2e;
      const float sc = exp2_ftz(d2);
      float z0, z1, s0, s1;
      upk(z, z0, z1);
      upk(s, s0, s1);
      s = pk(sc * (s0 + d2 * z0), sc * (s1 + d2 * z1));
      z = pk(sc * z0, sc * z1);
    }
    m = cm;
  }

  // Folds one stage: kLaneF4 float4 of this lane (element indices
  // idx[u] * 4 + e, increasing).  Padding slots hold -FLT_MAX.  Called by
  // all 32 lanes of a warp together (it votes).
  __device__ __forceinline__ void add(const float4 (&x)[kLaneF4], const int (&idx)[kLaneF4]) {
    float cm = -FLT_MAX;
#pragma unroll
    for (int u = 0; u < kLaneF4; ++u)
      cm = fmaxf(cm, fmaxf(fmaxf(x[u].x, x[u].y), fmaxf(x[u].z, x[u].w)));
    const bool live = cm > -FLT_MAX;  // false past the end of the range
    if (live && cm > m) {  // a new maximum: its first index in this stage
      rescale(cm);
      int first = 0x7fffffff;
#pragma unroll
      for (int u = kLaneF4 - 1; u >= 0; --u) {  // the last hit from the end is the first
        if (x[u].w == cm) first = idx[u] * 4 + 3;
        if (x[u].z == cm) first = idx[u] * 4 + 2;
        if (x[u].y == cm) first = idx[u] * 4 + 1;
        if (x[u].x == cm) first = idx[u] * 4;
      }
      am = first;
    }
    float thr = fmaxf(tl.v[KM - 1], lb);
    if (__any_sync(0xffffffffu, live && cm >= thr)) {
#pragma unroll
      for (int u = 0; u < kLaneF4; ++u) {
        const float xs[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          if (live && xs[e] >= thr) {  // per-lane list: no vote needed
            tl.push(xs[e], idx[u] * 4 + e);
            thr = fmaxf(tl.v[KM - 1], lb);
          }
        }
      }
    }
    if (live) {
      const uint64_t l2 = pk(kLog2e, kLog2e);
      const uint64_t nmb = pk(-m * kLog2e, -m * kLog2e);
      uint64_t z2 = 0, s2 = 0;  // second chain
#pragma unroll
      for (int u = 0; u < kLaneF4; ++u) {
        float t0, t1, t2, t3;
        upk(fma2(pk(x[u].x, x[u].y), l2, nmb), t0, t1);
        upk(fma2(pk(x[u].z, x[u].w), l2, nmb), t2, t3);
        t0 = fmaxf(t0, -250.0f);  // exp underflows to 0 below
        t1 = fmaxf(t1, -250.0f);
        t2 = fmaxf(t2, -250.0f);
        t3 = fmaxf(t3, -250.0f);
        const uint64_t ea = pk(exp2_ftz(t0), exp2_ftz(t1));
        const uint64_t eb = pk(exp2_ftz(t2), exp2_ftz(t3));
        z = add2(z, ea);
        s = fma2(pk(t0, t1), ea, s);
        z2 = add2(z2, eb);
        s2 = fma2(pk(t2, t3), eb, s2);
      }
      z = add2(z, z2);
      s = add2(s, s2);
    }
  }
};

// Warp-wide best (value desc, index asc) in two warp reductions: the
// largest order-preserving value code, then the smallest index holding it
// (-0 and +0 share a code, as they compare equal).
__device__ __forceinline__ ArgMax warp_best(ArgMax a) {
  const uint32_t c = score_code(a.v);
  const uint32_t cm = __reduce_max_sync(0xffffffffu, c);
  const uint32_t im = __reduce_min_sync(0xffffffffu, c == cm ? (uint32_t)a.i : 0xffffffffu);
  return ArgMax{code_score(cm), (int)im};
}

// Bounded wait on an mbarrier phase; false after ~2 s.
__device__ __forceinline__ bool wait_phase(uint32_t bar, uint32_t parity) {
  if (ptx::mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!ptx::mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > kWaitCycles) return false;
  }
  return true;
}

// kappa-th largest value of the warp's lists (each lane's list sorted):
// kappa rounds of a warp-wide best over the list heads.
template <int KM>
__device__ __forceinline__ float warp_kth(const TopList<KM>& tl, int kappa) {
  float hv[KM];
  int hx[KM];
#pragma unroll
  for (int t = 0; t < KM; ++t) {
    hv[t] = tl.v[t];
    hx[t] = tl.i[t];
  }
  float kth = -FLT_MAX;
  for (int r = 0; r < kappa; ++r) {
    const ArgMax w = warp_best(ArgMax{hv[0], hx[0]});
    kth = w.v;
    if (hx[0] == w.i && hv[0] == w.v) {
#pragma unroll
      for (int t = 0; t < KM - 1; ++t) {
        hv[t] = hv[t + 1];
        hx[t] = hx[t + 1];
      }
      hv[KM - 1] = -FLT_MAX;
      hx[KM - 1] = 0x7fffffff;
    }
  }
  return kth;
}

// Statistics of one segment of a row, merged by the row's last warp.
struct Partial {
  float z, s;  // relative to m
  float m;
  float bv;
  int bi;
  int pad;
  float tv[SENSE_MAX_KAPPA];
  int ti[SENSE_MAX_KAPPA];
};

// Row statistics from its segment partials, written to out.  Called by a
// whole warp: each lane brings one partial (p, or none when p is null),
// then warp reductions.
__device__ void finish_row(const Partial* p, int vocab, int kappa, float thr, int unnormalized,
                           int32_t* __restrict__ out) {
  const int lane = threadIdx.x & 31;
  const bool has = p != nullptr;
  float m = -FLT_MAX, bv = -FLT_MAX;
  float pz = 0.0f, ps = 0.0f;
  int bi = 0x7fffffff;
  float tv[SENSE_MAX_KAPPA];
  int ti[SENSE_MAX_KAPPA];
  if (has) {
    m = p->m;
    pz = p->z;
    ps = p->s;
    bv = p->bv;
    bi = p->bi;
  }
#pragma unroll
  for (int r = 0; r < SENSE_MAX_KAPPA; ++r) {
    tv[r] = (has && r < kappa) ? p->tv[r] : -FLT_MAX;
    ti[r] = (has && r < kappa) ? p->ti[r] : 0x7fffffff;
  }
  float M = m;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
  float Z = 0.0f, Sx = 0.0f;
  if (has && pz > 0.0f) {
    const float d = m - M;
    const float sc = exp2_ftz(d * kLog2e);
    Z = pz * sc;
    Sx = sc * (ps + d * pz);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    Z += __shfl_xor_sync(0xffffffffu, Z, off);
    Sx += __shfl_xor_sync(0xffffffffu, Sx, off);
  }
  const ArgMax b = warp_best(ArgMax{bv, bi});
  int head = 0;
  for (int r = 0; r < kappa; ++r) {
    float hv = -FLT_MAX;
    int hx = 0x7fffffff;
#pragma unroll
    for (int t = 0; t < SENSE_MAX_KAPPA; ++t)
      if (t == head) {
        hv = tv[t];
        hx = ti[t];
      }
    const ArgMax w = warp_best(ArgMax{hv, hx});
    if (lane == 0) out[2 + r] = w.i;
    if (hx == w.i && hv == w.v) ++head;
  }
  if (lane == 0) {
    const float H = logf(Z) - Sx / Z;
    const float score = unnormalized ? H : H / logf((float)vocab);
    out[0] = b.i;
    out[1] = (score > thr) ? 1 : 0;
    for (int r = kappa; r < SENSE_MAX_KAPPA; ++r) out[2 + r] = -1;
  }
}

// One segment [lo4, hi4) of a row (float4 indices), streamed by one warp
// through its ring.  `seq` counts the warp's stages across tasks (it fixes
// buffer and phase of every stage).  Lane 0 receives the partial; returns
// false (whole warp) if a stage never arrived.
template <int KM>
__device__ bool warp_segment(const float* __restrict__ row, int lo4, int hi4, int kappa,
                             float4* ring, uint64_t* bars, uint32_t& seq, uint64_t pol,
                             Partial* out) {
  const int lane = threadIdx.x & 31;
  const float4* row4 = reinterpret_cast<const float4*>(row) + lo4;
  const int n4 = hi4 - lo4;
  const int n = (n4 + kWStageF4 - 1) / kWStageF4;
  auto issue = [&](int j) {  // lane 0: stage j of this row
    const uint32_t g = seq + (uint32_t)j;
    const int f0 = j * kWStageF4;
    const int nf = min(kWStageF4, n4 - f0);
    const uint32_t bar = ptx::smem_u32(bars + (g % kWStages));
    ptx::mbar_arrive_expect_tx(bar, (uint32_t)nf * 16u);
    ptx::bulk_load(ptx::smem_u32(ring + (size_t)(g % kWStages) * kWStageF4), row4 + f0,
                   (uint32_t)nf * 16u, bar, pol);
  };
  int next = min(kWStages - 1, n);  // stages issued (same value in every lane)
  if (lane == 0)
    for (int j = 0; j < next; ++j) issue(j);

  RowAcc<KM> acc;
  acc.tl.init();
  const float4 pad = make_float4(-FLT_MAX, -FLT_MAX, -FLT_MAX, -FLT_MAX);
  bool ok = true;
  for (int i = 0; i < n; ++i) {
    const uint32_t g = seq + (uint32_t)i;
    const bool got = wait_phase(ptx::smem_u32(bars + (g % kWStages)), (g / kWStages) & 1u);
    if (!__all_sync(0xffffffffu, got)) {
      if (lane == 0)  // let the copies in flight land before giving up
        for (int j = i; j < next; ++j) {
          const uint32_t gj = seq + (uint32_t)j;
          wait_phase(ptx::smem_u32(bars + (gj % kWStages)), (gj / kWStages) & 1u);
        }
      ok = false;
      break;
    }
    if (next < n) {  // every lane is past stage i-1: refill its buffer
      if (lane == 0) issue(next);
      ++next;
    }
    const float4* st = ring + (size_t)(g % kWStages) * kWStageF4;
    const int f0 = i * kWStageF4;
    const int nf = min(kWStageF4, n4 - f0);
    float4 x[kLaneF4];
    int idx[kLaneF4];
    if (nf == kWStageF4) {
#pragma unroll
      for (int u = 0; u < kLaneF4; ++u) {
        x[u] = st[lane + 32 * u];
        idx[u] = lo4 + f0 + lane + 32 * u;
      }
    } else {
#pragma unroll
      for (int u = 0; u < kLaneF4; ++u) {
        const int j = lane + 32 * u;
        x[u] = (j < nf) ? st[j] : pad;
        idx[u] = lo4 + f0 + j;
      }
    }
    if (i == 0) {
      // seed the bound: the kappa-th largest lane maximum of the first stage
      float cm = -FLT_MAX;
#pragma unroll
      for (int u = 0; u < kLaneF4; ++u)
        cm = fmaxf(cm, fmaxf(fmaxf(x[u].x, x[u].y), fmaxf(x[u].z, x[u].w)));
      float b = -FLT_MAX;
      for (int r = 0; r < kappa; ++r) {
        const ArgMax w = warp_best(ArgMax{cm, lane});
        b = w.v;
        if (lane == w.i) cm = -FLT_MAX;
      }
      acc.lb = b;
    }
    acc.add(x, idx);
    if (((i + 2) & (i + 1)) == 0 && i < 32 && i + 1 < n)  // after stages 1, 3, 7, 15, 31
      acc.lb = fmaxf(acc.lb, warp_kth<KM>(acc.tl, kappa));
  }
  seq += (uint32_t)n;
  if (!ok) return false;
  float z0, z1, s0, s1;
  upk(acc.z, z0, z1);
  upk(acc.s, s0, s1);
  const float lz = z0 + z1;
  const float ls = (s0 + s1) * (1.0f / kLog2e);  // natural-log units
  float M = acc.m;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
  float z = 0.0f, s = 0.0f;
  if (lz > 0.0f) {  // rescale this lane's sums to the row max
    const float d = acc.m - M;
    const float sc = exp2_ftz(d * kLog2e);
    z = lz * sc;
    s = sc * (ls + d * lz);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    z += __shfl_xor_sync(0xffffffffu, z, off);
    s += __shfl_xor_sync(0xffffffffu, s, off);
  }
  const ArgMax am = warp_best(ArgMax{acc.m, acc.am});
  if (lane == 0) {
    out->z = z;
    out->s = s;
    out->m = M;
    out->bv = am.v;
    out->bi = am.i;
  }
  // top-kappa: kappa rounds of a warp-wide best over the list heads
  for (int r = 0; r < kappa; ++r) {
    const ArgMax w = warp_best(ArgMax{acc.tl.v[0], acc.tl.i[0]});
    if (lane == 0) {
      out->tv[r] = w.v;
      out->ti[r] = w.i;
    }
    if (acc.tl.i[0] == w.i && acc.tl.v[0] == w.v) {
#pragma unroll
      for (int t = 0; t < KM - 1; ++t) {
        acc.tl.v[t] = acc.tl.v[t + 1];
        acc.tl.i[t] = acc.tl.i[t + 1];
      }
      acc.tl.v[KM - 1] = -FLT_MAX;
      acc.tl.i[KM - 1] = 0x7fffffff;
    }
  }
  __syncwarp();
  return true;
}

template <int KM>
__global__ void __launch_bounds__(kRowThreads, 1)
gate_rows_kernel(const int32_t* __restrict__ parent, const int32_t* __restrict__ num_nodes,
                 int q_count, int cap, const float* __restrict__ root_logits,
                 const float* __restrict__ node_logits, int vocab, int kappa, float thr,
                 int unnormalized, int segs, int seg4, unsigned* __restrict__ next_task,
                 Partial* __restrict__ parts, unsigned* __restrict__ done,
                 int32_t* __restrict__ stats, uint32_t* status) {
  extern __shared__ __align__(128) float4 ring_all[];
  __shared__ __align__(8) uint64_t bars_all[kWarps * kWStages];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  pdl_wait();
  pdl_launch_dependents();
  if (threadIdx.x == 0) {
    for (int b = 0; b < kWarps * kWStages; ++b) ptx::mbar_init(ptx::smem_u32(bars_all + b), 1);
    ptx::fence_barrier_init();
  }
  __syncthreads();
  float4* ring = ring_all + (size_t)wid * kWStages * kWStageF4;
  uint64_t* bars = bars_all + wid * kWStages;
  const uint64_t pol = (lane == 0) ? ptx::policy_evict_first() : 0ull;
  __shared__ Partial s_part[kWarps];  // the partial of a one-piece row
  const unsigned n_tasks = (unsigned)q_count * (unsigned)(cap + 1) * (unsigned)segs;
  const int n4 = vocab >> 2;
  uint32_t seq = 0;
  while (true) {
    unsigned t = 0;
    if (lane == 0) t = atomicAdd(next_task, 1u);
    t = __shfl_sync(0xffffffffu, t, 0);
    if (t >= n_tasks) break;
    const unsigned rid = t / (unsigned)segs;  // row task: q * (cap + 1) + slot
    const int seg = (int)(t - rid * (unsigned)segs);
    const int q = (int)(rid / (unsigned)(cap + 1));
    const int slot = (int)(rid - (unsigned)q * (unsigned)(cap + 1));  // 0 = root, 1 + n = node n
    const float* row;
    if (slot == 0) {
      row = root_logits + (int64_t)q * vocab;
    } else {
      const int nd = slot - 1;
      const int nn = min(num_nodes[q], cap);
      const bool inner = (nd + 1 < nn) && parent[(int64_t)q * cap + nd + 1] == nd;
      if (!inner) continue;
      row = node_logits + ((int64_t)q * cap + nd) * vocab;
    }
    const int lo4 = seg * seg4;
    const int hi4 = min(n4, lo4 + seg4);
    Partial* slot_out = (segs == 1) ? &s_part[wid] : parts + (int64_t)rid * segs + seg;
    if (!warp_segment<KM>(row, lo4, hi4, kappa, ring, bars, seq, pol, slot_out)) {
      if (lane == 0) raise_status(status, SENSE_DEVST_TIMEOUT);
      break;
    }
    int32_t* out = stats + (int64_t)rid * kStatsInts;
    if (segs == 1) {
      __syncwarp();
      finish_row(lane == 0 ? &s_part[wid] : nullptr, vocab, kappa, thr, unnormalized, out);
    } else {
      // the row's last segment to finish merges the partials
      unsigned last = 0;
      if (lane == 0) {
        __threadfence();
        last = atomicAdd(&done[rid], 1u) == (unsigned)segs - 1u;
      }
      last = __shfl_sync(0xffffffffu, last, 0);
      if (last) {
        __threadfence();
        finish_row(lane < segs ? parts + (int64_t)rid * segs + lane : nullptr, vocab, kappa, thr,
                   unnormalized, out);
        if (lane == 0) done[rid] = 0u;
      }
    }
    __syncwarp();
  }
}

constexpr int kDecideThreads = 1024;

// Shared memory of a staged decide block: Gamma, tokens, parents and the
// row statistics of one query, then the flags.
size_t decide_stage_bytes(int k, int m, int cap) {
  return sizeof(int32_t) * ((size_t)k * m + 2 * (size_t)cap + (size_t)(cap + 1) * kStatsInts) +
         (size_t)k * m;
}
constexpr size_t kDecideStageMax = 96 * 1024;

// 4-byte asynchronous global -> shared copy (no register round trip: every
// copy of a thread is in flight at once); cp_async_wait_all() completes them.
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(ptx::smem_u32(dst)), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_all;" ::: "memory");
}

// Issues the asynchronous copies of query q's Gamma, tokens and parents into
// a staged decide block's shared memory (completed by the same threads'
// cp_async_wait_all() in decide_block).
__device__ __forceinline__ void decide_stage_inputs(const GateArgs& a, int q, int32_t* s_dyn) {
  const int km = a.k * a.m, cap = a.cap;
  int32_t* sg = s_dyn;
  int32_t* stk = sg + km;
  int32_t* spr = stk + cap;
  const int32_t* gam = a.gamma + (int64_t)q * km;
  const int32_t* tok = a.tokens + (int64_t)q * cap;
  const int32_t* par = a.parent + (int64_t)q * cap;
  for (int i = threadIdx.x; i < km; i += blockDim.x) cp_async4(sg + i, gam + i);
  for (int i = threadIdx.x; i < cap; i += blockDim.x) {
    cp_async4(stk + i, tok + i);
    cp_async4(spr + i, par + i);
  }
}

// The decision of query q by one block (any multiple of 32 threads up to
// 1024).  s_dyn: staged ? [Gamma k*m][tokens cap][parents cap][stats
// (cap+1) rows] : nothing, then flags [k*m]: bit0 valid, bit1 em, bit2 ent,
// bit3 topk, bit4 G.  `fresh` (staged only): the statistics were written
// by other blocks of the running grid, so they are read from L2 with plain
// loads rather than copied through L1.  `prestaged`: the same threads
// already issued decide_stage_inputs into s_dyn.
__device__ __forceinline__ void decide_block(const GateArgs& a, const int32_t* __restrict__ stats, int staged,
                             int q, int32_t* s_dyn, bool fresh, bool prestaged = false) {
  __shared__ int s_L[SENSE_MAX_K];
  __shared__ int s_best[32];
  __shared__ int s_istar, s_lstar, s_next, s_nn;
  __shared__ ArgMax s_w[32];
  const int k = a.k, m = a.m, cap = a.cap, km = k * m;
  const int32_t* gam = a.gamma + (int64_t)q * km;
  const int32_t* tok = a.tokens + (int64_t)q * cap;
  const int32_t* par = a.parent + (int64_t)q * cap;
  const int32_t* st = stats + (int64_t)q * (cap + 1) * kStatsInts;
  uint8_t* s_flags = reinterpret_cast<uint8_t*>(s_dyn);
  if (staged) {  // one round trip for everything the block reads more than once
    int32_t* sg = s_dyn;
    int32_t* stk = sg + km;
    int32_t* spr = stk + cap;
    int32_t* sst = spr + cap;
    if (!prestaged) decide_stage_inputs(a, q, s_dyn);
    if (fresh) {  // four loads per thread in flight before their stores
      const int ns = (cap + 1) * kStatsInts;
      for (int i0 = threadIdx.x; i0 < ns; i0 += 4 * blockDim.x) {
        int32_t v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int i = i0 + u * blockDim.x;
          v[u] = i < ns ? __ldcg(st + i) : 0;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int i = i0 + u * blockDim.x;
          if (i < ns) sst[i] = v[u];
        }
      }
    } else
      for (int i = threadIdx.x; i < (cap + 1) * kStatsInts; i += blockDim.x) cp_async4(sst + i, st + i);
    if (threadIdx.x == 0) cp_async4(&s_nn, a.num_nodes + q);
    cp_async_wait_all();
    s_flags = reinterpret_cast<uint8_t*>(sst + (cap + 1) * kStatsInts);
    gam = sg;
    tok = stk;
    par = spr;
    st = sst;
    __syncthreads();
  } else if (threadIdx.x == 0) {
    s_nn = a.num_nodes[q];
  }

  for (int e = threadIdx.x; e < km; e += blockDim.x) {
    const int j = e % m;
    const int nd = gam[e];
    const int pn = (j == 0) ? -1 : gam[e - 1];
    uint8_t f = 0;
    if (nd >= cap || pn >= cap || (j > 0 && nd >= 0 && pn < 0)) {
      raise_status(a.status, SENSE_DEVST_INTERNAL);  // malformed tree: position dropped
    } else if (nd >= 0) {
      const int slot = 1 + pn;
      const int32_t* rs = st + (int64_t)slot * kStatsInts;
      const int t = tok[nd];
      f |= 1;
      if (rs[0] == t) f |= 2;
      if (rs[1]) f |= 4;
      for (int r = 0; r < a.kappa; ++r) {
        if (rs[2 + r] == t) {
          f |= 8;
          break;
        }
      }
    }
    s_flags[e] = f;
  }
  __syncthreads();
  // B_con over the strictly-future window j+1..j+W; positions past the span
  // and dropped positions count as mismatches.  Then G.
  {
    // bit 4 (G) of a position is written in place: readers of other
    // positions only use bits 0-1, which no thread changes here
    for (int e = threadIdx.x; e < km; e += blockDim.x) {
      const int i = e / m, j = e - i * m;
      const uint8_t f = s_flags[e];
      int mism = 0;
      for (int u = j + 1; u <= j + a.window; ++u) {
        if (u >= m) {
          mism += j + a.window - u + 1;
          break;
        }
        const uint8_t fu = s_flags[i * m + u];
        mism += ((fu & 1) && (fu & 2)) ? 0 : 1;
      }
      const bool con = mism <= a.tau;
      const bool valid = f & 1, em = f & 2, ent = f & 4, tk = f & 8;
      if (valid && (em || (ent && (tk || con)))) s_flags[e] = f | 16;
    }
    __syncthreads();
  }
  if (a.G) {
    for (int e = threadIdx.x; e < km; e += blockDim.x)
      a.G[(int64_t)q * km + e] = (s_flags[e] >> 4) & 1;
  }
  // L_i and i* = lowest i with the largest L_i.
  for (int i = threadIdx.x; i < k; i += blockDim.x) {
    int run = 0;
    while (run < m && (s_flags[i * m + run] & 16)) ++run;
    s_L[i] = run - 1;
  }
  __syncthreads();
  {
    int bl = -2, bi = 0x7fffffff;
    for (int i = threadIdx.x; i < k; i += blockDim.x) {
      if (s_L[i] > bl || (s_L[i] == bl && i < bi)) {
        bl = s_L[i];
        bi = i;
      }
    }
    // pack (L desc, i asc) into one int: larger = better
    int key = ((bl + 2) << 11) | (2047 - min(bi, 2047));
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) key = max(key, __shfl_xor_sync(0xffffffffu, key, off));
    if ((threadIdx.x & 31) == 0) s_best[threadIdx.x >> 5] = key;
    __syncthreads();
    if (threadIdx.x < 32) {
      int kk = (threadIdx.x < (int)(blockDim.x >> 5)) ? s_best[threadIdx.x] : 0;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) kk = max(kk, __shfl_xor_sync(0xffffffffu, kk, off));
      if (threadIdx.x == 0) {
        const int istar = 2047 - (kk & 2047);
        const int lstar = (kk >> 11) - 2;
        s_istar = istar;
        s_lstar = lstar;
        s_next = (lstar >= 0) ? gam[istar * m + lstar] : -1;
        a.i_star[q] = istar;
        a.L_star[q] = lstar;
        a.n_accept[q] = lstar + 1;
        a.next_node[q] = s_next;
      }
    }
    __syncthreads();
  }
  const int istar = s_istar, lstar = s_lstar, nxt = s_next;
  for (int j = threadIdx.x; j < m; j += blockDim.x)
    a.accepted[(int64_t)q * m + j] = (j <= lstar) ? tok[gam[istar * m + j]] : -1;
  // h_next: the hidden state of the next node (root state when nxt == -1).
  {
    const uint16_t* hs = (nxt < 0) ? a.root_hidden + (int64_t)q * a.d
                                   : a.node_hidden + ((int64_t)q * cap + nxt) * a.d;
    const uint4* h4 = reinterpret_cast<const uint4*>(hs);
    uint4* o4 = reinterpret_cast<uint4*>(a.h_next + (int64_t)q * a.d);
    for (int i = threadIdx.x; i < (a.d >> 3); i += blockDim.x) o4[i] = h4[i];
  }
  // next anchor: argmax of the next node's logits row.
  const int nn = min(s_nn, cap);
  const bool have = (nxt < 0) || ((nxt + 1 < nn) && par[nxt + 1] == nxt);
  if (have) {
    if (threadIdx.x == 0) a.next_anchor[q] = st[(int64_t)(nxt + 1) * kStatsInts];
    return;
  }
  const float4* r4 = reinterpret_cast<const float4*>(a.node_logits + ((int64_t)q * cap + nxt) * a.vocab);
  float bv = -FLT_MAX;
  int bi = 0x7fffffff;
  for (int c = threadIdx.x; c < (a.vocab >> 2); c += blockDim.x) {
    const float4 x = __ldcs(r4 + c);
    const float xs[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      if (xs[e] > bv) {
        bv = xs[e];
        bi = c * 4 + e;
      }
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
    if (better(ov, oi, bv, bi)) {
      bv = ov;
      bi = oi;
    }
  }
  if ((threadIdx.x & 31) == 0) s_w[threadIdx.x >> 5] = ArgMax{bv, bi};
  __syncthreads();
  if (threadIdx.x < 32) {
    ArgMax w = (threadIdx.x < (int)(blockDim.x >> 5)) ? s_w[threadIdx.x] : ArgMax{-FLT_MAX, 0x7fffffff};
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, w.v, off);
      const int oi = __shfl_xor_sync(0xffffffffu, w.i, off);
      if (better(ov, oi, w.v, w.i)) {
        w.v = ov;
        w.i = oi;
      }
    }
    if (threadIdx.x == 0) a.next_anchor[q] = w.i;
  }
}

// The streaming pass of one row by the NC blocks of its cluster (all of
// them call it); warp 0 of block 0 writes the row's statistics to `out`.
template <int KM, int NC>
__device__ void row_block_pass(const float* __restrict__ row, int vocab, int kappa, float thr,
                               int unnormalized, int seg4, int32_t* __restrict__ out,
                               uint32_t* status, int crank, float4* ring_all, uint64_t* bars_all,
                               Partial* s_part, int& s_fail) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    for (int b = 0; b < kWarps * kWStages; ++b) ptx::mbar_init(ptx::smem_u32(bars_all + b), 1);
    ptx::fence_barrier_init();
    s_fail = 0;
  }
  __syncthreads();
  const int n4 = vocab >> 2;
  const int lo4 = min(n4, (crank * kWarps + wid) * seg4);
  const int hi4 = min(n4, lo4 + seg4);
  if (lo4 < hi4) {
    float4* ring = ring_all + (size_t)wid * kWStages * kWStageF4;
    uint64_t* bars = bars_all + wid * kWStages;
    const uint64_t pol = (lane == 0) ? ptx::policy_evict_first() : 0ull;
    uint32_t seq = 0;
    if (!warp_segment<KM>(row, lo4, hi4, kappa, ring, bars, seq, pol, &s_part[wid])) {
      if (lane == 0) {
        raise_status(status, SENSE_DEVST_TIMEOUT);
        s_fail = 1;
      }
    }
  } else if (lane == 0) {  // empty slice: a neutral partial
    Partial& p = s_part[wid];
    p.z = 0.0f;
    p.s = 0.0f;
    p.m = -FLT_MAX;
    p.bv = -FLT_MAX;
    p.bi = 0x7fffffff;
    for (int r = 0; r < SENSE_MAX_KAPPA; ++r) {
      p.tv[r] = -FLT_MAX;
      p.ti[r] = 0x7fffffff;
    }
  }
  if constexpr (NC == 1) {
    __syncthreads();
    if (wid == 0 && !s_fail)
      finish_row(lane < kWarps ? &s_part[lane] : nullptr, vocab, kappa, thr, unnormalized, out);
  } else {
    cg::cluster_group cl = cg::this_cluster();
    cl.sync();  // every block's partials (and failure flag) are written
    if (crank == 0 && wid == 0) {
      const int src = lane / kWarps;  // block holding this lane's partial
      const Partial* pp = cl.map_shared_rank(&s_part[lane - src * kWarps], src);
      bool fail = false;
      for (int r = 0; r < NC; ++r) fail |= *cl.map_shared_rank(&s_fail, r) != 0;
      if (!fail) finish_row(lane < NC * kWarps ? pp : nullptr, vocab, kappa, thr, unnormalized, out);
    }
    cl.sync();  // the other blocks' shared memory stays alive until it is read
  }
}

// Few rows with short slices: NC blocks per row (a cluster of NC blocks
// when NC > 1), whose kWarps * NC warps stream consecutive slices of seg4
// float4 each through their own rings.  Each block keeps its warps'
// partials in shared memory; warp 0 of the cluster's first block merges
// them all, reading the other block's partials through distributed shared
// memory.  No task counter, no partials in global memory, no grid-wide
// atomics: the row's latency is one streaming pass plus block and cluster
// barriers.  With `decide_done` set, the decision of each query runs in the
// same launch: every row slot of query q (rows without logits included)
// counts itself on decide_done[q] after its statistics are written, and the
// first block of the slot that arrives last runs the decide block and
// resets the counter to zero for the next call.
template <int KM, int NC>
__global__ void __launch_bounds__(kRowThreads, 1)
gate_row_block_kernel(const int32_t* __restrict__ parent, const int32_t* __restrict__ num_nodes,
                      int cap, const float* __restrict__ root_logits,
                      const float* __restrict__ node_logits, int vocab, int kappa, float thr,
                      int unnormalized, int seg4, int32_t* __restrict__ stats, uint32_t* status,
                      GateArgs a, int staged, unsigned* __restrict__ decide_done, int prestage) {
  static_assert(NC >= 1 && NC * kWarps <= 32, "one merging warp holds every partial");
  extern __shared__ __align__(128) float4 ring_all[];
  __shared__ __align__(8) uint64_t bars_all[kWarps * kWStages];
  __shared__ Partial s_part[kWarps];
  __shared__ int s_fail;
  __shared__ int s_last;
  pdl_wait();  // the tree (and everything before it) is complete
  pdl_launch_dependents();
  const int rid = blockIdx.x / NC;  // q * (cap + 1) + slot
  const int crank = blockIdx.x - rid * NC;  // rank in the cluster (clusters of NC along x)
  const int q = rid / (cap + 1);
  const int slot = rid - q * (cap + 1);  // 0 = root, 1 + n = node n
  const float* row = nullptr;
  if (slot == 0) {
    row = root_logits + (int64_t)q * vocab;
  } else {
    const int nd = slot - 1;
    const int nn = min(num_nodes[q], cap);
    const bool inner = (nd + 1 < nn) && parent[(int64_t)q * cap + nd + 1] == nd;
    // depends on the row only: the whole cluster skips the row
    if (inner) row = node_logits + ((int64_t)q * cap + nd) * vocab;
  }
  // the decision's inputs that the trie wrote go to shared memory past the
  // ring now, so the block that runs the decision waits only for the stats
  int32_t* s_dec = reinterpret_cast<int32_t*>(reinterpret_cast<char*>(ring_all) + kRingBytes);
  if (decide_done != nullptr && prestage && crank == 0) decide_stage_inputs(a, q, s_dec);
  if (row) row_block_pass<KM, NC>(row, vocab, kappa, thr, unnormalized, seg4,
                                  stats + (int64_t)rid * kStatsInts, status, crank, ring_all,
                                  bars_all, s_part, s_fail);
  if (decide_done == nullptr || crank != 0) return;
  __threadfence();  // this block's statistics before its count
  __syncthreads();
  if (threadIdx.x == 0) {
    const bool last = atomicAdd(&decide_done[q], 1u) == (unsigned)cap;  // cap + 1 slots
    if (last) atomicExch(&decide_done[q], 0u);
    s_last = last;
  }
  __syncthreads();
  if (!s_last) {
    if (prestage) cp_async_wait_all();  // no copy into this block's memory outlives it
    return;
  }
  __threadfence();  // every slot's statistics are visible
  if (prestage) decide_block(a, stats, staged, q, s_dec, true, true);
  else decide_block(a, stats, staged, q, reinterpret_cast<int32_t*>(ring_all), true);
}

__global__ void __launch_bounds__(kDecideThreads)
gate_decide_kernel(GateArgs a, const int32_t* __restrict__ stats, int staged) {
  extern __shared__ __align__(16) int32_t s_dyn[];
  pdl_wait();  // every row statistic is written
  decide_block(a, stats, staged, blockIdx.x, s_dyn, false);
}

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

}  // namespace

// Segments per row: enough row pieces for every streaming warp of the
// grid, each piece at least two stages long.
int gate_segments(int q, int cap, int vocab) {
  const int64_t rows = (int64_t)q * (cap + 1);
  const int64_t warps = (int64_t)sm_count() * kWarps;
  int64_t segs = (warps + rows - 1) / rows;
  const int64_t by_len = (vocab >> 2) / (2 * kWStageF4);
  if (segs > by_len) segs = by_len;
  if (segs > kMaxSegs) segs = kMaxSegs;
  if (segs < 1) segs = 1;
  return (int)segs;
}

size_t gate_workspace_bytes(int q, int cap, int kappa) {
  (void)kappa;
  const size_t rows = (size_t)q * (cap + 1);
  const int segs = gate_segments(q, cap, 1 << 30);  // upper bound over vocabularies
  size_t b = align256(rows * kStatsInts * sizeof(int32_t));
  b += 256;                                      // task counter
  b += align256((size_t)q * sizeof(unsigned));  // per-query decide counters
  if (segs > 1) b += align256(rows * segs * sizeof(Partial)) + align256(rows * sizeof(unsigned));
  return b;
}

sense_status launch_gate(const GateArgs& a, cudaStream_t s) {
  const size_t rows = (size_t)a.q * (a.cap + 1);
  char* ws = static_cast<char*>(a.workspace);
  int32_t* stats = reinterpret_cast<int32_t*>(ws);
  ws += align256(rows * kStatsInts * sizeof(int32_t));
  unsigned* next_task = reinterpret_cast<unsigned*>(ws);
  ws += 256;
  unsigned* decide_done = reinterpret_cast<unsigned*>(ws);  // zero between calls
  ws += align256((size_t)a.q * sizeof(unsigned));
  const int n4 = a.vocab >> 2;
  const size_t staged_smem = decide_stage_bytes(a.k, a.m, a.cap);
  const int staged = staged_smem <= kDecideStageMax ? 1 : 0;
  sense_status st = SENSE_OK;
  // Few rows, each warp's slice inside its ring: blocks per row (two as a
  // cluster when the rows leave room for it).
  const int64_t sms = sm_count();
  const bool pair = 2 * (int64_t)rows <= sms &&
                    (n4 + 2 * kWarps - 1) / (2 * kWarps) <= kWStages * kWStageF4;
  const bool single = (int64_t)rows <= sms && (n4 + kWarps - 1) / kWarps <= kWStages * kWStageF4;
  if (pair || single) {
    const int nc = pair ? 2 : 1;
    const int slice4 = (n4 + nc * kWarps - 1) / (nc * kWarps);
    void (*kern)(const int32_t*, const int32_t*, int, const float*, const float*, int, int, float,
                 int, int, int32_t*, uint32_t*, GateArgs, int, unsigned*, int);
    if (pair) kern = (a.kappa <= 4) ? gate_row_block_kernel<4, 2>
                                     : gate_row_block_kernel<SENSE_MAX_KAPPA, 2>;
    else kern = (a.kappa <= 4) ? gate_row_block_kernel<4, 1>
                               : gate_row_block_kernel<SENSE_MAX_KAPPA, 1>;
    // the decision's staged inputs past the ring when they fit beside it
    const size_t dec_bytes = (staged_smem + 15) & ~(size_t)15;
    const int prestage = (staged && kRingBytes + dec_bytes <= kRowSmemMax) ? 1 : 0;
    const size_t row_smem = kRingBytes + (prestage ? dec_bytes : 0);
    st = cuda_check(
        func_smem(reinterpret_cast<const void*>(kern), (int)row_smem),
        "cudaFuncSetAttribute(gate_row_block)");
    if (st != SENSE_OK) return st;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(rows * nc));
    cfg.blockDim = dim3(kRowThreads);
    cfg.dynamicSmemBytes = row_smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)nc;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    // the decision runs in the same launch (in the last row slot of each
    // query) when its staged inputs fit the ring's shared memory
    unsigned* fuse = staged ? decide_done : nullptr;
    LaunchScope ls(K_GATE_ROWS, s);
    st = cuda_check(cudaLaunchKernelEx(&cfg, kern, a.parent, a.num_nodes, a.cap, a.root_logits,
                                       a.node_logits, a.vocab, a.kappa, a.thr, a.unnormalized,
                                       slice4, stats, a.status, a, staged, fuse, prestage),
                    "launch gate_row_block");
    if (st != SENSE_OK) return st;
    if (fuse) return SENSE_OK;
  } else {
    const int segs = gate_segments(a.q, a.cap, a.vocab);
    const int seg4 = (n4 + segs - 1) / segs;
    Partial* parts = reinterpret_cast<Partial*>(ws);
    unsigned* done = nullptr;
    if (segs > 1) done = reinterpret_cast<unsigned*>(ws + align256(rows * segs * sizeof(Partial)));
    st = cuda_check(cudaMemsetAsync(next_task, 0, sizeof(unsigned), s), "clear gate task counter");
    if (st != SENSE_OK) return st;
    if (segs > 1) {
      st = cuda_check(cudaMemsetAsync(done, 0, rows * sizeof(unsigned), s), "clear gate counters");
      if (st != SENSE_OK) return st;
    }
    auto k4 = gate_rows_kernel<4>;
    auto k16 = gate_rows_kernel<SENSE_MAX_KAPPA>;
    auto kern = (a.kappa <= 4) ? k4 : k16;
    st = cuda_check(
        func_smem(reinterpret_cast<const void*>(kern), (int)kRingBytes),
        "cudaFuncSetAttribute(gate_rows)");
    if (st != SENSE_OK) return st;
    // persistent: one block of kWarps row-streaming warps per SM; with few
    // row pieces, spread them over as many SMs as there are pieces
    int64_t blocks = sm_count();
    if (blocks > (int64_t)rows * segs) blocks = (int64_t)rows * segs;
    LaunchScope ls(K_GATE_ROWS, s);
    kern<<<(unsigned)blocks, kRowThreads, kRingBytes, s>>>(
        a.parent, a.num_nodes, a.q, a.cap, a.root_logits, a.node_logits, a.vocab, a.kappa, a.thr,
        a.unnormalized, segs, seg4, next_task, parts, done, stats, a.status);
    st = cuda_check(cudaGetLastError(), "launch gate_rows");
    if (st != SENSE_OK) return st;
  }
  const size_t smem = staged ? staged_smem : (size_t)a.k * a.m;
  if (smem > 48 * 1024) {
    st = cuda_check(func_smem(reinterpret_cast<const void*>(gate_decide_kernel), (int)smem),
                    "cudaFuncSetAttribute(gate_decide)");
    if (st != SENSE_OK) return st;
  }
  const int threads = (a.k * a.m <= 4096) ? 256 : kDecideThreads;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)a.q);
  cfg.blockDim = dim3((unsigned)threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  LaunchScope ls(K_GATE_DECIDE, s);
  return cuda_check(cudaLaunchKernelEx(&cfg, gate_decide_kernel, a, (const int32_t*)stats, staged),
                    "launch gate_decide");
}

}  // namespace sense
