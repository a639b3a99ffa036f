// Soft-gated evaluation (Sec. 3.3, Eqs. 12-19; App. C.4 Alg. 4).
//
// Alg. 4 evaluates argmax, softmax entropy and top-k on every aligned row
// P_align[i, j].  Many (i, j) share a row: position j of candidate i is
// predicted by the row of node gamma[i, j-1] (the root row for j = 0), so the
// distinct rows are the root and the tree's inner nodes.  The gate therefore
// runs in two kernels:
//  1. gate_rows: each needed row is cut into `segs` segments, one block per
//     segment.  Thread 0 streams the segment through a 4-stage shared-memory
//     ring with 1-D bulk copies (cp.async.bulk, 16 KB per stage, completion
//     on an mbarrier; every wait is bounded by clock64 and a timeout sets
//     SENSE_DEVST_TIMEOUT).  From shared memory each thread keeps the running
//     max, sum exp(x - max) and sum (x - max) exp(x - max) (entropy
//     H = log Z - S / Z, accumulated with ex2 in base-2 units), the argmax
//     (lowest index among maxima) and a top-kappa list under (logit desc,
//     index asc); after the first stage the block's kappa-th largest value
//     bounds the row's kappa-th largest from below, and warp votes keep list
//     updates off the common path.  The block combines its threads (fp64),
//     writes a partial, and the last block of a row to finish (an atomic
//     counter per row) merges the segments into the row's statistics.  A
//     node is an inner node iff the next node in preorder is its child, so
//     the test is O(1).
//  2. gate_decide: one block per query evaluates B_em, B_ent, B_topk, the
//     lookahead B_con, G, the accepted prefix lengths L_i, i*, and writes
//     the accepted tokens, the next node, its argmax (streaming that row if
//     it is a leaf) and h_next.
#include <float.h>

#include "common.cuh"
#include "launch.h"
#include "tc_ptx.cuh"

namespace sense {
namespace {

constexpr int kRowThreads = 256;
constexpr int kStageBytes = 16384;                 // one ring stage
constexpr int kStageF4 = kStageBytes / 16;         // float4 per stage
constexpr int kStages = 4;
constexpr int kVec = kStageF4 / kRowThreads;       // float4 per thread per stage
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

// Statistics of one segment of a row (workspace).
struct Partial {
  double z, s;  // relative to m
  float m;
  float bv;
  int bi;
  int pad;
  float tv[SENSE_MAX_KAPPA];
  int ti[SENSE_MAX_KAPPA];
};

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

constexpr float kLog2e = 1.4426950408889634f;  // log2(e)

template <int KM>
struct RowAcc {
  float m = -FLT_MAX;  // running max (also the argmax value)
  float z0 = 0.0f, z1 = 0.0f;    // sum exp(x - m), two chains
  float s0 = 0.0f, s1 = 0.0f;    // sum ((x - m) log2 e) exp(x - m), two chains
  int mstage = -1;     // stage holding this thread's first maximum
  float lb = -FLT_MAX; // lower bound of the row's kappa-th largest value
  TopList<KM> tl;

  // Folds kVec float4 (element indices idx[u] * 4 + e, increasing) of stage
  // `st` into the state.  Padding slots hold -FLT_MAX and contribute
  // nothing.  Called by all 32 lanes of a warp together (it votes).
  __device__ __forceinline__ void add(const float4 (&x)[kVec], const int (&idx)[kVec], int st) {
    float cm = -FLT_MAX;
#pragma unroll
    for (int u = 0; u < kVec; ++u)
      cm = fmaxf(cm, fmaxf(fmaxf(x[u].x, x[u].y), fmaxf(x[u].z, x[u].w)));
    const bool live = cm > -FLT_MAX;  // false past the end of the segment
    if (live && cm > m) {
      if (m > -FLT_MAX) {
        const float d2 = (m - cm) * kLog2e;
        const float sc = exp2_ftz(d2);
        s0 = sc * (s0 + d2 * z0);
        s1 = sc * (s1 + d2 * z1);
        z0 *= sc;
        z1 *= sc;
      }
      m = cm;
      mstage = st;
    }
    float thr = fmaxf(tl.v[KM - 1], lb);
    if (__any_sync(0xffffffffu, live && cm >= thr)) {
#pragma unroll
      for (int u = 0; u < kVec; ++u) {
        const float xs[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const bool want = live && xs[e] >= thr;
          if (__any_sync(0xffffffffu, want)) {
            if (want) {
              tl.push(xs[e], idx[u] * 4 + e);
              thr = fmaxf(tl.v[KM - 1], lb);
            }
          }
        }
      }
    }
    if (live) {
      const float mb = m * kLog2e;
#pragma unroll
      for (int u = 0; u < kVec; ++u) {
        const float xs[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
#pragma unroll
        for (int e = 0; e < 4; e += 2) {
          const float ta = fmaxf(fmaf(xs[e], kLog2e, -mb), -250.0f);
          const float tb = fmaxf(fmaf(xs[e + 1], kLog2e, -mb), -250.0f);
          const float ea = exp2_ftz(ta);
          const float eb = exp2_ftz(tb);
          z0 += ea;
          z1 += eb;
          s0 = fmaf(ta, ea, s0);
          s1 = fmaf(tb, eb, s1);
        }
      }
    }
  }
};

__device__ __forceinline__ ArgMax warp_best(ArgMax a) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, a.v, off);
    const int oi = __shfl_xor_sync(0xffffffffu, a.i, off);
    if (better(ov, oi, a.v, a.i)) {
      a.v = ov;
      a.i = oi;
    }
  }
  return a;
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

// Reduces one segment [lo4, hi4) of a row (float4 indices) over the block
// and writes the block's partial to *out.  Returns false (uniformly) if a
// stage never arrived.
template <int KM>
__device__ bool segment_stats(const float* __restrict__ row, int lo4, int hi4, int kappa,
                              Partial* out, float4* ring, uint64_t* full) {
  __shared__ float s_m[kRowThreads / 32];
  __shared__ double s_z[kRowThreads / 32], s_s[kRowThreads / 32];
  __shared__ ArgMax s_w[kRowThreads / 32];
  __shared__ ArgMax s_pick;
  __shared__ float s_top[(kRowThreads / 32) * SENSE_MAX_KAPPA];

  const int tid = threadIdx.x;
  const float4* row4 = reinterpret_cast<const float4*>(row);
  const int n_st = (hi4 - lo4 + kStageF4 - 1) / kStageF4;
  uint64_t pol = 0;
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) ptx::mbar_init(ptx::smem_u32(full + s), 1);
    ptx::fence_barrier_init();
    pol = ptx::policy_evict_first();
  }
  __syncthreads();
  auto issue = [&](int i) {
    const int f0 = lo4 + i * kStageF4;
    const int nf = min(kStageF4, hi4 - f0);
    const uint32_t bar = ptx::smem_u32(full + (i % kStages));
    ptx::mbar_arrive_expect_tx(bar, (uint32_t)nf * 16u);
    ptx::bulk_load(ptx::smem_u32(ring + (size_t)(i % kStages) * kStageF4), row4 + f0,
                   (uint32_t)nf * 16u, bar, pol);
  };
  if (tid == 0)
    for (int i = 0; i < kStages - 1 && i < n_st; ++i) issue(i);

  RowAcc<KM> acc;
  acc.tl.init();
  const float4 pad = make_float4(-FLT_MAX, -FLT_MAX, -FLT_MAX, -FLT_MAX);
  bool ok = true;
  for (int i = 0; i < n_st; ++i) {
    const bool got = wait_phase(ptx::smem_u32(full + (i % kStages)), (uint32_t)((i / kStages) & 1));
    if (__syncthreads_or(!got)) {  // uniform: every thread leaves together
      ok = false;
      if (tid == 0) {  // let the copies in flight land before the block exits
        for (int j = i; j < i + kStages - 1 && j < n_st; ++j)
          wait_phase(ptx::smem_u32(full + (j % kStages)), (uint32_t)((j / kStages) & 1));
      }
      break;
    }
    // every thread is past stage i-1, so its buffer may be refilled
    if (tid == 0 && i + kStages - 1 < n_st) issue(i + kStages - 1);
    const float4* st = ring + (size_t)(i % kStages) * kStageF4;
    const int f0 = lo4 + i * kStageF4;
    const int nf = min(kStageF4, hi4 - f0);
    float4 x[kVec];
    int idx[kVec];
#pragma unroll
    for (int u = 0; u < kVec; ++u) {
      const int j = tid + u * kRowThreads;
      idx[u] = f0 + j;
      x[u] = (j < nf) ? st[j] : pad;
    }
    acc.add(x, idx, i);
    if (i == 0 && n_st > 1) {
      // The block's kappa-th largest value so far bounds the row's kappa-th
      // largest from below: later values under it cannot enter.
      float hv[KM];
      int hx[KM];
#pragma unroll
      for (int t = 0; t < KM; ++t) {
        hv[t] = acc.tl.v[t];
        hx[t] = acc.tl.i[t];
      }
      for (int r = 0; r < kappa; ++r) {
        const ArgMax w = warp_best(ArgMax{hv[0], hx[0]});
        if ((tid & 31) == 0) s_top[(tid >> 5) * SENSE_MAX_KAPPA + r] = w.v;
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
      __syncthreads();
      float best[SENSE_MAX_KAPPA];
      for (int r = 0; r < kappa; ++r) best[r] = -FLT_MAX;
      for (int w = 0; w < kRowThreads / 32; ++w) {
        for (int r = 0; r < kappa; ++r) {
          float v = s_top[w * SENSE_MAX_KAPPA + r];
          for (int t = 0; t < kappa; ++t) {
            if (v > best[t]) {
              const float tmp = best[t];
              best[t] = v;
              v = tmp;
            }
          }
        }
      }
      acc.lb = best[kappa - 1];
    }
  }
  if (!ok) return false;
  // argmax index: the first element equal to the maximum in its stage
  int bi = 0x7fffffff;
  if (acc.mstage >= 0) {
    const int f0 = lo4 + acc.mstage * kStageF4;
    for (int u = 0; u < kVec && bi == 0x7fffffff; ++u) {
      const int j = f0 + tid + u * kRowThreads;
      if (j >= hi4) break;
      const float4 v = row4[j];
      if (v.x == acc.m) bi = j * 4;
      else if (v.y == acc.m) bi = j * 4 + 1;
      else if (v.z == acc.m) bi = j * 4 + 2;
      else if (v.w == acc.m) bi = j * 4 + 3;
    }
  }
  const float acc_z = acc.z0 + acc.z1;
  const float acc_s = (acc.s0 + acc.s1) * (1.0f / kLog2e);  // natural-log units
  const int lane = tid & 31, wid = tid >> 5;
  constexpr int NW = kRowThreads / 32;
  float mm = acc.m;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mm = fmaxf(mm, __shfl_xor_sync(0xffffffffu, mm, off));
  if (lane == 0) s_m[wid] = mm;
  __syncthreads();
  float M = s_m[0];
#pragma unroll
  for (int w = 1; w < NW; ++w) M = fmaxf(M, s_m[w]);
  double z = 0.0, s = 0.0;
  if (acc_z > 0.0f) {  // rescale this thread's sums to the block max (fp32)
    const float d = acc.m - M;
    const float sc = exp2_ftz(d * kLog2e);
    z = (double)(acc_z * sc);
    s = (double)(sc * (acc_s + d * acc_z));
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    z += __shfl_xor_sync(0xffffffffu, z, off);
    s += __shfl_xor_sync(0xffffffffu, s, off);
  }
  ArgMax a = warp_best(ArgMax{acc.m, bi});
  if (lane == 0) {
    s_z[wid] = z;
    s_s[wid] = s;
    s_w[wid] = a;
  }
  __syncthreads();
  if (tid == 0) {
    double Z = 0.0, Sx = 0.0;
    ArgMax b = s_w[0];
    for (int w = 0; w < NW; ++w) {
      Z += s_z[w];
      Sx += s_s[w];
      if (better(s_w[w].v, s_w[w].i, b.v, b.i)) b = s_w[w];
    }
    out->z = Z;
    out->s = Sx;
    out->m = M;
    out->bv = b.v;
    out->bi = b.i;
  }
  // top-kappa of the segment: kappa rounds of a block-wide best over heads
  for (int r = 0; r < kappa; ++r) {
    ArgMax h = warp_best(ArgMax{acc.tl.v[0], acc.tl.i[0]});
    __syncthreads();
    if (lane == 0) s_w[wid] = h;
    __syncthreads();
    if (tid == 0) {
      ArgMax b = s_w[0];
      for (int w = 1; w < NW; ++w)
        if (better(s_w[w].v, s_w[w].i, b.v, b.i)) b = s_w[w];
      s_pick = b;
      out->tv[r] = b.v;
      out->ti[r] = b.i;
    }
    __syncthreads();
    if (acc.tl.i[0] == s_pick.i && acc.tl.v[0] == s_pick.v) {
#pragma unroll
      for (int t = 0; t < KM - 1; ++t) {
        acc.tl.v[t] = acc.tl.v[t + 1];
        acc.tl.i[t] = acc.tl.i[t + 1];
      }
      acc.tl.v[KM - 1] = -FLT_MAX;
      acc.tl.i[KM - 1] = 0x7fffffff;
    }
  }
  return true;
}

// Merges the segment partials of one row into its statistics (one thread).
__device__ void finish_row(const Partial* parts, int segs, int vocab, int kappa, float thr,
                           int unnormalized, int32_t* __restrict__ out) {
  float M = -FLT_MAX;
  for (int g = 0; g < segs; ++g) M = fmaxf(M, parts[g].m);
  double Z = 0.0, Sx = 0.0;
  ArgMax b{-FLT_MAX, 0x7fffffff};
  for (int g = 0; g < segs; ++g) {
    const Partial& p = parts[g];
    if (p.z > 0.0) {
      const float d = p.m - M;
      const double sc = (double)exp2_ftz(d * kLog2e);
      Z += p.z * sc;
      Sx += sc * (p.s + (double)d * p.z);
    }
    if (better(p.bv, p.bi, b.v, b.i)) b = ArgMax{p.bv, p.bi};
  }
  const float H = logf((float)Z) - (float)(Sx / Z);
  const float score = unnormalized ? H : H / logf((float)vocab);
  out[0] = b.i;
  out[1] = (score > thr) ? 1 : 0;
  int head[kMaxSegs];
  for (int g = 0; g < segs; ++g) head[g] = 0;
  for (int r = 0; r < kappa; ++r) {
    int bg = -1;
    ArgMax bb{-FLT_MAX, 0x7fffffff};
    for (int g = 0; g < segs; ++g) {
      if (head[g] >= kappa) continue;
      const float v = parts[g].tv[head[g]];
      const int ix = parts[g].ti[head[g]];
      if (bg < 0 || better(v, ix, bb.v, bb.i)) {
        bb = ArgMax{v, ix};
        bg = g;
      }
    }
    out[2 + r] = bb.i;
    if (bg >= 0) ++head[bg];
  }
  for (int r = kappa; r < SENSE_MAX_KAPPA; ++r) out[2 + r] = -1;
}

template <int KM>
__global__ void __launch_bounds__(kRowThreads)
gate_rows_kernel(const int32_t* __restrict__ parent, const int32_t* __restrict__ num_nodes,
                 int cap, const float* __restrict__ root_logits,
                 const float* __restrict__ node_logits, int vocab, int kappa, float thr,
                 int unnormalized, int segs, int seg4, Partial* __restrict__ parts,
                 unsigned* __restrict__ done, int32_t* __restrict__ stats, uint32_t* status) {
  extern __shared__ __align__(128) float4 ring[];
  __shared__ __align__(8) uint64_t full[kStages];
  __shared__ int s_last;
  const int slot = blockIdx.x / segs;  // 0 = root, 1 + n = node n
  const int seg = blockIdx.x - slot * segs;
  const int q = blockIdx.y;
  const float* row;
  if (slot == 0) {
    row = root_logits + (int64_t)q * vocab;
  } else {
    const int n = slot - 1;
    const int nn = min(num_nodes[q], cap);
    const bool inner = (n + 1 < nn) && parent[(int64_t)q * cap + n + 1] == n;
    if (!inner) return;
    row = node_logits + ((int64_t)q * cap + n) * vocab;
  }
  const int n4 = vocab >> 2;
  const int lo4 = seg * seg4;
  const int hi4 = min(n4, lo4 + seg4);
  const int64_t rid = (int64_t)q * (cap + 1) + slot;
  Partial* rp = parts + rid * segs;
  if (!segment_stats<KM>(row, lo4, hi4, kappa, rp + seg, ring, full)) {
    if (threadIdx.x == 0) raise_status(status, SENSE_DEVST_TIMEOUT);
    return;
  }
  if (segs == 1) {
    __syncthreads();
    if (threadIdx.x == 0) finish_row(rp, 1, vocab, kappa, thr, unnormalized, stats + rid * kStatsInts);
    return;
  }
  // last block of the row to finish merges the segments
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = (atomicAdd(&done[rid], 1u) == (unsigned)segs - 1u);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (threadIdx.x == 0) {
    finish_row(rp, segs, vocab, kappa, thr, unnormalized, stats + rid * kStatsInts);
    done[rid] = 0u;
  }
}

constexpr int kDecideThreads = 1024;

__global__ void __launch_bounds__(kDecideThreads)
gate_decide_kernel(GateArgs a, const int32_t* __restrict__ stats) {
  extern __shared__ uint8_t s_flags[];  // [k*m]: bit0 valid, bit1 em, bit2 ent, bit3 topk, bit4 G
  __shared__ int s_L[SENSE_MAX_K];
  __shared__ int s_best[32];
  __shared__ int s_istar, s_lstar, s_next;
  __shared__ ArgMax s_w[32];
  const int q = blockIdx.x;
  const int k = a.k, m = a.m, cap = a.cap, km = k * m;
  const int32_t* gam = a.gamma + (int64_t)q * km;
  const int32_t* tok = a.tokens + (int64_t)q * cap;
  const int32_t* st = stats + (int64_t)q * (cap + 1) * kStatsInts;

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
  const int nn = min(a.num_nodes[q], cap);
  const bool have = (nxt < 0) || ((nxt + 1 < nn) && a.parent[(int64_t)q * cap + nxt + 1] == nxt);
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

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

int gate_segments(int q, int cap, int vocab) {
  const int64_t rows = (int64_t)q * (cap + 1);
  const int n4 = vocab >> 2;
  int64_t segs = (2LL * sm_count() + rows - 1) / rows;
  const int64_t by_len = n4 / (2 * kStageF4);  // at least two stages per segment
  if (segs > by_len) segs = by_len;
  if (segs > kMaxSegs) segs = kMaxSegs;
  if (segs < 1) segs = 1;
  return (int)segs;
}

}  // namespace

size_t gate_workspace_bytes(int q, int cap, int kappa) {
  (void)kappa;
  const size_t rows = (size_t)q * (cap + 1);
  size_t b = align256(rows * kStatsInts * sizeof(int32_t));
  b += align256(rows * kMaxSegs * sizeof(Partial));
  b += align256(rows * sizeof(unsigned));
  return b;
}

sense_status launch_gate(const GateArgs& a, cudaStream_t s) {
  const size_t rows = (size_t)a.q * (a.cap + 1);
  char* ws = static_cast<char*>(a.workspace);
  int32_t* stats = reinterpret_cast<int32_t*>(ws);
  ws += align256(rows * kStatsInts * sizeof(int32_t));
  Partial* parts = reinterpret_cast<Partial*>(ws);
  ws += align256(rows * kMaxSegs * sizeof(Partial));
  unsigned* done = reinterpret_cast<unsigned*>(ws);
  const int segs = gate_segments(a.q, a.cap, a.vocab);
  const int n4 = a.vocab >> 2;
  const int seg4 = (n4 + segs - 1) / segs;
  if (segs > 1) {
    sense_status st = cuda_check(cudaMemsetAsync(done, 0, rows * sizeof(unsigned), s),
                                 "clear gate counters");
    if (st != SENSE_OK) return st;
  }
  {
    dim3 grid((unsigned)((a.cap + 1) * segs), a.q);
    const size_t ring = (size_t)kStages * kStageBytes;
    auto k4 = gate_rows_kernel<4>;
    auto k16 = gate_rows_kernel<SENSE_MAX_KAPPA>;
    auto kern = (a.kappa <= 4) ? k4 : k16;
    sense_status st = cuda_check(
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ring),
        "cudaFuncSetAttribute(gate_rows)");
    if (st != SENSE_OK) return st;
    LaunchScope ls(K_GATE_ROWS, s);
    kern<<<grid, kRowThreads, ring, s>>>(a.parent, a.num_nodes, a.cap, a.root_logits,
                                         a.node_logits, a.vocab, a.kappa, a.thr, a.unnormalized,
                                         segs, seg4, parts, done, stats, a.status);
    st = cuda_check(cudaGetLastError(), "launch gate_rows");
    if (st != SENSE_OK) return st;
  }
  const size_t smem = (size_t)a.k * a.m;
  LaunchScope ls(K_GATE_DECIDE, s);
  const int threads = (a.k * a.m <= 4096) ? 256 : kDecideThreads;
  gate_decide_kernel<<<a.q, threads, smem, s>>>(a, stats);
  return cuda_check(cudaGetLastError(), "launch gate_decide");
}

}  // namespace sense
