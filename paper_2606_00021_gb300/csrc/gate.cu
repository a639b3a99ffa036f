// Soft-gated evaluation (Sec. 3.3, Eqs. 12-19; App. C.4 Alg. 4).
//
// Alg. 4 evaluates argmax, softmax entropy and top-k on every aligned row
// P_align[i, j].  Many (i, j) share a row: position j of candidate i is
// predicted by the row of node gamma[i, j-1] (the root row for j = 0), so the
// distinct rows are the root and the tree's inner nodes.  The gate therefore
// runs in two kernels:
//  1. gate_rows: each needed row is cut into `segs` segments, one block per
//     segment.  A block streams its V/segs fp32 logits once (eight 128-bit
//     loads in flight per thread) and keeps, per thread, the running max,
//     sum exp(x - max) and sum (x - max) exp(x - max) (entropy H = log Z -
//     S / Z), the argmax (lowest index among maxima) and a top-kappa list
//     under (logit desc, index asc); the maximum of each 32-value chunk gates
//     the rare updates of the argmax and the list.  The block combines its
//     threads (fp64), writes a partial, and the last block of a row to
//     finish (an atomic counter per row) merges the segments into the row's
//     statistics.  A node is an inner node iff the next node in preorder is
//     its child, so the test is O(1).
//  2. gate_decide: one block per query evaluates B_em, B_ent, B_topk, the
//     lookahead B_con, G, the accepted prefix lengths L_i, i*, and writes
//     the accepted tokens, the next node, its argmax (streaming that row if
//     it is a leaf) and h_next.
#include <float.h>

#include "common.cuh"
#include "launch.h"

namespace sense {
namespace {

constexpr int kRowThreads = 256;
constexpr int kVec = 8;                          // float4 loads per thread per step
constexpr int kStatsInts = 2 + SENSE_MAX_KAPPA;  // argmax, ent flag, top list
constexpr int kMaxSegs = 16;

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

template <int KM>
struct RowAcc {
  float m = -FLT_MAX;  // running max
  float z = 0.0f;      // sum exp(x - m)
  float s = 0.0f;      // sum (x - m) exp(x - m)
  float bv = -FLT_MAX; // argmax value / index (lowest index among maxima)
  int bi = 0x7fffffff;
  TopList<KM> tl;

  // Folds kVec float4 (element indices idx[u] * 4 + e, increasing) into the
  // state.  Padding slots hold -FLT_MAX and contribute nothing.
  __device__ __forceinline__ void add(const float4 (&x)[kVec], const int (&idx)[kVec]) {
    float cm = -FLT_MAX;
#pragma unroll
    for (int u = 0; u < kVec; ++u)
      cm = fmaxf(cm, fmaxf(fmaxf(x[u].x, x[u].y), fmaxf(x[u].z, x[u].w)));
    if (cm > m) {
      const float sc = __expf(m - cm);
      s = sc * (s + (m - cm) * z);
      z = sc * z;
      m = cm;
    }
    if (cm > bv) {
      bv = cm;
      bool found = false;
#pragma unroll
      for (int u = 0; u < kVec; ++u) {
        const float xs[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          if (!found && xs[e] == cm) {
            bi = idx[u] * 4 + e;
            found = true;
          }
        }
      }
    }
    if (cm > tl.v[KM - 1]) {
#pragma unroll
      for (int u = 0; u < kVec; ++u) {
        const float xs[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) tl.push(xs[e], idx[u] * 4 + e);
      }
    }
#pragma unroll
    for (int u = 0; u < kVec; ++u) {
      const float xs[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float t = fmaxf(xs[e] - m, -200.0f);  // exp underflows to 0 below
        const float ex = __expf(t);
        z += ex;
        s = fmaf(t, ex, s);
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

// Reduces one segment [lo4, hi4) of a row (float4 indices) over the block
// and writes the block's partial to *out (thread 0 writes scalars).
template <int KM>
__device__ void segment_stats(const float* __restrict__ row, int lo4, int hi4, int kappa,
                              Partial* out) {
  __shared__ float s_m[kRowThreads / 32];
  __shared__ double s_z[kRowThreads / 32], s_s[kRowThreads / 32];
  __shared__ ArgMax s_w[kRowThreads / 32];
  __shared__ ArgMax s_pick;

  RowAcc<KM> acc;
  acc.tl.init();
  const float4* r4 = reinterpret_cast<const float4*>(row);
  const float4 pad = make_float4(-FLT_MAX, -FLT_MAX, -FLT_MAX, -FLT_MAX);
  for (int c = lo4 + threadIdx.x; c < hi4; c += kVec * kRowThreads) {
    float4 x[kVec];
    int idx[kVec];
#pragma unroll
    for (int u = 0; u < kVec; ++u) {
      idx[u] = c + u * kRowThreads;
      x[u] = (idx[u] < hi4) ? __ldcs(r4 + idx[u]) : pad;
    }
    acc.add(x, idx);
  }
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  constexpr int NW = kRowThreads / 32;
  // block max
  float mm = acc.m;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mm = fmaxf(mm, __shfl_xor_sync(0xffffffffu, mm, off));
  if (lane == 0) s_m[wid] = mm;
  __syncthreads();
  float M = s_m[0];
#pragma unroll
  for (int w = 1; w < NW; ++w) M = fmaxf(M, s_m[w]);
  // rescale (z, s) to M in fp64 and sum
  double z = 0.0, s = 0.0;
  if (acc.z > 0.0f) {
    const double d = (double)acc.m - (double)M;
    const double sc = exp(d);
    z = (double)acc.z * sc;
    s = sc * ((double)acc.s + d * (double)acc.z);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    z += __shfl_xor_sync(0xffffffffu, z, off);
    s += __shfl_xor_sync(0xffffffffu, s, off);
  }
  ArgMax a = warp_best(ArgMax{acc.bv, acc.bi});
  if (lane == 0) {
    s_z[wid] = z;
    s_s[wid] = s;
    s_w[wid] = a;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
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
    if (threadIdx.x == 0) {
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
      const double d = (double)p.m - (double)M;
      const double sc = exp(d);
      Z += p.z * sc;
      Sx += sc * (p.s + d * p.z);
    }
    if (better(p.bv, p.bi, b.v, b.i)) b = ArgMax{p.bv, p.bi};
  }
  const double H = log(Z) - Sx / Z;
  const double score = unnormalized ? H : H / log((double)vocab);
  out[0] = b.i;
  out[1] = (score > (double)thr) ? 1 : 0;
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
                 unsigned* __restrict__ done, int32_t* __restrict__ stats) {
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
  segment_stats<KM>(row, lo4, hi4, kappa, rp + seg);
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
  uint8_t g_val[(SENSE_MAX_TREE_TOKENS + kDecideThreads - 1) / kDecideThreads];
  {
    int c = 0;
    for (int e = threadIdx.x; e < km; e += blockDim.x, ++c) {
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
      g_val[c] = (valid && (em || (ent && (tk || con)))) ? 1 : 0;
    }
    __syncthreads();
    c = 0;
    for (int e = threadIdx.x; e < km; e += blockDim.x, ++c) s_flags[e] |= g_val[c] << 4;
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
  int64_t segs = (4LL * sm_count() + rows - 1) / rows;
  const int64_t by_len = n4 / 512;  // at least 8 KB of logits per segment
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
    LaunchScope ls(K_GATE_ROWS, s);
    if (a.kappa <= 4) {
      gate_rows_kernel<4><<<grid, kRowThreads, 0, s>>>(
          a.parent, a.num_nodes, a.cap, a.root_logits, a.node_logits, a.vocab, a.kappa, a.thr,
          a.unnormalized, segs, seg4, parts, done, stats);
    } else {
      gate_rows_kernel<SENSE_MAX_KAPPA><<<grid, kRowThreads, 0, s>>>(
          a.parent, a.num_nodes, a.cap, a.root_logits, a.node_logits, a.vocab, a.kappa, a.thr,
          a.unnormalized, segs, seg4, parts, done, stats);
    }
    sense_status st = cuda_check(cudaGetLastError(), "launch gate_rows");
    if (st != SENSE_OK) return st;
  }
  const size_t smem = (size_t)a.k * a.m;
  LaunchScope ls(K_GATE_DECIDE, s);
  gate_decide_kernel<<<a.q, kDecideThreads, smem, s>>>(a, stats);
  return cuda_check(cudaGetLastError(), "launch gate_decide");
}

}  // namespace sense
