// Soft-gated evaluation (Sec. 3.3, Eqs. 12-19; App. C.4 Alg. 4).
//
// Alg. 4 evaluates argmax, softmax entropy and top-k on every aligned row
// P_align[i, j].  Many (i, j) share a row: position j of candidate i is
// predicted by the row of node gamma[i, j-1] (the root row for j = 0), so the
// distinct rows are the root and the tree's inner nodes.  The gate therefore
// runs in two kernels:
//  1. gate_rows: one block per needed row streams its V fp32 logits once
//     (128-bit loads) and produces argmax (lowest index among maxima), the
//     entropy of softmax (online max / sum-exp / sum (x-max) exp, combined
//     across threads in fp64: H = log Z - S / Z) and the top-kappa list
//     under the order (logit desc, index asc).  A node is an inner node iff
//     the next node in preorder is its child, so the test is O(1).
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
constexpr int kStatsInts = 2 + SENSE_MAX_KAPPA;  // argmax, ent flag, top list

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

struct Online {
  float m, z, s;  // running max, sum exp(x-m), sum (x-m) exp(x-m)
};
__device__ __forceinline__ void online_add(Online& o, float x) {
  if (x > o.m) {
    const float sc = __expf(o.m - x);
    o.s = sc * (o.s + (o.m - x) * o.z);
    o.z = sc * o.z + 1.0f;
    o.m = x;
  } else {
    const float e = __expf(x - o.m);
    o.z += e;
    o.s = fmaf(x - o.m, e, o.s);
  }
}

template <int KM>
__device__ void row_stats(const float* __restrict__ row, int vocab, int kappa, float thr,
                          int unnormalized, int32_t* __restrict__ out) {
  __shared__ float s_m[kRowThreads];
  __shared__ double s_z[kRowThreads], s_s[kRowThreads];
  __shared__ ArgMax s_w[32];
  __shared__ int s_pick;

  Online o;
  o.m = -FLT_MAX;
  o.z = 0.0f;
  o.s = 0.0f;
  float bv = -FLT_MAX;
  int bi = 0x7fffffff;
  TopList<KM> tl;
  tl.init();

  const int n4 = vocab >> 2;
  const float4* r4 = reinterpret_cast<const float4*>(row);
  int c = threadIdx.x;
  for (; c + 3 * kRowThreads < n4; c += 4 * kRowThreads) {
    float4 x[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) x[u] = __ldcs(r4 + c + u * kRowThreads);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int base = (c + u * kRowThreads) * 4;
      const float xs[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        online_add(o, xs[e]);
        if (xs[e] > bv) {
          bv = xs[e];
          bi = base + e;
        }
        tl.push(xs[e], base + e);
      }
    }
  }
  for (; c < n4; c += kRowThreads) {
    const float4 x = __ldcs(r4 + c);
    const float xs[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      online_add(o, xs[e]);
      if (xs[e] > bv) {
        bv = xs[e];
        bi = c * 4 + e;
      }
      tl.push(xs[e], c * 4 + e);
    }
  }

  // Entropy: combine (m, z, s) across the block in fp64.
  s_m[threadIdx.x] = o.m;
  __syncthreads();
  if (threadIdx.x < 32) {
    float mm = -FLT_MAX;
    for (int t = threadIdx.x; t < kRowThreads; t += 32) mm = fmaxf(mm, s_m[t]);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) mm = fmaxf(mm, __shfl_xor_sync(0xffffffffu, mm, off));
    if (threadIdx.x == 0) s_m[0] = mm;  // safe: all lanes read s_m before
  }
  __syncthreads();
  const double M = (double)s_m[0];
  {
    double z = 0.0, s = 0.0;
    if (o.z > 0.0f) {
      const double sc = exp((double)o.m - M);
      z = (double)o.z * sc;
      s = sc * ((double)o.s + ((double)o.m - M) * (double)o.z);
    }
    s_z[threadIdx.x] = z;
    s_s[threadIdx.x] = s;
  }
  // Argmax: warp reduce then block reduce.
  {
    float v = bv;
    int i = bi;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, v, off);
      const int oi = __shfl_xor_sync(0xffffffffu, i, off);
      if (better(ov, oi, v, i)) {
        v = ov;
        i = oi;
      }
    }
    if ((threadIdx.x & 31) == 0) s_w[threadIdx.x >> 5] = ArgMax{v, i};
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    double z = 0.0, s = 0.0;
    for (int t = threadIdx.x; t < kRowThreads; t += 32) {
      z += s_z[t];
      s += s_s[t];
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      z += __shfl_xor_sync(0xffffffffu, z, off);
      s += __shfl_xor_sync(0xffffffffu, s, off);
    }
    ArgMax a = (threadIdx.x < kRowThreads / 32) ? s_w[threadIdx.x] : ArgMax{-FLT_MAX, 0x7fffffff};
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, a.v, off);
      const int oi = __shfl_xor_sync(0xffffffffu, a.i, off);
      if (better(ov, oi, a.v, a.i)) {
        a.v = ov;
        a.i = oi;
      }
    }
    if (threadIdx.x == 0) {
      const double H = log(z) - s / z;
      const double score = unnormalized ? H : H / log((double)vocab);
      out[0] = a.i;
      out[1] = (score > (double)thr) ? 1 : 0;
    }
  }
  // Top-kappa: kappa rounds of a block-wide best over the thread heads.
  int head = 0;
  for (int r = 0; r < kappa; ++r) {
    float v = (head < KM) ? tl.v[0] : -FLT_MAX;
    int i = (head < KM) ? tl.i[0] : 0x7fffffff;
    // (tl is kept shifted so that slot 0 is the current head)
    float wv = v;
    int wi = i;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, wv, off);
      const int oi = __shfl_xor_sync(0xffffffffu, wi, off);
      if (better(ov, oi, wv, wi)) {
        wv = ov;
        wi = oi;
      }
    }
    __syncthreads();
    if ((threadIdx.x & 31) == 0) s_w[threadIdx.x >> 5] = ArgMax{wv, wi};
    __syncthreads();
    if (threadIdx.x < 32) {
      ArgMax a = (threadIdx.x < kRowThreads / 32) ? s_w[threadIdx.x] : ArgMax{-FLT_MAX, 0x7fffffff};
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, a.v, off);
        const int oi = __shfl_xor_sync(0xffffffffu, a.i, off);
        if (better(ov, oi, a.v, a.i)) {
          a.v = ov;
          a.i = oi;
        }
      }
      if (threadIdx.x == 0) {
        s_pick = a.i;
        out[2 + r] = a.i;
      }
    }
    __syncthreads();
    if (head < KM && tl.i[0] == s_pick) {
#pragma unroll
      for (int s = 0; s < KM - 1; ++s) {
        tl.v[s] = tl.v[s + 1];
        tl.i[s] = tl.i[s + 1];
      }
      tl.v[KM - 1] = -FLT_MAX;
      tl.i[KM - 1] = 0x7fffffff;
      ++head;
    }
  }
  for (int r = kappa + threadIdx.x; r < SENSE_MAX_KAPPA; r += kRowThreads) out[2 + r] = -1;
}

template <int KM>
__global__ void __launch_bounds__(kRowThreads)
gate_rows_kernel(const int32_t* __restrict__ parent, const int32_t* __restrict__ num_nodes,
                 int cap, const float* __restrict__ root_logits,
                 const float* __restrict__ node_logits, int vocab, int kappa, float thr,
                 int unnormalized, int32_t* __restrict__ stats) {
  const int slot = blockIdx.x;  // 0 = root, 1 + n = node n
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
  row_stats<KM>(row, vocab, kappa, thr, unnormalized,
                stats + ((int64_t)q * (cap + 1) + slot) * kStatsInts);
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

}  // namespace

size_t gate_workspace_bytes(int q, int cap, int kappa) {
  (void)kappa;
  const size_t b = (size_t)q * (cap + 1) * kStatsInts * sizeof(int32_t);
  return (b + 255) & ~(size_t)255;
}

sense_status launch_gate(const GateArgs& a, cudaStream_t s) {
  int32_t* stats = static_cast<int32_t*>(a.workspace);
  {
    dim3 grid(a.cap + 1, a.q);
    LaunchScope ls(K_GATE_ROWS, s);
    if (a.kappa <= 4) {
      gate_rows_kernel<4><<<grid, kRowThreads, 0, s>>>(a.parent, a.num_nodes, a.cap, a.root_logits,
                                                       a.node_logits, a.vocab, a.kappa, a.thr,
                                                       a.unnormalized, stats);
    } else {
      gate_rows_kernel<SENSE_MAX_KAPPA><<<grid, kRowThreads, 0, s>>>(
          a.parent, a.num_nodes, a.cap, a.root_logits, a.node_logits, a.vocab, a.kappa, a.thr,
          a.unnormalized, stats);
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
