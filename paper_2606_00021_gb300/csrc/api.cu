// C-ABI layer of libsense: argument validation, workspace planning, the
// per-device status word, launch profiling and the datastore handle.
#include <cuda_bf16.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <map>
#include <mutex>
#include <string>
#include <vector>

#include "common.cuh"
#include "launch.h"

namespace sense {

namespace {
thread_local char g_err[512] = "";
std::mutex g_mu;
constexpr int kMaxDevices = 64;
uint32_t* g_status[kMaxDevices] = {nullptr};
int g_sms[kMaxDevices] = {0};

struct ProfRec {
  int id;
  cudaEvent_t a, b;
};
bool g_prof_on = false;
bool g_prof_family[K_COUNT];  // families bracketed while profiling is on
std::vector<ProfRec> g_prof;
std::vector<cudaEvent_t> g_ev_pool;
const char* const kKernelNames[K_COUNT] = {
    "normalize", "scan_gemv", "scan_tc", "threshold", "merge",
    "gather",    "tree",      "gate_rows", "gate_decide", "pad_queries",
    "tree_mask", "project",  "kmeans",    "ivf_build", "ivf_coarse",
    "ivf_scan",  "ctx",       "tree_attn", "rescore",   "draft"};

cudaEvent_t take_event() {
  if (!g_ev_pool.empty()) {
    cudaEvent_t e = g_ev_pool.back();
    g_ev_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int current_device() {
  int dev = 0;
  cudaGetDevice(&dev);
  return dev;
}
}  // namespace

sense_status fail(sense_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return s;
}

sense_status cuda_check(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return SENSE_OK;
  if (e == cudaErrorMemoryAllocation)
    return fail(SENSE_ERR_OOM, "%s: %s", what, cudaGetErrorString(e));
  return fail(SENSE_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

uint32_t* device_status_word() {
  const int dev = current_device();
  if (dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_status[dev]) {
    void* p = nullptr;
    if (cudaMalloc(&p, 256) != cudaSuccess) {
      fail(SENSE_ERR_OOM, "cannot allocate the device status word");
      return nullptr;
    }
    if (cudaMemset(p, 0, 256) != cudaSuccess) {
      cudaFree(p);
      fail(SENSE_ERR_CUDA, "cannot clear the device status word");
      return nullptr;
    }
    g_status[dev] = static_cast<uint32_t*>(p);
  }
  return g_status[dev];
}

cudaError_t func_smem(const void* f, int bytes) {
  static std::mutex mu;
  static std::map<std::pair<const void*, int>, int> done;
  const int dev = current_device();
  std::lock_guard<std::mutex> lk(mu);
  auto it = done.find({f, dev});
  if (it != done.end() && it->second >= bytes) return cudaSuccess;
  const cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done[{f, dev}] = bytes;
  return e;
}

int sm_count() {
  const int dev = current_device();
  if (dev >= 0 && dev < kMaxDevices && g_sms[dev] > 0) return g_sms[dev];
  int v = 0;
  cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
  if (v <= 0) v = 1;
  if (dev >= 0 && dev < kMaxDevices) g_sms[dev] = v;
  return v;
}

LaunchScope::LaunchScope(KernelId id, cudaStream_t s) : id_(id), s_(s), slot_(-1) {
  if (!g_prof_on || !g_prof_family[id]) return;
  std::lock_guard<std::mutex> lk(g_mu);
  ProfRec r{id, take_event(), take_event()};
  cudaEventRecord(r.a, s);
  g_prof.push_back(r);
  slot_ = (int)g_prof.size() - 1;
}

LaunchScope::~LaunchScope() {
  if (slot_ < 0) return;
  std::lock_guard<std::mutex> lk(g_mu);
  if (slot_ < (int)g_prof.size()) cudaEventRecord(g_prof[slot_].b, s_);
}

// ---------------------------------------------------------------------------
// Datastore normalisation (SENSE_DS_NORMALIZE)
// ---------------------------------------------------------------------------
namespace {
__global__ void normalize_kernel(const float* __restrict__ src, int64_t n, int d,
                                 __nv_bfloat16* __restrict__ dst) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t r = warp; r < n; r += nw) {
    const float* x = src + r * d;
    double ss = 0.0;
    for (int j = lane; j < d; j += 32) ss = fma((double)x[j], (double)x[j], ss);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    const double nrm = sqrt(ss);
    __nv_bfloat16* y = dst + r * d;
    for (int j = lane; j < d; j += 32)
      y[j] = (nrm > 0.0) ? __double2bfloat16((double)x[j] / nrm) : __double2bfloat16(0.0);
  }
}
}  // namespace

sense_status launch_normalize(const float* src, int64_t n, int d, uint16_t* dst, cudaStream_t s) {
  int64_t blocks = (n + 7) / 8;
  const int64_t cap = (int64_t)sm_count() * 8;
  if (blocks > cap) blocks = cap;
  LaunchScope ls(K_NORMALIZE, s);
  normalize_kernel<<<(unsigned)blocks, 256, 0, s>>>(src, n, d, reinterpret_cast<__nv_bfloat16*>(dst));
  return cuda_check(cudaGetLastError(), "launch normalize");
}

// ---------------------------------------------------------------------------
// Retrieval plan
// ---------------------------------------------------------------------------
namespace {
size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }
}  // namespace

RetrievePlan make_plan(const sense_datastore* ds, int q, int k) {
  RetrievePlan p{};
  p.tc = q > 8;
  p.group = p.tc ? (q < 128 ? q : 128) : q;
  p.fused = !p.tc && q <= kFusedMaxQ && k <= kFusedMaxK &&
            fused_smem_bytes(q, ds->d, k) <= 110 * 1024;  // two blocks per SM
  p.fused_blocks = p.fused ? fused_blocks() : 0;
  p.s_rows = sample_tiles(ds->n) * (int64_t)kTileRows;
  p.r_rows = rest_tiles(ds->n) * (int64_t)kTileRows;
  p.sampling = sample_tiles(ds->n) >= 4 && p.s_rows >= 4LL * k && p.s_rows >= 2048;
  p.pool_cap = p.fused ? (int64_t)p.fused_blocks * k : ds->n;
  if (p.fused) p.sampling = false;
  const int g = p.group;
  size_t off = 0;
  p.off_counts = off;
  off = align256(off + sizeof(uint32_t) * g);
  p.off_thresh = off;
  off = align256(off + sizeof(uint64_t) * g);
  p.off_sample = off;
  if (p.sampling) off = align256(off + sizeof(uint64_t) * g * (size_t)p.s_rows);
  p.off_cand = off;
  if (p.sampling) off = align256(off + sizeof(uint64_t) * g * (size_t)chunk_count(p.s_rows) * k);
  p.off_pool = off;
  off = align256(off + sizeof(uint64_t) * g * (size_t)p.pool_cap);
  p.off_qpad = off;
  if (p.tc) off = align256(off + sizeof(uint16_t) * (size_t)((g + 15) / 16 * 16) * ds->d);
  p.total = off;
  return p;
}

sense_status run_retrieve(const RetrievePlan& p, const sense_datastore* ds,
                          const uint16_t* queries, int q, int k, float* out_scores,
                          int32_t* out_idx, char* ws, uint32_t* status, cudaStream_t stream) {
  uint32_t* counts = reinterpret_cast<uint32_t*>(ws + p.off_counts);
  uint64_t* thresh = reinterpret_cast<uint64_t*>(ws + p.off_thresh);
  uint64_t* sample = reinterpret_cast<uint64_t*>(ws + p.off_sample);
  uint64_t* cand = reinterpret_cast<uint64_t*>(ws + p.off_cand);
  uint64_t* pool = reinterpret_cast<uint64_t*>(ws + p.off_pool);
  uint16_t* qpad = reinterpret_cast<uint16_t*>(ws + p.off_qpad);
  const int64_t n = ds->n;
  const int d = ds->d;
  sense_status st = SENSE_OK;
  if (p.fused) {
    st = launch_scan_gemv_topk(ds->keys, n, d, queries, q, k, p.fused_blocks, pool, stream);
    if (st != SENSE_OK) return st;
    return launch_merge_lists(pool, p.fused_blocks, q, k, out_scores, out_idx, status, stream);
  }
  for (int g0 = 0; g0 < q; g0 += p.group) {
    const int gq = (q - g0 < p.group) ? (q - g0) : p.group;
    const int nq = (gq + 15) / 16 * 16;
    const uint16_t* qg = queries + (int64_t)g0 * d;
    st = cuda_check(cudaMemsetAsync(counts, 0, sizeof(uint32_t) * gq, stream), "clear pool counts");
    if (st != SENSE_OK) return st;
    if (p.tc) {
      st = launch_pad_queries(qg, gq, d, qpad, nq, stream);
      if (st != SENSE_OK) return st;
    }
    // scan(mode): the work set of `mode` against `thr`, into `out`
    auto scan = [&](int mode, const uint64_t* thr, uint64_t* out, int64_t cap) -> sense_status {
      const int64_t halves = (mode == SCAN_SAMPLE) ? sample_tiles(n)
                           : (mode == SCAN_REST)   ? rest_tiles(n)
                                                   : num_tiles(n);
      if (p.tc)
        return launch_scan_tc(ds->keys, n, d, qpad, gq, nq, mode, halves, thr, out, counts, cap,
                              status, stream);
      const int64_t rows = (mode == SCAN_ALL) ? n : halves * kTileRows;
      return launch_scan_gemv(ds->keys, n, d, qg, gq, mode, rows, thr, out, counts, cap, status,
                              stream);
    };
    if (p.sampling) {
      st = scan(SCAN_SAMPLE, nullptr, sample, 0);
      if (st != SENSE_OK) return st;
      st = launch_threshold(sample, p.s_rows, gq, k, cand, thresh, pool, counts, p.pool_cap,
                            status, stream);
      if (st != SENSE_OK) return st;
      st = scan(SCAN_REST, thresh, pool, p.pool_cap);
    } else {
      st = scan(SCAN_ALL, nullptr, pool, p.pool_cap);
    }
    if (st != SENSE_OK) return st;
    st = launch_merge(pool, counts, p.pool_cap, gq, k, out_scores + (int64_t)g0 * k,
                      out_idx + (int64_t)g0 * k, status, stream);
    if (st != SENSE_OK) return st;
  }
  return SENSE_OK;
}

namespace {
sense_status check_ds(const sense_datastore* ds) {
  if (!ds) return fail(SENSE_ERR_INVALID_ARG, "datastore handle is NULL");
  if (ds->device != current_device())
    return fail(SENSE_ERR_INVALID_ARG, "datastore was built on device %d, current device is %d",
                ds->device, current_device());
  return SENSE_OK;
}
}  // namespace

}  // namespace sense

using namespace sense;

// ---------------------------------------------------------------------------
// Exported functions
// ---------------------------------------------------------------------------
extern "C" {

int32_t sense_version(void) { return 10000; }

const char* sense_status_string(sense_status s) {
  switch (s) {
    case SENSE_OK: return "SENSE_OK";
    case SENSE_ERR_INVALID_ARG: return "SENSE_ERR_INVALID_ARG";
    case SENSE_ERR_UNSUPPORTED: return "SENSE_ERR_UNSUPPORTED";
    case SENSE_ERR_OOM: return "SENSE_ERR_OOM";
    case SENSE_ERR_CUDA: return "SENSE_ERR_CUDA";
    case SENSE_ERR_DEVICE_STATUS: return "SENSE_ERR_DEVICE_STATUS";
    case SENSE_ERR_TIMEOUT: return "SENSE_ERR_TIMEOUT";
  }
  return "SENSE_ERR_UNKNOWN";
}

const char* sense_last_error(void) { return g_err; }

sense_status sense_device_status(sense_stream_t stream, uint32_t* out_bits, int32_t clear) {
  if (!out_bits) return fail(SENSE_ERR_INVALID_ARG, "out_bits is NULL");
  uint32_t* w = device_status_word();
  if (!w) return SENSE_ERR_OOM;
  sense_status st = cuda_check(cudaStreamSynchronize(stream), "cudaStreamSynchronize");
  if (st != SENSE_OK) return st;
  uint32_t v = 0;
  st = cuda_check(cudaMemcpy(&v, w, sizeof(v), cudaMemcpyDeviceToHost), "read status word");
  if (st != SENSE_OK) return st;
  if (clear) {
    st = cuda_check(cudaMemset(w, 0, sizeof(uint32_t)), "clear status word");
    if (st != SENSE_OK) return st;
  }
  *out_bits = v;
  if (v & SENSE_DEVST_TIMEOUT) return fail(SENSE_ERR_TIMEOUT, "a device wait hit its limit (bits 0x%x)", v);
  if (v) return fail(SENSE_ERR_DEVICE_STATUS, "device status bits 0x%x", v);
  return SENSE_OK;
}

sense_status sense_datastore_build(const void* keys, int32_t key_dtype, int64_t n, int32_t d,
                                   const int32_t* spans, int32_t m, uint32_t flags,
                                   sense_stream_t stream, sense_datastore** out) {
  if (!out) return fail(SENSE_ERR_INVALID_ARG, "out is NULL");
  if (!keys || !spans) return fail(SENSE_ERR_INVALID_ARG, "keys and spans must be non-NULL");
  if (n < 1 || n > 2147483647LL) return fail(SENSE_ERR_INVALID_ARG, "n=%lld outside [1, 2^31-1]", (long long)n);
  if (d < 8 || d > 65536 || (d % 8) != 0) return fail(SENSE_ERR_INVALID_ARG, "d=%d must be a multiple of 8 in [8, 65536]", d);
  if (m < 1 || m > SENSE_MAX_M) return fail(SENSE_ERR_INVALID_ARG, "m=%d outside [1, %d]", m, SENSE_MAX_M);
  if (!aligned(keys, 16) || !aligned(spans, 16)) return fail(SENSE_ERR_INVALID_ARG, "keys and spans must be 16-byte aligned");
  if (flags & ~SENSE_DS_NORMALIZE) return fail(SENSE_ERR_INVALID_ARG, "unknown datastore flags 0x%x", flags);
  const bool norm = (flags & SENSE_DS_NORMALIZE) != 0;
  if (norm && key_dtype != SENSE_KEY_F32) return fail(SENSE_ERR_INVALID_ARG, "SENSE_DS_NORMALIZE needs SENSE_KEY_F32 keys");
  if (!norm && key_dtype != SENSE_KEY_BF16) return fail(SENSE_ERR_INVALID_ARG, "borrowed keys must be SENSE_KEY_BF16");
  if (!device_status_word()) return SENSE_ERR_OOM;
  sense_datastore* ds = new (std::nothrow) sense_datastore();
  if (!ds) return fail(SENSE_ERR_OOM, "host allocation failed");
  ds->n = n;
  ds->d = d;
  ds->m = m;
  ds->spans = spans;
  ds->owned = nullptr;
  ds->device = current_device();
  if (norm) {
    void* p = nullptr;
    const size_t bytes = (size_t)n * d * sizeof(uint16_t);
    sense_status st = cuda_check(cudaMalloc(&p, bytes), "cudaMalloc(normalised keys)");
    if (st != SENSE_OK) {
      delete ds;
      return st;
    }
    ds->owned = static_cast<uint16_t*>(p);
    st = launch_normalize(static_cast<const float*>(keys), n, d, ds->owned, stream);
    if (st != SENSE_OK) {
      cudaFree(p);
      delete ds;
      return st;
    }
    ds->keys = ds->owned;
  } else {
    ds->keys = static_cast<const uint16_t*>(keys);
  }
  *out = ds;
  return SENSE_OK;
}

sense_status sense_datastore_destroy(sense_datastore* ds) {
  if (!ds) return SENSE_OK;
  sense_status st = SENSE_OK;
  if (ds->owned) {
    st = cuda_check(cudaDeviceSynchronize(), "cudaDeviceSynchronize");
    cudaFree(ds->owned);
  }
  delete ds;
  return st;
}

const uint16_t* sense_datastore_keys(const sense_datastore* ds) { return ds ? ds->keys : nullptr; }

size_t sense_retrieve_workspace_bytes(const sense_datastore* ds, int32_t q, int32_t k) {
  if (!ds || q < 1 || k < 1) return 0;
  return make_plan(ds, q, k).total;
}

sense_status sense_retrieve_topk(const sense_datastore* ds, const uint16_t* queries, int32_t q,
                                 int32_t k, float* out_scores, int32_t* out_idx,
                                 void* workspace, size_t workspace_bytes, sense_stream_t stream) {
  sense_status st = check_ds(ds);
  if (st != SENSE_OK) return st;
  if (!queries || !out_scores || !out_idx || !workspace)
    return fail(SENSE_ERR_INVALID_ARG, "queries, outputs and workspace must be non-NULL");
  if (q < 1) return fail(SENSE_ERR_INVALID_ARG, "q=%d must be >= 1", q);
  if (k < 1 || k > SENSE_MAX_K || (int64_t)k > ds->n)
    return fail(SENSE_ERR_INVALID_ARG, "k=%d outside [1, min(n=%lld, %d)]", k, (long long)ds->n, SENSE_MAX_K);
  if (!aligned(queries, 16)) return fail(SENSE_ERR_INVALID_ARG, "queries must be 16-byte aligned");
  if (q > 8 && ds->n > 2147483647LL - 1024)
    return fail(SENSE_ERR_UNSUPPORTED, "batched (q > 8) retrieval supports n <= 2^31 - 1025");
  if (!aligned(workspace, 256)) return fail(SENSE_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  const RetrievePlan p = make_plan(ds, q, k);
  if (workspace_bytes < p.total)
    return fail(SENSE_ERR_INVALID_ARG, "workspace has %zu bytes, needs %zu", workspace_bytes, p.total);
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  return run_retrieve(p, ds, queries, q, k, out_scores, out_idx, static_cast<char*>(workspace),
                      status, stream);
}

sense_status sense_rescore_topk(const sense_datastore* ds, const uint16_t* queries, int32_t q,
                                const int32_t* cand_idx, int32_t n_cand, int32_t k,
                                float* out_scores, int32_t* out_idx, sense_stream_t stream) {
  sense_status st = check_ds(ds);
  if (st != SENSE_OK) return st;
  if (!queries || !cand_idx || !out_scores || !out_idx)
    return fail(SENSE_ERR_INVALID_ARG, "queries, candidates and outputs must be non-NULL");
  if (q < 1 || q > 65535) return fail(SENSE_ERR_INVALID_ARG, "q=%d outside [1, 65535]", q);
  if (n_cand < 1 || n_cand > SENSE_MAX_RESCORE)
    return fail(SENSE_ERR_INVALID_ARG, "n_cand=%d outside [1, %d]", n_cand, SENSE_MAX_RESCORE);
  if (k < 1 || k > n_cand) return fail(SENSE_ERR_INVALID_ARG, "k=%d outside [1, n_cand=%d]", k, n_cand);
  if (!aligned(queries, 16)) return fail(SENSE_ERR_INVALID_ARG, "queries must be 16-byte aligned");
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  return launch_rescore(ds->keys, ds->n, ds->d, queries, q, cand_idx, n_cand, k, out_scores,
                        out_idx, status, stream);
}

sense_status sense_gather_drafts(const sense_datastore* ds, const int32_t* idx, int32_t q,
                                 int32_t k, const int32_t* anchor, int32_t n_keep, uint32_t flags,
                                 int32_t* out_spans, sense_stream_t stream) {
  sense_status st = check_ds(ds);
  if (st != SENSE_OK) return st;
  if (!idx || !out_spans) return fail(SENSE_ERR_INVALID_ARG, "idx and out_spans must be non-NULL");
  if (q < 1) return fail(SENSE_ERR_INVALID_ARG, "q=%d must be >= 1", q);
  if (k < 1 || k > SENSE_MAX_K) return fail(SENSE_ERR_INVALID_ARG, "k=%d outside [1, %d]", k, SENSE_MAX_K);
  if (n_keep < 1 || n_keep > k) return fail(SENSE_ERR_INVALID_ARG, "n_keep=%d outside [1, k=%d]", n_keep, k);
  if (!anchor && n_keep != k) return fail(SENSE_ERR_INVALID_ARG, "n_keep must equal k without an anchor");
  if (flags & ~SENSE_GATHER_FORCE_ANCHOR) return fail(SENSE_ERR_INVALID_ARG, "unknown gather flags 0x%x", flags);
  if (!aligned(out_spans, 16)) return fail(SENSE_ERR_INVALID_ARG, "out_spans must be 16-byte aligned");
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  return launch_gather(ds->spans, ds->n, ds->m, idx, q, k, anchor, n_keep,
                       (flags & SENSE_GATHER_FORCE_ANCHOR) ? 1 : 0, out_spans, status, stream);
}

sense_status sense_build_tree(const int32_t* spans, int32_t q, int32_t k, int32_t m,
                              int32_t node_cap, uint32_t flags, int32_t* out_num_nodes,
                              int32_t* out_tokens, int32_t* out_parent, int32_t* out_depth,
                              int32_t* out_gamma, uint32_t* out_mask_bits, sense_stream_t stream) {
  if (!spans || !out_num_nodes || !out_tokens || !out_parent || !out_depth || !out_gamma)
    return fail(SENSE_ERR_INVALID_ARG, "spans and outputs must be non-NULL");
  if (q < 1) return fail(SENSE_ERR_INVALID_ARG, "q=%d must be >= 1", q);
  if (k < 1 || k > SENSE_MAX_K) return fail(SENSE_ERR_INVALID_ARG, "k=%d outside [1, %d]", k, SENSE_MAX_K);
  if (m < 1 || m > SENSE_MAX_M) return fail(SENSE_ERR_INVALID_ARG, "m=%d outside [1, %d]", m, SENSE_MAX_M);
  if ((int64_t)k * m > SENSE_MAX_TREE_TOKENS)
    return fail(SENSE_ERR_INVALID_ARG, "k*m=%d exceeds %d", k * m, SENSE_MAX_TREE_TOKENS);
  if (node_cap < 0) return fail(SENSE_ERR_INVALID_ARG, "node_cap=%d must be >= 0", node_cap);
  if (flags & ~SENSE_TREE_MASK_BITS) return fail(SENSE_ERR_INVALID_ARG, "unknown tree flags 0x%x", flags);
  const bool bits = (flags & SENSE_TREE_MASK_BITS) != 0;
  if (bits && !out_mask_bits) return fail(SENSE_ERR_INVALID_ARG, "SENSE_TREE_MASK_BITS needs out_mask_bits");
  const int cap = node_cap > 0 ? node_cap : k * m;
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  return launch_tree(spans, q, k, m, cap, bits ? 1 : 0, out_num_nodes, out_tokens, out_parent,
                     out_depth, out_gamma, out_mask_bits, status, stream);
}

sense_status sense_draft(const sense_datastore* ds, const uint16_t* queries, int32_t q, int32_t k,
                         void* workspace, size_t workspace_bytes, int32_t node_cap, uint32_t flags,
                         float* out_scores, int32_t* out_idx, int32_t* out_spans,
                         int32_t* out_num_nodes, int32_t* out_tokens, int32_t* out_parent,
                         int32_t* out_depth, int32_t* out_gamma, uint32_t* out_mask_bits,
                         sense_stream_t stream) {
  sense_status st = check_ds(ds);
  if (st != SENSE_OK) return st;
  if (!queries || !out_scores || !out_idx || !workspace || !out_spans || !out_num_nodes ||
      !out_tokens || !out_parent || !out_depth || !out_gamma)
    return fail(SENSE_ERR_INVALID_ARG, "queries, workspace and outputs must be non-NULL");
  if (q < 1) return fail(SENSE_ERR_INVALID_ARG, "q=%d must be >= 1", q);
  if (k < 1 || k > SENSE_MAX_K || (int64_t)k > ds->n)
    return fail(SENSE_ERR_INVALID_ARG, "k=%d outside [1, min(n=%lld, %d)]", k, (long long)ds->n, SENSE_MAX_K);
  const int m = ds->m;
  if ((int64_t)k * m > SENSE_MAX_TREE_TOKENS)
    return fail(SENSE_ERR_INVALID_ARG, "k*m=%d exceeds %d", k * m, SENSE_MAX_TREE_TOKENS);
  if (node_cap < 0) return fail(SENSE_ERR_INVALID_ARG, "node_cap=%d must be >= 0", node_cap);
  if (flags & ~SENSE_TREE_MASK_BITS) return fail(SENSE_ERR_INVALID_ARG, "unknown tree flags 0x%x", flags);
  const bool bits = (flags & SENSE_TREE_MASK_BITS) != 0;
  if (bits && !out_mask_bits) return fail(SENSE_ERR_INVALID_ARG, "SENSE_TREE_MASK_BITS needs out_mask_bits");
  if (!aligned(queries, 16) || !aligned(out_spans, 16))
    return fail(SENSE_ERR_INVALID_ARG, "queries and out_spans must be 16-byte aligned");
  if (q > 8 && ds->n > 2147483647LL - 1024)
    return fail(SENSE_ERR_UNSUPPORTED, "batched (q > 8) retrieval supports n <= 2^31 - 1025");
  if (!aligned(workspace, 256)) return fail(SENSE_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  const RetrievePlan p = make_plan(ds, q, k);
  if (workspace_bytes < p.total)
    return fail(SENSE_ERR_INVALID_ARG, "workspace has %zu bytes, needs %zu", workspace_bytes, p.total);
  const int cap = node_cap > 0 ? node_cap : k * m;
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  char* ws = static_cast<char*>(workspace);
  if (p.fused && draft_fused_fits(k, m)) {
    // single-pass scan, then merge + gather + trie in one kernel per query
    uint64_t* pool = reinterpret_cast<uint64_t*>(ws + p.off_pool);
    st = launch_scan_gemv_topk(ds->keys, ds->n, ds->d, queries, q, k, p.fused_blocks, pool, stream);
    if (st != SENSE_OK) return st;
    return launch_draft_fused(pool, p.fused_blocks, q, k, out_scores, out_idx, ds->spans, ds->n, m,
                              out_spans, cap, bits ? 1 : 0, out_num_nodes, out_tokens, out_parent,
                              out_depth, out_gamma, out_mask_bits, status, stream);
  }
  st = run_retrieve(p, ds, queries, q, k, out_scores, out_idx, ws, status, stream);
  if (st != SENSE_OK) return st;
  st = launch_gather(ds->spans, ds->n, m, out_idx, q, k, nullptr, k, 0, out_spans, status, stream);
  if (st != SENSE_OK) return st;
  return launch_tree(out_spans, q, k, m, cap, bits ? 1 : 0, out_num_nodes, out_tokens, out_parent,
                     out_depth, out_gamma, out_mask_bits, status, stream);
}

sense_status sense_tree_mask_full(const uint32_t* mask_bits, const int32_t* num_nodes, int32_t q,
                                  int32_t cap, const int32_t* prefix_len, int32_t cache_len,
                                  float* out, sense_stream_t stream) {
  if (!mask_bits || !num_nodes || !prefix_len || !out)
    return fail(SENSE_ERR_INVALID_ARG, "mask_bits, num_nodes, prefix_len and out must be non-NULL");
  if (q < 1) return fail(SENSE_ERR_INVALID_ARG, "q=%d must be >= 1", q);
  if (cap < 1 || cap > SENSE_MAX_TREE_TOKENS)
    return fail(SENSE_ERR_INVALID_ARG, "cap=%d outside [1, %d]", cap, SENSE_MAX_TREE_TOKENS);
  if (cache_len < 1) return fail(SENSE_ERR_INVALID_ARG, "cache_len=%d must be >= 1", cache_len);
  if (!aligned(mask_bits, 4) || !aligned(num_nodes, 4) || !aligned(prefix_len, 4) || !aligned(out, 4))
    return fail(SENSE_ERR_INVALID_ARG, "arrays must be 4-byte aligned");
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  return launch_tree_mask_full(mask_bits, num_nodes, prefix_len, q, cap, cache_len, out, status,
                               stream);
}

size_t sense_soft_gate_workspace_bytes(int32_t q, int32_t cap, int32_t kappa) {
  if (q < 1 || cap < 1) return 0;
  return gate_workspace_bytes(q, cap, kappa);
}

sense_status sense_soft_gate(const int32_t* tokens, const int32_t* parent,
                             const int32_t* num_nodes, const int32_t* gamma, int32_t q, int32_t k,
                             int32_t m, int32_t cap, const float* root_logits,
                             const float* node_logits, int32_t vocab, const uint16_t* root_hidden,
                             const uint16_t* node_hidden, int32_t d,
                             const sense_gate_params* params, int32_t* out_i_star,
                             int32_t* out_L_star, int32_t* out_n_accept, int32_t* out_accepted,
                             int32_t* out_next_node, int32_t* out_next_anchor,
                             uint16_t* out_h_next, uint8_t* out_G, void* workspace,
                             size_t workspace_bytes, sense_stream_t stream) {
  if (!tokens || !parent || !num_nodes || !gamma || !root_logits || !node_logits ||
      !root_hidden || !node_hidden || !params || !out_i_star || !out_L_star || !out_n_accept ||
      !out_accepted || !out_next_node || !out_next_anchor || !out_h_next || !workspace)
    return fail(SENSE_ERR_INVALID_ARG, "a required pointer is NULL");
  if (q < 1) return fail(SENSE_ERR_INVALID_ARG, "q=%d must be >= 1", q);
  if (k < 1 || k > SENSE_MAX_K) return fail(SENSE_ERR_INVALID_ARG, "k=%d outside [1, %d]", k, SENSE_MAX_K);
  if (m < 1 || m > SENSE_MAX_M) return fail(SENSE_ERR_INVALID_ARG, "m=%d outside [1, %d]", m, SENSE_MAX_M);
  if ((int64_t)k * m > SENSE_MAX_TREE_TOKENS)
    return fail(SENSE_ERR_INVALID_ARG, "k*m=%d exceeds %d", k * m, SENSE_MAX_TREE_TOKENS);
  if (cap < 1) return fail(SENSE_ERR_INVALID_ARG, "cap=%d must be >= 1", cap);
  const sense_gate_params gp = *params;
  if (gp.topk < 1 || gp.topk > SENSE_MAX_KAPPA) return fail(SENSE_ERR_INVALID_ARG, "topk=%d outside [1, %d]", gp.topk, SENSE_MAX_KAPPA);
  if (gp.window < 1 || gp.window > SENSE_MAX_WINDOW) return fail(SENSE_ERR_INVALID_ARG, "window=%d outside [1, %d]", gp.window, SENSE_MAX_WINDOW);
  if (gp.tau < 0) return fail(SENSE_ERR_INVALID_ARG, "tau=%d must be >= 0", gp.tau);
  if (gp.flags & ~SENSE_GATE_UNNORMALIZED_ENTROPY) return fail(SENSE_ERR_INVALID_ARG, "unknown gate flags 0x%x", gp.flags);
  if (!(gp.gamma == gp.gamma)) return fail(SENSE_ERR_INVALID_ARG, "gamma is NaN");
  if (vocab < gp.topk || vocab < 4 || (vocab % 4) != 0) return fail(SENSE_ERR_INVALID_ARG, "vocab=%d must be a multiple of 4 and >= topk", vocab);
  if (d < 8 || (d % 8) != 0) return fail(SENSE_ERR_INVALID_ARG, "d=%d must be a positive multiple of 8", d);
  if (!aligned(root_logits, 16) || !aligned(node_logits, 16) || !aligned(root_hidden, 16) ||
      !aligned(node_hidden, 16) || !aligned(out_h_next, 16))
    return fail(SENSE_ERR_INVALID_ARG, "logits and hidden states must be 16-byte aligned");
  if (!aligned(workspace, 256)) return fail(SENSE_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  const size_t need = gate_workspace_bytes(q, cap, gp.topk);
  if (workspace_bytes < need) return fail(SENSE_ERR_INVALID_ARG, "workspace has %zu bytes, needs %zu", workspace_bytes, need);
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  GateArgs a{};
  a.tokens = tokens;
  a.parent = parent;
  a.num_nodes = num_nodes;
  a.gamma = gamma;
  a.q = q;
  a.k = k;
  a.m = m;
  a.cap = cap;
  a.root_logits = root_logits;
  a.node_logits = node_logits;
  a.vocab = vocab;
  a.root_hidden = root_hidden;
  a.node_hidden = node_hidden;
  a.d = d;
  a.thr = gp.gamma;
  a.kappa = gp.topk;
  a.window = gp.window;
  a.tau = gp.tau;
  a.unnormalized = (gp.flags & SENSE_GATE_UNNORMALIZED_ENTROPY) ? 1 : 0;
  a.i_star = out_i_star;
  a.L_star = out_L_star;
  a.n_accept = out_n_accept;
  a.accepted = out_accepted;
  a.next_node = out_next_node;
  a.next_anchor = out_next_anchor;
  a.h_next = out_h_next;
  a.G = out_G;
  a.workspace = workspace;
  a.status = status;
  return launch_gate(a, stream);
}

sense_status sense_selftest_timeout(sense_stream_t stream, int64_t limit_cycles) {
  if (limit_cycles < 1 || limit_cycles > (1LL << 34))
    return fail(SENSE_ERR_INVALID_ARG, "limit_cycles=%lld outside [1, 2^34]", (long long)limit_cycles);
  uint32_t* status = device_status_word();
  if (!status) return SENSE_ERR_OOM;
  return launch_selftest_wait(limit_cycles, status, stream);
}

sense_status sense_profile_enable(int32_t on) {
  std::lock_guard<std::mutex> lk(g_mu);
  for (auto& r : g_prof) {
    g_ev_pool.push_back(r.a);
    g_ev_pool.push_back(r.b);
  }
  g_prof.clear();
  g_prof_on = on != 0;
  for (int i = 0; i < K_COUNT; ++i) g_prof_family[i] = true;
  return SENSE_OK;
}

sense_status sense_profile_filter(const char* names) {
  bool sel[K_COUNT];
  for (int i = 0; i < K_COUNT; ++i) sel[i] = (names == nullptr || names[0] == 0);
  if (names && names[0]) {
    const char* p = names;
    while (*p) {
      const char* e = strchr(p, ',');
      const size_t len = e ? (size_t)(e - p) : strlen(p);
      int id = -1;
      for (int i = 0; i < K_COUNT; ++i)
        if (strlen(kKernelNames[i]) == len && strncmp(p, kKernelNames[i], len) == 0) id = i;
      if (id < 0) return fail(SENSE_ERR_INVALID_ARG, "unknown kernel family in '%s'", names);
      sel[id] = true;
      p = e ? e + 1 : p + len;
    }
  }
  std::lock_guard<std::mutex> lk(g_mu);
  for (int i = 0; i < K_COUNT; ++i) g_prof_family[i] = sel[i];
  return SENSE_OK;
}

int32_t sense_profile_count(void) { return K_COUNT; }

const char* sense_profile_name(int32_t i) {
  if (i < 0 || i >= K_COUNT) return "";
  return kKernelNames[i];
}

sense_status sense_profile_query(const char* name, double* total_ms, int64_t* launches) {
  if (!name || !total_ms || !launches) return fail(SENSE_ERR_INVALID_ARG, "NULL argument");
  int id = -1;
  for (int i = 0; i < K_COUNT; ++i)
    if (strcmp(name, kKernelNames[i]) == 0) id = i;
  if (id < 0) return fail(SENSE_ERR_INVALID_ARG, "unknown kernel name '%s'", name);
  std::lock_guard<std::mutex> lk(g_mu);
  double tot = 0.0;
  int64_t cnt = 0;
  for (auto& r : g_prof) {
    if (r.id != id) continue;
    sense_status st = cuda_check(cudaEventSynchronize(r.b), "cudaEventSynchronize");
    if (st != SENSE_OK) return st;
    float ms = 0.0f;
    st = cuda_check(cudaEventElapsedTime(&ms, r.a, r.b), "cudaEventElapsedTime");
    if (st != SENSE_OK) return st;
    tot += ms;
    ++cnt;
  }
  *total_ms = tot;
  *launches = cnt;
  return SENSE_OK;
}

}  // extern "C"
