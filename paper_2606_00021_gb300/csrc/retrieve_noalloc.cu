// Top-k retrieval for callers that cannot allocate device memory.
//
// sense_retrieve_topk needs a caller-provided device workspace.  Some
// callers have none to give and may not call cudaMalloc either: a serving
// process whose whole device memory is carved up in advance by another
// allocator, or a plug-in that runs inside a host application which exposes
// no device allocator to it (cudaMalloc can synchronise the device and fail
// in the middle of a request, which such hosts forbid).  This entry point
// runs the same kernels with their scratch taken from one file-scope device
// array of fixed size instead.
//
// The array lives in this file's module: every GPU that loads the library
// and uses this entry point holds its kNoallocScratchBytes until the process
// exits.  Its device address is looked up once per device, on the first
// call made with that device current, and kept for the life of the process
// (no call of this library may span a cudaDeviceReset).  All calls share the
// array and it keeps the previous call's contents: the per-query counters
// are cleared on every call, and calls whose work overlaps on the GPU
// (different streams with no ordering between them) race on the array.
//
// The first 256 bytes of the array hold this entry point's own device
// status word: the kernels' device-side checks (an internal consistency
// check, a bounded wait that ran out) set bits there.  Every call clears it
// first; sense_retrieve_noalloc_status reads it after the call.
#include <mutex>

#include "common.cuh"
#include "launch.h"

namespace sense {
namespace {

constexpr size_t kNoallocScratchBytes = SENSE_NOALLOC_SCRATCH_BYTES;
// First 256 bytes: the status word of this entry point; the rest: workspace.
constexpr size_t kStatusBytes = 256;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

constexpr int kMaxDev = 64;
std::mutex g_mu;
char* g_ptr[kMaxDev] = {nullptr};

// Device address of the array on the current device (looked up once).
sense_status scratch_address(char** out) {
  int dev = 0;
  sense_status st = cuda_check(cudaGetDevice(&dev), "cudaGetDevice");
  if (st != SENSE_OK) return st;
  if (dev < 0 || dev >= kMaxDev) return fail(SENSE_ERR_UNSUPPORTED, "device ordinal %d too large", dev);
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_ptr[dev]) {
    void* p = nullptr;
    st = cuda_check(cudaGetSymbolAddress(&p, g_noalloc_scratch), "cudaGetSymbolAddress(scratch)");
    if (st != SENSE_OK) return st;
    g_ptr[dev] = static_cast<char*>(p);
  }
  *out = g_ptr[dev];
  return SENSE_OK;
}

bool is_aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace
}  // namespace sense

using namespace sense;

extern "C" sense_status sense_retrieve_topk_noalloc(const sense_datastore* ds,
                                                    const uint16_t* queries, int32_t q, int32_t k,
                                                    float* out_scores, int32_t* out_idx,
                                                    sense_stream_t stream) {
  if (!ds) return fail(SENSE_ERR_INVALID_ARG, "datastore handle is NULL");
  int dev = 0;
  sense_status st = cuda_check(cudaGetDevice(&dev), "cudaGetDevice");
  if (st != SENSE_OK) return st;
  if (ds->device != dev)
    return fail(SENSE_ERR_INVALID_ARG, "datastore was built on device %d, current device is %d",
                ds->device, dev);
  if (!queries || !out_scores || !out_idx)
    return fail(SENSE_ERR_INVALID_ARG, "queries and outputs must be non-NULL");
  if (q < 1) return fail(SENSE_ERR_INVALID_ARG, "q=%d must be >= 1", q);
  if (k < 1 || k > SENSE_MAX_K || (int64_t)k > ds->n)
    return fail(SENSE_ERR_INVALID_ARG, "k=%d outside [1, min(n=%lld, %d)]", k,
                (long long)ds->n, SENSE_MAX_K);
  if (!is_aligned(queries, 16)) return fail(SENSE_ERR_INVALID_ARG, "queries must be 16-byte aligned");
  if (q > 8 && ds->n > 2147483647LL - 1024)
    return fail(SENSE_ERR_UNSUPPORTED, "batched (q > 8) retrieval supports n <= 2^31 - 1025");
  const RetrievePlan p = make_plan(ds, q, k);
  if (p.total > kNoallocScratchBytes - kStatusBytes)
    return fail(SENSE_ERR_UNSUPPORTED,
                "this request needs %zu bytes of scratch but the static scratch holds %zu; "
                "use sense_retrieve_topk with a workspace, or fewer queries or keys",
                p.total, kNoallocScratchBytes - kStatusBytes);
  char* base = nullptr;
  st = scratch_address(&base);
  if (st != SENSE_OK) return st;
  uint32_t* status = reinterpret_cast<uint32_t*>(base);
  st = cuda_check(cudaMemsetAsync(status, 0, sizeof(uint32_t), stream), "clear status word");
  if (st != SENSE_OK) return st;
  return run_retrieve(p, ds, queries, q, k, out_scores, out_idx, base + kStatusBytes, status,
                      stream);
}

extern "C" sense_status sense_retrieve_noalloc_status(sense_stream_t stream, uint32_t* out_bits,
                                                      int32_t clear) {
  if (!out_bits) return fail(SENSE_ERR_INVALID_ARG, "out_bits is NULL");
  char* base = nullptr;
  sense_status st = scratch_address(&base);
  if (st != SENSE_OK) return st;
  st = cuda_check(cudaStreamSynchronize(stream), "cudaStreamSynchronize");
  if (st != SENSE_OK) return st;
  uint32_t v = 0;
  st = cuda_check(cudaMemcpy(&v, base, sizeof(v), cudaMemcpyDeviceToHost), "read status word");
  if (st != SENSE_OK) return st;
  if (clear) {
    st = cuda_check(cudaMemset(base, 0, sizeof(uint32_t)), "clear status word");
    if (st != SENSE_OK) return st;
  }
  *out_bits = v;
  if (v & SENSE_DEVST_TIMEOUT)
    return fail(SENSE_ERR_TIMEOUT, "a device wait of the allocation-free retrieval hit its limit "
                "(bits 0x%x)", v);
  if (v) return fail(SENSE_ERR_DEVICE_STATUS, "allocation-free retrieval status bits 0x%x", v);
  return SENSE_OK;
}

extern "C" sense_status sense_retrieve_noalloc_selftest(sense_stream_t stream,
                                                        int64_t limit_cycles) {
  if (limit_cycles < 1 || limit_cycles > (1LL << 34))
    return fail(SENSE_ERR_INVALID_ARG, "limit_cycles=%lld outside [1, 2^34]",
                (long long)limit_cycles);
  char* base = nullptr;
  sense_status st = scratch_address(&base);
  if (st != SENSE_OK) return st;
  return launch_selftest_wait(limit_cycles, reinterpret_cast<uint32_t*>(base), stream);
}
