// Shared declarations of libsense: host-side plumbing (errors, status word,
// launch profiling) and small device helpers used by several kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "sense.h"

namespace sense {

// ---------------------------------------------------------------------------
// Host plumbing (defined in api.cu)
// ---------------------------------------------------------------------------

// Records a formatted message for sense_last_error() and returns `s`.
sense_status fail(sense_status s, const char* fmt, ...);
// Maps a CUDA error to SENSE_ERR_CUDA with a message; cudaSuccess -> SENSE_OK.
sense_status cuda_check(cudaError_t e, const char* what);
// Device pointer of the status word of the current device (allocated on the
// first call per device).  Returns nullptr and sets the error on failure.
uint32_t* device_status_word();
// Number of SMs of the current device (cached per device).
int sm_count();
// cudaFuncSetAttribute(f, MaxDynamicSharedMemorySize, bytes), skipped when
// a value at least as large was already set for f on the current device
// (the attribute call costs host time on every launch otherwise).
cudaError_t func_smem(const void* f, int bytes);

enum KernelId {
  K_NORMALIZE = 0,
  K_SCAN_GEMV,
  K_SCAN_TC,
  K_THRESHOLD,
  K_MERGE,
  K_GATHER,
  K_TREE,
  K_GATE_ROWS,
  K_GATE_DECIDE,
  K_PAD_QUERIES,
  K_TREE_MASK,
  K_PROJECT,
  K_KMEANS,
  K_IVF_BUILD,
  K_IVF_COARSE,
  K_IVF_SCAN,
  K_CTX,
  K_TREE_ATTN,
  K_RESCORE,
  K_DRAFT,
  K_COUNT
};

// Brackets one kernel launch with CUDA events when profiling is enabled.
struct LaunchScope {
  LaunchScope(KernelId id, cudaStream_t s);
  ~LaunchScope();
  KernelId id_;
  cudaStream_t s_;
  int slot_;
};

// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------

// Order-preserving map of an fp32 score to uint32 (larger score -> larger
// code).  -0 is folded onto +0 so that equal scores give equal codes.
__device__ __forceinline__ uint32_t score_code(float s) {
  uint32_t b = __float_as_uint(s == 0.0f ? 0.0f : s);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float code_score(uint32_t c) {
  uint32_t b = (c & 0x80000000u) ? (c & 0x7fffffffu) : ~c;
  return __uint_as_float(b);
}
// Candidate key: score code in the high word, bitwise-inverted key index in
// the low word, so that a larger key means (higher score, then lower index).
__device__ __forceinline__ uint64_t cand_key(float s, uint32_t idx) {
  return ((uint64_t)score_code(s) << 32) | (uint64_t)(~idx);
}
__device__ __forceinline__ uint32_t cand_index(uint64_t c) { return ~(uint32_t)c; }

// Programmatic dependent launch: a kernel launched with
// cudaLaunchAttributeProgrammaticStreamSerialization may be scheduled
// before the kernel ahead of it in the stream has finished; pdl_wait()
// blocks until that kernel has completed and its memory is visible (a
// no-op for a normal launch).  pdl_launch_dependents() lets the next such
// kernel be scheduled while this one still runs.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launches `kern` with programmatic stream serialization (see pdl_wait).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

__device__ __forceinline__ void raise_status(uint32_t* st, uint32_t bits) {
  if (st) atomicOr(st, bits);
}

// 128-bit streaming load that bypasses L1 (data read once).
__device__ __forceinline__ uint4 ld_stream_v4(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// bf16x2 word -> two floats (bf16 is the top half of an fp32 word).
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Warp-aggregated increment of a counter: returns this lane's slot.
__device__ __forceinline__ uint32_t warp_append(uint32_t* counter, bool want) {
  const unsigned act = __activemask();
  const unsigned m = __ballot_sync(act, want);
  if (!want) return 0;
  const int lane = threadIdx.x & 31;
  const int leader = __ffs(m) - 1;
  uint32_t base = 0;
  if (lane == leader) base = atomicAdd(counter, (uint32_t)__popc(m));
  base = __shfl_sync(m, base, leader);
  return base + __popc(m & ((1u << lane) - 1u));
}

// Sorted list of KPL * 32 candidate keys spread over a warp: position
// r = s * 32 + lane lives in v[s] of that lane, larger keys first.  Inserts
// the warp-uniform key c (distinct from every key in the list); the last
// entry drops out.
template <int KPL>
__device__ __forceinline__ void list_insert(uint64_t (&v)[KPL], uint64_t c, int lane) {
  int p = 0;  // keys ahead of c (all keys are distinct)
#pragma unroll
  for (int s = 0; s < KPL; ++s) p += __popc(__ballot_sync(0xffffffffu, v[s] > c));
  uint64_t up[KPL], last[KPL];
#pragma unroll
  for (int s = 0; s < KPL; ++s) {
    up[s] = __shfl_up_sync(0xffffffffu, v[s], 1);
    last[s] = __shfl_sync(0xffffffffu, v[s], 31);
  }
#pragma unroll
  for (int s = 0; s < KPL; ++s) {
    const int r = s * 32 + lane;
    const uint64_t prev = (lane == 0) ? (s > 0 ? last[s > 0 ? s - 1 : 0] : 0ull) : up[s];
    v[s] = (r < p) ? v[s] : (r == p ? c : prev);
  }
}

}  // namespace sense
