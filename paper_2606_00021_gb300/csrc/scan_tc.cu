// Key scoring for batched queries on tcgen05 tensor cores (written next).
#include "common.cuh"
#include "launch.h"

namespace sense {

size_t scan_tc_smem_bytes(int d, int q) {
  (void)d;
  (void)q;
  return 0;
}

sense_status launch_scan_tc(const uint16_t*, int64_t, int, const uint16_t*, int, int, int64_t,
                            const uint64_t*, uint64_t*, uint32_t*, int64_t, uint32_t*,
                            cudaStream_t) {
  return fail(SENSE_ERR_UNSUPPORTED, "tensor-core scan not built");
}

}  // namespace sense
