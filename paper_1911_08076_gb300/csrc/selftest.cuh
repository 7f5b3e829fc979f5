// Failure-path self-test: one warp waits on an mbarrier phase that nothing completes, bounded by a
// caller-given wall-time limit, and on running out records IFQ_ETIMEOUT in the device status word,
// exactly as every bounded wait of the conv kernels does (2 s there).  The kernel then returns
// normally: no trap, no fault, and the context stays usable.
#pragma once
#include <cstdint>

#include "ptx.cuh"

namespace ifq {

__global__ void wait_selftest_kernel(unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  const uint32_t b = smem_u32(&bar);
  if (threadIdx.x == 0) {
    mbar_init(b, 1);   // one arrival completes phase 0, and none is ever made
    fence_mbar_init();
  }
  __syncwarp();
  const unsigned long long t0 = global_ns();
  bool done = false;
  for (uint32_t it = 0; it < kWaitLimit && !done; ++it) {
    done = mbar_try(b, 0);
    if (!done && (it & 255u) == 0 && global_ns() - t0 > limit_ns) break;
  }
  if (!__all_sync(0xffffffffu, done) && threadIdx.x == 0) set_status(IFQ_ETIMEOUT);
}

}  // namespace ifq
