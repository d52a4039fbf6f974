// wait.cuh — bounded mbarrier waits.  No wait in this library can spin
// forever: past its time limit a wait records DA_ERR_TIMEOUT in the device
// status word, raises the CTA's abort flag and returns false.
#pragma once
#include <stdint.h>

#include "ptx.cuh"

namespace da {

constexpr int kStatusTimeout = -6;  // DA_ERR_TIMEOUT
constexpr uint64_t WAIT_LIMIT_NS = 1000000000ull;

__device__ __forceinline__ bool wait_bounded(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                             int* status, uint64_t limit_ns = WAIT_LIMIT_NS) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255u) == 0) {
      if (*abort_flag) return false;
      if (globaltimer_ns() - t0 > limit_ns) {
        *abort_flag = 1;
        atomicCAS(status, 0, kStatusTimeout);
        return false;
      }
    }
  }
}

// For waits that span a whole work item (the epilogue's): polls with a short
// sleep so the waiting warp leaves the issue slots to the busy warps.
__device__ __forceinline__ bool wait_sleepy(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* status) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
    __nanosleep(200);
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) {
      *abort_flag = 1;
      atomicCAS(status, 0, kStatusTimeout);
      return false;
    }
  }
}

// Used on the way out: waits for this CTA's own copies/MMAs even after an
// abort, still with a time limit.
__device__ __forceinline__ void wait_drain(uint64_t* bar, uint32_t parity, int* status) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) {
      atomicCAS(status, 0, kStatusTimeout);
      return;
    }
  }
}

}  // namespace da
