// Self-test of the bounded mbarrier wait (the failure detection of every
// pipelined kernel): a wait on a phase that nothing completes must end after
// its limit with DEVERR_TIMEOUT recorded, and the CTA's abort flag must release
// the other waiting roles early.
#include "common.cuh"
#include "kernels.h"

namespace aiq {
namespace {

__global__ void __launch_bounds__(64) k_wait_expiry(uint64_t limit_ns, int* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_word;
  volatile int* abort_flag = &abort_word;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  // nothing arrives on `bar`, so its phase 0 never completes
  const uint64_t limit = threadIdx.x < 32 ? limit_ns : 4 * limit_ns;
  mbar_wait_bounded(&bar, 0, abort_flag, err, limit);
  __syncthreads();
}

}  // namespace

int launch_wait_expiry(uint64_t limit_ns, int* err, cudaStream_t s) {
  k_wait_expiry<<<1, 64, 0, s>>>(limit_ns, err);
  return cudaGetLastError();
}

}  // namespace aiq
