// Diagnostic of the failure-detection path (not part of the paper's method).
//
// Every kernel of the library waits on mbarriers through mbar_wait_for
// (common.cuh): when a phase has not completed within the limit, the wait
// records TK_DEVERR_TIMEOUT in the device error word and returns false, and
// the kernel winds down instead of spinning.  This kernel drives that path on
// purpose, with a short limit: one thread waits on a barrier that nothing
// ever arrives at, so the wait must run out, record the code and return.
#include "common.cuh"
#include "kernels.h"

namespace tk {
namespace {

__global__ void wait_timeout_kernel(int* err, uint64_t limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);  // one arrival would complete phase 0; none comes
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const bool completed = mbar_wait_for(&bar, 0, err, limit_ns);
    // the barrier cannot have completed; a true here would be a logic error
    if (completed) record_error(err, TK_DEVERR_INDEX);
  }
  __syncthreads();
}

}  // namespace

cudaError_t launch_wait_timeout(int* err, uint64_t limit_ns, cudaStream_t stream) {
  wait_timeout_kernel<<<1, 32, 0, stream>>>(err, limit_ns);
  return cudaGetLastError();
}

}  // namespace tk
