// Test entry for the bounded pipeline waits: one CTA waits on an mbarrier that
// nothing ever arrives at, through the same bounded wait (tc::mbar_wait) every
// pipelined kernel of the library uses.  The wait gives up after the given
// time and the kernel reports FLARE_DEV_WAIT_TIMEOUT in the status word; the
// context stays usable.  No fault, no trap, no unbounded spin.
#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace flare {

namespace {
__global__ void debug_wait_timeout_kernel(int32_t* status, unsigned long long limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar, 1);
    tc::fence_mbar_init();
  }
  __syncthreads();
  const bool ok = tc::mbar_wait(&bar, 0u, nullptr, limit_ns);  // phase 0 never completes
  if (!ok && threadIdx.x == 0) flag(status, FLARE_DEV_WAIT_TIMEOUT);
}
}  // namespace

cudaError_t launch_debug_wait_timeout(int32_t* status, uint64_t limit_ns, cudaStream_t stream) {
  debug_wait_timeout_kernel<<<1, 32, 0, stream>>>(status, (unsigned long long)limit_ns);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace flare
