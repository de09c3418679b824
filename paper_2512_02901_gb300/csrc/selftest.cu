// Self-test of the device-side failure detection: the bounded mbarrier wait that every pipeline
// barrier of the matmul kernels uses, run on a barrier that nothing completes. The wait gives up
// after its limit, latches the timeout bit in the status word and the kernel returns normally,
// so the context stays usable.
#include <cuda_runtime.h>

#include "common.cuh"
#include "ptx.cuh"
#include "tc.cuh"

namespace fairy2i {

__global__ void selftest_wait_kernel(unsigned int* status, uint64_t limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (!mbar_wait_timed(&bar, 0, limit_ns)) latch_status(status, kStatusTimeout);
    mbar_arrive(&bar);   // complete the phase: the barrier is left consistent
  }
}

fairy2i_status launch_selftest_wait(uint32_t limit_us, cudaStream_t stream) {
  unsigned int* st = device_status_word();
  if (!st) return FAIRY2I_ERR_CUDA;
  selftest_wait_kernel<<<1, 32, 0, stream>>>(st, (uint64_t)limit_us * 1000ull);
  return cudaGetLastError() == cudaSuccess ? FAIRY2I_OK : FAIRY2I_ERR_CUDA;
}

}  // namespace fairy2i
