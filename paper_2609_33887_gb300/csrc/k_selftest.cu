// Self-test of the failure detection of the kernels' bounded waits: one
// thread waits, through the same bounded mbarrier wait the LM-head kernels
// use, on a barrier that nothing ever completes. After the wait limit it
// records DEV_TIMEOUT in the device status word and the kernel returns, so
// the context stays usable and the host reads the failure with
// bd_get_device_status.
#include "kernels.h"

namespace bd {

__global__ void timeout_selftest_kernel(uint32_t* status) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // no thread arrives on `bar`, so its phase 0 never completes: the wait
    // gives up after WAIT_LIMIT_NS and reports the timeout
    (void)mbar_wait(smem_u32(&bar), 0, &abort_flag, status);
  }
}

cudaError_t launch_timeout_selftest(uint32_t* status, cudaStream_t st) {
  timeout_selftest_kernel<<<1, 32, 0, st>>>(status);
  return cudaGetLastError();
}

}  // namespace bd
