// Diagnostic: a bounded wait that runs out.  One thread waits on an mbarrier that nothing
// arrives on, through the same bounded wait every kernel of the library uses; after its
// %globaltimer limit the wait records PTD_ERR_TIMEOUT in the status word and the kernel
// returns, leaving the context usable.  No fault, trap or endless loop is involved.
#include <cuda_runtime.h>

#include <cstdint>

#include "ptd_device.cuh"

namespace ptd {
namespace st {

__global__ void bounded_wait_kernel(int32_t* __restrict__ dev_status) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // phase 0 of a fresh barrier with one expected arrival never completes
    mbar_wait(smem_u32(&bar), 0u, &abort_flag, dev_status);
  }
}

}  // namespace st

cudaError_t launch_bounded_wait_check(int32_t* dev_status, cudaStream_t stream) {
  st::bounded_wait_kernel<<<1, 32, 0, stream>>>(dev_status);
  return cudaGetLastError();
}

}  // namespace ptd
