// Failure-path check: a bounded wait that runs out.  The tensor-core
// pipelines hand data between roles through mbarriers and every wait on them
// gives up after ~2 s (mbar_wait_bounded), raising EBD_DEV_TIMEOUT instead of
// spinning forever.  This kernel exercises exactly that path on a barrier
// phase that nothing completes, so the status and the context's survival can
// be checked without stalling a real pipeline.
#include <cuda_runtime.h>

#include "common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace ebd {

__global__ void stalled_wait_kernel(int32_t* dev_status) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
  }
  __syncthreads();
  // no thread arrives on `bar`: its phase 0 never completes
  if (threadIdx.x == 0 && !mbar_wait_bounded(&bar, 0)) raise_status(dev_status, EBD_DEV_TIMEOUT);
}

}  // namespace ebd

using namespace ebd;

extern "C" ebd_status ebd_check_stalled_wait(int32_t* dev_status, void* stream) {
  if (!dev_status) return EBD_ERR_INVALID;
  stalled_wait_kernel<<<1, 32, 0, (cudaStream_t)stream>>>(dev_status);
  return launch_status();
}
