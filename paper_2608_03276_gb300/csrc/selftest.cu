// Self-test of the failure path shared by every kernel: a bounded mbarrier
// wait that gives up, records TP_ERR_TIMEOUT in the status word and lets the
// kernel return normally, so the context stays usable.
#include <cuda_runtime.h>
#include <stdint.h>

#include "tp_device.cuh"
#include "tp_internal.h"

namespace tp {

namespace {

// One thread waits, through the waits' common routine, on an mbarrier that
// nothing ever arrives at; after limit_ns it gives up.
__global__ void tp_wait_selftest_kernel(int* status, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && !mbar_wait_limit(&bar, 0, &abort_flag, limit_ns))
    set_status(status, TP_ERR_TIMEOUT);
}

}  // namespace

cudaError_t launch_wait_selftest(int* status, uint64_t limit_ns, cudaStream_t s) {
  tp_wait_selftest_kernel<<<1, 32, 0, s>>>(status, limit_ns);
  return cudaGetLastError();
}

}  // namespace tp
