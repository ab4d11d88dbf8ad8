// Failure-detection self-test: every device-side wait of the library is
// bounded and reports BOUTE_ERR_TIMEOUT when its bound runs out (instead of
// hanging). This kernel makes one such wait run out on purpose, with a short
// bound, on an mbarrier that nothing arrives on, through the same bounded
// wait the kernels use; with `complete` the one expected arrival is made and
// the wait succeeds. No fault, no trap: the waiting thread gives up, records
// the status and the kernel returns.
#include "internal.h"

namespace boute {

namespace {

__global__ void wait_selftest_kernel(int complete, unsigned long long limit_ns, int *status) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (complete) mbar_arrive_count(&bar);
    if (!mbar_wait_ns(&bar, 0, limit_ns)) set_status(status, BOUTE_ERR_TIMEOUT);
  }
}

}  // namespace

int launch_wait_selftest(int complete, unsigned long long limit_ns, int *status, cudaStream_t s) {
  wait_selftest_kernel<<<1, 32, 0, s>>>(complete, limit_ns, status);
  count_launch();
  return last_launch_status();
}

}  // namespace boute
