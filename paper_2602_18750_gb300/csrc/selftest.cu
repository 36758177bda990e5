// selftest.cu -- exercises the bounded-wait path every kernel relies on.
//
// One warp arms an mbarrier for bytes that no copy will ever deliver and
// waits on it with the same bounded wait (mbar_wait) as the scoring and
// attention kernels, but with a caller-given limit.  The wait must give up,
// raise kErrTimeout in the device error word and let the kernel return, so
// that hill_sync_status() reports HILL_ERR_TIMEOUT and the context stays
// usable.  Nothing here faults, traps or spins without a bound.
#include "hill_internal.h"

namespace hill {
namespace {

__global__ void hill_selftest_wait_kernel(unsigned long long limit_ns, unsigned* err) {
  __shared__ __align__(8) uint64_t bar;
  const uint32_t b = smem_addr(&bar);
  if (threadIdx.x == 0) {
    mbar_init(b, 1);
    fence_barrier_init();
    mbar_arrive_expect_tx(b, 16u);   // 16 bytes that never arrive: phase 0 cannot complete
  }
  __syncwarp();
  (void)mbar_wait(b, 0u, err, limit_ns);
}

}  // namespace

cudaError_t launch_selftest_wait(unsigned long long limit_ns, unsigned* err, cudaStream_t st) {
  hill_selftest_wait_kernel<<<1, 32, 0, st>>>(limit_ns, err);
  return cudaGetLastError();
}

}  // namespace hill
