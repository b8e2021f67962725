// Self-test of the failure path every kernel of the library shares: a wait
// that is never satisfied gives up after its limit, records the timeout in
// the device status word and returns, leaving the context usable.  The
// kernel waits on purpose for something that never happens: an mbarrier
// that no thread and no copy completes (kind 0), or a global flag that
// nothing sets, polled with acquire loads (kind 1).
#include "kernels.cuh"

namespace mpc {

__global__ void __launch_bounds__(64) wait_selftest_kernel(int kind, const int* never_set, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  if (kind == 0) {
    (void)mbar_wait_bounded(&bar, 0, limit_ns);  // sets the timeout flag itself
    return;
  }
  const uint64_t t0 = global_timer_ns();
  while (ld_acquire(never_set) == 0) {
    if (global_timer_ns() - t0 > limit_ns) {
      atomicOr(&g_mpc_status, kStatusWaitTimeout);
      return;
    }
    __nanosleep(256);
  }
}

cudaError_t launch_wait_selftest(int kind, const int* never_set, uint64_t limit_ns, cudaStream_t st) {
  wait_selftest_kernel<<<1, 64, 0, st>>>(kind, never_set, limit_ns);
  return cudaGetLastError();
}

int take_status_selftest() { return take_status(); }

}  // namespace mpc
