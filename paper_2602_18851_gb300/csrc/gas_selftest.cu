// Self-test of the device-side failure detection (gas_selftest_wait_timeout, include/gas.h).
//
// The Gram and write-back kernels never wait without a limit: every mbarrier wait and
// every wait on another CTA's key-tile flag gives up after kWaitLimitNs, raises the
// CTA's abort word, sets GAS_DEV_WAIT_TIMEOUT in the handle's status word and returns.
// This kernel makes those same two waits run out on purpose: an mbarrier phase that no
// thread or copy ever completes, and a global flag that nothing ever writes.  It holds
// no tensor memory and issues no asynchronous copies, so giving up leaves nothing in
// flight and the context stays usable.

#include "gas_device.cuh"

namespace gas {

namespace {

__device__ unsigned g_never_set_flag = 0u;  // no kernel writes it: waiting for 1 runs out

__global__ void __launch_bounds__(32, 1) wait_selftest_kernel(unsigned* status, int which) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_word;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);  // one arrival completes phase 0; none comes
    abort_word = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  volatile int* abort = &abort_word;
  if (which == 0)
    mbar_wait(smem_u32(&bar), 0u, abort, status);
  else
    wait_flag(&g_never_set_flag, 1u, abort, status);
}

}  // namespace

cudaError_t launch_wait_selftest(unsigned* status, int which, cudaStream_t st) {
  wait_selftest_kernel<<<1, 32, 0, st>>>(status, which);
  return cudaGetLastError();
}

}  // namespace gas
