// Diagnostic: the bounded mbarrier wait every tcgen05 kernel of the library uses, made
// to run out.  One warp waits on an mbarrier nothing arrives on; after the bound (about
// a second) the wait gives up, ORs HD_DEVBIT_TIMEOUT into the status word and the kernel
// returns normally, so the failure path is exercised without a fault and the context
// stays usable.
#include "tc_common.cuh"

namespace hdsfa {

__global__ void __launch_bounds__(32) bounded_wait_selftest_kernel(int32_t* status, int32_t* result) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncwarp();
  // phase 0 of the barrier never completes: the wait can only end by its bound
  const bool ok = __all_sync(0xffffffffu, mbar_wait(&bar, 0, &abort_flag, status));
  if (threadIdx.x == 0) *result = ok ? 1 : 0;
}

cudaError_t launch_bounded_wait_selftest(int32_t* status, int32_t* result, cudaStream_t st) {
  bounded_wait_selftest_kernel<<<1, 32, 0, st>>>(status, result);
  return cudaGetLastError();
}

}  // namespace hdsfa
