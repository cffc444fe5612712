// Failure-detection self-test: a kernel whose one wait can never be satisfied.
//
// Every wait the library's kernels do on an mbarrier is bounded; when one
// gives up it sets a bit in the handle's error word and returns instead of
// hanging, so the CUDA context stays usable and the host learns of it at the
// next dqgan_synchronize.  This kernel exercises exactly that path on demand,
// without a fault: thread 0 initialises an mbarrier that expects one arrival,
// nobody arrives, and the bounded poll loop runs out.
#include "device_common.cuh"
#include "internal.cuh"

namespace dq {

__global__ void __launch_bounds__(32) wait_selftest_kernel(uint32_t polls, uint32_t* err) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    mbar_fence_init();
  }
  __syncwarp();
  if (threadIdx.x != 0) return;
  bool done = false;
  // Phase 0 of a fresh barrier completes only after one arrival, which never comes.
  for (uint32_t it = 0; it < polls && !done; ++it) done = mbar_try_wait(&bar, 0);
  if (!done) atomicOr(err, kErrTimeout);
}

cudaError_t launch_wait_selftest(uint32_t polls, uint32_t* err, cudaStream_t stream, uint64_t* launches) {
  wait_selftest_kernel<<<1, 32, 0, stream>>>(polls, err);
  *launches += 1;
  return cudaGetLastError();
}

uint32_t wait_selftest_max_polls() { return kSpinLimit; }

}  // namespace dq
