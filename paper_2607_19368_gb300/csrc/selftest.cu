// Self-test of the device-side wait limits, the failure path that every
// long-running kernel of the library relies on: a wait that is never
// satisfied -- an mbarrier nothing arrives at, a group barrier one CTA of the
// group never reaches -- gives up after about a second of clock cycles,
// records SLS_ERR_TIMEOUT in the status word and returns, so the context
// stays usable.  The kernels below use the same wait routines as the
// Lanczos, feature-map and segment kernels.
#include "common.cuh"
#include "kernels.cuh"

namespace sls {

namespace {

__global__ void selftest_mbar_kernel(int* status) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);  // one arrival completes phase 0; none is made
    mbar_fence_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && !mbar_wait(&bar, 0)) atomicExch(status, SLS_ERR_TIMEOUT);
}

// A cooperative grid of two CTAs: CTA 1 leaves without arriving, CTA 0 waits
// at the group barrier until the limit.
__global__ void selftest_group_kernel(unsigned* barw, int* status) {
  __shared__ int sflag;
  __shared__ volatile int serr;
  if (threadIdx.x == 0) serr = 0;
  __syncthreads();
  if (blockIdx.x == 1) return;
  const GroupBarrier bar{barw, barw + 32, gridDim.x};
  unsigned gen = 0;
  group_sync_named(bar, gen, status, &sflag, &serr, 1, blockDim.x);
}

}  // namespace

int launch_selftest_wait_limit(int which, int* status, unsigned* barw, cudaStream_t stream) {
  SLS_CUDA_TRY(cudaMemsetAsync(status, 0, sizeof(int), stream));
  if (which == 0) {
    selftest_mbar_kernel<<<1, 32, 0, stream>>>(status);
    SLS_LAUNCH_CHECK();
    return SLS_OK;
  }
  SLS_CUDA_TRY(cudaMemsetAsync(barw, 0, 256, stream));
  void* args[] = {(void*)&barw, (void*)&status};
  SLS_CUDA_TRY(cudaLaunchCooperativeKernel((const void*)selftest_group_kernel, dim3(2), dim3(32),
                                           args, 0, stream));
  count_launch(1);
  return SLS_OK;
}

}  // namespace sls
