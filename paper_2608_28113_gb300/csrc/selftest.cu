// selftest.cu -- exercises the failure path of the library's bounded waits on the GPU
// without a fault: one CTA waits on an mbarrier that nothing arrives on, with a small poll
// limit, and reports the timeout through the device error flags exactly as the TMA
// pipelines do (mbar_wait_bounded, then a sticky flag bit), after which the kernel ends
// normally and the context stays usable.
#include "hscale_internal.h"
#include "tma.cuh"

namespace hscale {
namespace {

__device__ uint32_t g_selftest_flags = 0;

__global__ void bounded_wait_kernel(uint32_t polls) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    mbar_fence_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && !mbar_wait_bounded(&bar, 0u, polls)) atomicOr(&g_selftest_flags, kErrMbarTimeout);
}

}  // namespace

cudaError_t launch_bounded_wait_selftest(uint32_t polls, cudaStream_t stream) {
  bounded_wait_kernel<<<1, 32, 0, stream>>>(polls);
  return cudaGetLastError();
}

cudaError_t read_selftest_device_error(uint32_t* flags) {
  uint32_t v = 0;
  cudaError_t err = cudaMemcpyFromSymbol(&v, g_selftest_flags, sizeof v);
  if (err != cudaSuccess) return err;
  *flags = v;
  if (v) {
    const uint32_t zero = 0;
    err = cudaMemcpyToSymbol(g_selftest_flags, &zero, sizeof zero);
  }
  return err;
}

}  // namespace hscale
