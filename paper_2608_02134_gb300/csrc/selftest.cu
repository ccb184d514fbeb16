// gmc_selftest_bounded_wait: the failure path of the library's bounded waits,
// exercised on purpose.  A one-block kernel initialises an mbarrier that
// nothing ever arrives on and waits for its first phase with the same
// clock-bounded helper every TMA / tcgen05 kernel uses (tc::mbar_wait); when
// the limit passes it records GMC_STATUS_TIMEOUT and returns, leaving the
// context usable.  No paper counterpart: it tests the error reporting.
#include "common.cuh"
#include "kernels.cuh"
#include "tc.cuh"

namespace gmc {

__global__ void k_wait_selftest(long long cycles, uint32_t* status) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar, 1);
    tc::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const long long deadline = clock64() + cycles;
    // phase 0 completes only after one arrival, and none is made
    if (!tc::mbar_wait(&bar, 0u, deadline)) set_status(status, GMC_STATUS_TIMEOUT);
  }
}

}  // namespace gmc

extern "C" int gmc_selftest_bounded_wait(long long cycles, void* workspace, size_t ws_bytes,
                                         gmc_stream_t stream_) {
  // at most about two seconds at the GB300's 2.07 GHz, like the kernels' own limit
  if (cycles < 0 || cycles > 4000000000LL || !workspace || ws_bytes < sizeof(uint32_t) ||
      ((uintptr_t)workspace % 256) != 0)
    return GMC_ERR_ARG;
  cudaStream_t st = (cudaStream_t)stream_;
  uint32_t* status = static_cast<uint32_t*>(workspace);
  if (cudaMemsetAsync(status, 0, sizeof(uint32_t), st) != cudaSuccess) {
    cudaGetLastError();
    return GMC_ERR_CUDA;
  }
  gmc::k_wait_selftest<<<1, 32, 0, st>>>(cycles, status);
  if (cudaGetLastError() != cudaSuccess) return GMC_ERR_CUDA;
  return GMC_OK;
}
