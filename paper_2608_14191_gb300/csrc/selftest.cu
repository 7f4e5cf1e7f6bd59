// Test hook for the bounded waits of this library's kernels (failure detection without a GPU
// fault): one CTA waits on an mbarrier that nothing ever arrives on, with the same bounded wait
// the encode, decode and prefill kernels use.  The wait gives up after the limit, the CTA records
// bit 1 of the device flags exactly as those kernels do on a timeout, and the kernel returns
// normally, so the context stays usable.
#include <cstdint>

#include "aatc_internal.h"
#include "ptx.cuh"

namespace aatc {
namespace {

__global__ void aatc_bounded_wait_kernel(int* flags, unsigned long long limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    ptx::mbar_init(&bar, 1);                 // one arrival expected; none is ever made
    abort_flag = 0;
    ptx::fence_mbar_init();
  }
  __syncthreads();
  if (!ptx::mbar_wait_bounded(&bar, 0, &abort_flag, limit_ns)) {
    abort_flag = 1;                          // the other threads stop waiting too
    atomicOr(flags, 2);
  }
}

}  // namespace
}  // namespace aatc

extern "C" aatc_status_t aatc_selftest_bounded_wait(int32_t limit_us, int32_t* dev_flags, void* stream) {
  if (!dev_flags || limit_us < 1 || limit_us > 2000000) return AATC_ERR_INVALID_ARG;
  aatc::aatc_bounded_wait_kernel<<<1, 64, 0, static_cast<cudaStream_t>(stream)>>>(
      reinterpret_cast<int*>(dev_flags), static_cast<unsigned long long>(limit_us) * 1000ull);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? AATC_OK : AATC_ERR_CUDA;
}
