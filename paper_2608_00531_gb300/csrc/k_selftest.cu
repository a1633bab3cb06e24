// Failure-detection self-test: the library's bounded pipeline wait, run on a
// barrier that nothing ever completes.  The wait must give up after its limit,
// raise CURE_DEVERR_TIMEOUT in the device error word and return, leaving the
// context usable.  No fault, trap or hang is involved.
#include "common.cuh"
#include "tc_ptx.cuh"

namespace cure {
namespace {

__global__ void selftest_wait_kernel(int* err, long long limit) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    tc::mbar_init(tc::smem_u32(&bar), 1);  // one arrival completes a phase; none ever comes
    abort_flag = 0;
    tc::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) tc::wait_bounded(tc::smem_u32(&bar), 0, &abort_flag, err, true, limit);
}

}  // namespace
}  // namespace cure

using namespace cure;

extern "C" cure_status cure_selftest_wait_timeout(int64_t limit_cycles, void* stream) {
  if (limit_cycles < 1 || limit_cycles > tc::kWaitTimeoutCycles) return CURE_ERR_INVALID_ARG;
  selftest_wait_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(device_error_word(), limit_cycles);
  return cudaGetLastError() == cudaSuccess ? CURE_OK : CURE_ERR_CUDA;
}
