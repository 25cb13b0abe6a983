// Self-tests of the failure paths:
//   - the pipelined kernels' bounded wait: one CTA waits, with the same bounded mbarrier wait every
//     tcgen05 kernel uses, on a barrier phase that nothing will ever complete. The wait gives up
//     after its limit, raises JAB_ERR_TIMEOUT in the device status word and the kernel returns
//     normally, leaving the context usable;
//   - the checked build's bounds checks: writes to indices 0 .. n of an n-element extent, each
//     behind in_bounds; the last is skipped and raises JAB_ERR_DEVICE_ASSERT.
#include "tc.cuh"

namespace jab {
namespace {

__global__ void selftest_wait_kernel(int* status) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar, 1);  // expects one arrival; none is ever made
    abort_flag = 0;
    tc::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) tc::mbar_wait(&bar, 0, &abort_flag, status);
}

#if JAB_CHECKED
__global__ void selftest_bounds_kernel(int32_t* buf, int32_t n, int* status) {
  for (int32_t i = threadIdx.x; i <= n; i += blockDim.x)
    if (in_bounds(i, n, status)) buf[i] = i;
}
#endif

}  // namespace

// Declared in jab.h; the device status word lives in api.cu.
jab_status device_status_ptr(int** status);

}  // namespace jab

extern "C" jab_status jab_selftest_wait_timeout(jab_stream_t stream) {
  int* status = nullptr;
  const jab_status s = jab::device_status_ptr(&status);
  if (s != JAB_OK) return s;
  jab::selftest_wait_kernel<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(status);
  return cudaGetLastError() == cudaSuccess ? JAB_OK : JAB_ERR_CUDA;
}

extern "C" jab_status jab_selftest_bounds_check(int32_t* buf_dev, int32_t n, jab_stream_t stream) {
  if (buf_dev == nullptr || n < 1) return JAB_ERR_INVALID_ARG;
#if JAB_CHECKED
  int* status = nullptr;
  const jab_status s = jab::device_status_ptr(&status);
  if (s != JAB_OK) return s;
  jab::selftest_bounds_kernel<<<1, 128, 0, reinterpret_cast<cudaStream_t>(stream)>>>(buf_dev, n,
                                                                                    status);
  return cudaGetLastError() == cudaSuccess ? JAB_OK : JAB_ERR_CUDA;
#else
  (void)stream;
  return JAB_ERR_UNSUPPORTED;  // the normal build has no checks: its kernel would write past n
#endif
}
