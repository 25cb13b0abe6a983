// Self-test of the failure path of the pipelined kernels: one CTA waits, with the same bounded
// mbarrier wait every tcgen05 kernel uses, on a barrier phase that nothing will ever complete. The
// wait gives up after its limit, raises JAB_ERR_TIMEOUT in the device status word and the kernel
// returns normally, leaving the context usable.
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
