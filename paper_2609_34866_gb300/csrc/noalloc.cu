// Forward L_JAB for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc (or any allocating library routine) at the point where they
// want a loss: a process whose device memory is fully reserved up front by another allocator, code
// running inside a CUDA-graph capture or a real-time loop where allocation is forbidden, or a
// host that must not grow its device footprint after start-up. This entry point gives them the
// candidate-loss forward without a caller workspace: the scratch lives in one fixed, file-scope
// device array that every GPU loading this library holds until the process exits.
//
// It is the same computation as jab_loss_forward: it calls that entry point with the array as its
// workspace and changes nothing else.
#include <mutex>

#include "common.cuh"

namespace jab {
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(JAB_NOALLOC_SCRATCH_BYTES);

// The scratch. In host code this name is only a host-side stand-in for the device symbol: its
// device address is looked up with cudaGetSymbolAddress (below) and only that address is passed on.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch on the current device; looked up once per device.
jab_status scratch_address(void** ptr) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return JAB_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr)
      return JAB_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *ptr = g_scratch_ptr[dev];
  return JAB_OK;
}

}  // namespace
}  // namespace jab

extern "C" jab_status jab_loss_forward_noalloc(const jab_block_desc* desc, int32_t B, int32_t T,
                                               const void* X_dev, const void* W_dev,
                                               const float* A_ref_dev, int32_t n_cand,
                                               const int32_t* bits_host,
                                               const float* const* scales_host, double* loss_dev,
                                               double* sse_parts_dev, jab_stream_t stream) {
  const size_t need = jab_workspace_size(desc, B, T, n_cand, 0);
  if (need > jab::kNoAllocScratchBytes) return JAB_ERR_SCRATCH_LIMIT;
  void* scratch = nullptr;
  const jab_status s = jab::scratch_address(&scratch);
  if (s != JAB_OK) return s;
  // need == 0 means invalid arguments: jab_loss_forward reports which.
  return jab_loss_forward(desc, B, T, X_dev, W_dev, A_ref_dev, n_cand, bits_host, scales_host,
                          loss_dev, sse_parts_dev, scratch, jab::kNoAllocScratchBytes, stream);
}
