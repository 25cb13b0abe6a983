// Selection between the tensor-core (tcgen05) kernels and the CUDA-core reference kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include "kernels.h"

namespace jab {

// JAB_PATH=simple selects the CUDA-core kernels; anything else (the default) the tcgen05 kernels.
inline bool use_tc_path() {
  static const bool tc = [] {
    const char* p = getenv("JAB_PATH");
    return !(p != nullptr && strcmp(p, "simple") == 0);
  }();
  return tc;
}

// gemm_tc.cu
cudaError_t launch_proj_gemm_tc(const void* A, const void* Bw, void* C, int64_t M, int Nn, int K,
                                int D, int n_rot, int dh, int T, const float* cos_t,
                                const float* sin_t, int* status, cudaStream_t st);
// x: bf16 [N, d] as the caller stores it (no transposed copy)
cudaError_t launch_wgrad_lsq_tc(const void* dqkvt, int64_t ldt, const void* x, const void* w,
                                const float* s, int64_t N, int D, int d, int G, int bits,
                                float coef, float* ds, int* status, cudaStream_t st);
// coef * dQKV^T X stored fp32 [D, d] (dw may be NULL) and its squared norm added to *sqnorm (may be
// NULL; the caller zeroes it)
cudaError_t launch_wgrad_store_tc(const void* dqkvt, int64_t ldt, const void* x, int64_t N, int D,
                                  int d, float coef, float* dw, double* sqnorm, int* status,
                                  cudaStream_t st);
// attn_tc.cu
int attn_fwd_tc_rows(int Hq, int Hkv);  // query rows per loss partial of the forward kernel
cudaError_t launch_attn_fwd_tc(const AttnLaunch& L, int mode);
cudaError_t launch_attn_bwd_tc(const AttnLaunch& L, const float* cos_t, const float* sin_t,
                               int use_rope, void* dqkvt);

}  // namespace jab
