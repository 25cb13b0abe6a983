// Tensor-core entry points not yet built: each delegates to the CUDA-core kernel of the same op.
#include "path.h"

namespace jab {

cudaError_t launch_proj_gemm_tc(const void* A, const void* Bw, void* C, int64_t M, int Nn, int K,
                                int D, int n_rot, int dh, int T, const float* cos_t,
                                const float* sin_t, cudaStream_t st) {
  return launch_proj_gemm_simple(A, Bw, C, M, Nn, K, D, n_rot, dh, T, cos_t, sin_t, st);
}
cudaError_t launch_wgrad_lsq_tc(const void* dqkvt, const void* xt, const void* w, const float* s,
                                int64_t N, int D, int d, int G, int bits, float coef, float* ds,
                                cudaStream_t st) {
  return launch_wgrad_lsq_simple(dqkvt, xt, w, s, N, D, d, G, bits, coef, ds, st);
}
cudaError_t launch_attn_fwd_tc(const AttnLaunch& L, int mode) { return launch_attn_fwd_simple(L, mode); }
cudaError_t launch_attn_bwd_tc(const AttnLaunch& L, const float* cos_t, const float* sin_t,
                               int use_rope, void* dqkvt) {
  return launch_attn_bwd_simple(L, cos_t, sin_t, use_rope, dqkvt);
}

}  // namespace jab
