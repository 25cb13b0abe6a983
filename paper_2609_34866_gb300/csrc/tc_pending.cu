// Tensor-core attention entry points not yet built: each delegates to the CUDA-core kernel.
#include "path.h"

namespace jab {

cudaError_t launch_attn_bwd_tc(const AttnLaunch& L, const float* cos_t, const float* sin_t,
                               int use_rope, void* dqkvt) {
  return launch_attn_bwd_simple(L, cos_t, sin_t, use_rope, dqkvt);
}

}  // namespace jab
