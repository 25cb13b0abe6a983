// Host-side launchers of the L_JAB kernels (internal to libjab; not part of the C ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace jab {

struct AttnLaunch {
  const void* qkv;      // fp16 [N, ldq]
  int64_t ldq;          // C * D
  int D, B, T, Hq, Hkv, dh, C;
  float scale;
  int nP;
  double* part;         // [C, B, Hq, nP]
  const float* a_ref;   // fp32 [N, Hq*dh]
  float* a_out;         // fp32 [N, Hq*dh] (teacher)
  float* lse;           // fp32 [B, Hq, T] or null
  void* d_o;            // fp16 [N, Hq*dh] (backward)
  float* dvec;          // fp32 [B, Hq, T] (backward)
  int64_t ldt;          // row pitch of the transposed dQKV^T (backward)
  int lse_pitch;        // row pitch of lse and dvec ([B, Hq, lse_pitch])
  int* status;
  cudaStream_t stream;
};

// prep.cu
cudaError_t launch_convert_x(const void* x, void* xh, int64_t n, int* status, int sms, cudaStream_t st);
cudaError_t launch_transpose_x(const void* x, void* xt, int64_t N, int64_t ldt, int d, cudaStream_t st);
cudaError_t launch_quantize(const void* w, const float* s, int D, int d, int G, int bits, void* w16,
                            int8_t* codes, float* w_hat32, int* status, int sms, cudaStream_t st);
cudaError_t launch_init_scales(const void* w, int D, int d, int G, int bits, int mode, float* s_out,
                               cudaStream_t st);
cudaError_t launch_rope_table(int T, int dh, double theta, float* cos_t, float* sin_t, cudaStream_t st);

// gemm_simple.cu
cudaError_t launch_proj_gemm_simple(const void* A, const void* Bw, void* C, int64_t M, int Nn, int K,
                                    int D, int n_rot, int dh, int T, const float* cos_t,
                                    const float* sin_t, cudaStream_t st);
cudaError_t launch_wgrad_lsq_simple(const void* dqkvt, const void* xt, int64_t ldt, const void* w,
                                    const float* s, int64_t N, int D, int d, int G, int bits,
                                    float coef, float* ds, cudaStream_t st);

// attn_simple.cu
cudaError_t launch_attn_fwd_simple(const AttnLaunch& L, int mode);
cudaError_t launch_attn_bwd_simple(const AttnLaunch& L, const float* cos_t, const float* sin_t,
                                   int use_rope, void* dqkvt);

// reduce.cu
cudaError_t launch_loss_reduce(const double* part, int C, int B, int Hq, int nP, double inv_n,
                               double* out, double* parts_out, cudaStream_t st);
cudaError_t launch_check_finite(const float* x, int64_t n, int* status, cudaStream_t st);

}  // namespace jab
