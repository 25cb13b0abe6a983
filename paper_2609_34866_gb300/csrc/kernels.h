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
  void* ds;             // fp16 dS^T tiles (backward): [B, Hq, nq (nq + 1) / 2, 128 keys, 128 queries]
  int* status;
  cudaStream_t stream;
};

// prep.cu
cudaError_t launch_convert_x(const void* x, void* xh, int64_t n, int* status, int sms, cudaStream_t st);
cudaError_t launch_quantize(const void* w, const float* s, int D, int d, int G, int bits, void* w16,
                            int8_t* codes, float* w_hat32, int* status, int sms, cudaStream_t st);
// codes a, b: int8 [n], 16-byte aligned; *count (int64, device) = #{i : a[i] != b[i]}
cudaError_t launch_flip_count(const int8_t* a, const int8_t* b, int64_t n, int64_t* count,
                              int sms, cudaStream_t st);
cudaError_t launch_init_scales(const void* w, int D, int d, int G, int bits, int mode, float* s_out,
                               cudaStream_t st);
cudaError_t launch_rope_table(int T, int dh, double theta, float* cos_t, float* sin_t, cudaStream_t st);

// gemm_tc.cu
cudaError_t launch_proj_gemm_tc(const void* A, const void* Bw, void* C, int64_t M, int Nn, int K,
                                int D, int n_rot, int dh, int T, const float* cos_t,
                                const float* sin_t, int* status, cudaStream_t st);
// x: bf16 [N, d] as the caller stores it (no transposed copy)
// ds: the scale gradient, written (fp32 [D, d/G]); dspart: fp32 [kMaxSplits, D, d/G] scratch
cudaError_t launch_wgrad_lsq_tc(const void* dqkvt, int64_t ldt, const void* x, const void* w,
                                const float* s, int64_t N, int D, int d, int G, int bits,
                                float coef, float* ds, float* dspart, int* status, cudaStream_t st);
// coef * dQKV^T X stored fp32 [D, d] in dw, or in scratch (fp32 [D, d]) when dw is NULL, and its
// squared norm in *sqnorm (may be NULL) by a fixed-order reduction (red: fp64 [kRedBlocks]). A split
// K adds partial tiles with atomics; deterministic keeps one unit per tile (bit-identical dW).
cudaError_t launch_wgrad_store_tc(const void* dqkvt, int64_t ldt, const void* x, int64_t N, int D,
                                  int d, float coef, float* dw, double* sqnorm, float* scratch,
                                  double* red, bool deterministic, int* status, cudaStream_t st);
// split count of a K-split GEMM: whole waves of units on the persistent grid
int choose_splits(int tiles, int k_blocks, int sms);
// attn_tc.cu
int attn_fwd_tc_rows(int Hq, int Hkv);  // query rows per loss partial of the forward kernel
cudaError_t launch_attn_fwd_tc(const AttnLaunch& L, int mode);
// kl_ab: null for the MSE term alone; else {a, b}: dS = a P (dP - D) + b (P - P_teacher) with the
// teacher's probabilities read from the dS^T tile buffer (launch_attn_teacher_p_tc), dV times a
cudaError_t launch_attn_bwd_tc(const AttnLaunch& L, const float* cos_t, const float* sin_t,
                               int use_rope, void* dqkvt, const float* kl_ab = nullptr);
// The teacher's probabilities P^T of every (query block, key block <= query block) tile into the
// dS^T tile buffer `ds` (layout of AttnLaunch::ds) and one KL partial per CTA in part
// [Hkv, B, ceil(T / 128)]: the sum of P (s_t - s_s) over its entries plus, in key block 0, of
// lse_s - lse_t over its query rows (natural units). qkv_s / qkv_t: student and teacher projections,
// fp16 [B*T, ldq]; lse2_t / lse2_s: log-sum-exp in log2 units, [B, Hq, lse_pitch].
cudaError_t launch_attn_teacher_p_tc(const void* qkv_s, int64_t ldq_s, const void* qkv_t,
                                     int64_t ldq_t, int B, int T, int Hq, int Hkv, int dh,
                                     float scale, const float* lse2_t, const float* lse2_s,
                                     int lse_pitch, void* ds, double* part, int* status,
                                     cudaStream_t st);
// out[b, h, t] = in[b, h, t] * log2(e) for t < T: [B, Hq, T] -> [B, Hq, pitch]
cudaError_t launch_lse_to_log2(const float* in, int BH, int T, int pitch, float* out,
                               cudaStream_t st);
// *out = scale * sum of part[0 .. n - 1], in order (fp64)
cudaError_t launch_sum_scaled(const double* part, int n, double scale, double* out, cudaStream_t st);

// attn_kl_tc.cu: KL attention-map term (Eq. 3). qkv_s: student fp16 [B*T, ldq] (candidate c at
// column c * D); qkv_t: teacher fp16 [B*T, D]. part [C, B, Hq, nP] (nP >= ceil(T / rows)), kl_rows
// fp32 [C, B, Hq, T] or null.
int attn_kl_tc_rows();
cudaError_t launch_attn_kl_tc(const void* qkv_s, int64_t ldq, const void* qkv_t, int B, int T,
                              int C, int Hq, int Hkv, int dh, float scale, double* part, int nP,
                              float* kl_rows, int* status, cudaStream_t st);

// attn_jvp_tc.cu: ||J_A v||^2 partials of the forward-mode attention product (Section 2.4). qkv and
// tqkv: primal and tangent projections, fp16 [B*T, D]; lse: teacher log-sum-exp (natural log)
// [B, Hq, lse_pitch]; a_ref: teacher output fp32 [B*T, Hq*dh]; part [B, Hq, nP].
int attn_jvp_tc_rows();
cudaError_t launch_attn_jvp_tc(const void* qkv, const void* tqkv, const float* lse, int lse_pitch,
                               const float* a_ref, int B, int T, int Hq, int Hkv, int dh,
                               float scale, double* part, int nP, int* status, cudaStream_t st);

// prep.cu: Rademacher probe entries first .. first + n - 1 of the SplitMix64 sequence of `seed` as
// fp16 +-2^-log2_scale (n a multiple of 8, 0 <= log2_scale <= 14); partial sums of the squared
// quantisation error, one per block.
cudaError_t launch_rademacher_probe(uint64_t seed, uint64_t first, int64_t n, int log2_scale,
                                    void* out, int sms, cudaStream_t st);
cudaError_t launch_qerr_partial(const void* w, const float* s, int D, int d, int G, int bits,
                                double* part, int nblocks, int* status, cudaStream_t st);

// reduce.cu
// A non-finite total raises JAB_ERR_NONFINITE in *status.
cudaError_t launch_loss_reduce(const double* part, int C, int B, int Hq, int nP, double inv_n,
                               double* out, double* parts_out, int* status, cudaStream_t st);
// out[c] = a[c] + lam * b[c] for c < C
cudaError_t launch_loss_combine(const double* a, const double* b, double lam, int C, double* out,
                                cudaStream_t st);
cudaError_t launch_omega_finish(const double* part, int nblocks, int C, const double* trace,
                                double layers_after, double* c1, double* c2, cudaStream_t st);
cudaError_t launch_mean(const double* x, int n, double* out, cudaStream_t st);
cudaError_t launch_check_finite(const float* x, int64_t n, int* status, cudaStream_t st);
// *out = sum of x[i]^2 in fp64, fixed order (part: fp64 [kRedBlocks])
cudaError_t launch_sumsq(const float* x, int64_t n, double* part, double* out, cudaStream_t st);
// out[i] = sum over s < splits of part[s n + i], in order of s (fp64 sum, fp32 result)
cudaError_t launch_split_sum(const float* part, int splits, int64_t n, float* out, cudaStream_t st);

}  // namespace jab
