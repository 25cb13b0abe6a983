// C ABI of libjab (include/jab.h): argument validation, workspace carving and kernel sequencing.
// Every step of the computation runs in the kernels of this library; there is no host fallback.
#include <math.h>

#include <cmath>
#include <stdlib.h>
#include <string.h>

#include <mutex>

#include <vector>

#include "common.cuh"
#include "kernels.h"
#include "timing.h"
#include "workspace.h"

namespace jab {

// Deterministic-reduction mode (jab_set_deterministic): process-wide, read when a call is issued.
int g_deterministic = 0;

__device__ int g_status;  // one per device context: first device-side problem since the last read

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mu;
int* g_status_ptr[kMaxDevices] = {};
int g_sms[kMaxDevices] = {};

jab_status device_info(int** status, int* sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return JAB_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_status_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status) != cudaSuccess) return JAB_ERR_CUDA;
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return JAB_ERR_CUDA;
    g_status_ptr[dev] = static_cast<int*>(p);
    g_sms[dev] = n;
  }
  *status = g_status_ptr[dev];
  *sms = g_sms[dev];
  return JAB_OK;
}

}  // namespace

// The device status word of the current device (for kernels launched outside this file).
jab_status device_status_ptr(int** status) {
  int sms = 0;
  return device_info(status, &sms);
}

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

jab_status check_desc(const jab_block_desc* d) {
  if (d == nullptr) return JAB_ERR_INVALID_ARG;
  if (d->d_model <= 0 || d->n_q_heads <= 0 || d->n_kv_heads <= 0 || d->head_dim <= 0 ||
      d->group_size <= 0)
    return JAB_ERR_INVALID_ARG;
  if (d->use_rope && !(d->rope_theta > 0.f)) return JAB_ERR_INVALID_ARG;
  if (d->n_q_heads % d->n_kv_heads != 0) return JAB_ERR_UNSUPPORTED;
  if (d->head_dim != 64 && d->head_dim != 128) return JAB_ERR_UNSUPPORTED;
  if (d->d_model % 64 != 0 || d->group_size % 64 != 0 || d->d_model % d->group_size != 0)
    return JAB_ERR_UNSUPPORTED;
  if (block_rows(d) % 128 != 0) return JAB_ERR_UNSUPPORTED;
  return JAB_OK;
}

jab_status check_bt(int32_t B, int32_t T) {
  if (B < 1 || T < 1) return JAB_ERR_INVALID_ARG;
  if ((int64_t)B * T > (int64_t)1 << 31) return JAB_ERR_UNSUPPORTED;
  return JAB_OK;
}

float softmax_scale(const jab_block_desc* d) {
  return d->softmax_scale > 0.f ? d->softmax_scale : (float)(1.0 / sqrt((double)d->head_dim));
}

#define JAB_TRY(expr)                                   \
  do {                                                  \
    if ((expr) != cudaSuccess) return JAB_ERR_CUDA;     \
  } while (0)

// A timed launch site: `nk` kernels launched by `expr` on stream `st`.
#define JAB_SITE(name, nk, expr)                        \
  do {                                                  \
    TimedSite site_(name, st, nk);                      \
    if ((expr) != cudaSuccess) return JAB_ERR_CUDA;     \
  } while (0)

// Projection X W^T (+ RoPE) for C candidates stacked along the output dimension.
jab_status run_projection(const jab_block_desc* d, int64_t N, int T, int C, const void* x16,
                          const void* w16, void* qkv, const float* cos_t, const float* sin_t,
                          int* status, cudaStream_t st) {
  const int D = (int)block_rows(d);
  const int n_rot = d->use_rope ? (d->n_q_heads + d->n_kv_heads) * d->head_dim : 0;
  JAB_SITE("proj_gemm", 1, launch_proj_gemm_tc(x16, w16, qkv, N, C * D, d->d_model, D, n_rot,
                                               d->head_dim, T, cos_t, sin_t, status, st));
  return JAB_OK;
}

AttnLaunch attn_launch(const jab_block_desc* d, int B, int T, int C, char* ws,
                       const Workspace& wp, int* status, cudaStream_t st) {
  AttnLaunch L{};
  L.qkv = ws + wp.qkv;
  L.D = (int)block_rows(d);
  L.ldq = (int64_t)C * L.D;
  L.B = B;
  L.T = T;
  L.Hq = d->n_q_heads;
  L.Hkv = d->n_kv_heads;
  L.dh = d->head_dim;
  L.C = C;
  L.scale = softmax_scale(d);
  const int rows = attn_fwd_tc_rows(d->n_q_heads, d->n_kv_heads);
  L.nP = (T + rows - 1) / rows;
  L.lse_pitch = T;
  L.part = reinterpret_cast<double*>(ws + wp.part);
  L.status = status;
  L.stream = st;
  return L;
}

// Which X each workspace holds in fp16 (its x16 slot): written by every call that converts X into
// a workspace, read by the *_prepared entry points, which skip the conversion.
struct PreparedX {
  const void* ws;
  const void* x;
  int32_t B, T, d;
};
std::mutex g_prep_mu;
std::vector<PreparedX> g_prep;

void note_prepared(const void* ws, const void* x, int32_t B, int32_t T, int32_t d) {
  std::lock_guard<std::mutex> lk(g_prep_mu);
  for (auto& e : g_prep)
    if (e.ws == ws) {
      e = PreparedX{ws, x, B, T, d};
      return;
    }
  g_prep.push_back(PreparedX{ws, x, B, T, d});
}

bool is_prepared(const void* ws, const void* x, int32_t B, int32_t T, int32_t d) {
  std::lock_guard<std::mutex> lk(g_prep_mu);
  for (const auto& e : g_prep)
    if (e.ws == ws) return e.x == x && e.B == B && e.T == T && e.d == d;
  return false;
}

// X (bf16) -> the workspace's fp16 copy, with the fp16 range check; records it for *_prepared.
jab_status convert_x_into(const jab_block_desc* desc, int32_t B, int32_t T, const void* X_dev,
                          void* ws, const Workspace& wp, int* status, int sms, cudaStream_t st) {
  const int64_t N = (int64_t)B * T;
  JAB_SITE("convert_x", 1, launch_convert_x(X_dev, static_cast<char*>(ws) + wp.x16,
                                            N * desc->d_model, status, sms, st));
  note_prepared(ws, X_dev, B, T, desc->d_model);
  return JAB_OK;
}

}  // namespace
}  // namespace jab

using namespace jab;

extern "C" {

size_t jab_workspace_size(const jab_block_desc* desc, int32_t B, int32_t T, int32_t n_cand,
                          int32_t with_bwd) {
  if (check_desc(desc) != JAB_OK || check_bt(B, T) != JAB_OK || n_cand < 1) return 0;
  return plan_workspace(desc, B, T, n_cand, with_bwd != 0).total;
}

jab_status jab_reference_forward(const jab_block_desc* desc, int32_t B, int32_t T,
                                 const void* X_dev, const void* W_dev, float* A_ref_dev,
                                 float* lse_dev, double* a_sqnorm_dev, void* ws, size_t ws_bytes,
                                 jab_stream_t stream) {
  jab_status s = check_desc(desc);
  if (s != JAB_OK) return s;
  if ((s = check_bt(B, T)) != JAB_OK) return s;
  if (!X_dev || !W_dev || !A_ref_dev || !ws) return JAB_ERR_INVALID_ARG;
  if (!aligned16(X_dev) || !aligned16(W_dev) || !aligned16(A_ref_dev) ||
      (reinterpret_cast<uintptr_t>(ws) & 255u))
    return JAB_ERR_INVALID_ARG;
  const Workspace wp = plan_workspace(desc, B, T, 1, false);
  if (ws_bytes < wp.total) return JAB_ERR_INVALID_ARG;
  int* status;
  int sms;
  if ((s = device_info(&status, &sms)) != JAB_OK) return s;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  const int64_t N = (int64_t)B * T;
  const int D = (int)block_rows(desc), dm = desc->d_model, dh = desc->head_dim;
  float* cos_t = reinterpret_cast<float*>(w + wp.rope);
  float* sin_t = cos_t + (int64_t)T * (dh / 2);
  if ((s = convert_x_into(desc, B, T, X_dev, ws, wp, status, sms, st)) != JAB_OK) return s;
  JAB_SITE("quantize", 1, launch_quantize(W_dev, nullptr, D, dm, desc->group_size, 0, w + wp.w16, nullptr, nullptr,
                          status, sms, st));
  if (desc->use_rope) JAB_SITE("rope_table", 1, launch_rope_table(T, dh, desc->rope_theta, cos_t, sin_t, st));
  if ((s = run_projection(desc, N, T, 1, w + wp.x16, w + wp.w16, w + wp.qkv, cos_t, sin_t, status, st)) !=
      JAB_OK)
    return s;
  AttnLaunch L = attn_launch(desc, B, T, 1, w, wp, status, st);
  L.a_out = A_ref_dev;
  L.lse = lse_dev;
  JAB_SITE("attn_fwd", 1, launch_attn_fwd_tc(L, 0));
  if (a_sqnorm_dev)
    JAB_SITE("loss_reduce", 1, launch_loss_reduce(L.part, 1, B, desc->n_q_heads, L.nP, 1.0,
                                                  a_sqnorm_dev, nullptr, status, st));
  return JAB_OK;
}

}  // extern "C"

// The candidate forward of jab_loss_forward: quantise every candidate, one projection GEMM over all
// of them (+ RoPE), the attention forward with the MSE epilogue, the loss per candidate into
// mse_dev. On success *wp_out / *status_out describe the workspace and the status word.
static jab_status forward_candidates(const jab_block_desc* desc, int32_t B, int32_t T,
                                     const void* X_dev, const void* W_dev, const float* A_ref_dev,
                                     int32_t n_cand, const int32_t* bits_host,
                                     const float* const* scales_host, double* mse_dev,
                                     double* sse_parts_dev, void* ws, size_t ws_bytes,
                                     cudaStream_t st, Workspace* wp_out, int** status_out) {
  jab_status s = check_desc(desc);
  if (s != JAB_OK) return s;
  if ((s = check_bt(B, T)) != JAB_OK) return s;
  if (n_cand < 1 || !bits_host || !scales_host || !X_dev || !W_dev || !A_ref_dev || !mse_dev ||
      !ws)
    return JAB_ERR_INVALID_ARG;
  if (!aligned16(X_dev) || !aligned16(W_dev) || !aligned16(A_ref_dev) ||
      (reinterpret_cast<uintptr_t>(ws) & 255u))
    return JAB_ERR_INVALID_ARG;
  for (int c = 0; c < n_cand; ++c) {
    if (bits_host[c] < 2 || bits_host[c] > 8 || scales_host[c] == nullptr)
      return JAB_ERR_INVALID_ARG;
    if (!aligned16(scales_host[c])) return JAB_ERR_INVALID_ARG;
  }
  const Workspace wp = plan_workspace(desc, B, T, n_cand, false);
  if (ws_bytes < wp.total) return JAB_ERR_INVALID_ARG;
  int* status;
  int sms;
  if ((s = device_info(&status, &sms)) != JAB_OK) return s;
  char* w = static_cast<char*>(ws);
  const int64_t N = (int64_t)B * T;
  const int D = (int)block_rows(desc), dm = desc->d_model, dh = desc->head_dim;
  float* cos_t = reinterpret_cast<float*>(w + wp.rope);
  float* sin_t = cos_t + (int64_t)T * (dh / 2);
  if ((s = convert_x_into(desc, B, T, X_dev, ws, wp, status, sms, st)) != JAB_OK) return s;
  for (int c = 0; c < n_cand; ++c)
    JAB_SITE("quantize", 1, launch_quantize(W_dev, scales_host[c], D, dm, desc->group_size, bits_host[c],
                            w + wp.w16 + (size_t)c * D * dm * 2, nullptr, nullptr, status, sms, st));
  if (desc->use_rope) JAB_SITE("rope_table", 1, launch_rope_table(T, dh, desc->rope_theta, cos_t, sin_t, st));
  if ((s = run_projection(desc, N, T, n_cand, w + wp.x16, w + wp.w16, w + wp.qkv, cos_t, sin_t,
                          status, st)) != JAB_OK)
    return s;
  AttnLaunch L = attn_launch(desc, B, T, n_cand, w, wp, status, st);
  L.a_ref = A_ref_dev;
  JAB_SITE("attn_fwd", 1, launch_attn_fwd_tc(L, 1));
  const double inv_n = 1.0 / ((double)N * desc->n_q_heads * dh);
  JAB_SITE("loss_reduce", 1, launch_loss_reduce(L.part, n_cand, B, desc->n_q_heads, L.nP, inv_n,
                                                mse_dev, sse_parts_dev, status, st));
  *wp_out = wp;
  *status_out = status;
  return JAB_OK;
}

extern "C" {

jab_status jab_loss_forward(const jab_block_desc* desc, int32_t B, int32_t T, const void* X_dev,
                            const void* W_dev, const float* A_ref_dev, int32_t n_cand,
                            const int32_t* bits_host, const float* const* scales_host,
                            double* loss_dev, double* sse_parts_dev, void* ws, size_t ws_bytes,
                            jab_stream_t stream) {
  Workspace wp;
  int* status;
  return forward_candidates(desc, B, T, X_dev, W_dev, A_ref_dev, n_cand, bits_host, scales_host,
                            loss_dev, sse_parts_dev, ws, ws_bytes,
                            reinterpret_cast<cudaStream_t>(stream), &wp, &status);
}

jab_status jab_reference_projection(const jab_block_desc* desc, int32_t B, int32_t T,
                                    const void* X_dev, const void* W_dev, void* QKV_ref_dev,
                                    void* ws, size_t ws_bytes, jab_stream_t stream) {
  jab_status s = check_desc(desc);
  if (s != JAB_OK) return s;
  if ((s = check_bt(B, T)) != JAB_OK) return s;
  if (!X_dev || !W_dev || !QKV_ref_dev || !ws) return JAB_ERR_INVALID_ARG;
  if (!aligned16(X_dev) || !aligned16(W_dev) || !aligned16(QKV_ref_dev) ||
      (reinterpret_cast<uintptr_t>(ws) & 255u))
    return JAB_ERR_INVALID_ARG;
  const Workspace wp = plan_workspace(desc, B, T, 1, false);
  if (ws_bytes < wp.total) return JAB_ERR_INVALID_ARG;
  int* status;
  int sms;
  if ((s = device_info(&status, &sms)) != JAB_OK) return s;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  const int64_t N = (int64_t)B * T;
  const int D = (int)block_rows(desc), dm = desc->d_model, dh = desc->head_dim;
  float* cos_t = reinterpret_cast<float*>(w + wp.rope);
  float* sin_t = cos_t + (int64_t)T * (dh / 2);
  if ((s = convert_x_into(desc, B, T, X_dev, ws, wp, status, sms, st)) != JAB_OK) return s;
  JAB_SITE("quantize", 1, launch_quantize(W_dev, nullptr, D, dm, desc->group_size, 0, w + wp.w16,
                                          nullptr, nullptr, status, sms, st));
  if (desc->use_rope) JAB_SITE("rope_table", 1, launch_rope_table(T, dh, desc->rope_theta, cos_t, sin_t, st));
  return run_projection(desc, N, T, 1, w + wp.x16, w + wp.w16, QKV_ref_dev, cos_t, sin_t, status,
                        st);
}

jab_status jab_loss_forward_kl(const jab_block_desc* desc, int32_t B, int32_t T, const void* X_dev,
                               const void* W_dev, const float* A_ref_dev, const void* QKV_ref_dev,
                               int32_t n_cand, const int32_t* bits_host,
                               const float* const* scales_host, float lambda_kl, double* loss_dev,
                               double* mse_dev, double* kl_dev, float* kl_rows_dev, void* ws,
                               size_t ws_bytes, jab_stream_t stream) {
  if (!QKV_ref_dev || !aligned16(QKV_ref_dev) || !loss_dev || !(lambda_kl >= 0.f) ||
      !isfinite(lambda_kl)) {
    const jab_status s = check_desc(desc);
    return s != JAB_OK ? s : JAB_ERR_INVALID_ARG;
  }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (n_cand >= 1 && desc != nullptr && check_desc(desc) == JAB_OK && check_bt(B, T) == JAB_OK) {
    const Workspace wp0 = plan_workspace(desc, B, T, n_cand, false);
    if (ws != nullptr && ws_bytes >= wp0.total && !mse_dev)
      mse_dev = reinterpret_cast<double*>(static_cast<char*>(ws) + wp0.scal);
  }
  Workspace wp;
  int* status;
  jab_status s = forward_candidates(desc, B, T, X_dev, W_dev, A_ref_dev, n_cand, bits_host,
                                    scales_host, mse_dev, nullptr, ws, ws_bytes, st, &wp, &status);
  if (s != JAB_OK) return s;
  char* w = static_cast<char*>(ws);
  double* kl = kl_dev ? kl_dev : reinterpret_cast<double*>(w + wp.scal) + n_cand;
  double* part = reinterpret_cast<double*>(w + wp.part);
  const int nP = (T + attn_kl_tc_rows() - 1) / attn_kl_tc_rows();
  JAB_SITE("attn_kl", 1, launch_attn_kl_tc(w + wp.qkv, (int64_t)n_cand * block_rows(desc),
                                           QKV_ref_dev, B, T, n_cand, desc->n_q_heads,
                                           desc->n_kv_heads, desc->head_dim, softmax_scale(desc),
                                           part, nP, kl_rows_dev, status, st));
  // batchmean (App. B "Effective weight of the KL term"): the sum over rows divided by B
  JAB_SITE("loss_reduce", 1, launch_loss_reduce(part, n_cand, B, desc->n_q_heads, nP, 1.0 / B, kl,
                                                nullptr, status, st));
  JAB_SITE("loss_combine", 1, launch_loss_combine(mse_dev, kl, (double)lambda_kl, n_cand, loss_dev,
                                                  st));
  return JAB_OK;
}

jab_status jab_hutchinson_trace(const jab_block_desc* desc, int32_t B, int32_t T,
                                const void* X_dev, const void* W_dev, const float* A_ref_dev,
                                const float* lse_ref_dev, int32_t n_probes, uint64_t seed,
                                double* trace_dev, double* vhv_dev, void* ws, size_t ws_bytes,
                                jab_stream_t stream) {
  jab_status s = check_desc(desc);
  if (s != JAB_OK) return s;
  if ((s = check_bt(B, T)) != JAB_OK) return s;
  if (n_probes < 1 || !X_dev || !W_dev || !A_ref_dev || !lse_ref_dev || !trace_dev || !ws)
    return JAB_ERR_INVALID_ARG;
  if (!aligned16(X_dev) || !aligned16(W_dev) || !aligned16(A_ref_dev) ||
      (reinterpret_cast<uintptr_t>(lse_ref_dev) & 3u) || (reinterpret_cast<uintptr_t>(ws) & 255u))
    return JAB_ERR_INVALID_ARG;
  const Workspace wp = plan_workspace(desc, B, T, 2, false);
  if (ws_bytes < wp.total) return JAB_ERR_INVALID_ARG;
  int* status;
  int sms;
  if ((s = device_info(&status, &sms)) != JAB_OK) return s;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  const int64_t N = (int64_t)B * T;
  const int D = (int)block_rows(desc), dm = desc->d_model, dh = desc->head_dim;
  float* cos_t = reinterpret_cast<float*>(w + wp.rope);
  float* sin_t = cos_t + (int64_t)T * (dh / 2);
  char* qkv = w + wp.qkv;                      // primal [N, D]
  char* tqkv = qkv + (size_t)N * D * 2;        // tangent [N, D]
  double* part = reinterpret_cast<double*>(w + wp.part);
  double* tmp = reinterpret_cast<double*>(w + wp.scal);
  const int nP = (T + attn_jvp_tc_rows() - 1) / attn_jvp_tc_rows();
  const double n_el = (double)N * desc->n_q_heads * dh;
  if ((s = convert_x_into(desc, B, T, X_dev, ws, wp, status, sms, st)) != JAB_OK) return s;
  JAB_SITE("quantize", 1, launch_quantize(W_dev, nullptr, D, dm, desc->group_size, 0, w + wp.w16,
                                          nullptr, nullptr, status, sms, st));
  if (desc->use_rope) JAB_SITE("rope_table", 1, launch_rope_table(T, dh, desc->rope_theta, cos_t, sin_t, st));
  if ((s = run_projection(desc, N, T, 1, w + wp.x16, w + wp.w16, qkv, cos_t, sin_t, status, st)) !=
      JAB_OK)
    return s;
  // The probe enters scaled by c = 2^-k, k = floor(log2(sqrt(d_model))): the tangent projections
  // X (c v)^T are then of the order of the activations, inside the fp16 range of the tensor-core
  // operands; v^T H v = ||J_A (c v)||^2 * 2 / (n c^2) is rescaled exactly (a power of two).
  int k2 = 0;
  while ((1 << (2 * (k2 + 1))) <= dm && k2 < 14) ++k2;
  const double rescale = std::ldexp(1.0, 2 * k2);
  JAB_SITE("memset_grad", 0, cudaMemsetAsync(trace_dev, 0, sizeof(double), st));
  for (int pr = 0; pr < n_probes; ++pr) {
    // probe pr: entries pr * D * d .. of the seed's sequence, the tangent projection X V^T + RoPE
    JAB_SITE("probe", 1, launch_rademacher_probe(seed, (uint64_t)pr * D * dm, (int64_t)D * dm, k2,
                                                 w + wp.w16, sms, st));
    if ((s = run_projection(desc, N, T, 1, w + wp.x16, w + wp.w16, tqkv, cos_t, sin_t, status,
                            st)) != JAB_OK)
      return s;
    JAB_SITE("attn_jvp", 1, launch_attn_jvp_tc(qkv, tqkv, lse_ref_dev, T, A_ref_dev, B, T,
                                               desc->n_q_heads, desc->n_kv_heads, dh,
                                               softmax_scale(desc), part, nP, status, st));
    double* vhv = vhv_dev ? vhv_dev + pr : tmp;
    // v^T H v = 2 ||J_A v||^2 / n (Eq. 5 at the float weights, MSE term)
    JAB_SITE("loss_reduce", 1, launch_loss_reduce(part, 1, B, desc->n_q_heads, nP,
                                                  2.0 * rescale / n_el, vhv, nullptr, status, st));
    JAB_SITE("loss_combine", 1, launch_loss_combine(trace_dev, vhv, 1.0 / n_probes, 1, trace_dev,
                                                    st));
  }
  return JAB_OK;
}

jab_status jab_rademacher_probes(uint64_t seed, int64_t first, int64_t n, void* out_dev,
                                 jab_stream_t stream) {
  if (!out_dev || n < 0 || first < 0 || (n & 7) || !aligned16(out_dev)) return JAB_ERR_INVALID_ARG;
  if (n == 0) return JAB_OK;
  int* status;
  int sms;
  const jab_status s = device_info(&status, &sms);
  if (s != JAB_OK) return s;
  JAB_TRY(launch_rademacher_probe(seed, (uint64_t)first, n, 0, out_dev, sms,
                                  reinterpret_cast<cudaStream_t>(stream)));
  return JAB_OK;
}

jab_status jab_omega_scores(const jab_block_desc* desc, const void* W_dev, int32_t n_cand,
                            const int32_t* bits_host, const float* const* scales_host,
                            const double* trace_dev, int32_t layers_after, double* c1_dev,
                            double* c2_dev, void* ws, size_t ws_bytes, jab_stream_t stream) {
  jab_status s = check_desc(desc);
  if (s != JAB_OK) return s;
  if (n_cand < 1 || !W_dev || !bits_host || !scales_host || !trace_dev || !c1_dev || !ws ||
      layers_after < 0 || !aligned16(W_dev) || (reinterpret_cast<uintptr_t>(ws) & 255u))
    return JAB_ERR_INVALID_ARG;
  for (int c = 0; c < n_cand; ++c)
    if (bits_host[c] < 2 || bits_host[c] > 8 || scales_host[c] == nullptr)
      return JAB_ERR_INVALID_ARG;
  const Workspace wp = plan_workspace(desc, 1, 1, n_cand, false);
  if (ws_bytes < wp.total) return JAB_ERR_INVALID_ARG;
  int* status;
  int sms;
  if ((s = device_info(&status, &sms)) != JAB_OK) return s;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  double* red = reinterpret_cast<double*>(static_cast<char*>(ws) + wp.red);
  const int D = (int)block_rows(desc), dm = desc->d_model;
  for (int c = 0; c < n_cand; ++c)
    JAB_SITE("qerr", 1, launch_qerr_partial(W_dev, scales_host[c], D, dm, desc->group_size,
                                            bits_host[c], red + (size_t)c * kRedBlocks, kRedBlocks,
                                            status, st));
  JAB_SITE("omega", 1, launch_omega_finish(red, kRedBlocks, n_cand, trace_dev,
                                           (double)layers_after, c1_dev, c2_dev, st));
  return JAB_OK;
}

// The KL term of Eq. 3 in the backward (App. B "Effective weight of the KL term"): the teacher's
// projection and log-sum-exp, lambda_KL, where the KL value goes, and the two factors of the
// combined score gradient dS = a P (dP - D) + b (P - P_teacher) (b / a = lambda n / (2 B), with
// n = B T Hq d_h; a <= 1 keeps b <= 1024 so that the fp16 dS tiles hold the KL part in range).
struct KlTerm {
  const void* qkv_ref;
  const float* lse_ref;
  double lambda;
  double* kl_out;
  float ab[2];
};

// Steps shared by the backward entry points (App. B, STE): quantise, project (+ RoPE), attention
// forward in mode 2 (loss partials, dO = A_hat - A_ref, lse, D), the loss, and the attention backward
// into dQKV^T (bf16 [D, ldt]) in the workspace; with a KL term also the teacher's probability tiles
// and the KL value. Checks the arguments common to all.
static jab_status backward_to_dqkvt(const jab_block_desc* desc, int32_t B, int32_t T,
                                    const void* X_dev, const void* W_dev, const float* A_ref_dev,
                                    int32_t bits, const float* scales_dev, double* loss_dev,
                                    void* ws, size_t ws_bytes, bool x_prepared, cudaStream_t st,
                                    Workspace* wp_out, int** status_out,
                                    const KlTerm* kl = nullptr) {
  jab_status s = check_desc(desc);
  if (s != JAB_OK) return s;
  if ((s = check_bt(B, T)) != JAB_OK) return s;
  if (bits < 2 || bits > 8 || !X_dev || !W_dev || !A_ref_dev || !scales_dev || !loss_dev || !ws)
    return JAB_ERR_INVALID_ARG;
  if (!aligned16(X_dev) || !aligned16(W_dev) || !aligned16(A_ref_dev) || !aligned16(scales_dev) ||
      (reinterpret_cast<uintptr_t>(ws) & 255u))
    return JAB_ERR_INVALID_ARG;
  const Workspace wp = plan_workspace(desc, B, T, 1, true);
  if (ws_bytes < wp.total) return JAB_ERR_INVALID_ARG;
  int* status;
  int sms;
  if ((s = device_info(&status, &sms)) != JAB_OK) return s;
  char* w = static_cast<char*>(ws);
  const int64_t N = (int64_t)B * T;
  const int D = (int)block_rows(desc), dm = desc->d_model, dh = desc->head_dim;
  const int G = desc->group_size;
  float* cos_t = reinterpret_cast<float*>(w + wp.rope);
  float* sin_t = cos_t + (int64_t)T * (dh / 2);
  if (x_prepared) {  // the workspace already holds this X in fp16 (jab_prepare_x)
    if (!is_prepared(ws, X_dev, B, T, dm)) return JAB_ERR_INVALID_ARG;
  } else if ((s = convert_x_into(desc, B, T, X_dev, ws, wp, status, sms, st)) != JAB_OK) {
    return s;
  }
  JAB_SITE("quantize", 1, launch_quantize(W_dev, scales_dev, D, dm, G, bits, w + wp.w16, nullptr, nullptr, status,
                          sms, st));
  if (desc->use_rope) JAB_SITE("rope_table", 1, launch_rope_table(T, dh, desc->rope_theta, cos_t, sin_t, st));
  if ((s = run_projection(desc, N, T, 1, w + wp.x16, w + wp.w16, w + wp.qkv, cos_t, sin_t, status, st)) !=
      JAB_OK)
    return s;
  AttnLaunch L = attn_launch(desc, B, T, 1, w, wp, status, st);
  L.a_ref = A_ref_dev;
  L.lse = reinterpret_cast<float*>(w + wp.lse);
  L.d_o = w + wp.d_o;
  L.dvec = reinterpret_cast<float*>(w + wp.dvec);
  L.ldt = wp.ldt;
  L.lse_pitch = (int)wp.tp;
  L.ds = w + wp.ds;
  JAB_SITE("attn_fwd", 1, launch_attn_fwd_tc(L, 2));
  const double n_el = (double)N * desc->n_q_heads * dh;
  JAB_SITE("loss_reduce", 1, launch_loss_reduce(L.part, 1, B, desc->n_q_heads, L.nP, 1.0 / n_el,
                                                loss_dev, nullptr, status, st));
  const float* kl_ab = nullptr;
  if (kl != nullptr) {
    const int Hq = desc->n_q_heads, Hkv = desc->n_kv_heads;
    float* lse_t = reinterpret_cast<float*>(w + wp.lse_t);
    double* klpart = reinterpret_cast<double*>(w + wp.klpart);
    double* klv = kl->kl_out ? kl->kl_out : reinterpret_cast<double*>(w + wp.scal) + 1;
    JAB_SITE("lse_log2", 1, launch_lse_to_log2(kl->lse_ref, B * Hq, T, (int)wp.tp, lse_t, st));
    JAB_SITE("teacher_p", 1, launch_attn_teacher_p_tc(w + wp.qkv, D, kl->qkv_ref, D, B, T, Hq, Hkv,
                                                      dh, L.scale, lse_t, L.lse, (int)wp.tp, L.ds,
                                                      klpart, status, st));
    // batchmean (reading R18): the sum over sequences, heads, rows and keys divided by B
    JAB_SITE("kl_reduce", 1, launch_sum_scaled(klpart, Hkv * B * ((T + 127) / 128), 1.0 / B, klv,
                                               st));
    JAB_SITE("loss_combine", 1, launch_loss_combine(loss_dev, klv, kl->lambda, 1, loss_dev, st));
    kl_ab = kl->ab;
  }
  JAB_SITE("attn_bwd", 2, launch_attn_bwd_tc(L, cos_t, sin_t, desc->use_rope, w + wp.dqkvt, kl_ab));
  *wp_out = wp;
  *status_out = status;
  return JAB_OK;
}

}  // extern "C"

// jab_loss_backward_scales with the fp16 conversion of X either done here or taken from the
// workspace (x_prepared).
static jab_status backward_scales(const jab_block_desc* desc, int32_t B, int32_t T,
                                  const void* X_dev, const void* W_dev, const float* A_ref_dev,
                                  int32_t bits, const float* scales_dev, float kappa,
                                  double* loss_dev, float* grad_scales_dev, void* ws,
                                  size_t ws_bytes, bool x_prepared, jab_stream_t stream,
                                  const KlTerm* kl = nullptr) {
  if (!grad_scales_dev || !aligned16(grad_scales_dev)) {
    const jab_status s = check_desc(desc);
    return s != JAB_OK ? s : JAB_ERR_INVALID_ARG;
  }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  Workspace wp;
  int* status;
  jab_status s = backward_to_dqkvt(desc, B, T, X_dev, W_dev, A_ref_dev, bits, scales_dev, loss_dev,
                                   ws, ws_bytes, x_prepared, st, &wp, &status, kl);
  if (s != JAB_OK) return s;
  char* w = static_cast<char*>(ws);
  const int64_t N = (int64_t)B * T;
  const int D = (int)block_rows(desc), dm = desc->d_model, G = desc->group_size;
  const double n_el = (double)N * desc->n_q_heads * desc->head_dim;
  const double k = kappa > 0.f ? (double)kappa : 1.0 / sqrt((double)G * qmax_of(bits));
  // with the KL term the attention backward's dQKV^T is a times the MSE term's units
  const float coef = (float)(k * 2.0 / n_el / (kl ? (double)kl->ab[0] : 1.0));
  // per-split partials summed in order: the scale gradient is bit-identical between calls
  JAB_SITE("wgrad_lsq", 1, launch_wgrad_lsq_tc(w + wp.dqkvt, wp.ldt, X_dev, W_dev, scales_dev, N, D,
                                               dm, G, bits, coef, grad_scales_dev,
                                               reinterpret_cast<float*>(w + wp.gpart), status, st));
  JAB_SITE("check_finite", 1, launch_check_finite(grad_scales_dev, (int64_t)D * (dm / G), status, st));
  return JAB_OK;
}

extern "C" {

jab_status jab_loss_backward_scales(const jab_block_desc* desc, int32_t B, int32_t T,
                                    const void* X_dev, const void* W_dev, const float* A_ref_dev,
                                    int32_t bits, const float* scales_dev, float kappa,
                                    double* loss_dev, float* grad_scales_dev, void* ws,
                                    size_t ws_bytes, jab_stream_t stream) {
  return backward_scales(desc, B, T, X_dev, W_dev, A_ref_dev, bits, scales_dev, kappa, loss_dev,
                         grad_scales_dev, ws, ws_bytes, false, stream);
}

jab_status jab_prepare_x(const jab_block_desc* desc, int32_t B, int32_t T, const void* X_dev,
                         void* ws, size_t ws_bytes, jab_stream_t stream) {
  jab_status s = check_desc(desc);
  if (s != JAB_OK) return s;
  if ((s = check_bt(B, T)) != JAB_OK) return s;
  if (!X_dev || !ws || !aligned16(X_dev) || (reinterpret_cast<uintptr_t>(ws) & 255u))
    return JAB_ERR_INVALID_ARG;
  const Workspace wp = plan_workspace(desc, B, T, 1, false);
  if (ws_bytes < wp.x16 + (size_t)B * T * desc->d_model * 2) return JAB_ERR_INVALID_ARG;
  int* status;
  int sms;
  if ((s = device_info(&status, &sms)) != JAB_OK) return s;
  return convert_x_into(desc, B, T, X_dev, ws, wp, status, sms,
                        reinterpret_cast<cudaStream_t>(stream));
}

jab_status jab_loss_backward_scales_prepared(const jab_block_desc* desc, int32_t B, int32_t T,
                                             const void* X_dev, const void* W_dev,
                                             const float* A_ref_dev, int32_t bits,
                                             const float* scales_dev, float kappa,
                                             double* loss_dev, float* grad_scales_dev, void* ws,
                                             size_t ws_bytes, jab_stream_t stream) {
  return backward_scales(desc, B, T, X_dev, W_dev, A_ref_dev, bits, scales_dev, kappa, loss_dev,
                         grad_scales_dev, ws, ws_bytes, true, stream);
}

jab_status jab_flip_rate(const int8_t* codes_a_dev, const int8_t* codes_b_dev, int64_t n,
                         int64_t* count_dev, jab_stream_t stream) {
  if (!count_dev || n < 0 || (reinterpret_cast<uintptr_t>(count_dev) & 7u))
    return JAB_ERR_INVALID_ARG;
  if (n > 0 && (!codes_a_dev || !codes_b_dev || !aligned16(codes_a_dev) || !aligned16(codes_b_dev)))
    return JAB_ERR_INVALID_ARG;
  int* status;
  int sms;
  const jab_status s = device_info(&status, &sms);
  if (s != JAB_OK) return s;
  JAB_TRY(launch_flip_count(codes_a_dev, codes_b_dev, n, count_dev, sms,
                            reinterpret_cast<cudaStream_t>(stream)));
  return JAB_OK;
}

jab_status jab_loss_backward_scales_kl(const jab_block_desc* desc, int32_t B, int32_t T,
                                       const void* X_dev, const void* W_dev,
                                       const float* A_ref_dev, const void* QKV_ref_dev,
                                       const float* lse_ref_dev, int32_t bits,
                                       const float* scales_dev, float kappa, float lambda_kl,
                                       double* loss_dev, double* kl_dev, float* grad_scales_dev,
                                       void* ws, size_t ws_bytes, jab_stream_t stream) {
  jab_status s = check_desc(desc);
  if (s != JAB_OK) return s;
  if ((s = check_bt(B, T)) != JAB_OK) return s;
  if (!QKV_ref_dev || !aligned16(QKV_ref_dev) || !lse_ref_dev ||
      (reinterpret_cast<uintptr_t>(lse_ref_dev) & 3u) || !(lambda_kl >= 0.f) || !isfinite(lambda_kl))
    return JAB_ERR_INVALID_ARG;
  const double n_el = (double)B * T * desc->n_q_heads * desc->head_dim;
  const double c = (double)lambda_kl * n_el / (2.0 * B);
  const double a = c > 1024.0 ? 1024.0 / c : 1.0;
  KlTerm kl{QKV_ref_dev, lse_ref_dev, (double)lambda_kl, kl_dev, {(float)a, (float)(a * c)}};
  return backward_scales(desc, B, T, X_dev, W_dev, A_ref_dev, bits, scales_dev, kappa, loss_dev,
                         grad_scales_dev, ws, ws_bytes, false, stream, &kl);
}

jab_status jab_loss_backward_weights(const jab_block_desc* desc, int32_t B, int32_t T,
                                     const void* X_dev, const void* W_dev, const float* A_ref_dev,
                                     int32_t bits, const float* scales_dev, double* loss_dev,
                                     float* grad_w_dev, double* grad_sqnorm_dev, void* ws,
                                     size_t ws_bytes, jab_stream_t stream) {
  jab_status s = check_desc(desc);
  if (s != JAB_OK) return s;
  if ((!grad_w_dev && !grad_sqnorm_dev) || (grad_w_dev && !aligned16(grad_w_dev)))
    return JAB_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  Workspace wp;
  int* status;
  s = backward_to_dqkvt(desc, B, T, X_dev, W_dev, A_ref_dev, bits, scales_dev, loss_dev, ws,
                        ws_bytes, false, st, &wp, &status);
  if (s != JAB_OK) return s;
  char* w = static_cast<char*>(ws);
  const int64_t N = (int64_t)B * T;
  const int D = (int)block_rows(desc), dm = desc->d_model;
  const double n_el = (double)N * desc->n_q_heads * desc->head_dim;
  JAB_SITE("wgrad_store", 1, launch_wgrad_store_tc(w + wp.dqkvt, wp.ldt, X_dev, N, D, dm,
                                                   (float)(2.0 / n_el), grad_w_dev, grad_sqnorm_dev,
                                                   reinterpret_cast<float*>(w + wp.dwscr),
                                                   reinterpret_cast<double*>(w + wp.red),
                                                   g_deterministic != 0, status, st));
  if (grad_w_dev)
    JAB_SITE("check_finite", 1, launch_check_finite(grad_w_dev, (int64_t)D * dm, status, st));
  return JAB_OK;
}

jab_status jab_quantize(const jab_block_desc* desc, int32_t bits, const void* W_dev,
                        const float* scales_dev, int8_t* codes_dev, float* w_hat_dev,
                        jab_stream_t stream) {
  jab_status s = check_desc(desc);
  if (s != JAB_OK) return s;
  if (bits < 2 || bits > 8 || !W_dev || !scales_dev || (!codes_dev && !w_hat_dev))
    return JAB_ERR_INVALID_ARG;
  if (!aligned16(W_dev) || !aligned16(scales_dev) || (codes_dev && !aligned16(codes_dev)) ||
      (w_hat_dev && !aligned16(w_hat_dev)))
    return JAB_ERR_INVALID_ARG;
  int* status;
  int sms;
  if ((s = device_info(&status, &sms)) != JAB_OK) return s;
  JAB_TRY(launch_quantize(W_dev, scales_dev, (int)block_rows(desc), desc->d_model,
                          desc->group_size, bits, nullptr, codes_dev, w_hat_dev, status, sms,
                          reinterpret_cast<cudaStream_t>(stream)));
  return JAB_OK;
}

jab_status jab_init_scales(const jab_block_desc* desc, int32_t bits, int32_t mode,
                           const void* W_dev, float* scales_dev, jab_stream_t stream) {
  jab_status s = check_desc(desc);
  if (s != JAB_OK) return s;
  if (bits < 2 || bits > 8 || (mode != 0 && mode != 1) || !W_dev || !scales_dev)
    return JAB_ERR_INVALID_ARG;
  JAB_TRY(launch_init_scales(W_dev, (int)block_rows(desc), desc->d_model, desc->group_size, bits,
                             mode, scales_dev, reinterpret_cast<cudaStream_t>(stream)));
  return JAB_OK;
}

jab_status jab_set_deterministic(int32_t on) {
  if (on != 0 && on != 1) return JAB_ERR_INVALID_ARG;
  jab::g_deterministic = on;
  return JAB_OK;
}

jab_status jab_get_device_status(jab_stream_t stream) {
  int* status;
  int sms;
  jab_status s = device_info(&status, &sms);
  if (s != JAB_OK) return s;
  JAB_TRY(cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)));
  int v = 0;
  JAB_TRY(cudaMemcpyFromSymbol(&v, g_status, sizeof(int)));
  const int zero = 0;
  JAB_TRY(cudaMemcpyToSymbol(g_status, &zero, sizeof(int)));
  return static_cast<jab_status>(v);
}

const char* jab_status_string(jab_status status) {
  switch (status) {
    case JAB_OK: return "ok";
    case JAB_ERR_INVALID_ARG: return "invalid argument";
    case JAB_ERR_UNSUPPORTED: return "unsupported shape";
    case JAB_ERR_CUDA: return "CUDA error";
    case JAB_ERR_NONFINITE: return "non-finite or non-positive value";
    case JAB_ERR_RANGE: return "input outside the fp16 range";
    case JAB_ERR_TIMEOUT: return "device wait timed out";
    case JAB_ERR_SCRATCH_LIMIT: return "problem larger than the fixed no-allocation scratch";
    case JAB_ERR_INTERNAL: return "internal device invariant failed";
    case JAB_ERR_DEVICE_ASSERT: return "index outside its buffer (checked build)";
  }
  return "unknown status";
}

}  // extern "C"
