// Loss reduction (Eq. 3, MSE term): per-tile fp64 partials -> SSE per (candidate, sequence, head)
// and L = SSE / (B T Hq d_h). Fixed summation order, so repeated calls give identical bits.
#include "common.cuh"
#include "kernels.h"
#include "workspace.h"

namespace jab {

__global__ void __launch_bounds__(256) loss_reduce_kernel(const double* __restrict__ part, int B,
                                                          int Hq, int nP, double inv_n,
                                                          double* __restrict__ out,
                                                          double* __restrict__ parts_out,
                                                          int* status) {
  __shared__ double red[8];
  const int c = blockIdx.x;
  const int nbh = B * Hq;
  double acc = 0.0;
  for (int i = threadIdx.x; i < nbh; i += blockDim.x) {
    const double* p = part + ((int64_t)c * nbh + i) * nP;
    double s = 0.0;
    for (int k = 0; k < nP; ++k) s += p[k];
    if (parts_out) parts_out[(int64_t)c * nbh + i] = s;
    acc += s;
  }
  const double tot = block_sum<256>(acc, red);
  if (threadIdx.x == 0) {
    out[c] = tot * inv_n;
    if (!isfinite(tot)) report(status, JAB_ERR_NONFINITE);
  }
}

__global__ void loss_combine_kernel(const double* __restrict__ a, const double* __restrict__ b,
                                    double lam, int C, double* __restrict__ out) {
  for (int c = threadIdx.x; c < C; c += blockDim.x) out[c] = a[c] + lam * b[c];
}

// Omega of Eq. 6 per candidate: c1[c] = Tr(H) * sum of the candidate's quantisation-error partials
// (fixed order), c2[c] = layers_after * c1[c].
__global__ void omega_finish_kernel(const double* __restrict__ part, int nblocks, int C,
                                    const double* __restrict__ trace, double layers_after,
                                    double* __restrict__ c1, double* __restrict__ c2) {
  for (int c = threadIdx.x; c < C; c += blockDim.x) {
    double e = 0.0;
    for (int k = 0; k < nblocks; ++k) e += part[(int64_t)c * nblocks + k];
    const double v = *trace * e;
    c1[c] = v;
    if (c2) c2[c] = layers_after * v;
  }
}

// mean over n of a fp64 array (the Hutchinson estimate over its probes), fixed order
__global__ void mean_kernel(const double* __restrict__ x, int n, double* __restrict__ out) {
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int i = 0; i < n; ++i) t += x[i];
    *out = t / n;
  }
}

__global__ void check_finite_kernel(const float* __restrict__ x, int64_t n, int* status) {
  bool bad = false;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    bad |= !isfinite(x[i]);
  if (__syncthreads_or(bad) && threadIdx.x == 0) report(status, JAB_ERR_NONFINITE);
}

// Sum of squares in fp64: block b sums its contiguous chunk (fixed per-thread order, fixed tree),
// then one thread adds the kRedBlocks partials in order.
__global__ void __launch_bounds__(256) sumsq_partial_kernel(const float* __restrict__ x, int64_t n,
                                                            double* __restrict__ part) {
  __shared__ double red[8];
  const int64_t chunk = (n + gridDim.x - 1) / gridDim.x;
  const int64_t lo = blockIdx.x * chunk, hi = lo + chunk < n ? lo + chunk : n;
  double acc = 0.0;
  for (int64_t i = lo + threadIdx.x; i < hi; i += blockDim.x) {
    const double v = x[i];
    acc += v * v;
  }
  const double t = block_sum<256>(acc, red);
  if (threadIdx.x == 0) part[blockIdx.x] = t;
}

__global__ void sum_in_order_kernel(const double* __restrict__ part, int n, double* __restrict__ out) {
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int i = 0; i < n; ++i) t += part[i];
    *out = t;
  }
}

// One block: thread t adds its contiguous chunk in order, then a fixed tree (block_sum), so the
// result is the same on every call.
__global__ void __launch_bounds__(256) sum_scaled_kernel(const double* __restrict__ part, int n,
                                                         double scale, double* __restrict__ out) {
  __shared__ double red[8];
  const int chunk = (n + blockDim.x - 1) / blockDim.x;
  const int lo = threadIdx.x * chunk, hi = min(lo + chunk, n);
  double t = 0.0;
  for (int i = lo; i < hi; ++i) t += part[i];
  const double tot = block_sum<256>(t, red);
  if (threadIdx.x == 0) *out = scale * tot;
}

// Natural-log log-sum-exp rows [BH, T] to log2 units with the row pitch of the backward workspace.
__global__ void lse_to_log2_kernel(const float* __restrict__ in, int BH, int T, int pitch,
                                   float* __restrict__ out) {
  const int64_t n = (int64_t)BH * T;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / T, t = i - r * T;
    out[r * pitch + t] = in[i] * 1.4426950408889634f;
  }
}

// Sum of the K-split partials of a gradient in the order of the splits (one thread per element).
__global__ void split_sum_kernel(const float* __restrict__ part, int splits, int64_t n,
                                 float* __restrict__ out) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    double t = 0.0;
    for (int s = 0; s < splits; ++s) t += part[(int64_t)s * n + i];
    out[i] = (float)t;
  }
}

cudaError_t launch_loss_reduce(const double* part, int C, int B, int Hq, int nP, double inv_n,
                               double* out, double* parts_out, int* status, cudaStream_t st) {
  loss_reduce_kernel<<<C, 256, 0, st>>>(part, B, Hq, nP, inv_n, out, parts_out, status);
  return cudaGetLastError();
}

cudaError_t launch_loss_combine(const double* a, const double* b, double lam, int C, double* out,
                                cudaStream_t st) {
  loss_combine_kernel<<<1, 128, 0, st>>>(a, b, lam, C, out);
  return cudaGetLastError();
}

cudaError_t launch_omega_finish(const double* part, int nblocks, int C, const double* trace,
                                double layers_after, double* c1, double* c2, cudaStream_t st) {
  omega_finish_kernel<<<1, 128, 0, st>>>(part, nblocks, C, trace, layers_after, c1, c2);
  return cudaGetLastError();
}

cudaError_t launch_mean(const double* x, int n, double* out, cudaStream_t st) {
  mean_kernel<<<1, 32, 0, st>>>(x, n, out);
  return cudaGetLastError();
}

cudaError_t launch_sumsq(const float* x, int64_t n, double* part, double* out, cudaStream_t st) {
  sumsq_partial_kernel<<<kRedBlocks, 256, 0, st>>>(x, n, part);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  sum_in_order_kernel<<<1, 32, 0, st>>>(part, kRedBlocks, out);
  return cudaGetLastError();
}

cudaError_t launch_split_sum(const float* part, int splits, int64_t n, float* out, cudaStream_t st) {
  int64_t blocks = (n + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  if (blocks < 1) blocks = 1;
  split_sum_kernel<<<(unsigned)blocks, 256, 0, st>>>(part, splits, n, out);
  return cudaGetLastError();
}

cudaError_t launch_sum_scaled(const double* part, int n, double scale, double* out, cudaStream_t st) {
  sum_scaled_kernel<<<1, 256, 0, st>>>(part, n, scale, out);
  return cudaGetLastError();
}

cudaError_t launch_lse_to_log2(const float* in, int BH, int T, int pitch, float* out,
                               cudaStream_t st) {
  int64_t blocks = ((int64_t)BH * T + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  if (blocks < 1) blocks = 1;
  lse_to_log2_kernel<<<(unsigned)blocks, 256, 0, st>>>(in, BH, T, pitch, out);
  return cudaGetLastError();
}

cudaError_t launch_check_finite(const float* x, int64_t n, int* status, cudaStream_t st) {
  int64_t blocks = (n + 255) / 256;
  if (blocks > 1024) blocks = 1024;
  check_finite_kernel<<<(unsigned)blocks, 256, 0, st>>>(x, n, status);
  return cudaGetLastError();
}

}  // namespace jab
