// Shared device helpers for the JAB kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/jab.h"

namespace jab {

using half_t = __half;
using bf16_t = __nv_bfloat16;

// Records the first device-side problem in the per-device status word (0 = OK).
__device__ __forceinline__ void report(int* status, int code) {
  if (status != nullptr) atomicCAS(status, 0, code);
}

// Checked build (nvcc -DJAB_CHECKED=1, libjab_checked.so): the kernels test the last index of each
// computed global access against its buffer's extent before making it; a failed test reports
// JAB_ERR_DEVICE_ASSERT and the caller skips the access (no trap, no fault). Compiled out otherwise.
#ifndef JAB_CHECKED
#define JAB_CHECKED 0
#endif
__device__ __forceinline__ bool in_bounds(int64_t last, int64_t extent, int* status) {
#if JAB_CHECKED
  if (last < 0 || last >= extent) {
    report(status, JAB_ERR_DEVICE_ASSERT);
    return false;
  }
#else
  (void)last;
  (void)extent;
  (void)status;
#endif
  return true;
}

// Non-zero when either half of a packed fp16 pair has every exponent bit set: an infinity (the
// rounded value was outside the fp16 range) or a NaN. Integer SIMD compare, no FP instructions.
__device__ __forceinline__ uint32_t half2_exp_all_ones(uint32_t h2) {
  return __vcmpeq2(h2 & 0x7C007C00u, 0x7C007C00u);
}

__host__ __device__ __forceinline__ int qmax_of(int bits) { return (1 << (bits - 1)) - 1; }

// Eq. 2 with reading R1: v = fl32(w / s) (IEEE round-to-nearest division), q = clip(rint(v)).
__device__ __forceinline__ float quant_code(float w, float s, int qmax, float* v_out) {
  const float v = __fdiv_rn(w, s);
  float q = rintf(v);  // round half to even
  q = fminf(fmaxf(q, -(float)qmax), (float)qmax);
  if (v_out) *v_out = v;
  return q;
}

// Eq. 13: d w_hat / d s = q - v if |v| <= qmax, else sign(v) * qmax.
__device__ __forceinline__ float lsq_factor(float w, float s, int qmax) {
  float v;
  const float q = quant_code(w, s, qmax, &v);
  return (fabsf(v) <= (float)qmax) ? (q - v) : copysignf((float)qmax, v);
}

__device__ __forceinline__ double warp_sum(double x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}
__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// Block-wide sum in a fixed order (deterministic); every thread gets the result.
template <int NT>
__device__ __forceinline__ double block_sum(double x, double* smem /* >= NT/32 */) {
  x = warp_sum(x);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) smem[w] = x;
  __syncthreads();
  double t = 0.0;
#pragma unroll
  for (int i = 0; i < NT / 32; ++i) t += smem[i];
  return t;
}

// Static schedule of a persistent kernel: the tile a CTA takes in round i when `ntiles` tiles,
// ordered from the most work to the least, are dealt to `grid` CTAs. Rounds alternate direction
// (CTA x takes position x, then grid - 1 - x, ...), so every CTA gets a similar total; the tile
// index grows with i, so a CTA is done at its first index >= ntiles.
__device__ __forceinline__ int sched_tile(int i, int grid, int cta) {
  return i * grid + ((i & 1) ? grid - 1 - cta : cta);
}

}  // namespace jab
