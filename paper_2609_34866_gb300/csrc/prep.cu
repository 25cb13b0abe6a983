// Elementwise and small kernels of the L_JAB path: X conversion, the quantiser (Eq. 2), scale
// initialisation, the RoPE table. All are HBM-bound: 16-byte vector loads and stores, grids sized
// in multiples of the SM count.
#include "common.cuh"
#include "kernels.h"

namespace jab {

// ---------------------------------------------------------------- X: bf16 -> fp16 (+ range check)
__global__ void convert_x_kernel(const uint4* __restrict__ x, uint4* __restrict__ xh, int64_t n8,
                                 int* status) {
  int bad = 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n8;
       i += (int64_t)gridDim.x * blockDim.x) {
    uint4 v = __ldg(x + i);
    const bf16_t* b = reinterpret_cast<const bf16_t*>(&v);
    uint4 o;
    half_t* h = reinterpret_cast<half_t*>(&o);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float f = __bfloat162float(b[k]);
      h[k] = __float2half_rn(f);
      if (!isfinite(f)) bad |= 2;
      else if (__hisinf(h[k])) bad |= 1;
    }
    xh[i] = o;
  }
  if (bad & 2) report(status, JAB_ERR_NONFINITE);
  else if (bad & 1) report(status, JAB_ERR_RANGE);
}

// ---------------------------------------------------------------- quantiser (Section 2.1, Eq. 2)
// bits == 0: plain bf16 -> fp16 conversion of W (the teacher's weights).
__global__ void quantize_kernel(const uint4* __restrict__ w, const float* __restrict__ s, int D,
                                int d, int G, int bits, uint4* __restrict__ w16,
                                int8_t* __restrict__ codes, float* __restrict__ w_hat32,
                                int* status) {
  const int64_t n8 = (int64_t)D * d / 8;
  const int qmax = bits > 0 ? qmax_of(bits) : 0;
  const int ng = d / G;
  int bad = 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n8;
       i += (int64_t)gridDim.x * blockDim.x) {
    uint4 v = __ldg(w + i);
    const bf16_t* b = reinterpret_cast<const bf16_t*>(&v);
    const int64_t e0 = i * 8;
    const int64_t row = e0 / d;
    const int col = (int)(e0 - row * d);
    float out[8];
    if (bits == 0) {
#pragma unroll
      for (int k = 0; k < 8; ++k) out[k] = __bfloat162float(b[k]);
    } else {
      float sc = __ldg(s + row * ng + col / G);
      if (!(sc > 0.f) || !isfinite(sc)) {  // reading: scales must be finite and > 0
        bad = 1;
        sc = 1.f;
      }
      char cq[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float q = quant_code(__bfloat162float(b[k]), sc, qmax, nullptr);
        cq[k] = (char)(int)q;
        out[k] = __fmul_rn(q, sc);
      }
      if (codes) *reinterpret_cast<uint2*>(codes + e0) = *reinterpret_cast<uint2*>(cq);
      if (w_hat32) {
        reinterpret_cast<float4*>(w_hat32 + e0)[0] = make_float4(out[0], out[1], out[2], out[3]);
        reinterpret_cast<float4*>(w_hat32 + e0)[1] = make_float4(out[4], out[5], out[6], out[7]);
      }
    }
    if (w16) {
      uint4 o;
      half_t* h = reinterpret_cast<half_t*>(&o);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        h[k] = __float2half_rn(out[k]);
        if (__hisinf(h[k]) || __hisnan(h[k])) bad |= 2;  // not representable as an fp16 operand
      }
      w16[i] = o;
    }
  }
  if (bad & 1) report(status, JAB_ERR_NONFINITE);
  else if (bad & 2) report(status, JAB_ERR_RANGE);
}

// ---------------------------------------------------------------- Rademacher probes (Section 2.4)
// SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom number generators", 2014) used as
// a counter-based generator: entry n of the probe sequence (n = probe * D * d + flat index) takes
// the (n + 1)-th output of the stream seeded with `seed`; its top bit selects -1, else +1.
__device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t n) {
  uint64_t z = seed + (n + 1) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Entries are written as +-2^-k (fp16: exponent field 15 - k, zero mantissa), an exact scaling.
__global__ void rademacher_probe_kernel(uint64_t seed, uint64_t first, int64_t n8, int k2,
                                        uint4* __restrict__ out) {
  const uint16_t pos = (uint16_t)((15 - k2) << 10), neg = (uint16_t)(0x8000u | pos);
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n8;
       i += (int64_t)gridDim.x * blockDim.x) {
    uint4 o;
    uint16_t* h = reinterpret_cast<uint16_t*>(&o);
#pragma unroll
    for (int k = 0; k < 8; ++k)
      h[k] = (splitmix64_at(seed, first + (uint64_t)(i * 8 + k)) >> 63) ? neg : pos;
    out[i] = o;
  }
}

// ---------------------------------------------------------------- quantisation error (Eq. 6)
// Partial sums of (Q_b(w) - w)^2 over a grid-stride range, one per block (fp64, each term exact as
// the oracle forms it: q s - w in double); reduced in fixed order by omega_finish_kernel.
__global__ void __launch_bounds__(256) qerr_partial_kernel(const uint4* __restrict__ w,
                                                           const float* __restrict__ s, int D,
                                                           int d, int G, int bits,
                                                           double* __restrict__ part, int* status) {
  __shared__ double red[8];
  const int64_t n8 = (int64_t)D * d / 8;
  const int qmax = qmax_of(bits);
  const int ng = d / G;
  double acc = 0.0;
  int bad = 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n8;
       i += (int64_t)gridDim.x * blockDim.x) {
    uint4 v = __ldg(w + i);
    const bf16_t* b = reinterpret_cast<const bf16_t*>(&v);
    const int64_t e0 = i * 8;
    const int64_t row = e0 / d;
    const int col = (int)(e0 - row * d);
    float sc = __ldg(s + row * ng + col / G);
    if (!(sc > 0.f) || !isfinite(sc)) {
      bad = 1;
      sc = 1.f;
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float wv = __bfloat162float(b[k]);
      const double e = (double)quant_code(wv, sc, qmax, nullptr) * (double)sc - (double)wv;
      acc += e * e;
    }
  }
  const double t = block_sum<256>(acc, red);
  if (threadIdx.x == 0) part[blockIdx.x] = t;
  if (bad) report(status, JAB_ERR_NONFINITE);
}

// ---------------------------------------------------------------- flip count (App. B, Eq. 15)
// Number of positions where two int8 code arrays differ; 16 bytes per thread and step, one 64-bit
// atomic per block (integer sums: the result does not depend on the order).
__global__ void __launch_bounds__(256) flip_count_kernel(const uint4* __restrict__ a,
                                                         const uint4* __restrict__ b, int64_t n16,
                                                         const int8_t* __restrict__ a_tail,
                                                         const int8_t* __restrict__ b_tail,
                                                         int tail,
                                                         unsigned long long* __restrict__ count) {
  __shared__ unsigned long long red[8];
  unsigned long long c = 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n16;
       i += (int64_t)gridDim.x * blockDim.x) {
    const uint4 x = __ldg(a + i), y = __ldg(b + i);
    // __vcmpne4: 0xff in each byte that differs
    c += __popc(__vcmpne4(x.x, y.x)) + __popc(__vcmpne4(x.y, y.y)) + __popc(__vcmpne4(x.z, y.z)) +
         __popc(__vcmpne4(x.w, y.w));
  }
  c >>= 3;  // eight set bits per differing byte
  if (blockIdx.x == 0 && (int)threadIdx.x < tail) c += a_tail[threadIdx.x] != b_tail[threadIdx.x];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long t = 0;
    for (int w = 0; w < 8; ++w) t += red[w];
    atomicAdd(count, t);
  }
}

// ---------------------------------------------------------------- starting scales
// One warp per (row, group). mode 0: absmax / qmax. mode 1: min-MSE over s_k = fl32(s0*(100-k)/100).
__global__ void init_scales_kernel(const bf16_t* __restrict__ w, int D, int d, int G, int bits,
                                   int mode, float* __restrict__ s_out) {
  const int ng = d / G;
  const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= (int64_t)D * ng) return;
  const int64_t row = warp / ng;
  const int g = (int)(warp - row * ng);
  const bf16_t* wp = w + row * d + (int64_t)g * G;
  float amax = 0.f;
  for (int i = lane; i < G; i += 32) amax = fmaxf(amax, fabsf(__bfloat162float(wp[i])));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  const int qmax = qmax_of(bits);
  float s0 = (amax > 0.f) ? __fdiv_rn(amax, (float)qmax) : 1.f;
  float best = s0;
  if (mode == 1 && amax > 0.f) {
    double best_err = INFINITY;
    for (int k = 0; k < 80; ++k) {
      const float sk = (float)((double)s0 * (double)(100 - k) / 100.0);
      double err = 0.0;
      for (int i = lane; i < G; i += 32) {
        const float wv = __bfloat162float(wp[i]);
        const float q = quant_code(wv, sk, qmax, nullptr);
        const double e = (double)q * (double)sk - (double)wv;
        err += e * e;
      }
      err = warp_sum(err);
      if (err < best_err) {
        best_err = err;
        best = sk;
      }
    }
  }
  if (lane == 0) s_out[warp] = best;
}

// ---------------------------------------------------------------- RoPE table (reading R7)
__global__ void rope_table_kernel(int T, int dh, double theta, float* __restrict__ cos_t,
                                  float* __restrict__ sin_t) {
  const int half = dh / 2;
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= (int64_t)T * half) return;
  const int t = (int)(i / half), j = (int)(i % half);
  const double inv_freq = pow(theta, -2.0 * (double)j / (double)dh);
  const double phi = (double)t * inv_freq;
  double sn, cs;
  sincos(phi, &sn, &cs);
  cos_t[i] = (float)cs;
  sin_t[i] = (float)sn;
}

// ---------------------------------------------------------------- host launchers
static int grid_for(int64_t n, int threads, int sms) {
  int64_t g = (n + threads - 1) / threads;
  const int64_t cap = (int64_t)sms * 8;
  return (int)(g < cap ? (g < 1 ? 1 : g) : cap);
}

cudaError_t launch_convert_x(const void* x, void* xh, int64_t n, int* status, int sms,
                             cudaStream_t st) {
  const int64_t n8 = n / 8;
  convert_x_kernel<<<grid_for(n8, 256, sms), 256, 0, st>>>((const uint4*)x, (uint4*)xh, n8, status);
  return cudaGetLastError();
}

cudaError_t launch_quantize(const void* w, const float* s, int D, int d, int G, int bits,
                            void* w16, int8_t* codes, float* w_hat32, int* status, int sms,
                            cudaStream_t st) {
  const int64_t n8 = (int64_t)D * d / 8;
  quantize_kernel<<<grid_for(n8, 256, sms), 256, 0, st>>>(
      (const uint4*)w, s, D, d, G, bits, (uint4*)w16, codes, w_hat32, status);
  return cudaGetLastError();
}

cudaError_t launch_flip_count(const int8_t* a, const int8_t* b, int64_t n, int64_t* count,
                              int sms, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(count, 0, sizeof(int64_t), st);
  if (e != cudaSuccess) return e;
  const int64_t n16 = n / 16;
  const int tail = (int)(n - n16 * 16);
  flip_count_kernel<<<grid_for(n16 > 0 ? n16 : 1, 256, sms), 256, 0, st>>>(
      (const uint4*)a, (const uint4*)b, n16, a + n16 * 16, b + n16 * 16, tail,
      reinterpret_cast<unsigned long long*>(count));
  return cudaGetLastError();
}

cudaError_t launch_rademacher_probe(uint64_t seed, uint64_t first, int64_t n, int log2_scale,
                                    void* out, int sms, cudaStream_t st) {
  const int64_t n8 = n / 8;
  if (log2_scale < 0 || log2_scale > 14) return cudaErrorInvalidValue;
  rademacher_probe_kernel<<<grid_for(n8, 256, sms), 256, 0, st>>>(seed, first, n8, log2_scale,
                                                                 (uint4*)out);
  return cudaGetLastError();
}

cudaError_t launch_qerr_partial(const void* w, const float* s, int D, int d, int G, int bits,
                                double* part, int nblocks, int* status, cudaStream_t st) {
  qerr_partial_kernel<<<nblocks, 256, 0, st>>>((const uint4*)w, s, D, d, G, bits, part, status);
  return cudaGetLastError();
}

cudaError_t launch_init_scales(const void* w, int D, int d, int G, int bits, int mode,
                               float* s_out, cudaStream_t st) {
  const int64_t warps = (int64_t)D * (d / G);
  const int64_t blocks = (warps * 32 + 255) / 256;
  init_scales_kernel<<<(unsigned)blocks, 256, 0, st>>>((const bf16_t*)w, D, d, G, bits, mode, s_out);
  return cudaGetLastError();
}

cudaError_t launch_rope_table(int T, int dh, double theta, float* cos_t, float* sin_t,
                              cudaStream_t st) {
  const int64_t n = (int64_t)T * (dh / 2);
  rope_table_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(T, dh, theta, cos_t, sin_t);
  return cudaGetLastError();
}

}  // namespace jab
