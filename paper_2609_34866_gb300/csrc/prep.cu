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

// X [N, d] bf16 -> X^T [d, N] bf16 through a 64x64 shared-memory tile.
__global__ void transpose_bf16_kernel(const bf16_t* __restrict__ x, bf16_t* __restrict__ xt,
                                      int64_t N, int64_t ldt, int d) {
  __shared__ bf16_t tile[64][65];
  const int64_t n0 = (int64_t)blockIdx.x * 64;
  const int c0 = blockIdx.y * 64;
  for (int r = threadIdx.y; r < 64; r += blockDim.y) {
    const int64_t n = n0 + r;
    const int c = c0 + threadIdx.x;
    tile[r][threadIdx.x] = (n < N && c < d) ? x[n * d + c] : __float2bfloat16(0.f);
  }
  __syncthreads();
  for (int r = threadIdx.y; r < 64; r += blockDim.y) {
    const int c = c0 + r;
    const int64_t n = n0 + threadIdx.x;
    if (n < N && c < d) xt[(int64_t)c * ldt + n] = tile[threadIdx.x][r];
  }
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
      for (int k = 0; k < 8; ++k) h[k] = __float2half_rn(out[k]);
      w16[i] = o;
    }
  }
  if (bad) report(status, JAB_ERR_NONFINITE);
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

cudaError_t launch_transpose_x(const void* x, void* xt, int64_t N, int64_t ldt, int d,
                               cudaStream_t st) {
  dim3 grid((unsigned)((N + 63) / 64), (unsigned)((d + 63) / 64));
  transpose_bf16_kernel<<<grid, dim3(64, 8), 0, st>>>((const bf16_t*)x, (bf16_t*)xt, N, ldt, d);
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
