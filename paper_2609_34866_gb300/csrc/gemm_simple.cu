// CUDA-core GEMMs of the L_JAB path: a correctness-first implementation kept as the portable
// reference path of the library (selected with JAB_PATH=simple). The tensor-core (tcgen05) kernels
// in gemm_tc.cu compute the same outputs.
//
//  proj:  C[m, n] = sum_k A[m, k] B[n, k]   A = X fp16 [M, K], B = w_hat fp16 [Nn, K], C fp16 [M, Nn]
//         epilogue: rotate-half RoPE on the Q and K columns of each candidate, then fp16 store.
//  wgrad: G[o, i] = sum_n dQKV^T[o, n] X^T[i, n]   (bf16 operands, fp32 accumulation)
//         epilogue: ds[o, g] += coef * sum_{i in g} G[o, i] * r(w[o, i], s[o, g])   (Eq. 13)
#include "common.cuh"
#include "kernels.h"

namespace jab {

// ---------------------------------------------------------------- projection + RoPE
// Tile 64 x 128 x 32, 256 threads. Thread (ty, tx) owns rows ty + 16 i and columns tx + 16 j, so the
// RoPE partner column (+-d_h/2, a multiple of 16) of every output it holds is also in its registers.
__global__ void __launch_bounds__(256) proj_gemm_simple_kernel(
    const half_t* __restrict__ A, const half_t* __restrict__ Bw, half_t* __restrict__ C, int64_t M,
    int Nn, int K, int D, int n_rot, int dh, int T, const float* __restrict__ cos_t,
    const float* __restrict__ sin_t) {
  __shared__ float As[32][64 + 1];
  __shared__ float Bs[32][128 + 1];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int64_t m0 = (int64_t)blockIdx.y * 64;
  const int n0 = blockIdx.x * 128;
  float acc[4][8];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

  for (int k0 = 0; k0 < K; k0 += 32) {
    {  // A tile: 64 rows x 32 k = 256 x 8 halves
      const int r = tid >> 2, kk = (tid & 3) * 8;
      const int64_t m = m0 + r;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (m < M) v = *reinterpret_cast<const uint4*>(A + m * K + k0 + kk);
      const half_t* h = reinterpret_cast<const half_t*>(&v);
#pragma unroll
      for (int e = 0; e < 8; ++e) As[kk + e][r] = __half2float(h[e]);
    }
#pragma unroll
    for (int p = 0; p < 2; ++p) {  // B tile: 128 rows x 32 k
      const int r = (tid >> 2) + p * 64, kk = (tid & 3) * 8;
      const int n = n0 + r;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (n < Nn) v = *reinterpret_cast<const uint4*>(Bw + (int64_t)n * K + k0 + kk);
      const half_t* h = reinterpret_cast<const half_t*>(&v);
#pragma unroll
      for (int e = 0; e < 8; ++e) Bs[kk + e][r] = __half2float(h[e]);
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < 32; ++kk) {
      float a[4], b[8];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < 8; ++j) b[j] = Bs[kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }

  const int half = dh / 2, hstep = half / 16;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t m = m0 + ty + 16 * i;
    if (m >= M) continue;
    const int t = (int)(m % T);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int n = n0 + tx + 16 * j;
      if (n >= Nn) continue;
      float out = acc[i][j];
      const int o = n % D;
      if (n_rot > 0 && o < n_rot) {
        const int jj = o % dh;
        const int pj = (jj < half) ? j + hstep : j - hstep;  // partner column, same thread
        float partner = 0.f;
#pragma unroll
        for (int q = 0; q < 8; ++q)
          if (q == pj) partner = acc[i][q];
        const float c = cos_t[(int64_t)t * half + (jj % half)];
        const float s = sin_t[(int64_t)t * half + (jj % half)];
        out = (jj < half) ? out * c - partner * s : out * c + partner * s;
      }
      C[m * Nn + n] = __float2half_rn(out);
    }
  }
}

// ---------------------------------------------------------------- weight gradient + LSQ
// Tile 64 (o) x 64 (i) x 32 (n), 256 threads, thread owns rows ty + 16 a, columns tx + 16 b.
// The 64 columns of a tile lie in one quantisation group (G is a multiple of 64).
__global__ void __launch_bounds__(256) wgrad_lsq_simple_kernel(
    const bf16_t* __restrict__ dqkvt, const bf16_t* __restrict__ xt, int64_t ldt,
    const bf16_t* __restrict__ w, const float* __restrict__ s, int64_t N, int D, int d, int G,
    int bits, float coef, float* __restrict__ ds) {
  __shared__ float As[32][64 + 1];
  __shared__ float Bs[32][64 + 1];
  __shared__ float red[64][17];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int o0 = blockIdx.y * 64, i0 = blockIdx.x * 64;
  float acc[4][4];
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;
  const bool vec = (ldt % 8) == 0;
  for (int64_t n0 = 0; n0 < N; n0 += 32) {
    {  // 64 rows x 32 n of each operand: thread loads 8 consecutive n of one row
      const int r = tid >> 2, nn = (tid & 3) * 8;
      const int64_t n = n0 + nn;
      float va[8], vb[8];
      if (vec && n + 8 <= N) {  // 16-byte loads need row starts aligned: ldt % 8 == 0
        uint4 ua = *reinterpret_cast<const uint4*>(dqkvt + (int64_t)(o0 + r) * ldt + n);
        uint4 ub = *reinterpret_cast<const uint4*>(xt + (int64_t)(i0 + r) * ldt + n);
        const bf16_t* ha = reinterpret_cast<const bf16_t*>(&ua);
        const bf16_t* hb = reinterpret_cast<const bf16_t*>(&ub);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          va[e] = __bfloat162float(ha[e]);
          vb[e] = __bfloat162float(hb[e]);
        }
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const bool ok = n + e < N;
          va[e] = ok ? __bfloat162float(dqkvt[(int64_t)(o0 + r) * ldt + n + e]) : 0.f;
          vb[e] = ok ? __bfloat162float(xt[(int64_t)(i0 + r) * ldt + n + e]) : 0.f;
        }
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        As[nn + e][r] = va[e];
        Bs[nn + e][r] = vb[e];
      }
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < 32; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        a[q] = As[kk][ty + 16 * q];
        b[q] = Bs[kk][tx + 16 * q];
      }
#pragma unroll
      for (int p = 0; p < 4; ++p)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[p][q] = fmaf(a[p], b[q], acc[p][q]);
    }
    __syncthreads();
  }
  const int qmax = qmax_of(bits);
  const int ng = d / G;
  const int g = i0 / G;
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    const int o = o0 + ty + 16 * a;
    const float sc = s[(int64_t)o * ng + g];
    float sum = 0.f;
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const int i = i0 + tx + 16 * b;
      sum += acc[a][b] * lsq_factor(__bfloat162float(w[(int64_t)o * d + i]), sc, qmax);
    }
    red[ty + 16 * a][tx] = sum;
  }
  __syncthreads();
  if (tid < 64) {
    float t = 0.f;
#pragma unroll
    for (int k = 0; k < 16; ++k) t += red[tid][k];
    atomicAdd(ds + (int64_t)(o0 + tid) * ng + g, coef * t);
  }
}

cudaError_t launch_proj_gemm_simple(const void* A, const void* Bw, void* C, int64_t M, int Nn,
                                    int K, int D, int n_rot, int dh, int T, const float* cos_t,
                                    const float* sin_t, cudaStream_t st) {
  dim3 grid((unsigned)((Nn + 127) / 128), (unsigned)((M + 63) / 64));
  proj_gemm_simple_kernel<<<grid, 256, 0, st>>>((const half_t*)A, (const half_t*)Bw, (half_t*)C,
                                                M, Nn, K, D, n_rot, dh, T, cos_t, sin_t);
  return cudaGetLastError();
}

cudaError_t launch_wgrad_lsq_simple(const void* dqkvt, const void* xt, int64_t ldt, const void* w,
                                    const float* s, int64_t N, int D, int d, int G, int bits,
                                    float coef, float* ds, cudaStream_t st) {
  dim3 grid((unsigned)(d / 64), (unsigned)(D / 64));
  wgrad_lsq_simple_kernel<<<grid, 256, 0, st>>>((const bf16_t*)dqkvt, (const bf16_t*)xt, ldt,
                                                (const bf16_t*)w, s, N, D, d, G, bits, coef, ds);
  return cudaGetLastError();
}

}  // namespace jab
