// CUDA-core causal GQA attention of the L_JAB path (correctness-first reference path, selected with
// JAB_PATH=simple; attn_tc.cu holds the tensor-core kernels).
//
// Layouts: QKV fp16 [N, ldq] with the candidate's Q|K|V at column offset c*D; query head h at
// h*d_h, key/value head g at Hq*d_h + g*d_h and (Hq+Hkv)*d_h + g*d_h (nn.Linear row order).
// Four threads share one query (or key) row; thread quarter qd owns dims [qd*d_h/4, (qd+1)*d_h/4),
// so the RoPE partner dimension j +- d_h/2 lives in lane ^ 2.
#include "common.cuh"
#include "kernels.h"

namespace jab {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

struct AttnArgs {
  const half_t* qkv;
  int64_t ldq;     // row stride of qkv (C * D)
  int D;           // rows of the joint weight (columns per candidate)
  int B, T, Hq, Hkv;
  float scale;     // softmax scale
  int nP;          // partial tiles per (c, b, h)
  double* part;    // [C, B, Hq, nP]
  const float* a_ref;   // [N, Hq*d_h] fp32 (modes 1, 2)
  float* a_out;         // teacher output (mode 0)
  float* lse;           // [B, Hq, T] or null
  half_t* d_o;          // mode 2: e = A_hat - A_ref, fp16 [N, Hq*d_h]
  float* dvec;          // mode 2: rowsum(dO * O) [B, Hq, T]
  int* status;
  int lse_pitch;        // row pitch of lse / dvec
};

__device__ __forceinline__ float quad_sum(float x) {
  x += __shfl_xor_sync(0xffffffffu, x, 1);
  x += __shfl_xor_sync(0xffffffffu, x, 2);
  return x;
}

template <int DH>
__device__ __forceinline__ void load_tile(half_t (*dst)[DH], const half_t* src, int64_t ld,
                                          int64_t row0, int rows_valid) {
  // 64 rows x DH halves, 16-byte vectors
  constexpr int V = DH / 8;
  for (int i = threadIdx.x; i < 64 * V; i += blockDim.x) {
    const int r = i / V, c = (i % V) * 8;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (r < rows_valid) v = *reinterpret_cast<const uint4*>(src + (row0 + r) * ld + c);
    *reinterpret_cast<uint4*>(&dst[r][c]) = v;
  }
}

// MODE 0: teacher (write A and lse, partial ||A||^2); 1: loss (partial SSE); 2: loss + backward
// inputs (dO = e in fp16, lse in log2 units, rowsum(dO * O)).
template <int DH, int MODE>
__global__ void __launch_bounds__(256) attn_fwd_simple_kernel(AttnArgs a) {
  constexpr int DQ = DH / 4;
  __shared__ __align__(16) half_t Ks[64][DH];
  __shared__ __align__(16) half_t Vs[64][DH];
  __shared__ double red[8];
  const int qb = blockIdx.x, h = blockIdx.y;
  const int b = blockIdx.z % a.B, c = blockIdx.z / a.B;
  const int g = h / (a.Hq / a.Hkv);
  const int ql = threadIdx.x >> 2, qd = threadIdx.x & 3;
  const int t = qb * 64 + ql;
  const bool valid = t < a.T;
  const int te = valid ? t : a.T - 1;
  const int64_t rowbase = (int64_t)b * a.T;
  const half_t* Qp = a.qkv + (int64_t)c * a.D + (int64_t)h * DH;
  const half_t* Kp = a.qkv + (int64_t)c * a.D + (int64_t)(a.Hq + g) * DH;
  const half_t* Vp = a.qkv + (int64_t)c * a.D + (int64_t)(a.Hq + a.Hkv + g) * DH;

  float q[DQ], o[DQ];
  const float qs = a.scale * kLog2e;
#pragma unroll
  for (int k = 0; k < DQ; ++k) {
    q[k] = __half2float(Qp[(rowbase + te) * a.ldq + qd * DQ + k]) * qs;
    o[k] = 0.f;
  }
  float m = -INFINITY, l = 0.f;
  for (int kb = 0; kb <= qb; ++kb) {
    const int rows = min(64, a.T - kb * 64);
    __syncthreads();
    load_tile<DH>(Ks, Kp, a.ldq, rowbase + kb * 64, rows);
    load_tile<DH>(Vs, Vp, a.ldq, rowbase + kb * 64, rows);
    __syncthreads();
    float s[64];
    float mt = m;
#pragma unroll
    for (int j = 0; j < 64; ++j) {
      float p = 0.f;
#pragma unroll
      for (int k = 0; k < DQ; ++k) p = fmaf(q[k], __half2float(Ks[j][qd * DQ + k]), p);
      p = quad_sum(p);
      const int key = kb * 64 + j;
      s[j] = (key <= te) ? p : -INFINITY;
      mt = fmaxf(mt, s[j]);
    }
    const float alpha = exp2f(m - mt);  // m = -inf on the first tile: alpha = 0
    l *= alpha;
#pragma unroll
    for (int k = 0; k < DQ; ++k) o[k] *= alpha;
#pragma unroll
    for (int j = 0; j < 64; ++j) {
      const float p = exp2f(s[j] - mt);
      l += p;
      const float p16 = __half2float(__float2half_rn(p));
#pragma unroll
      for (int k = 0; k < DQ; ++k) o[k] = fmaf(p16, __half2float(Vs[j][qd * DQ + k]), o[k]);
    }
    m = mt;
  }
  // Explicitly rounded ops: the teacher (mode 0) and the student (modes 1, 2) must produce the same
  // bits for the same inputs, so no FMA contraction may differ between the modes.
  const float inv_l = __fdiv_rn(1.f, l);
#pragma unroll
  for (int k = 0; k < DQ; ++k) o[k] = __fmul_rn(o[k], inv_l);
  const float lse = MODE == 2 ? m + log2f(l) : (m + log2f(l)) * kLn2;  // mode 2: log2 units
  const int64_t orow = (rowbase + te) * (int64_t)(a.Hq * DH) + (int64_t)h * DH + qd * DQ;
  double acc = 0.0;
  if (MODE == 0) {
    float sq = 0.f;
#pragma unroll
    for (int k = 0; k < DQ; ++k) sq += o[k] * o[k];
    if (valid) {
#pragma unroll
      for (int k = 0; k < DQ; ++k) a.a_out[orow + k] = o[k];
    }
    acc = valid ? (double)sq : 0.0;
  } else {
    float sq = 0.f, dsum = 0.f;
#pragma unroll
    for (int k = 0; k < DQ; ++k) {
      const float e = __fsub_rn(o[k], a.a_ref[orow + k]);
      sq += e * e;
      if (MODE == 2) {
        const half_t e16 = __float2half_rn(e);
        dsum += __half2float(e16) * o[k];
        if (valid) a.d_o[orow + k] = e16;
      }
    }
    acc = valid ? (double)sq : 0.0;
    if (MODE == 2) {
      dsum = quad_sum(dsum);
      if (valid && qd == 0) a.dvec[((int64_t)b * a.Hq + h) * a.lse_pitch + t] = dsum;
    }
  }
  if (a.lse != nullptr && MODE != 1 && valid && qd == 0) a.lse[((int64_t)b * a.Hq + h) * a.lse_pitch + t] = lse;
  const double tot = block_sum<256>(acc, red);
  if (threadIdx.x == 0)
    a.part[(((int64_t)c * a.B + b) * a.Hq + h) * a.nP + qb] = tot;
}

// dQ: one CTA per (64 queries, query head, sequence); recomputes P from lse.
template <int DH>
__global__ void __launch_bounds__(256) attn_bwd_dq_simple_kernel(AttnArgs a, const float* cos_t,
                                                                 const float* sin_t, int use_rope,
                                                                 bf16_t* dqkvt, int64_t N) {
  constexpr int DQ = DH / 4;
  __shared__ __align__(16) half_t Ks[64][DH];
  __shared__ __align__(16) half_t Vs[64][DH];
  const int qb = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int g = h / (a.Hq / a.Hkv);
  const int ql = threadIdx.x >> 2, qd = threadIdx.x & 3;
  const int t = qb * 64 + ql;
  const bool valid = t < a.T;
  const int te = valid ? t : a.T - 1;
  const int64_t rowbase = (int64_t)b * a.T;
  const half_t* Qp = a.qkv + (int64_t)h * DH;
  const half_t* Kp = a.qkv + (int64_t)(a.Hq + g) * DH;
  const half_t* Vp = a.qkv + (int64_t)(a.Hq + a.Hkv + g) * DH;
  float q[DQ], dO[DQ], dq[DQ];
  const float qs = a.scale * kLog2e;
  const int64_t orow = (rowbase + te) * (int64_t)(a.Hq * DH) + (int64_t)h * DH + qd * DQ;
#pragma unroll
  for (int k = 0; k < DQ; ++k) {
    q[k] = __half2float(Qp[(rowbase + te) * a.ldq + qd * DQ + k]) * qs;
    dO[k] = __half2float(a.d_o[orow + k]);
    dq[k] = 0.f;
  }
  const float lse2 = a.lse[((int64_t)b * a.Hq + h) * a.lse_pitch + te];  // log2 units
  const float Dt = a.dvec[((int64_t)b * a.Hq + h) * a.lse_pitch + te];
  for (int kb = 0; kb <= qb; ++kb) {
    const int rows = min(64, a.T - kb * 64);
    __syncthreads();
    load_tile<DH>(Ks, Kp, a.ldq, rowbase + kb * 64, rows);
    load_tile<DH>(Vs, Vp, a.ldq, rowbase + kb * 64, rows);
    __syncthreads();
    for (int j = 0; j < 64; ++j) {
      float s = 0.f, dp = 0.f;
#pragma unroll
      for (int k = 0; k < DQ; ++k) {
        s = fmaf(q[k], __half2float(Ks[j][qd * DQ + k]), s);
        dp = fmaf(dO[k], __half2float(Vs[j][qd * DQ + k]), dp);
      }
      s = quad_sum(s);
      dp = quad_sum(dp);
      const int key = kb * 64 + j;
      const float p = (key <= te) ? exp2f(s - lse2) : 0.f;
      const float dsv = p * (dp - Dt);
#pragma unroll
      for (int k = 0; k < DQ; ++k) dq[k] = fmaf(dsv, __half2float(Ks[j][qd * DQ + k]), dq[k]);
    }
  }
  const int half = DH / 2;
#pragma unroll
  for (int k = 0; k < DQ; ++k) {
    float v = dq[k] * a.scale;
    const float partner = __shfl_xor_sync(0xffffffffu, dq[k] * a.scale, 2);
    const int dim = qd * DQ + k;
    if (use_rope) {
      const float cs = cos_t[(int64_t)te * half + dim % half];
      const float sn = sin_t[(int64_t)te * half + dim % half];
      v = (dim < half) ? v * cs + partner * sn : v * cs - partner * sn;  // transpose of RoPE
    }
    if (valid) dqkvt[((int64_t)h * DH + dim) * N + rowbase + t] = __float2bfloat16_rn(v);
  }
}

// dK, dV: one CTA per (64 keys, key/value head, sequence); loops over the query heads of the group.
template <int DH>
__global__ void __launch_bounds__(256) attn_bwd_dkdv_simple_kernel(AttnArgs a, const float* cos_t,
                                                                   const float* sin_t,
                                                                   int use_rope, bf16_t* dqkvt,
                                                                   int64_t N) {
  constexpr int DQ = DH / 4;
  __shared__ __align__(16) half_t Qs[64][DH];
  __shared__ __align__(16) half_t Os[64][DH];  // dO tile
  __shared__ float Ls[64], Ds[64];
  const int kb = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int kl = threadIdx.x >> 2, qd = threadIdx.x & 3;
  const int j = kb * 64 + kl;
  const bool valid = j < a.T;
  const int je = valid ? j : a.T - 1;
  const int64_t rowbase = (int64_t)b * a.T;
  const half_t* Kp = a.qkv + (int64_t)(a.Hq + g) * DH;
  const half_t* Vp = a.qkv + (int64_t)(a.Hq + a.Hkv + g) * DH;
  float k[DQ], v[DQ], dk[DQ], dv[DQ];
  const float qs = a.scale * kLog2e;
#pragma unroll
  for (int i = 0; i < DQ; ++i) {
    k[i] = __half2float(Kp[(rowbase + je) * a.ldq + qd * DQ + i]) * qs;
    v[i] = __half2float(Vp[(rowbase + je) * a.ldq + qd * DQ + i]);
    dk[i] = dv[i] = 0.f;
  }
  const int r = a.Hq / a.Hkv;
  const int nqb = (a.T + 63) / 64;
  for (int hh = 0; hh < r; ++hh) {
    const int h = g * r + hh;
    const half_t* Qp = a.qkv + (int64_t)h * DH;
    const half_t* dOp = a.d_o + (int64_t)h * DH;
    for (int qb = kb; qb < nqb; ++qb) {
      const int rows = min(64, a.T - qb * 64);
      __syncthreads();
      load_tile<DH>(Qs, Qp, a.ldq, rowbase + qb * 64, rows);
      load_tile<DH>(Os, dOp, (int64_t)a.Hq * DH, rowbase + qb * 64, rows);
      if (threadIdx.x < 64) {
        const int tq = min(qb * 64 + (int)threadIdx.x, a.T - 1);
        Ls[threadIdx.x] = a.lse[((int64_t)b * a.Hq + h) * a.lse_pitch + tq];
        Ds[threadIdx.x] = a.dvec[((int64_t)b * a.Hq + h) * a.lse_pitch + tq];
      }
      __syncthreads();
      for (int i = 0; i < 64; ++i) {
        float s = 0.f, dp = 0.f;
#pragma unroll
        for (int x = 0; x < DQ; ++x) {
          s = fmaf(k[x], __half2float(Qs[i][qd * DQ + x]), s);
          dp = fmaf(v[x], __half2float(Os[i][qd * DQ + x]), dp);
        }
        s = quad_sum(s);
        dp = quad_sum(dp);
        const int tq = qb * 64 + i;
        const float p = (tq < a.T && je <= tq) ? exp2f(s - Ls[i]) : 0.f;
        const float dsv = p * (dp - Ds[i]);
#pragma unroll
        for (int x = 0; x < DQ; ++x) {
          dv[x] = fmaf(p, __half2float(Os[i][qd * DQ + x]), dv[x]);
          dk[x] = fmaf(dsv, __half2float(Qs[i][qd * DQ + x]), dk[x]);
        }
      }
    }
  }
  const int half = DH / 2;
  const int64_t n = rowbase + j;
#pragma unroll
  for (int i = 0; i < DQ; ++i) {
    float gk = dk[i] * a.scale;
    const float partner = __shfl_xor_sync(0xffffffffu, dk[i] * a.scale, 2);
    const int dim = qd * DQ + i;
    if (use_rope) {
      const float cs = cos_t[(int64_t)je * half + dim % half];
      const float sn = sin_t[(int64_t)je * half + dim % half];
      gk = (dim < half) ? gk * cs + partner * sn : gk * cs - partner * sn;
    }
    if (valid) {
      dqkvt[((int64_t)(a.Hq + g) * DH + dim) * N + n] = __float2bfloat16_rn(gk);
      dqkvt[((int64_t)(a.Hq + a.Hkv + g) * DH + dim) * N + n] = __float2bfloat16_rn(dv[i]);
    }
  }
}

// ---------------------------------------------------------------- launchers
cudaError_t launch_attn_fwd_simple(const AttnLaunch& L, int mode) {
  AttnArgs a{(const half_t*)L.qkv, L.ldq, L.D, L.B, L.T, L.Hq, L.Hkv, L.scale, L.nP, L.part,
             L.a_ref, L.a_out, L.lse, (half_t*)L.d_o, L.dvec, L.status, L.lse_pitch};
  dim3 grid((unsigned)((L.T + 63) / 64), (unsigned)L.Hq, (unsigned)(L.B * L.C));
#define JAB_FWD(DH_, M_) attn_fwd_simple_kernel<DH_, M_><<<grid, 256, 0, L.stream>>>(a)
  if (L.dh == 128) {
    if (mode == 0) JAB_FWD(128, 0); else if (mode == 1) JAB_FWD(128, 1); else JAB_FWD(128, 2);
  } else {
    if (mode == 0) JAB_FWD(64, 0); else if (mode == 1) JAB_FWD(64, 1); else JAB_FWD(64, 2);
  }
#undef JAB_FWD
  return cudaGetLastError();
}

cudaError_t launch_attn_bwd_simple(const AttnLaunch& L, const float* cos_t, const float* sin_t,
                                   int use_rope, void* dqkvt) {
  AttnArgs a{(const half_t*)L.qkv, L.ldq, L.D, L.B, L.T, L.Hq, L.Hkv, L.scale, L.nP, L.part,
             L.a_ref, L.a_out, L.lse, (half_t*)L.d_o, L.dvec, L.status, L.lse_pitch};
  const int64_t N = L.ldt;  // row pitch of dQKV^T
  dim3 gq((unsigned)((L.T + 63) / 64), (unsigned)L.Hq, (unsigned)L.B);
  dim3 gk((unsigned)((L.T + 63) / 64), (unsigned)L.Hkv, (unsigned)L.B);
  if (L.dh == 128) {
    attn_bwd_dq_simple_kernel<128><<<gq, 256, 0, L.stream>>>(a, cos_t, sin_t, use_rope, (bf16_t*)dqkvt, N);
    attn_bwd_dkdv_simple_kernel<128><<<gk, 256, 0, L.stream>>>(a, cos_t, sin_t, use_rope, (bf16_t*)dqkvt, N);
  } else {
    attn_bwd_dq_simple_kernel<64><<<gq, 256, 0, L.stream>>>(a, cos_t, sin_t, use_rope, (bf16_t*)dqkvt, N);
    attn_bwd_dkdv_simple_kernel<64><<<gk, 256, 0, L.stream>>>(a, cos_t, sin_t, use_rope, (bf16_t*)dqkvt, N);
  }
  return cudaGetLastError();
}

}  // namespace jab
