// Tensor-core (tcgen05) causal GQA flash attention with the L_JAB epilogue, sm_103a.
//
// One CTA = 128 query rows of one (candidate, sequence, query head); keys in blocks of 128.
//   warp 0      TMA: the Q tile once, then K and V tiles of each key block (2-stage ring)
//   warp 1      TMEM owner, UMMA issuer (one thread):
//                 S_j = Q K_j^T            M128 N128 K=d_h     A, B K-major (smem)
//                 O  += P_j V_j            M128 N=d_h K128     A = P (smem, K-major), B = V MN-major
//               S is double-buffered in TMEM so S_{j+1} runs while the softmax works on S_j.
//   warps 2..9  softmax, two warps per TMEM lane quarter: a thread owns one query row and half of
//               its 128 scores (the halves exchange row maxima through shared memory): tcgen05.ld of
//               the S row, causal mask, online
//               softmax in the log2 domain with lazy rescaling (O is rescaled in TMEM only when the
//               running max grows by more than 2^8), P in fp16 to shared memory; after the last
//               block the epilogue of the calling mode:
//                 mode 0 (teacher)  A_ref = O (fp32), lse, partial ||A||^2
//                 mode 1 (loss)     partial SSE = sum (O - A_ref)^2                     (Eq. 3)
//                 mode 2 (loss+bwd) also dO = O - A_ref (fp16), lse in log2 units, D = rowsum(dO * O)
// The SSE partials are per (candidate, sequence, head, 128-row block), fp64, reduced in fixed order.
#include <cudaTypedefs.h>

#include "path.h"
#include "tc.cuh"

namespace jab {
namespace {

constexpr int BQ = 128, BKV = 128;
constexpr int NUM_THREADS = 320;  // warp 0 TMA, warp 1 UMMA, warps 2..9 softmax (2 per lane quarter)
constexpr int EW_WARPS = 8;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kRescaleLog2 = 8.f;  // rescale O only when the row max grows by more than 2^8

template <int DH>
struct FwdLayout {
  static constexpr int TILE = BQ * DH * 2;  // a 128-row tile of Q, K or V (fp16)
  static constexpr int CHUNK = BQ * 128;    // one 64-column (128-byte) swizzle chunk of a tile
  static constexpr int Q_OFF = 0;
  static constexpr int K_OFF = Q_OFF + TILE;
  static constexpr int V_OFF = K_OFF + 2 * TILE;
  static constexpr int P_OFF = V_OFF + 2 * TILE;
  static constexpr int P_BYTES = BQ * BKV * 2;
  static constexpr int BAR_OFF = P_OFF + P_BYTES;
  static constexpr int USED = BAR_OFF + 8192 + 1024;
  // At least half of the SM's shared memory, so that one CTA (and its 512 TMEM columns) owns the SM.
  static constexpr int SMEM = USED > 118 * 1024 ? USED : 118 * 1024;
};

struct FwdBars {
  uint64_t q_full, kv_full[2], kv_empty[2], s_full[2], s_empty[2], p_full, p_empty, o_full, drain;
  uint32_t tmem_base;
  int abort;
  double red[EW_WARPS];
  float xmax[2][2][BQ];  // [iteration parity][column half][row]: partial row maxima
  float xl[2][BQ];       // partial row sums, exchanged once at the end
  float xd[2][BQ];       // partial rowsum(dO * O)
  int flag[2][BQ];       // [column half][row]: sequence number of the last value posted
};

// Pair exchange between the two threads that own the halves of one row: post a value under a
// monotonically increasing sequence number, then read the partner's value of the same number.
// The wait is time-bounded like every mbarrier wait (no barrier that could hang if one side left).
__device__ __forceinline__ void pair_post(FwdBars* bars, int half, int row, int seq) {
  __threadfence_block();
  reinterpret_cast<volatile int*>(&bars->flag[half][row])[0] = seq;
}
__device__ __forceinline__ void pair_wait(FwdBars* bars, int half, int row, int seq,
                                          volatile int* abort, int* status) {
  volatile int* f = &bars->flag[half ^ 1][row];
  if (*f < seq) {
    const uint64_t t0 = tc::globaltimer();
    for (uint32_t it = 0; *f < seq; ++it) {
      if ((it & 63u) == 0) {
        if (*abort) break;
        if (tc::globaltimer() - t0 > tc::kWaitLimitNs) {
          *abort = 1;
          report(status, JAB_ERR_TIMEOUT);
          break;
        }
      }
    }
  }
  __threadfence_block();
}

struct FwdParams {
  int T, B, Hq, Hkv, D, nqb, nP, lse_pitch;
  float sl2;  // softmax scale * log2(e)
  double* part;
  const float* a_ref;
  float* a_out;
  float* lse;
  half_t* d_o;
  float* dvec;
  int* status;
};

__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = tc::globaltimer();
  while (!tc::mbar_test(bar, parity))
    if (tc::globaltimer() - t0 > tc::kWaitLimitNs) break;
}

template <int DH, int MODE>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    attn_fwd_tc_kernel(const __grid_constant__ CUtensorMap tm, const FwdParams p) {
  using L = FwdLayout<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  FwdBars* bars = reinterpret_cast<FwdBars*>(smem + L::BAR_OFF);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &bars->abort;

  const int qb = p.nqb - 1 - (int)blockIdx.z;  // slowest grid index: longest rows start first
  const int h = blockIdx.x;
  const int b = (int)blockIdx.y % p.B, c = (int)blockIdx.y / p.B;
  const int g = h / (p.Hq / p.Hkv);
  const int q0 = qb * BQ;
  const int nkb = min(qb + 1, (p.T + BKV - 1) / BKV);
  const int row0 = b * p.T;
  const int qcol = c * p.D + h * DH;
  const int kcol = c * p.D + (p.Hq + g) * DH;
  const int vcol = c * p.D + (p.Hq + p.Hkv + g) * DH;

  if (threadIdx.x == 0) {
    tc::mbar_init(&bars->q_full, 1);
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&bars->kv_full[i], 1);
      tc::mbar_init(&bars->kv_empty[i], 1);
      tc::mbar_init(&bars->s_full[i], 1);
      tc::mbar_init(&bars->s_empty[i], EW_WARPS);
    }
    tc::mbar_init(&bars->p_full, EW_WARPS);
    tc::mbar_init(&bars->p_empty, 1);
    tc::mbar_init(&bars->o_full, 1);
    tc::mbar_init(&bars->drain, 1);
    bars->abort = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&tm);
  }
  for (int i = threadIdx.x; i < 2 * BQ; i += blockDim.x) (&bars->flag[0][0])[i] = 0;
  if (warp == 1) {
    tc::tmem_alloc(&bars->tmem_base, 512);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = bars->tmem_base;
  constexpr uint32_t O_COL = 2 * BKV;

  if (warp == 0) {
    if (lane == 0) {  // ---------------------------------------------------------------- TMA
      uint32_t issued = 0, last_par = 0;
      tc::mbar_expect_tx(&bars->q_full, L::TILE);
      for (int ch = 0; ch < DH / 64; ++ch)
        tc::tma_load_2d(smem + L::Q_OFF + ch * L::CHUNK, &tm, &bars->q_full, qcol + ch * 64,
                        row0 + q0);
      for (int j = 0; j < nkb; ++j) {
        const int st = j & 1;
        if (!tc::mbar_wait(&bars->kv_empty[st], ((j >> 1) & 1) ^ 1, abort, p.status)) break;
        tc::mbar_expect_tx(&bars->kv_full[st], 2 * L::TILE);
        for (int ch = 0; ch < DH / 64; ++ch) {
          tc::tma_load_2d(smem + L::K_OFF + st * L::TILE + ch * L::CHUNK, &tm, &bars->kv_full[st],
                          kcol + ch * 64, row0 + j * BKV);
          tc::tma_load_2d(smem + L::V_OFF + st * L::TILE + ch * L::CHUNK, &tm, &bars->kv_full[st],
                          vcol + ch * 64, row0 + j * BKV);
        }
        issued |= 1u << st;
        last_par = (last_par & ~(1u << st)) | (((uint32_t)(j >> 1) & 1u) << st);
      }
      if (*abort) {
        drain_wait(&bars->q_full, 0);
        for (int st = 0; st < 2; ++st)
          if (issued & (1u << st)) drain_wait(&bars->kv_full[st], (last_par >> st) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {  // ---------------------------------------------------------------- UMMA
      constexpr uint32_t ID_S = tc::idesc_f16(false, BQ, BKV);
      constexpr uint32_t ID_PV = tc::idesc_f16(false, BQ, DH) | (1u << 16);  // B = V, MN-major
      const uint32_t q_base = tc::smem_u32(smem + L::Q_OFF);
      const uint32_t p_base = tc::smem_u32(smem + L::P_OFF);
      bool ok = tc::mbar_wait(&bars->q_full, 0, abort, p.status);
      auto issue_pv = [&](int jj) -> bool {
        if (!tc::mbar_wait(&bars->p_full, jj & 1, abort, p.status)) return false;
        tc::fence_after_sync();
        const int st = jj & 1;
        const uint32_t v_base = tc::smem_u32(smem + L::V_OFF + st * L::TILE);
#pragma unroll
        for (int k = 0; k < BKV / 16; ++k) {
          const uint64_t a = tc::sdesc_kmajor_sw128(p_base + (k >> 2) * (BQ * 128) + (k & 3) * 32);
          const uint64_t bdesc = tc::sdesc_mnmajor_sw128(v_base + k * 16 * 128, L::CHUNK, 1024);
          tc::umma_f16(tmem + O_COL, a, bdesc, ID_PV, (jj > 0 || k > 0) ? 1u : 0u);
        }
        tc::umma_commit(&bars->kv_empty[st]);
        tc::umma_commit(&bars->p_empty);
        return true;
      };
      for (int j = 0; ok && j < nkb; ++j) {
        const int st = j & 1;
        if (!tc::mbar_wait(&bars->kv_full[st], (j >> 1) & 1, abort, p.status)) break;
        if (!tc::mbar_wait(&bars->s_empty[st], ((j >> 1) & 1) ^ 1, abort, p.status)) break;
        tc::fence_after_sync();
        const uint32_t k_base = tc::smem_u32(smem + L::K_OFF + st * L::TILE);
#pragma unroll
        for (int k = 0; k < DH / 16; ++k) {
          const uint32_t off = (k >> 2) * L::CHUNK + (k & 3) * 32;
          tc::umma_f16(tmem + st * BKV, tc::sdesc_kmajor_sw128(q_base + off),
                       tc::sdesc_kmajor_sw128(k_base + off), ID_S, k > 0 ? 1u : 0u);
        }
        tc::umma_commit(&bars->s_full[st]);
        if (j > 0 && !issue_pv(j - 1)) {
          ok = false;
          break;
        }
        if (j == nkb - 1) {
          if (issue_pv(j)) tc::umma_commit(&bars->o_full);
        }
      }
      tc::umma_commit(&bars->drain);
      drain_wait(&bars->drain, 0);
    }
  } else {  // ------------------------------------------------------------------------ softmax
    const int quarter = warp & 3;
    const int half = (warp - 2) >> 2;
    const int row = quarter * 32 + lane;
    const int t = q0 + row;
    const int col0 = half * (BKV / 2);  // this thread's 64 score columns
    const int ocol0 = half * (DH / 2);  // and DH/2 output columns
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    uint8_t* pbuf = smem + L::P_OFF;
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      const int sb = j & 1;
      if (!tc::mbar_wait(&bars->s_full[sb], (j >> 1) & 1, abort, p.status)) {
        ok = false;
        break;
      }
      tc::fence_after_sync();
      float s[BKV / 2];
#pragma unroll
      for (int ch = 0; ch < BKV / 64; ++ch) {
        uint32_t r[32];
        __syncwarp();
        tc::tmem_ld32(tmem + lane_base + sb * BKV + col0 + ch * 32, r);
        tc::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i) s[ch * 32 + i] = __uint_as_float(r[i]) * p.sl2;
      }
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->s_empty[sb]);
      const int k0 = j * BKV + col0;
      if (k0 + BKV / 2 - 1 > q0 || k0 + BKV / 2 > p.T) {  // diagonal or ragged block: mask
#pragma unroll
        for (int i = 0; i < BKV / 2; ++i)
          if (k0 + i > t || k0 + i >= p.T) s[i] = -INFINITY;
      }
      float mx8[8];  // 8 independent partial maxima: a short dependency chain
#pragma unroll
      for (int i = 0; i < 8; ++i) mx8[i] = s[i];
#pragma unroll
      for (int i = 8; i < BKV / 2; ++i) mx8[i & 7] = fmaxf(mx8[i & 7], s[i]);
      const float pmax = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                               fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
      bars->xmax[sb][half][row] = pmax;
      pair_post(bars, half, row, j + 1);
      pair_wait(bars, half, row, j + 1, abort, p.status);
      const float mx = fmaxf(pmax, reinterpret_cast<volatile float*>(&bars->xmax[sb][half ^ 1][row])[0]);
      const float m_new = fmaxf(m, mx);
      const bool resc = m_new > m + kRescaleLog2;
      const float m_use = resc ? m_new : m;
      const float alpha = resc ? tc::fast_exp2(m - m_new) : 1.f;
      float rs8[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int i = 0; i < BKV / 2; ++i) {
        s[i] = tc::fast_exp2(s[i] - m_use);
        rs8[i & 7] += s[i];
      }
      l = l * alpha + (((rs8[0] + rs8[1]) + (rs8[2] + rs8[3])) + ((rs8[4] + rs8[5]) + (rs8[6] + rs8[7])));
      m = m_use;
      // P_{j-1} V_{j-1} must be complete before O is rescaled or the P buffer is overwritten.
      if (!tc::mbar_wait(&bars->p_empty, (j & 1) ^ 1, abort, p.status)) {
        ok = false;
        break;
      }
      tc::fence_after_sync();
      if (j > 0 && __any_sync(0xffffffffu, resc)) {
#pragma unroll
        for (int ch = 0; ch < DH / 64; ++ch) {
          uint32_t r[32];
          __syncwarp();
          tc::tmem_ld32(tmem + lane_base + O_COL + ocol0 + ch * 32, r);
          tc::tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
          tc::tmem_st32(tmem + lane_base + O_COL + ocol0 + ch * 32, r);
        }
        tc::tmem_st_wait();
      }
      uint8_t* prow = pbuf + half * (BQ * 128) + row * 128;  // this half = one 64-key swizzle chunk
#pragma unroll
      for (int c8 = 0; c8 < 8; ++c8) {
        uint4 u;
        __half2* hp = reinterpret_cast<__half2*>(&u);
#pragma unroll
        for (int e = 0; e < 4; ++e) hp[e] = __floats2half2_rn(s[c8 * 8 + 2 * e], s[c8 * 8 + 2 * e + 1]);
        *reinterpret_cast<uint4*>(prow + ((c8 ^ (row & 7)) << 4)) = u;
      }
      tc::fence_proxy_async_smem();
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->p_full);
    }
    // ---------------------------------------------------------------- epilogue
    double acc = 0.0;
    bars->xl[half][row] = l;
    pair_post(bars, half, row, nkb + 1);
    pair_wait(bars, half, row, nkb + 1, abort, p.status);
    l += reinterpret_cast<volatile float*>(&bars->xl[half ^ 1][row])[0];
    if (ok && tc::mbar_wait(&bars->o_full, 0, abort, p.status)) {
      tc::fence_after_sync();
      const bool valid = t < p.T;
      const float inv_l = __fdiv_rn(1.f, l);
      const int64_t orow = ((int64_t)row0 + (valid ? t : 0)) * (int64_t)(p.Hq * DH) + h * DH + ocol0;
      float sq = 0.f, dsum = 0.f;
#pragma unroll 1
      for (int ch = 0; ch < DH / 64; ++ch) {
        uint32_t r[32];
        __syncwarp();
        tc::tmem_ld32(tmem + lane_base + O_COL + ocol0 + ch * 32, r);
        tc::tmem_ld_wait();
        float o[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) o[i] = __fmul_rn(__uint_as_float(r[i]), inv_l);
        if (!valid) continue;
        if (MODE == 0) {
          float4* dst = reinterpret_cast<float4*>(p.a_out + orow + ch * 32);
#pragma unroll
          for (int v = 0; v < 8; ++v) {
            dst[v] = make_float4(o[4 * v], o[4 * v + 1], o[4 * v + 2], o[4 * v + 3]);
            sq += o[4 * v] * o[4 * v] + o[4 * v + 1] * o[4 * v + 1] + o[4 * v + 2] * o[4 * v + 2] +
                  o[4 * v + 3] * o[4 * v + 3];
          }
        } else {
          const float4* ar = reinterpret_cast<const float4*>(p.a_ref + orow + ch * 32);
          float e[32];
#pragma unroll
          for (int v = 0; v < 8; ++v) {
            const float4 a4 = __ldg(ar + v);
            e[4 * v] = __fsub_rn(o[4 * v], a4.x);
            e[4 * v + 1] = __fsub_rn(o[4 * v + 1], a4.y);
            e[4 * v + 2] = __fsub_rn(o[4 * v + 2], a4.z);
            e[4 * v + 3] = __fsub_rn(o[4 * v + 3], a4.w);
          }
#pragma unroll
          for (int i = 0; i < 32; ++i) sq += e[i] * e[i];
          if (MODE == 2) {
            uint4* dst = reinterpret_cast<uint4*>(p.d_o + orow + ch * 32);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
              uint4 u;
              __half2* hp = reinterpret_cast<__half2*>(&u);
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                hp[k] = __floats2half2_rn(e[v * 8 + 2 * k], e[v * 8 + 2 * k + 1]);
                const float2 f = __half22float2(hp[k]);
                dsum += f.x * o[v * 8 + 2 * k] + f.y * o[v * 8 + 2 * k + 1];
              }
              dst[v] = u;
            }
          }
        }
      }
      if (MODE == 2) {
        bars->xd[half][row] = dsum;
        pair_post(bars, half, row, nkb + 2);
        pair_wait(bars, half, row, nkb + 2, abort, p.status);
        dsum += reinterpret_cast<volatile float*>(&bars->xd[half ^ 1][row])[0];
      }
      if (valid && half == 0) {
        if (MODE != 1 && p.lse != nullptr)
          p.lse[((int64_t)b * p.Hq + h) * p.lse_pitch + t] =
              MODE == 2 ? m + log2f(l) : (m + log2f(l)) * kLn2;  // mode 2: log2 units
        if (MODE == 2) p.dvec[((int64_t)b * p.Hq + h) * p.lse_pitch + t] = dsum;
      }
      if (valid) acc = (double)sq;
    }
    acc = warp_sum(acc);
    if (lane == 0) bars->red[warp - 2] = acc;
    tc::named_bar_sync(1, EW_WARPS * 32);
    if (warp == 2 && lane == 0) {
      double tot = 0.0;
      for (int w = 0; w < EW_WARPS; ++w) tot += bars->red[w];
      p.part[(((int64_t)c * p.B + b) * p.Hq + h) * p.nP + qb] = tot;
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  if (warp == 1) {
    __syncwarp();
    tc::tmem_dealloc(tmem, 512);
  }
}

// ============================================================================ head-pair kernel
// Two query heads of one KV group per CTA (GQA: they read the same K and V), 128 query rows each,
// keys in blocks of 64 through a 3-stage K/V ring. Per head: S double-buffered in TMEM (2 x 64
// columns), O in TMEM (128 columns), P in shared memory; four softmax warps per head, one row per
// thread. Every K/V byte loaded feeds twice the tensor work of the single-head kernel.
constexpr int PBQ = 128, PBK = 64, PSTAGES = 3;

template <int DH>
struct PairLayout {
  static constexpr int QTILE = PBQ * DH * 2;
  static constexpr int QCHUNK = PBQ * 128;
  static constexpr int KVTILE = PBK * DH * 2;
  static constexpr int KVCHUNK = PBK * 128;
  static constexpr int Q_OFF = 0;
  static constexpr int KV_OFF = Q_OFF + 2 * QTILE;
  static constexpr int STAGE = 2 * KVTILE;  // K then V
  static constexpr int P_OFF = KV_OFF + PSTAGES * STAGE;
  static constexpr int PTILE = PBQ * PBK * 2;
  static constexpr int BAR_OFF = P_OFF + 2 * PTILE;
  static constexpr int USED = BAR_OFF + 512 + 1024;
  static constexpr int SMEM = USED > 118 * 1024 ? USED : 118 * 1024;
};

struct PairBars {
  uint64_t q_full, kv_full[PSTAGES], kv_empty[PSTAGES];
  uint64_t s_full[2][2], s_empty[2][2], p_full[2], p_empty[2], o_full[2], drain;
  uint32_t tmem_base;
  int abort;
  double red[EW_WARPS];
};

template <int DH, int MODE>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    attn_fwd_pair_kernel(const __grid_constant__ CUtensorMap tm_q,
                         const __grid_constant__ CUtensorMap tm_kv, const FwdParams p) {
  using L = PairLayout<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  PairBars* bars = reinterpret_cast<PairBars*>(smem + L::BAR_OFF);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &bars->abort;

  const int qb = p.nqb - 1 - (int)blockIdx.z;  // slowest grid index: longest rows start first
  const int h0 = 2 * (int)blockIdx.x;
  const int b = (int)blockIdx.y % p.B, c = (int)blockIdx.y / p.B;
  const int g = h0 / (p.Hq / p.Hkv);
  const int q0 = qb * PBQ;
  const int nkb = (min(q0 + PBQ, p.T) + PBK - 1) / PBK;
  const int row0 = b * p.T;
  const int kcol = c * p.D + (p.Hq + g) * DH;
  const int vcol = c * p.D + (p.Hq + p.Hkv + g) * DH;

  if (threadIdx.x == 0) {
    tc::mbar_init(&bars->q_full, 1);
    for (int i = 0; i < PSTAGES; ++i) {
      tc::mbar_init(&bars->kv_full[i], 1);
      tc::mbar_init(&bars->kv_empty[i], 1);
    }
    for (int hd = 0; hd < 2; ++hd) {
      for (int i = 0; i < 2; ++i) {
        tc::mbar_init(&bars->s_full[hd][i], 1);
        tc::mbar_init(&bars->s_empty[hd][i], 4);
      }
      tc::mbar_init(&bars->p_full[hd], 4);
      tc::mbar_init(&bars->p_empty[hd], 1);
      tc::mbar_init(&bars->o_full[hd], 1);
    }
    tc::mbar_init(&bars->drain, 1);
    bars->abort = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&tm_q);
    tc::prefetch_tmap(&tm_kv);
  }
  if (warp == 1) {
    tc::tmem_alloc(&bars->tmem_base, 512);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = bars->tmem_base;
  auto s_col = [](int hd, int sb) { return (uint32_t)((hd * 2 + sb) * PBK); };
  auto o_col = [](int hd) { return (uint32_t)(4 * PBK + hd * 128); };

  if (warp == 0) {
    if (lane == 0) {  // ---------------------------------------------------------------- TMA
      uint32_t issued = 0, last_par = 0;
      tc::mbar_expect_tx(&bars->q_full, 2 * L::QTILE);
      for (int hd = 0; hd < 2; ++hd)
        for (int ch = 0; ch < DH / 64; ++ch)
          tc::tma_load_2d(smem + L::Q_OFF + hd * L::QTILE + ch * L::QCHUNK, &tm_q, &bars->q_full,
                          c * p.D + (h0 + hd) * DH + ch * 64, row0 + q0);
      for (int j = 0; j < nkb; ++j) {
        const int st = j % PSTAGES;
        const uint32_t ph = (j / PSTAGES) & 1;
        if (!tc::mbar_wait(&bars->kv_empty[st], ph ^ 1, abort, p.status)) break;
        uint8_t* sbase = smem + L::KV_OFF + st * L::STAGE;
        tc::mbar_expect_tx(&bars->kv_full[st], L::STAGE);
        for (int ch = 0; ch < DH / 64; ++ch) {
          tc::tma_load_2d(sbase + ch * L::KVCHUNK, &tm_kv, &bars->kv_full[st], kcol + ch * 64,
                          row0 + j * PBK);
          tc::tma_load_2d(sbase + L::KVTILE + ch * L::KVCHUNK, &tm_kv, &bars->kv_full[st],
                          vcol + ch * 64, row0 + j * PBK);
        }
        issued |= 1u << st;
        last_par = (last_par & ~(1u << st)) | (ph << st);
      }
      if (*abort) {
        drain_wait(&bars->q_full, 0);
        for (int st = 0; st < PSTAGES; ++st)
          if (issued & (1u << st)) drain_wait(&bars->kv_full[st], (last_par >> st) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {  // ---------------------------------------------------------------- UMMA
      constexpr uint32_t ID_S = tc::idesc_f16(false, PBQ, PBK);
      constexpr uint32_t ID_PV = tc::idesc_f16(false, PBQ, DH) | (1u << 16);  // B = V, MN-major
      bool ok = tc::mbar_wait(&bars->q_full, 0, abort, p.status);
      auto issue_pv = [&](int hd, int jj) -> bool {
        if (!tc::mbar_wait(&bars->p_full[hd], jj & 1, abort, p.status)) return false;
        tc::fence_after_sync();
        const uint32_t v_base =
            tc::smem_u32(smem + L::KV_OFF + (jj % PSTAGES) * L::STAGE + L::KVTILE);
        const uint32_t p_base = tc::smem_u32(smem + L::P_OFF + hd * L::PTILE);
#pragma unroll
        for (int k = 0; k < PBK / 16; ++k)
          tc::umma_f16(tmem + o_col(hd), tc::sdesc_kmajor_sw128(p_base + k * 32),
                       tc::sdesc_mnmajor_sw128(v_base + k * 16 * 128, L::KVCHUNK, 1024), ID_PV,
                       (jj > 0 || k > 0) ? 1u : 0u);
        tc::umma_commit(&bars->p_empty[hd]);
        if (hd == 1) tc::umma_commit(&bars->kv_empty[jj % PSTAGES]);
        return true;
      };
      for (int j = 0; ok && j < nkb; ++j) {
        const int st = j % PSTAGES, sb = j & 1;
        if (!tc::mbar_wait(&bars->kv_full[st], (j / PSTAGES) & 1, abort, p.status)) break;
        const uint32_t k_base = tc::smem_u32(smem + L::KV_OFF + st * L::STAGE);
        for (int hd = 0; hd < 2 && ok; ++hd) {
          if (!tc::mbar_wait(&bars->s_empty[hd][sb], ((j >> 1) & 1) ^ 1, abort, p.status)) {
            ok = false;
            break;
          }
          tc::fence_after_sync();
          const uint32_t q_base = tc::smem_u32(smem + L::Q_OFF + hd * L::QTILE);
#pragma unroll
          for (int k = 0; k < DH / 16; ++k)
            tc::umma_f16(tmem + s_col(hd, sb),
                         tc::sdesc_kmajor_sw128(q_base + (k >> 2) * L::QCHUNK + (k & 3) * 32),
                         tc::sdesc_kmajor_sw128(k_base + (k >> 2) * L::KVCHUNK + (k & 3) * 32),
                         ID_S, k > 0 ? 1u : 0u);
          tc::umma_commit(&bars->s_full[hd][sb]);
        }
        if (!ok) break;
        if (j > 0 && (!issue_pv(0, j - 1) || !issue_pv(1, j - 1))) break;
        if (j == nkb - 1) {
          for (int hd = 0; hd < 2; ++hd)
            if (issue_pv(hd, j)) tc::umma_commit(&bars->o_full[hd]);
        }
      }
      tc::umma_commit(&bars->drain);
      drain_wait(&bars->drain, 0);
    }
  } else {  // ------------------------------------------------------------------------ softmax
    const int hd = (warp - 2) >> 2;
    const int h = h0 + hd;
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const int t = q0 + row;
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    uint8_t* prow = smem + L::P_OFF + hd * L::PTILE + row * 128;
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      const int sb = j & 1;
      if (!tc::mbar_wait(&bars->s_full[hd][sb], (j >> 1) & 1, abort, p.status)) {
        ok = false;
        break;
      }
      tc::fence_after_sync();
      float s[PBK];
#pragma unroll
      for (int ch = 0; ch < PBK / 32; ++ch) {
        uint32_t r[32];
        __syncwarp();
        tc::tmem_ld32(tmem + lane_base + s_col(hd, sb) + ch * 32, r);
        tc::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i) s[ch * 32 + i] = __uint_as_float(r[i]) * p.sl2;
      }
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->s_empty[hd][sb]);
      const int k0 = j * PBK;
      if (k0 + PBK - 1 > q0 || k0 + PBK > p.T) {  // diagonal or ragged block: mask
#pragma unroll
        for (int i = 0; i < PBK; ++i)
          if (k0 + i > t || k0 + i >= p.T) s[i] = -INFINITY;
      }
      float mx8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx8[i] = s[i];
#pragma unroll
      for (int i = 8; i < PBK; ++i) mx8[i & 7] = fmaxf(mx8[i & 7], s[i]);
      const float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                             fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
      const float m_new = fmaxf(m, mx);
      const bool resc = m_new > m + kRescaleLog2;
      const float m_use = resc ? m_new : m;
      const float alpha = resc ? tc::fast_exp2(m - m_new) : 1.f;
      float rs8[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int i = 0; i < PBK; ++i) {
        s[i] = tc::fast_exp2(s[i] - m_use);
        rs8[i & 7] += s[i];
      }
      l = l * alpha + (((rs8[0] + rs8[1]) + (rs8[2] + rs8[3])) + ((rs8[4] + rs8[5]) + (rs8[6] + rs8[7])));
      m = m_use;
      // P V of the previous block must be complete before O is rescaled or P is overwritten.
      if (!tc::mbar_wait(&bars->p_empty[hd], (j & 1) ^ 1, abort, p.status)) {
        ok = false;
        break;
      }
      tc::fence_after_sync();
      if (j > 0 && __any_sync(0xffffffffu, resc)) {
#pragma unroll
        for (int ch = 0; ch < DH / 32; ++ch) {
          uint32_t r[32];
          __syncwarp();
          tc::tmem_ld32(tmem + lane_base + o_col(hd) + ch * 32, r);
          tc::tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
          tc::tmem_st32(tmem + lane_base + o_col(hd) + ch * 32, r);
        }
        tc::tmem_st_wait();
      }
#pragma unroll
      for (int c8 = 0; c8 < 8; ++c8) {
        uint4 u;
        __half2* hp = reinterpret_cast<__half2*>(&u);
#pragma unroll
        for (int e = 0; e < 4; ++e) hp[e] = __floats2half2_rn(s[c8 * 8 + 2 * e], s[c8 * 8 + 2 * e + 1]);
        *reinterpret_cast<uint4*>(prow + ((c8 ^ (row & 7)) << 4)) = u;
      }
      tc::fence_proxy_async_smem();
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->p_full[hd]);
    }
    // ---------------------------------------------------------------- epilogue
    double acc = 0.0;
    if (ok && tc::mbar_wait(&bars->o_full[hd], 0, abort, p.status)) {
      tc::fence_after_sync();
      const bool valid = t < p.T;
      const float inv_l = __fdiv_rn(1.f, l);
      const int64_t orow = ((int64_t)row0 + (valid ? t : 0)) * (int64_t)(p.Hq * DH) + h * DH;
      float sq = 0.f, dsum = 0.f;
#pragma unroll 1
      for (int ch = 0; ch < DH / 32; ++ch) {
        uint32_t r[32];
        __syncwarp();
        tc::tmem_ld32(tmem + lane_base + o_col(hd) + ch * 32, r);
        tc::tmem_ld_wait();
        float o[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) o[i] = __fmul_rn(__uint_as_float(r[i]), inv_l);
        if (!valid) continue;
        if (MODE == 0) {
          float4* dst = reinterpret_cast<float4*>(p.a_out + orow + ch * 32);
#pragma unroll
          for (int v = 0; v < 8; ++v) {
            dst[v] = make_float4(o[4 * v], o[4 * v + 1], o[4 * v + 2], o[4 * v + 3]);
            sq += o[4 * v] * o[4 * v] + o[4 * v + 1] * o[4 * v + 1] + o[4 * v + 2] * o[4 * v + 2] +
                  o[4 * v + 3] * o[4 * v + 3];
          }
        } else {
          const float4* ar = reinterpret_cast<const float4*>(p.a_ref + orow + ch * 32);
          float e[32];
#pragma unroll
          for (int v = 0; v < 8; ++v) {
            const float4 a4 = __ldg(ar + v);
            e[4 * v] = __fsub_rn(o[4 * v], a4.x);
            e[4 * v + 1] = __fsub_rn(o[4 * v + 1], a4.y);
            e[4 * v + 2] = __fsub_rn(o[4 * v + 2], a4.z);
            e[4 * v + 3] = __fsub_rn(o[4 * v + 3], a4.w);
          }
#pragma unroll
          for (int i = 0; i < 32; ++i) sq += e[i] * e[i];
          if (MODE == 2) {
            uint4* dst = reinterpret_cast<uint4*>(p.d_o + orow + ch * 32);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
              uint4 u;
              __half2* hp = reinterpret_cast<__half2*>(&u);
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                hp[k] = __floats2half2_rn(e[v * 8 + 2 * k], e[v * 8 + 2 * k + 1]);
                const float2 f = __half22float2(hp[k]);
                dsum += f.x * o[v * 8 + 2 * k] + f.y * o[v * 8 + 2 * k + 1];
              }
              dst[v] = u;
            }
          }
        }
      }
      if (valid) {
        if (MODE != 1 && p.lse != nullptr)
          p.lse[((int64_t)b * p.Hq + h) * p.lse_pitch + t] =
              MODE == 2 ? m + log2f(l) : (m + log2f(l)) * kLn2;  // mode 2: log2 units
        if (MODE == 2) p.dvec[((int64_t)b * p.Hq + h) * p.lse_pitch + t] = dsum;
        acc = (double)sq;
      }
    }
    acc = warp_sum(acc);
    if (lane == 0) bars->red[warp - 2] = acc;
    tc::named_bar_sync(1, EW_WARPS * 32);
    if (quarter == 0 && lane == 0) {  // one thread per head
      const int w0 = hd * 4;
      p.part[(((int64_t)c * p.B + b) * p.Hq + h) * p.nP + qb] =
          bars->red[w0] + bars->red[w0 + 1] + bars->red[w0 + 2] + bars->red[w0 + 3];
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  if (warp == 1) {
    __syncwarp();
    tc::tmem_dealloc(tmem, 512);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return (PFN_cuTensorMapEncodeTiled_v12000) nullptr;
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  }();
  return fn;
}

template <int DH, int MODE>
cudaError_t launch_fwd_pair(const CUtensorMap& tq, const CUtensorMap& tkv, const FwdParams& p,
                            dim3 grid, cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(attn_fwd_pair_kernel<DH, MODE>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         PairLayout<DH>::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  attn_fwd_pair_kernel<DH, MODE><<<grid, NUM_THREADS, PairLayout<DH>::SMEM, st>>>(tq, tkv, p);
  return cudaGetLastError();
}

template <int DH, int MODE>
cudaError_t launch_fwd(const CUtensorMap& tm, const FwdParams& p, dim3 grid, cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(attn_fwd_tc_kernel<DH, MODE>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         FwdLayout<DH>::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  attn_fwd_tc_kernel<DH, MODE><<<grid, NUM_THREADS, FwdLayout<DH>::SMEM, st>>>(tm, p);
  return cudaGetLastError();
}

}  // namespace

int attn_fwd_tc_rows() { return BQ; }

cudaError_t launch_attn_fwd_tc(const AttnLaunch& L, int mode) {
  auto fn = encode_fn();
  if (fn == nullptr) return cudaErrorNotSupported;
  const int64_t N = (int64_t)L.B * L.T;
  CUtensorMap tm;
  cuuint64_t dims[2] = {(cuuint64_t)L.ldq, (cuuint64_t)N};
  cuuint64_t strides[1] = {(cuuint64_t)L.ldq * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)BQ};
  cuuint32_t estr[2] = {1, 1};
  if (fn(&tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(L.qkv), dims, strides, box,
         estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  FwdParams p{};
  p.T = L.T;
  p.B = L.B;
  p.Hq = L.Hq;
  p.Hkv = L.Hkv;
  p.D = L.D;
  p.nqb = (L.T + BQ - 1) / BQ;
  p.nP = L.nP;
  p.lse_pitch = L.lse_pitch;
  p.sl2 = L.scale * kLog2e;
  p.part = L.part;
  p.a_ref = L.a_ref;
  p.a_out = L.a_out;
  p.lse = L.lse;
  p.d_o = static_cast<half_t*>(L.d_o);
  p.dvec = L.dvec;
  p.status = L.status;
  if ((L.Hq / L.Hkv) % 2 == 0) {  // head pairs of one KV group share every K/V tile
    CUtensorMap tkv;
    cuuint32_t box64[2] = {64, (cuuint32_t)PBK};
    if (fn(&tkv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(L.qkv), dims, strides, box64,
           estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
    dim3 pgrid((unsigned)(L.Hq / 2), (unsigned)(L.B * L.C), (unsigned)p.nqb);
#define JAB_FWD2(DH_, M_) return launch_fwd_pair<DH_, M_>(tm, tkv, p, pgrid, L.stream)
    if (L.dh == 128) {
      if (mode == 0) JAB_FWD2(128, 0);
      if (mode == 1) JAB_FWD2(128, 1);
      JAB_FWD2(128, 2);
    }
    if (mode == 0) JAB_FWD2(64, 0);
    if (mode == 1) JAB_FWD2(64, 1);
    JAB_FWD2(64, 2);
#undef JAB_FWD2
  }
  dim3 grid((unsigned)L.Hq, (unsigned)(L.B * L.C), (unsigned)p.nqb);
#define JAB_FWD(DH_, M_) return launch_fwd<DH_, M_>(tm, p, grid, L.stream)
  if (L.dh == 128) {
    if (mode == 0) JAB_FWD(128, 0);
    if (mode == 1) JAB_FWD(128, 1);
    JAB_FWD(128, 2);
  }
  if (mode == 0) JAB_FWD(64, 0);
  if (mode == 1) JAB_FWD(64, 1);
  JAB_FWD(64, 2);
#undef JAB_FWD
}

}  // namespace jab
