// Tensor-core (tcgen05) forward-mode product of causal GQA attention, sm_103a: ||J_A v||^2 for the
// Hutchinson estimate of Tr(H) (Section 2.4, Eq. 5). At the float weights w* the Hessian of the MSE
// term is H = 2 J_A^T J_A / n, so a probe v gives v^T H v = 2 ||J_A v||^2 / n, and only the
// forward-mode derivative of the block output along v is needed, not a second backward pass.
//
// With the primal projections Q, K, V, the tangent projections dQ, dK, dV (the same projection and
// RoPE applied to the probe), S = scale Q K^T, P = softmax(S) and O = P V:
//     dS = scale (dQ K^T + Q dK^T)               (visible keys)
//     dO = (P o dS) V + P dV - rowsum(P o dS) O
// The teacher pass already has the row log-sum-exp and O (= A_ref), so P = exp(S - lse) is exact
// tile by tile and one pass over the keys suffices (no online rescaling).
//
// One CTA = 128 query rows of one (sequence, query head); keys in blocks of 128. Tensor memory:
//   S at 0 (128 columns), T = dQ K^T + Q dK^T at 128 (128), Z = (P o dS) V + P dV at 256 (d_h),
//   Q and dQ after it (d_h / 2 each), copied in once by tcgen05.cp.
// Per key block: S = Q K^T and T (TS-form UMMAs, A from TMEM); the elementwise warps form P and
// U = P o dS, accumulate r = rowsum(U), and write P and U back as packed fp16 over the first 64
// columns of S and T, where the TS-form Z += U V and Z += P dV read them; the next block's S and T
// are issued once those have completed.
//   warp 0      TMA: Q and dQ once (into the V/dV slot), K/dK ring (2 stages), V/dV slot
//   warp 1      TMEM owner, tcgen05.cp, UMMA issuer (one thread)
//   warps 2..9  elementwise (16x256b TMEM shape, two rows per thread), then the epilogue
//               dO = Z - r O with O read from A_ref, and its squared norm
// Output: one fp64 partial per tile, summed in fixed order afterwards.
#include <cudaTypedefs.h>

#include <algorithm>

#include "kernels.h"
#include "tc.cuh"

namespace jab {
namespace {

constexpr int BQ = 128, BK = 128;
constexpr int NUM_THREADS = 320;  // warp 0 TMA, warp 1 UMMA, warps 2..9 elementwise
constexpr int EW_WARPS = 8;
constexpr float kLog2e = 1.4426950408889634f;

template <int DH>
struct JvpLayout {
  static constexpr int TILE = 128 * DH * 2;  // 128 rows of fp16
  static constexpr int CHUNK = 128 * 128;    // 64 columns of a 128-row tile (128-byte swizzle)
  static constexpr int VD_OFF = 0;           // V then dV of the current block (first Q then dQ)
  static constexpr int KD_OFF = 2 * TILE;    // stage st: K at KD_OFF + 2 st TILE, dK after it
  static constexpr int STAGES = 2;
  static constexpr int BAR_OFF = KD_OFF + STAGES * 2 * TILE;
  static constexpr int USED = BAR_OFF + 256 + 1024;
  static constexpr int SMEM = USED > 118 * 1024 ? USED : 118 * 1024;
  static constexpr uint32_t S_COL = 0, T_COL = 128, Z_COL = 256, Q_COL = 256 + DH,
                            DQ_COL = 256 + DH + DH / 2;
  static_assert(DQ_COL + DH / 2 <= 512, "TMEM budget");
  static_assert(USED <= 227 * 1024, "shared memory budget");
};

struct JvpBars {
  uint64_t q_full, stg_free, kd_full[2], kd_empty[2], vd_full, vd_empty, s_full, pu_full, z_done;
  uint64_t o_full, drain;
  uint32_t tmem_base;
  int abort;
  double red[EW_WARPS];
};

struct JvpParams {
  int T, B, Hq, Hkv, D, nqb, nP, lse_pitch;
  float scale, sl2;     // softmax scale; scale * log2(e)
  const float* lse;     // [B, Hq, lse_pitch] natural log (teacher)
  const float* a_ref;   // [B*T, Hq*DH] fp32: O of the teacher
  double* part;         // [B, Hq, nP]
  int* status;
};

__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = tc::globaltimer();
  while (!tc::mbar_test(bar, parity))
    if (tc::globaltimer() - t0 > tc::kWaitLimitNs) break;
}

template <int DH>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    attn_jvp_tc_kernel(const __grid_constant__ CUtensorMap tm_p,
                       const __grid_constant__ CUtensorMap tm_t, const JvpParams p) {
  using L = JvpLayout<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  JvpBars* bars = reinterpret_cast<JvpBars*>(smem + L::BAR_OFF);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &bars->abort;

  // CTA order: grouped by (sequence, KV group), so that the CTAs which stream the K blocks
  // of one KV head run close together (read from HBM about once); inside a group query blocks from
  // the last (most keys) to the first, the query heads of the group next to each other.
  const int ratio = p.Hq / p.Hkv;
  const int per_group = ratio * p.nqb;
  const int grp = (int)blockIdx.x / per_group, rem = (int)blockIdx.x - grp * per_group;
  const int qb = p.nqb - 1 - rem / ratio;
  const int g = grp % p.Hkv;
  const int h = g * ratio + rem % ratio;
  const int b = grp / p.Hkv;
  const int q0 = qb * BQ;
  const int nkb = min(qb + 1, (p.T + BK - 1) / BK);
  const int row0 = b * p.T;

  if (threadIdx.x == 0) {
    tc::mbar_init(&bars->q_full, 1);
    tc::mbar_init(&bars->stg_free, 1);
    for (int i = 0; i < L::STAGES; ++i) {
      tc::mbar_init(&bars->kd_full[i], 1);
      tc::mbar_init(&bars->kd_empty[i], 1);
    }
    tc::mbar_init(&bars->vd_full, 1);
    tc::mbar_init(&bars->vd_empty, 1);
    tc::mbar_init(&bars->s_full, 1);
    tc::mbar_init(&bars->pu_full, EW_WARPS);
    tc::mbar_init(&bars->z_done, 1);
    tc::mbar_init(&bars->o_full, 1);
    tc::mbar_init(&bars->drain, 1);
    bars->abort = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&tm_p);
    tc::prefetch_tmap(&tm_t);
  }
  if (warp == 1) {
    tc::tmem_alloc(&bars->tmem_base, 512);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = bars->tmem_base;

  if (warp == 0) {
    if (lane == 0) {  // ---------------------------------------------------------------- TMA
      const int qcol = h * DH, kcol = (p.Hq + g) * DH, vcol = (p.Hq + p.Hkv + g) * DH;
      uint32_t kd_issued = 0, kd_par = 0;
      bool vd_issued = false, ok = true;
      uint32_t vd_par = 0;
      tc::mbar_expect_tx(&bars->q_full, 2 * L::TILE);
      for (int ch = 0; ch < DH / 64; ++ch) {
        tc::tma_load_2d(smem + L::VD_OFF + ch * L::CHUNK, &tm_p, &bars->q_full, qcol + ch * 64,
                        row0 + q0);
        tc::tma_load_2d(smem + L::VD_OFF + L::TILE + ch * L::CHUNK, &tm_t, &bars->q_full,
                        qcol + ch * 64, row0 + q0);
      }
      for (int j = 0; ok && j < nkb; ++j) {
        const int st = j & 1;
        const uint32_t ph = (uint32_t)(j >> 1) & 1u;
        if (!tc::mbar_wait(&bars->kd_empty[st], ph ^ 1, abort, p.status)) break;
        uint8_t* kd = smem + L::KD_OFF + st * 2 * L::TILE;
        tc::mbar_expect_tx(&bars->kd_full[st], 2 * L::TILE);
        for (int ch = 0; ch < DH / 64; ++ch) {
          tc::tma_load_2d(kd + ch * L::CHUNK, &tm_p, &bars->kd_full[st], kcol + ch * 64,
                          row0 + j * BK);
          tc::tma_load_2d(kd + L::TILE + ch * L::CHUNK, &tm_t, &bars->kd_full[st], kcol + ch * 64,
                          row0 + j * BK);
        }
        kd_issued |= 1u << st;
        kd_par = (kd_par & ~(1u << st)) | (ph << st);
        // the single V/dV slot: free once Q and dQ are in TMEM (block 0), else once Z_{j-1} is done
        if (!(j == 0 ? tc::mbar_wait(&bars->stg_free, 0, abort, p.status)
                     : tc::mbar_wait(&bars->z_done, (uint32_t)(j - 1) & 1u, abort, p.status))) {
          ok = false;
          break;
        }
        tc::mbar_expect_tx(&bars->vd_full, 2 * L::TILE);
        for (int ch = 0; ch < DH / 64; ++ch) {
          tc::tma_load_2d(smem + L::VD_OFF + ch * L::CHUNK, &tm_p, &bars->vd_full,
                          vcol + ch * 64, row0 + j * BK);
          tc::tma_load_2d(smem + L::VD_OFF + L::TILE + ch * L::CHUNK, &tm_t, &bars->vd_full,
                          vcol + ch * 64, row0 + j * BK);
        }
        vd_issued = true;
        vd_par = (uint32_t)j & 1u;
      }
      if (*abort) {
        drain_wait(&bars->q_full, 0);
        for (int st = 0; st < L::STAGES; ++st)
          if (kd_issued & (1u << st)) drain_wait(&bars->kd_full[st], (kd_par >> st) & 1);
        if (vd_issued) drain_wait(&bars->vd_full, vd_par);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {  // ---------------------------------------------------------------- UMMA
      constexpr uint32_t ID_S = tc::idesc_f16(false, BQ, BK);
      constexpr uint32_t ID_Z = tc::idesc_f16(false, BQ, DH) | (1u << 16);  // B = V / dV, MN-major
      bool ok = tc::mbar_wait(&bars->q_full, 0, abort, p.status);
      if (ok) {
        tc::fence_after_sync();
        const uint32_t qs = tc::smem_u32(smem + L::VD_OFF);
        const uint32_t dqs = tc::smem_u32(smem + L::VD_OFF + L::TILE);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint32_t off = (kk >> 2) * L::CHUNK + (kk & 3) * 32;
          tc::tmem_cp_128x256b(tmem + L::Q_COL + kk * 8, tc::sdesc_kmajor_sw128(qs + off));
          tc::tmem_cp_128x256b(tmem + L::DQ_COL + kk * 8, tc::sdesc_kmajor_sw128(dqs + off));
        }
        tc::umma_commit(&bars->stg_free);  // the slot may take V / dV of block 0
      }
      const uint64_t vd = tc::sdesc_mnmajor_sw128(tc::smem_u32(smem + L::VD_OFF), L::CHUNK, 1024);
      const uint64_t dvd =
          tc::sdesc_mnmajor_sw128(tc::smem_u32(smem + L::VD_OFF + L::TILE), L::CHUNK, 1024);
      for (int j = 0; ok && j < nkb; ++j) {
        const int st = j & 1;
        // S_j and T_j once K_j, dK_j have landed and Z_{j-1} has read P_{j-1}, U_{j-1} out of the
        // S and T columns
        if (!tc::mbar_wait(&bars->kd_full[st], (j >> 1) & 1, abort, p.status) ||
            (j > 0 && !tc::mbar_wait(&bars->z_done, (j - 1) & 1, abort, p.status))) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        const uint64_t kd = tc::sdesc_kmajor_sw128(tc::smem_u32(smem + L::KD_OFF + st * 2 * L::TILE));
        const uint64_t dkd =
            tc::sdesc_kmajor_sw128(tc::smem_u32(smem + L::KD_OFF + st * 2 * L::TILE + L::TILE));
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint32_t off = (kk >> 2) * L::CHUNK + (kk & 3) * 32;
          tc::umma_f16_ts(tmem + L::S_COL, tmem + L::Q_COL + kk * 8, tc::sdesc_advance(kd, off),
                          ID_S, kk > 0 ? 1u : 0u);
          tc::umma_f16_ts(tmem + L::T_COL, tmem + L::DQ_COL + kk * 8, tc::sdesc_advance(kd, off),
                          ID_S, kk > 0 ? 1u : 0u);
        }
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint32_t off = (kk >> 2) * L::CHUNK + (kk & 3) * 32;
          tc::umma_f16_ts(tmem + L::T_COL, tmem + L::Q_COL + kk * 8, tc::sdesc_advance(dkd, off),
                          ID_S, 1u);
        }
        tc::umma_commit(&bars->s_full);
        tc::umma_commit(&bars->kd_empty[st]);
        // Z += U_j V_j + P_j dV_j once the elementwise warps have written P_j, U_j and V_j, dV_j
        // have landed
        if (!tc::mbar_wait(&bars->pu_full, j & 1, abort, p.status) ||
            !tc::mbar_wait(&bars->vd_full, j & 1, abort, p.status)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
#pragma unroll
        for (int k = 0; k < BK / 16; ++k)
          tc::umma_f16_ts(tmem + L::Z_COL, tmem + L::T_COL + k * 8,
                          tc::sdesc_advance(vd, k * 16 * 128), ID_Z, (j > 0 || k > 0) ? 1u : 0u);
#pragma unroll
        for (int k = 0; k < BK / 16; ++k)
          tc::umma_f16_ts(tmem + L::Z_COL, tmem + L::S_COL + k * 8,
                          tc::sdesc_advance(dvd, k * 16 * 128), ID_Z, 1u);
        tc::umma_commit(&bars->z_done);
        if (j == nkb - 1) tc::umma_commit(&bars->o_full);
      }
      tc::umma_commit(&bars->drain);
      drain_wait(&bars->drain, 0);
    }
  } else {  // -------------------------------------------------------------------- elementwise
    const int quarter = warp & 3;
    const int half = (warp - 2) >> 2;
    const int cq = lane & 3;
    const int rA = quarter * 32 + half * 16 + (lane >> 2), rB = rA + 8;
    const int tA = q0 + rA, tB = q0 + rB;
    const uint32_t lane16 = (uint32_t)(quarter * 32 + half * 16) << 16;
    const int64_t lbase = ((int64_t)b * p.Hq + h) * p.lse_pitch;
    // rows past T: P = 0 (lse = +inf)
    const float lA = tA < p.T ? p.lse[lbase + tA] * kLog2e : INFINITY;
    const float lB = tB < p.T ? p.lse[lbase + tB] * kLog2e : INFINITY;
    const float2 sl2 = make_float2(p.sl2, p.sl2), sc = make_float2(p.scale, p.scale);
    const float2 nlA = make_float2(tc::neg_bits(lA), tc::neg_bits(lA));
    const float2 nlB = make_float2(tc::neg_bits(lB), tc::neg_bits(lB));
    float rsA = 0.f, rsB = 0.f;  // this thread's share of rowsum(P o dS)
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      if (!tc::mbar_wait(&bars->s_full, j & 1, abort, p.status)) {
        ok = false;
        break;
      }
      tc::fence_after_sync();
      // x[hh][4n + e]: e < 2 row A, key 128 j + 64 hh + 8n + 2 cq + e; e = 2, 3 row B
      float xs[2][32], xt[2][32];
      {
        uint32_t r0[32], r1[32], r2[32], r3[32];
        __syncwarp();
        tc::tmem_ld_16x256b_x8(tmem + lane16 + L::S_COL, r0);
        tc::tmem_ld_16x256b_x8(tmem + lane16 + L::S_COL + 64, r1);
        tc::tmem_ld_16x256b_x8(tmem + lane16 + L::T_COL, r2);
        tc::tmem_ld_16x256b_x8(tmem + lane16 + L::T_COL + 64, r3);
        tc::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          xs[0][i] = __uint_as_float(r0[i]);
          xs[1][i] = __uint_as_float(r1[i]);
          xt[0][i] = __uint_as_float(r2[i]);
          xt[1][i] = __uint_as_float(r3[i]);
        }
      }
      const int k0 = j * BK + 2 * cq;
      const bool masked = j * BK + BK - 1 > q0 || j * BK + BK > p.T;  // diagonal or ragged block
      float2 uA = make_float2(0.f, 0.f), uB = uA;
      uint32_t inf_bits = 0;
      uint32_t pw[32], uw[32];  // packed P and U: [2m] row A, [2m + 1] row B, packed column 4m + cq
#pragma unroll
      for (int hh = 0; hh < 2; ++hh)
#pragma unroll
        for (int n = 0; n < 8; ++n) {
          const float2 ea = tc::fma2(make_float2(xs[hh][4 * n], xs[hh][4 * n + 1]), sl2, nlA);
          const float2 eb = tc::fma2(make_float2(xs[hh][4 * n + 2], xs[hh][4 * n + 3]), sl2, nlB);
          float2 pa = make_float2(tc::fast_exp2(ea.x), tc::fast_exp2(ea.y));
          float2 pb = make_float2(tc::fast_exp2(eb.x), tc::fast_exp2(eb.y));
          if (masked) {
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int key = k0 + 64 * hh + 8 * n + e;
              if (key > tA || key >= p.T) (e ? pa.y : pa.x) = 0.f;
              if (key > tB || key >= p.T) (e ? pb.y : pb.x) = 0.f;
            }
          }
          const float2 ua = tc::mul2(pa, tc::mul2(make_float2(xt[hh][4 * n], xt[hh][4 * n + 1]), sc));
          const float2 ub =
              tc::mul2(pb, tc::mul2(make_float2(xt[hh][4 * n + 2], xt[hh][4 * n + 3]), sc));
          uA = tc::add2(uA, ua);
          uB = tc::add2(uB, ub);
          const int m = 8 * hh + n;
          pw[2 * m] = tc::pack_half2(pa.x, pa.y);
          pw[2 * m + 1] = tc::pack_half2(pb.x, pb.y);
          uw[2 * m] = tc::pack_half2(ua.x, ua.y);
          uw[2 * m + 1] = tc::pack_half2(ub.x, ub.y);
          inf_bits |= half2_exp_all_ones(uw[2 * m]) | half2_exp_all_ones(uw[2 * m + 1]);
        }
      rsA += uA.x + uA.y;
      rsB += uB.x + uB.y;
      if (inf_bits) report(p.status, JAB_ERR_RANGE);  // U out of the fp16 range (or NaN)
      __syncwarp();
      tc::tmem_st_16x128b_x16(tmem + lane16 + L::S_COL, pw);
      tc::tmem_st_16x128b_x16(tmem + lane16 + L::T_COL, uw);
      tc::tmem_st_wait();
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->pu_full);
    }
    // ---------------------------------------------------------------- epilogue: dO = Z - r O
    double acc = 0.0;
    rsA += __shfl_xor_sync(0xffffffffu, rsA, 1);
    rsB += __shfl_xor_sync(0xffffffffu, rsB, 1);
    rsA += __shfl_xor_sync(0xffffffffu, rsA, 2);
    rsB += __shfl_xor_sync(0xffffffffu, rsB, 2);
    if (ok && tc::mbar_wait(&bars->o_full, 0, abort, p.status)) {
      tc::fence_after_sync();
      const float* oA = p.a_ref + ((int64_t)row0 + (tA < p.T ? tA : 0)) * (int64_t)(p.Hq * DH) + h * DH;
      const float* oB = p.a_ref + ((int64_t)row0 + (tB < p.T ? tB : 0)) * (int64_t)(p.Hq * DH) + h * DH;
      float2 qA = make_float2(0.f, 0.f), qB = qA;
      const float2 nrA = make_float2(tc::neg_bits(rsA), tc::neg_bits(rsA));
      const float2 nrB = make_float2(tc::neg_bits(rsB), tc::neg_bits(rsB));
#pragma unroll 1
      for (int hh = 0; hh < DH / 64; ++hh) {
        uint32_t z[32];
        __syncwarp();
        tc::tmem_ld_16x256b_x8(tmem + lane16 + L::Z_COL + 64 * hh, z);
        tc::tmem_ld_wait();
#pragma unroll
        for (int n = 0; n < 8; ++n) {
          const int col = 64 * hh + 8 * n + 2 * cq;
          const float2 a = __ldg(reinterpret_cast<const float2*>(oA + col));
          const float2 bb = __ldg(reinterpret_cast<const float2*>(oB + col));
          const float2 dA = tc::fma2(nrA, a, make_float2(__uint_as_float(z[4 * n]), __uint_as_float(z[4 * n + 1])));
          const float2 dB = tc::fma2(nrB, bb, make_float2(__uint_as_float(z[4 * n + 2]), __uint_as_float(z[4 * n + 3])));
          qA = tc::fma2(dA, dA, qA);
          qB = tc::fma2(dB, dB, qB);
        }
      }
      if (tA < p.T) acc += (double)qA.x + (double)qA.y;
      if (tB < p.T) acc += (double)qB.x + (double)qB.y;
    }
    acc = warp_sum(acc);
    if (lane == 0) bars->red[warp - 2] = acc;
    tc::named_bar_sync(1, EW_WARPS * 32);  // every elementwise warp reaches this exactly once
    if (warp == 2 && lane == 0 && ok) {
      double tot = 0.0;
      for (int w = 0; w < EW_WARPS; ++w) tot += bars->red[w];
      const int64_t pi = ((int64_t)b * p.Hq + h) * p.nP + qb;
      if (in_bounds(pi, (int64_t)p.B * p.Hq * p.nP, p.status)) p.part[pi] = tot;
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

// fp16 [rows, cols] row-major, 64 x 128 boxes with the 128-byte swizzle.
bool tmap_fp16(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, 128};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int DH>
cudaError_t launch_jvp(const CUtensorMap& tp, const CUtensorMap& tt, const JvpParams& p,
                       cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(attn_jvp_tc_kernel<DH>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         JvpLayout<DH>::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int64_t n = (int64_t)p.Hq * p.B * p.nqb;
  if (n >= (1ll << 31)) return cudaErrorInvalidValue;
  const dim3 grid((unsigned)n);
  attn_jvp_tc_kernel<DH><<<grid, NUM_THREADS, JvpLayout<DH>::SMEM, st>>>(tp, tt, p);
  return cudaGetLastError();
}

}  // namespace

int attn_jvp_tc_rows() { return BQ; }

cudaError_t launch_attn_jvp_tc(const void* qkv, const void* tqkv, const float* lse, int lse_pitch,
                               const float* a_ref, int B, int T, int Hq, int Hkv, int dh,
                               float scale, double* part, int nP, int* status, cudaStream_t st) {
  const int D = (Hq + 2 * Hkv) * dh;
  const int64_t N = (int64_t)B * T;
  CUtensorMap tp, tt;
  if (!tmap_fp16(&tp, qkv, (uint64_t)D, (uint64_t)N) || !tmap_fp16(&tt, tqkv, (uint64_t)D, (uint64_t)N))
    return cudaErrorInvalidValue;
  JvpParams p{};
  p.T = T;
  p.B = B;
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.D = D;
  p.nqb = (T + BQ - 1) / BQ;
  p.nP = nP;
  p.lse_pitch = lse_pitch;
  p.scale = scale;
  p.sl2 = scale * kLog2e;
  p.lse = lse;
  p.a_ref = a_ref;
  p.part = part;
  p.status = status;
  if (p.nqb > nP) return cudaErrorInvalidValue;
  return dh == 128 ? launch_jvp<128>(tp, tt, p, st) : launch_jvp<64>(tp, tt, p, st);
}

}  // namespace jab
