// Tensor-core (tcgen05) backward of causal GQA attention for the STE gradient of L_JAB, sm_103a.
//
// Inputs from the forward (mode 2): dO = O - A_ref (fp16; the factor 2/n is applied to the scale
// gradient at the end), the row log-sum-exp in log2 units and D = rowsum(dO * O). P is recomputed
// tile by tile:
//   P = exp(S - lse),  dP = dO V^T,  dS = P * (dP - D)
//   dV = P^T dO,  dK = scale * dS^T Q,  dQ = scale * dS K        (summed over the GQA group for K, V)
// Two kernels, no atomics:
//   dkdv  one CTA per (128-key block, KV head, sequence); loops over the query heads of the group and
//         over 128-query blocks: S^T = K Q^T, dP^T = V dO^T into TMEM, P^T and dS^T (fp16) written
//         back over them by 16 elementwise warps (16 key rows x 64 queries each), dV += P^T dO and
//         dK += dS^T Q (A operands in TMEM) accumulated in TMEM. Each dS^T tile is also staged in
//         shared memory and stored to HBM by TMA (a store warp).
//   dq    persistent, (128 query rows, query head, sequence) tiles: dQ = scale * sum_kb dS K from the
//         stored dS^T tiles, a plain tensor-core product per key block (no recomputation of S, P or
//         dP: two of the three products and all elementwise work of a recomputing dq are saved, for
//         one HBM write and one read of the fp16 dS tiles).
// Both epilogues apply the transpose of RoPE to dQ and dK and write dQKV^T (bf16, [D, ldt]), the
// K-major operand of the weight-gradient GEMM.
#include <cudaTypedefs.h>

#include "kernels.h"
#include "tc.cuh"

namespace jab {
namespace {

constexpr int EW_WARPS = 8;       // dq: epilogue warps
constexpr int DKDV_EW = 16;       // dK/dV: elementwise warps, 16 key rows x 64 queries each
// warp 0 TMA, 1 UMMA (S^T, dP^T), 2..17 elementwise, 18 stores, 19 UMMA (dV, dK)
constexpr int DKDV_THREADS = (2 + DKDV_EW + 2) * 32;
constexpr int DKDV_GRAD_WARP = 3 + DKDV_EW;
constexpr int kSuperGroup = 8;  // (KV head, sequence) pairs whose dK/dV CTAs are interleaved
constexpr float kLog2e = 1.4426950408889634f;
constexpr double kLn2 = 0.6931471805599453;

struct BwdParams {
  int T, B, Hq, Hkv, lse_pitch;
  int qcol0, kcol0, vcol0;  // column offsets of Q, K, V heads in the QKV matrix
  int64_t ldt;
  int npairs;  // (query block, key block) pairs of one (sequence, head): nq (nq + 1) / 2
  float scale, sl2;
  // KL term of Eq. 3 (dK/dV kernel with KL): dS = a_mse P (dP - D) + b_kl (P - P_teacher), dV times
  // a_mse; the caller's coefficient of the whole gradient is divided by a_mse
  float a_mse, b_kl;
  const float* lse;
  const float* dvec;
  const float* cos_t;
  const float* sin_t;
  int use_rope;
  bf16_t* dqkvt;
  int* status;
};

__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = tc::globaltimer();
  while (!tc::mbar_test(bar, parity))
    if (tc::globaltimer() - t0 > tc::kWaitLimitNs) break;
}

// Stages gradient rows of a TMEM accumulator (DH columns), times `mul`, optionally through the
// transpose of RoPE, into tile[dim][row] (bf16, 128 rows per dim). The calling warp handles the 16
// TMEM lanes addressed by `taddr` with the 16x256b shape: thread t holds rows row_a = first + t / 4
// and row_a + 8 and, in each 8-column group, the column pair 2 (t % 4), so the four threads of a row
// read 32 contiguous bytes of a cos / sin table row (pos_a, pos_b: table rows of row_a, row_a + 8).
template <int DH>
__device__ __forceinline__ void stage_grad_16(uint32_t taddr, float mul, bool rope, int pos_a,
                                              int pos_b, const float* cos_t, const float* sin_t,
                                              bf16_t* tile, int row_a) {
  constexpr int HALF = DH / 2;
  const int cq = threadIdx.x & 3;
#pragma unroll 1
  for (int c = 0; c < HALF / 32; ++c) {
    uint32_t r1[16], r2[16];
    __syncwarp();
    tc::tmem_ld_16x256b_x4(taddr + c * 32, r1);
    tc::tmem_ld_16x256b_x4(taddr + HALF + c * 32, r2);
    tc::tmem_ld_wait();
#pragma unroll
    for (int n = 0; n < 4; ++n) {
      const int j0 = c * 32 + 8 * n + 2 * cq;  // columns j0, j0 + 1 of the first half
      float2 ca = make_float2(1.f, 1.f), sa = make_float2(0.f, 0.f);
      float2 cb = make_float2(1.f, 1.f), sb = make_float2(0.f, 0.f);
      if (rope) {
        ca = __ldg(reinterpret_cast<const float2*>(cos_t + (int64_t)pos_a * HALF + j0));
        sa = __ldg(reinterpret_cast<const float2*>(sin_t + (int64_t)pos_a * HALF + j0));
        cb = __ldg(reinterpret_cast<const float2*>(cos_t + (int64_t)pos_b * HALF + j0));
        sb = __ldg(reinterpret_cast<const float2*>(sin_t + (int64_t)pos_b * HALF + j0));
      }
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const float csa = e ? ca.y : ca.x, sna = e ? sa.y : sa.x;
        const float csb = e ? cb.y : cb.x, snb = e ? sb.y : sb.x;
        float a1 = __uint_as_float(r1[4 * n + e]) * mul, a2 = __uint_as_float(r2[4 * n + e]) * mul;
        float b1 = __uint_as_float(r1[4 * n + 2 + e]) * mul;
        float b2 = __uint_as_float(r2[4 * n + 2 + e]) * mul;
        if (rope) {
          const float x1 = a1, x2 = a2, y1 = b1, y2 = b2;
          a1 = x1 * csa + x2 * sna;
          a2 = x2 * csa - x1 * sna;
          b1 = y1 * csb + y2 * snb;
          b2 = y2 * csb - y1 * snb;
        }
        tile[(j0 + e) * 128 + row_a] = __float2bfloat16_rn(a1);
        tile[(HALF + j0 + e) * 128 + row_a] = __float2bfloat16_rn(a2);
        tile[(j0 + e) * 128 + row_a + 8] = __float2bfloat16_rn(b1);
        tile[(HALF + j0 + e) * 128 + row_a + 8] = __float2bfloat16_rn(b2);
      }
    }
  }
}

// Cooperative store of tile[DH][128] to dst[d * ldt + n0 + r] for r < nvalid: 16-byte vectors when
// the token offset is 8-aligned (consecutive threads cover consecutive 16-byte chunks of a dim
// row), element-wise otherwise.
template <int DH>
// (checked build: every store is tested against [base, base + extent) of dQKV^T)
__device__ __forceinline__ void store_tile(const bf16_t* tile, bf16_t* dst, int64_t ldt, int64_t n0,
                                           int nvalid, int tid, int nthreads, const bf16_t* base,
                                           int64_t extent, int* status) {
  if ((n0 & 7) == 0) {
    for (int idx = tid; idx < DH * 16; idx += nthreads) {
      const int d = idx >> 4, r0 = (idx & 15) * 8;
      bf16_t* o = dst + (int64_t)d * ldt + n0 + r0;
      if (!in_bounds((o - base) + min(8, nvalid - r0) - 1, extent, status)) continue;
      if (r0 + 8 <= nvalid)
        *reinterpret_cast<uint4*>(o) = *reinterpret_cast<const uint4*>(tile + d * 128 + r0);
      else
        for (int r = r0; r < nvalid; ++r) o[r - r0] = tile[d * 128 + r];
    }
  } else {
    for (int idx = tid; idx < DH * 128; idx += nthreads) {
      const int d = idx >> 7, r = idx & 127;
      if (r < nvalid && in_bounds((dst - base) + (int64_t)d * ldt + n0 + r, extent, status))
        dst[(int64_t)d * ldt + n0 + r] = tile[d * 128 + r];
    }
  }
}

// ================================================================================ dK, dV
// One CTA per (128-key block, KV head, sequence); it loops over the query heads of the group and over
// 128-query blocks, so that every UMMA runs at N = 128 (an N = 64 UMMA costs the tensor pipe as much
// time as an N = 128 one). Tensor memory: S^T = K Q^T at column 0 and dP^T = V dO^T at 128 (SS form:
// K and V stay in shared memory for the whole tile), dV at 256, dK at 256 + DH. The elementwise warps
// write P^T and dS^T back as packed fp16 into S^T and dP^T, where the TS-form gradient UMMAs
// dV += P^T dO and dK += dS^T Q read them as their A operand: the 64 queries of half h (whose fp32
// scores are columns 64 h .. 64 h + 63, read by the warps of that half) go to packed columns
// 64 h .. 64 h + 31, so a warp writes only columns that it has itself read (warps of the two halves
// are not synchronised with each other). With no room for a second
// S^T / dP^T buffer, S^T(j+1) goes out once dV(j) has completed (it overwrites the P^T(j) columns)
// and dP^T(j+1) once dK(j) has; the elementwise warps compute P^T(j+1) while dK(j) and dP^T(j+1)
// run. The score products (S^T, dP^T) and the gradient products (dV, dK) are issued by two threads,
// so that neither waits behind the issue of the other; dK(j) enters the pipe only after S^T(j+1)
// has been issued, since the elementwise warps wait for S^T(j+1) and nothing waits for dK(j) sooner.

// TMEM column of the K-step k (queries 16 k .. 16 k + 15) of packed P^T or dS^T.
__device__ __forceinline__ uint32_t pk_col(int k) { return (uint32_t)((k >> 2) * 64 + (k & 3) * 8); }

template <int DH>
struct DkdvLayout {
  static constexpr int BK = 128, BQ = 128, STAGES = 2;
  static constexpr int PREFETCH = 2;  // blocks beyond the stage ring kept in flight to L2
  static constexpr int CHUNK = 128 * 128;  // 64 columns of a 128-row fp16 tile
  static constexpr int NCH = DH / 64;
  static constexpr int K_OFF = 0, V_OFF = NCH * CHUNK;
  static constexpr int ST_OFF = 2 * NCH * CHUNK;
  static constexpr int ST_Q = 0, ST_DO = NCH * CHUNK, ST_LSE = 2 * NCH * CHUNK,
                       ST_D = ST_LSE + BQ * 4, ST_BYTES = ST_D + BQ * 4;
  static constexpr int ST_STRIDE = (ST_BYTES + 1023) / 1024 * 1024;
  static constexpr int DSS_OFF = ST_OFF + STAGES * ST_STRIDE;  // dS^T staging: two 64-query halves
  static constexpr int BAR_OFF = DSS_OFF + 2 * CHUNK;
  // No slack for aligning the base: the kernel checks that it is 1024-byte aligned (it is, after the
  // per-CTA reserved shared memory) and returns with JAB_ERR_INTERNAL otherwise.
  static constexpr int USED = BAR_OFF + 256;
  static constexpr int SMEM = USED > 118 * 1024 ? USED : 118 * 1024;
  static constexpr uint32_t S_COL = 0, DP_COL = 128, DV_COL = 256, DK_COL = 256 + DH;
  static_assert(DK_COL + DH <= 512, "TMEM budget");
  static_assert(2 * DH * 128 * 2 <= STAGES * ST_STRIDE, "epilogue staging fits the stage ring");
  static_assert(USED <= 227 * 1024, "shared memory budget");
};

struct DkdvBars {
  uint64_t kv_full, ld_full[2], ld_empty[2], s_full, dp_full, p_full, ds_full, dv_done, dk_done;
  uint64_t o_full, drain, drain_g, dss_full, dss_free, s_issued, pt_full;
  uint32_t tmem_base;
  int abort;
};

// KL: the teacher's probabilities P^T of each (query block, key block) tile were stored in the dS^T
// tile buffer (attn_teacher_p_tc_kernel); the store warp loads the tile into the staging buffer
// before the block's dS, the elementwise warps add b_kl (P - P^T) to a_mse P (dP - D) and write
// dS^T over it, and the tile goes back to the same place.
template <int DH, bool KL>
__global__ void __launch_bounds__(DKDV_THREADS, 1)
    attn_bwd_dkdv_tc_kernel(const __grid_constant__ CUtensorMap tm_qkv,
                            const __grid_constant__ CUtensorMap tm_do,
                            const __grid_constant__ CUtensorMap tm_ds, const BwdParams p) {
  using L = DkdvLayout<DH>;
  constexpr int BK = L::BK, BQ = L::BQ, STAGES = L::STAGES;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if (tc::smem_u32(smem_raw) & 1023u) {  // the swizzled TMA tiles need a 1024-byte aligned base
    if (threadIdx.x == 0) report(p.status, JAB_ERR_INTERNAL);
    return;
  }
  uint8_t* smem = smem_raw;
  DkdvBars* bars = reinterpret_cast<DkdvBars*>(smem + L::BAR_OFF);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &bars->abort;

  const int r = p.Hq / p.Hkv;
  const int nq = (p.T + BQ - 1) / BQ;
  // CTA order: super-groups of kSuperGroup (KV head, sequence) pairs, key block slowest inside one,
  // so that the CTAs which stream the same Q and dO blocks run at the same time (their reads hit
  // L2) and the longest CTAs of a super-group start first.
  int kb, g, b;
  {
    const int pairs = p.Hkv * p.B;
    const int sg = blockIdx.x / (kSuperGroup * nq);
    const int sgs = min(kSuperGroup, pairs - sg * kSuperGroup);
    const int rem = blockIdx.x - sg * kSuperGroup * nq;
    kb = rem / sgs;
    const int pr = sg * kSuperGroup + rem % sgs;
    g = pr % p.Hkv;
    b = pr / p.Hkv;
  }
  const int per_head = nq - kb;  // query blocks kb .. nq - 1 see keys of block kb
  const int n_it = r * per_head;
  const int row0 = b * p.T;

  if (threadIdx.x == 0) {
    tc::mbar_init(&bars->kv_full, 1);
    for (int i = 0; i < STAGES; ++i) {
      tc::mbar_init(&bars->ld_full[i], 1);
      tc::mbar_init(&bars->ld_empty[i], 1);
    }
    tc::mbar_init(&bars->s_full, 1);
    tc::mbar_init(&bars->dp_full, 1);
    tc::mbar_init(&bars->p_full, DKDV_EW);
    tc::mbar_init(&bars->ds_full, DKDV_EW);
    tc::mbar_init(&bars->dv_done, 1);
    tc::mbar_init(&bars->dk_done, 1);
    tc::mbar_init(&bars->o_full, 1);
    tc::mbar_init(&bars->drain, 1);
    tc::mbar_init(&bars->drain_g, 1);
    tc::mbar_init(&bars->s_issued, 1);
    tc::mbar_init(&bars->dss_full, DKDV_EW);  // the block's dS^T is in the staging tile
    tc::mbar_init(&bars->dss_free, 1);         // the store warp's TMA stores have read it
    tc::mbar_init(&bars->pt_full, 1);          // KL: the block's P^T tile is in the staging tile
    bars->abort = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&tm_qkv);
    tc::prefetch_tmap(&tm_do);
    tc::prefetch_tmap(&tm_ds);
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
    if (lane == 0) {  // ------------------------------------------------------------- TMA
      uint32_t issued = 0, last_par = 0;
      tc::mbar_expect_tx(&bars->kv_full, 2 * BK * DH * 2);
      for (int ch = 0; ch < L::NCH; ++ch) {
        tc::tma_load_2d(smem + L::K_OFF + ch * L::CHUNK, &tm_qkv, &bars->kv_full,
                        p.kcol0 + g * DH + ch * 64, row0 + kb * BK);
        tc::tma_load_2d(smem + L::V_OFF + ch * L::CHUNK, &tm_qkv, &bars->kv_full,
                        p.vcol0 + g * DH + ch * 64, row0 + kb * BK);
      }
      // The stage ring holds two blocks; blocks further ahead are prefetched into L2 so that a
      // stage load, which can start only when dK of the block two back has completed, hits L2.
      auto prefetch = [&](int j) {
        const int hj = g * r + j / per_head, ij = kb + j % per_head;
        for (int ch = 0; ch < L::NCH; ++ch) {
          tc::tma_prefetch_2d(&tm_qkv, p.qcol0 + hj * DH + ch * 64, row0 + ij * BQ);
          tc::tma_prefetch_2d(&tm_do, hj * DH + ch * 64, row0 + ij * BQ);
        }
        const int64_t lrow = ((int64_t)b * p.Hq + hj) * p.lse_pitch + ij * BQ;
        tc::prefetch_l2(p.lse + lrow, BQ * 4);
        tc::prefetch_l2(p.dvec + lrow, BQ * 4);
        if constexpr (KL) {
          const int64_t tile = ((int64_t)b * p.Hq + hj) * p.npairs + (int64_t)ij * (ij + 1) / 2 + kb;
          tc::tma_prefetch_2d(&tm_ds, 0, (int32_t)(tile * BK));
          tc::tma_prefetch_2d(&tm_ds, 64, (int32_t)(tile * BK));
        }
      };
      for (int j = STAGES; j < STAGES + L::PREFETCH - 1 && j < n_it; ++j) prefetch(j);
      for (int it = 0; it < n_it; ++it) {
        const int st = it % STAGES;
        const uint32_t ph = (it / STAGES) & 1;
        const int h = g * r + it / per_head, i = kb + it % per_head;
        if (it + STAGES + L::PREFETCH - 1 < n_it) prefetch(it + STAGES + L::PREFETCH - 1);
        if (!tc::mbar_wait(&bars->ld_empty[st], ph ^ 1, abort, p.status)) break;
        uint8_t* sbase = smem + L::ST_OFF + st * L::ST_STRIDE;
        tc::mbar_expect_tx(&bars->ld_full[st], L::ST_BYTES);
        for (int ch = 0; ch < L::NCH; ++ch) {
          tc::tma_load_2d(sbase + L::ST_Q + ch * L::CHUNK, &tm_qkv, &bars->ld_full[st],
                          p.qcol0 + h * DH + ch * 64, row0 + i * BQ);
          tc::tma_load_2d(sbase + L::ST_DO + ch * L::CHUNK, &tm_do, &bars->ld_full[st],
                          h * DH + ch * 64, row0 + i * BQ);
        }
        const int64_t lrow = ((int64_t)b * p.Hq + h) * p.lse_pitch + i * BQ;
        // (checked build: a failed test leaves the stage incomplete; its consumers' bounded waits
        // then give up and the kernel returns with the status raised)
        if (in_bounds(lrow + BQ - 1, (int64_t)p.B * p.Hq * p.lse_pitch, p.status)) {
          tc::bulk_load(sbase + L::ST_LSE, p.lse + lrow, BQ * 4, &bars->ld_full[st]);
          tc::bulk_load(sbase + L::ST_D, p.dvec + lrow, BQ * 4, &bars->ld_full[st]);
        }
        issued |= 1u << st;
        last_par = (last_par & ~(1u << st)) | (ph << st);
      }
      if (*abort) {
        drain_wait(&bars->kv_full, 0);
        for (int st = 0; st < STAGES; ++st)
          if (issued & (1u << st)) drain_wait(&bars->ld_full[st], (last_par >> st) & 1);
      }
    }
  } else if (warp == 1 || warp == DKDV_GRAD_WARP) {
    if (lane == 0) {  // ---------------------- UMMA: S^T, dP^T (warp 1); dV, dK (DKDV_GRAD_WARP)
      // Two issuing threads, so that the score products of the next block are never held back
      // behind the issue of this block's gradient products, nor the other way round. Every
      // dependency between them goes through a barrier: S^T(j) overwrites P^T(j - 1), so it waits
      // for dV(j - 1); dP^T(j) overwrites dS^T(j - 1), so it waits for dK(j - 1).
      constexpr uint32_t ID_S = tc::idesc_f16(false, BK, BQ);
      constexpr uint32_t ID_G = tc::idesc_f16(false, BK, DH) | (1u << 16);  // B MN-major
      bool ok = tc::mbar_wait(&bars->kv_full, 0, abort, p.status);
      if (warp == 1) {
        const uint64_t ka = tc::sdesc_kmajor_sw128(tc::smem_u32(smem + L::K_OFF));
        const uint64_t va = tc::sdesc_kmajor_sw128(tc::smem_u32(smem + L::V_OFF));
        for (int j = 0; ok && j < n_it; ++j) {
          const int st = j % STAGES;
          // S^T(j) = K Q(j)^T: its Q has landed and dV(j - 1) has read P^T(j - 1).
          ok = tc::mbar_wait(&bars->ld_full[st], (j / STAGES) & 1, abort, p.status) &&
               (j == 0 || tc::mbar_wait(&bars->dv_done, (j - 1) & 1, abort, p.status));
          if (!ok) break;
          tc::fence_after_sync();
          const uint64_t bq = tc::sdesc_kmajor_sw128(
              tc::smem_u32(smem + L::ST_OFF + st * L::ST_STRIDE + L::ST_Q));
#pragma unroll
          for (int k = 0; k < DH / 16; ++k) {
            const uint32_t o = (k >> 2) * L::CHUNK + (k & 3) * 32;
            tc::umma_f16(tmem + L::S_COL, tc::sdesc_advance(ka, o), tc::sdesc_advance(bq, o), ID_S,
                         k > 0 ? 1u : 0u);
          }
          tc::umma_commit(&bars->s_full);
          tc::mbar_arrive(&bars->s_issued);  // dK(j - 1) may now queue behind S^T(j)
          // dP^T(j) = V dO(j)^T once dK(j - 1) has read dS^T(j - 1).
          ok = j == 0 || tc::mbar_wait(&bars->dk_done, (j - 1) & 1, abort, p.status);
          if (!ok) break;
          tc::fence_after_sync();
          const uint64_t bd = tc::sdesc_kmajor_sw128(
              tc::smem_u32(smem + L::ST_OFF + st * L::ST_STRIDE + L::ST_DO));
#pragma unroll
          for (int k = 0; k < DH / 16; ++k) {
            const uint32_t o = (k >> 2) * L::CHUNK + (k & 3) * 32;
            tc::umma_f16(tmem + L::DP_COL, tc::sdesc_advance(va, o), tc::sdesc_advance(bd, o), ID_S,
                         k > 0 ? 1u : 0u);
          }
          tc::umma_commit(&bars->dp_full);
        }
      } else {
        for (int j = 0; ok && j < n_it; ++j) {
          const int st = j % STAGES;
          // dV += P^T(j) dO(j) once the elementwise warps have written P^T(j).
          ok = tc::mbar_wait(&bars->p_full, j & 1, abort, p.status);
          if (!ok) break;
          tc::fence_after_sync();
          const uint64_t bd = tc::sdesc_mnmajor_sw128(
              tc::smem_u32(smem + L::ST_OFF + st * L::ST_STRIDE + L::ST_DO), L::CHUNK, 1024);
#pragma unroll
          for (int k = 0; k < BQ / 16; ++k)
            tc::umma_f16_ts(tmem + L::DV_COL, tmem + L::S_COL + pk_col(k), tc::sdesc_advance(bd, k * 16 * 128),
                            ID_G, (j > 0 || k > 0) ? 1u : 0u);
          tc::umma_commit(&bars->dv_done);
          // dK += dS^T(j) Q(j) once dS^T(j) is written.
          // dK(j) goes into the pipe behind S^T(j + 1), which the elementwise warps wait for
          ok = tc::mbar_wait(&bars->ds_full, j & 1, abort, p.status) &&
               (j + 1 == n_it || tc::mbar_wait(&bars->s_issued, (j + 1) & 1, abort, p.status));
          if (!ok) break;
          tc::fence_after_sync();
          const uint64_t bq = tc::sdesc_mnmajor_sw128(
              tc::smem_u32(smem + L::ST_OFF + st * L::ST_STRIDE + L::ST_Q), L::CHUNK, 1024);
#pragma unroll
          for (int k = 0; k < BQ / 16; ++k)
            tc::umma_f16_ts(tmem + L::DK_COL, tmem + L::DP_COL + pk_col(k), tc::sdesc_advance(bq, k * 16 * 128),
                            ID_G, (j > 0 || k > 0) ? 1u : 0u);
          tc::umma_commit(&bars->dk_done);
          // dV(j) and dK(j) are the stage's last readers (S^T(j) and dP^T(j) completed before the
          // elementwise warps released P^T(j) and dS^T(j))
          tc::umma_commit(&bars->ld_empty[st]);
          if (j == n_it - 1) tc::umma_commit(&bars->o_full);
        }
      }
      uint64_t* dr = warp == 1 ? &bars->drain : &bars->drain_g;
      tc::umma_commit(dr);
      drain_wait(dr, 0);
    }
  } else if (warp == 2 + DKDV_EW) {
    if (lane == 0) {  // ------------------------------------------ dS^T tiles to global memory
      // Tile (sequence b, head h, query block i, key block kb) is row block
      // (b Hq + h) npairs + i (i + 1) / 2 + kb of the dS^T buffer: 128 key rows of 128 queries.
      auto tile_of = [&](int it) {
        const int h = g * r + it / per_head, i = kb + it % per_head;
        return ((int64_t)b * p.Hq + h) * p.npairs + (int64_t)i * (i + 1) / 2 + kb;
      };
      int pt_issued = 0;  // KL: P^T tiles loaded into the staging tile so far
      auto load_pt = [&](int it) {  // KL: block it's P^T tile into the staging tile
        const int32_t y = (int32_t)(tile_of(it) * BK);
        tc::mbar_expect_tx(&bars->pt_full, 2 * L::CHUNK);
        tc::tma_load_2d(smem + L::DSS_OFF, &tm_ds, &bars->pt_full, 0, y);
        tc::tma_load_2d(smem + L::DSS_OFF + L::CHUNK, &tm_ds, &bars->pt_full, 64, y);
        ++pt_issued;
      };
      if constexpr (KL) load_pt(0);
      for (int it = 0; it < n_it; ++it) {
        if (!tc::mbar_wait(&bars->dss_full, it & 1, abort, p.status)) break;
        const int64_t tile = tile_of(it);
        tc::tma_store_2d(&tm_ds, smem + L::DSS_OFF, 0, (int32_t)(tile * BK));
        tc::tma_store_2d(&tm_ds, smem + L::DSS_OFF + L::CHUNK, 64, (int32_t)(tile * BK));
        tc::bulk_commit_group();
        tc::bulk_wait_group_read<0>();  // the staging tile may be rewritten
        if constexpr (KL) {
          if (it + 1 < n_it) load_pt(it + 1);
        } else {
          tc::mbar_arrive(&bars->dss_free);
        }
      }
      tc::bulk_wait_group<0>();
      // KL: a P^T load that nobody waited for (the loop gave up) lands before shared memory goes
      if (KL && pt_issued > 0) drain_wait(&bars->pt_full, (pt_issued - 1) & 1);
    }
  } else {  // ------------------------------------ elementwise: 16 key rows x 64 queries per warp
    // Warp w (2..17) may access TMEM lane quarter w % 4; the four warps of a quarter take its two
    // 16-row groups x the block's two 64-query halves. Nothing is reduced across queries here (the
    // row log-sum-exp and D come with the block), so a warp needs only its half.
    const int quarter = warp & 3;
    const int idx = (warp - 2) >> 2;
    const int half = idx & 1;   // 16-row group of the quarter
    const int chalf = idx >> 1; // 64-query half of the block
    const int cq = lane & 3;
    const int rA = quarter * 32 + half * 16 + (lane >> 2);  // key rows rA and rA + 8 of the block
    const int keyA = kb * BK + rA, keyB = keyA + 8;
    const uint32_t lane16 = (uint32_t)(quarter * 32 + half * 16) << 16;
    bool ok = true;
    for (int it = 0; it < n_it; ++it) {
      const int st = it % STAGES;
      const int i = kb + it % per_head;
      const float* lse_s =
          reinterpret_cast<const float*>(smem + L::ST_OFF + st * L::ST_STRIDE + L::ST_LSE) + 64 * chalf;
      const float* d_s =
          reinterpret_cast<const float*>(smem + L::ST_OFF + st * L::ST_STRIDE + L::ST_D) + 64 * chalf;
      if (!tc::mbar_wait(&bars->ld_full[st], (it / STAGES) & 1, abort, p.status) ||
          !tc::mbar_wait(&bars->s_full, it & 1, abort, p.status)) {
        ok = false;
        break;
      }
      tc::fence_after_sync();
      // x[4n + e] (e < 2): row A, query 64 chalf + 8n + 2 cq + e; e = 2, 3: row B
      float x[32];
      {
        uint32_t r0[32];
        __syncwarp();
        tc::tmem_ld_16x256b_x8(tmem + lane16 + L::S_COL + 64 * chalf, r0);
        tc::tmem_ld_wait();
#pragma unroll
        for (int c = 0; c < 32; ++c) x[c] = __uint_as_float(r0[c]);
      }
      const int qc0 = i * BQ + 64 * chalf + 2 * cq;  // query of x[0]
      const bool full = i > kb && i * BQ + BQ <= p.T;
      const float2 sl2 = make_float2(p.sl2, p.sl2);
#pragma unroll
      for (int n = 0; n < 8; ++n) {
        const float2 l2 = *reinterpret_cast<const float2*>(lse_s + 8 * n + 2 * cq);
        const float2 nl = make_float2(tc::neg_bits(l2.x), tc::neg_bits(l2.y));
        const float2 ea = tc::fma2(make_float2(x[4 * n], x[4 * n + 1]), sl2, nl);
        const float2 eb = tc::fma2(make_float2(x[4 * n + 2], x[4 * n + 3]), sl2, nl);
        float pa[2] = {tc::fast_exp2(ea.x), tc::fast_exp2(ea.y)};
        float pb[2] = {tc::fast_exp2(eb.x), tc::fast_exp2(eb.y)};
        if (!full) {
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const int q = qc0 + 8 * n + e;
            if (q >= p.T || q < keyA) pa[e] = 0.f;
            if (q >= p.T || q < keyB) pb[e] = 0.f;
          }
        }
        x[4 * n] = pa[0];
        x[4 * n + 1] = pa[1];
        x[4 * n + 2] = pb[0];
        x[4 * n + 3] = pb[1];
      }
      {
        uint32_t pw[16];  // pw[2n] row A, pw[2n + 1] row B: packed column 64 chalf + 4n + cq
#pragma unroll
        for (int n = 0; n < 8; ++n) {
          pw[2 * n] = tc::pack_half2(x[4 * n], x[4 * n + 1]);
          pw[2 * n + 1] = tc::pack_half2(x[4 * n + 2], x[4 * n + 3]);
        }
        __syncwarp();
        tc::tmem_st_16x128b_x8(tmem + lane16 + L::S_COL + 64 * chalf, pw);
        tc::tmem_st_wait();
      }
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->p_full);
      if (!tc::mbar_wait(&bars->dp_full, it & 1, abort, p.status)) {
        ok = false;
        break;
      }
      tc::fence_after_sync();
      uint32_t dw[16];
      // The staging tile's words of this thread: packed word n of key rows rA and rA + 8 of the
      // 64-query half chalf (128-byte swizzle).
      uint8_t* hb = smem + L::DSS_OFF + chalf * L::CHUNK;
      uint32_t* wa_p = reinterpret_cast<uint32_t*>(hb + rA * 128 + cq * 4);
      uint32_t* wb_p = reinterpret_cast<uint32_t*>(hb + (rA + 8) * 128 + cq * 4);
      const int swa = rA & 7, swb = (rA + 8) & 7;
      if (KL && !tc::mbar_wait(&bars->pt_full, it & 1, abort, p.status)) {
        ok = false;
        break;
      }
      {
        uint32_t rd[32];
        __syncwarp();
        tc::tmem_ld_16x256b_x8(tmem + lane16 + L::DP_COL + 64 * chalf, rd);
        tc::tmem_ld_wait();
#pragma unroll
        for (int n = 0; n < 8; ++n) {
          const float2 d2 = *reinterpret_cast<const float2*>(d_s + 8 * n + 2 * cq);
          const float2 ta = tc::sub2(make_float2(__uint_as_float(rd[4 * n]), __uint_as_float(rd[4 * n + 1])), d2);
          const float2 tb = tc::sub2(make_float2(__uint_as_float(rd[4 * n + 2]), __uint_as_float(rd[4 * n + 3])), d2);
          const float2 pa = make_float2(x[4 * n], x[4 * n + 1]);
          const float2 pb = make_float2(x[4 * n + 2], x[4 * n + 3]);
          float2 da = tc::mul2(pa, ta);
          float2 db = tc::mul2(pb, tb);
          if constexpr (KL) {
            // + b_kl (P - P^T): the teacher's probabilities of the same entries (0 where masked)
            const float2 qa = __half22float2(
                *reinterpret_cast<const __half2*>(&wa_p[(n ^ swa) << 2]));
            const float2 qb = __half22float2(
                *reinterpret_cast<const __half2*>(&wb_p[(n ^ swb) << 2]));
            const float2 am = make_float2(p.a_mse, p.a_mse), bk = make_float2(p.b_kl, p.b_kl);
            const float2 ka = tc::mul2(tc::sub2(pa, qa), bk), kb2 = tc::mul2(tc::sub2(pb, qb), bk);
            float2 ea = tc::fma2(da, am, ka), eb = tc::fma2(db, am, kb2);
            if (!full) {  // masked entries (P = P^T = 0; D past T is not written): dS = 0
              if (pa.x == 0.f && qa.x == 0.f) ea.x = 0.f;
              if (pa.y == 0.f && qa.y == 0.f) ea.y = 0.f;
              if (pb.x == 0.f && qb.x == 0.f) eb.x = 0.f;
              if (pb.y == 0.f && qb.y == 0.f) eb.y = 0.f;
            }
            da = ea;
            db = eb;
          } else if (!full) {  // masked entries (P = 0; D past T is not written): dS = 0
            if (x[4 * n] == 0.f) da.x = 0.f;
            if (x[4 * n + 1] == 0.f) da.y = 0.f;
            if (x[4 * n + 2] == 0.f) db.x = 0.f;
            if (x[4 * n + 3] == 0.f) db.y = 0.f;
          }
          dw[2 * n] = tc::pack_half2(da.x, da.y);
          dw[2 * n + 1] = tc::pack_half2(db.x, db.y);
        }
      }
      __syncwarp();
      tc::tmem_st_16x128b_x8(tmem + lane16 + L::DP_COL + 64 * chalf, dw);
      tc::tmem_st_wait();
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->ds_full);
      // The same dS^T words into the staging tile for the store warp, once it has stored the
      // previous block's: packed word n (queries 64 chalf + 8n + 2cq, +1) is 16-byte unit n of the
      // 64-query half chalf of its key row (128-byte swizzle). With KL they go over this thread's
      // own P^T words, loaded only after the previous block's store had read the tile.
      if (!KL && it > 0 && !tc::mbar_wait(&bars->dss_free, (it - 1) & 1, abort, p.status)) {
        ok = false;
        break;
      }
#pragma unroll
      for (int n = 0; n < 8; ++n) {
        wa_p[(n ^ swa) << 2] = dw[2 * n];
        wb_p[(n ^ swb) << 2] = dw[2 * n + 1];
      }
      tc::fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->dss_full);
    }
    // Epilogue: dV rows (warps of query half 0) and dK rows (half 1; transpose of RoPE) staged
    // transposed in the now idle stage buffers, then stored as dQKV^T columns with coalesced
    // 16-byte stores by all elementwise warps.
    const bool have = ok && tc::mbar_wait(&bars->o_full, 0, abort, p.status);
    bf16_t* tv = reinterpret_cast<bf16_t*>(smem + L::ST_OFF);
    bf16_t* tk = tv + DH * 128;
    if (have) {
      tc::fence_after_sync();
      const int kA = keyA < p.T ? keyA : 0, kB = keyB < p.T ? keyB : 0;
      if (chalf == 0)
        stage_grad_16<DH>(tmem + lane16 + L::DV_COL, KL ? p.a_mse : 1.f, false, 0, 0, p.cos_t,
                          p.sin_t, tv, rA);
      else
        stage_grad_16<DH>(tmem + lane16 + L::DK_COL, p.scale, p.use_rope != 0, kA, kB, p.cos_t,
                          p.sin_t, tk, rA);
    }
    tc::named_bar_sync(1, DKDV_EW * 32);  // every elementwise warp reaches this exactly once
    if (have) {
      const int nvalid = min(BK, p.T - kb * BK);
      const int64_t n0 = (int64_t)row0 + kb * BK;
      const int64_t ext_t = (int64_t)(p.Hq + 2 * p.Hkv) * DH * p.ldt;  // dQKV^T elements
      const int tid = threadIdx.x - 64;
      store_tile<DH>(tv, p.dqkvt + (int64_t)(p.vcol0 + g * DH) * p.ldt, p.ldt, n0, nvalid, tid,
                     DKDV_EW * 32, p.dqkvt, ext_t, p.status);
      store_tile<DH>(tk, p.dqkvt + (int64_t)(p.kcol0 + g * DH) * p.ldt, p.ldt, n0, nvalid, tid,
                     DKDV_EW * 32, p.dqkvt, ext_t, p.status);
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

// ================================================================================ teacher P tiles
// The KL term of Eq. 3 (D_KL(P || Q), P the teacher's map) for the STE gradient: its gradient with
// respect to the student's scaled scores is (lambda / B)(Q - P), so the backward needs the teacher's
// probabilities P of every (query, key) entry that the dS tiles hold. This kernel writes P^T into
// the dS^T tile buffer in the dS^T layout (the dK/dV kernel then reads each tile, forms dS and
// stores it back over it), and the KL value itself, using the two softmax normalisers of the
// forward passes (teacher: jab_reference_forward; student: the loss+backward forward):
//   KL_row i = sum_j P_ij (s^T_ij - s^S_ij) + lse^S_i - lse^T_i,  s = scale Q K^T (natural units),
//   P_ij = exp(s^T_ij - lse^T_i).
// Per CTA (128-key block, KV head, sequence), as the dK/dV kernel's walk over the group's query
// heads and query blocks: S_t^T = K_t Q_t^T and S_s^T = K_s Q_s^T into one of two TMEM buffers
// (the next block's products run while the elementwise warps read this one), P^T = exp2(s_t^T sl2 -
// lse2_t) with the causal mask, the CTA's partial sum of P (s_t - s_s) (and, in the key-block-0 CTAs
// that see every query row once, of lse^S - lse^T), and P^T staged and stored by TMA.
//   warp 0      TMA: K_t, K_s once; per block Q_t, Q_s and the two rows of lse (log2 units)
//   warp 1      TMEM owner, UMMA issuer
//   warps 2..17 elementwise, 16 key rows x 64 queries each (the dK/dV kernel's layout)
//   warp 18     P^T tiles to global memory
constexpr int TP_THREADS = (2 + DKDV_EW + 1) * 32;

struct TpParams {
  int T, B, Hq, Hkv, lse_pitch, npairs;
  int qcol0, kcol0;  // column offsets of the Q and K heads (the same in both projections)
  float scale, sl2;
  const float* lse2_t;  // teacher log-sum-exp, log2 units, [B, Hq, lse_pitch]
  const float* lse2_s;  // student log-sum-exp, log2 units, [B, Hq, lse_pitch]
  double* part;         // [gridDim.x] KL partial of each CTA (natural units)
  int* status;
};

template <int DH>
struct TpLayout {
  static constexpr int BK = 128, BQ = 128, STAGES = 2;
  static constexpr int CHUNK = 128 * 128;
  static constexpr int NCH = DH / 64;
  static constexpr int KT_OFF = 0, KS_OFF = NCH * CHUNK;
  static constexpr int ST_OFF = 2 * NCH * CHUNK;
  static constexpr int ST_QT = 0, ST_QS = NCH * CHUNK, ST_LT = 2 * NCH * CHUNK,
                       ST_LS = ST_LT + BQ * 4, ST_BYTES = ST_LS + BQ * 4;
  static constexpr int ST_STRIDE = (ST_BYTES + 1023) / 1024 * 1024;
  static constexpr int DSS_OFF = ST_OFF + STAGES * ST_STRIDE;
  static constexpr int BAR_OFF = DSS_OFF + 2 * CHUNK;
  static constexpr int USED = BAR_OFF + 512;  // base alignment checked in the kernel
  static constexpr int SMEM = USED > 118 * 1024 ? USED : 118 * 1024;
  static_assert(USED <= 227 * 1024, "shared memory budget");
};

struct TpBars {
  uint64_t kv_full, ld_full[2], ld_empty[2], s_full[2], s_free[2], dss_full, dss_free, drain;
  uint32_t tmem_base;
  int abort;
  double red[DKDV_EW];
};

template <int DH>
__global__ void __launch_bounds__(TP_THREADS, 1)
    attn_teacher_p_tc_kernel(const __grid_constant__ CUtensorMap tm_s,
                             const __grid_constant__ CUtensorMap tm_t,
                             const __grid_constant__ CUtensorMap tm_ds, const TpParams p) {
  using L = TpLayout<DH>;
  constexpr int BK = L::BK, BQ = L::BQ, STAGES = L::STAGES;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if (tc::smem_u32(smem_raw) & 1023u) {
    if (threadIdx.x == 0) report(p.status, JAB_ERR_INTERNAL);
    return;
  }
  uint8_t* smem = smem_raw;
  TpBars* bars = reinterpret_cast<TpBars*>(smem + L::BAR_OFF);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &bars->abort;

  const int r = p.Hq / p.Hkv;
  const int nq = (p.T + BQ - 1) / BQ;
  int kb, g, b;  // the dK/dV kernel's CTA order
  {
    const int pairs = p.Hkv * p.B;
    const int sg = blockIdx.x / (kSuperGroup * nq);
    const int sgs = min(kSuperGroup, pairs - sg * kSuperGroup);
    const int rem = blockIdx.x - sg * kSuperGroup * nq;
    kb = rem / sgs;
    const int pr = sg * kSuperGroup + rem % sgs;
    g = pr % p.Hkv;
    b = pr / p.Hkv;
  }
  const int per_head = nq - kb;
  const int n_it = r * per_head;
  const int row0 = b * p.T;

  if (threadIdx.x == 0) {
    tc::mbar_init(&bars->kv_full, 1);
    for (int i = 0; i < STAGES; ++i) {
      tc::mbar_init(&bars->ld_full[i], 1);
      tc::mbar_init(&bars->ld_empty[i], 1 + DKDV_EW);  // the products and the lse readers
      tc::mbar_init(&bars->s_full[i], 1);
      tc::mbar_init(&bars->s_free[i], DKDV_EW);
    }
    tc::mbar_init(&bars->dss_full, DKDV_EW);
    tc::mbar_init(&bars->dss_free, 1);
    tc::mbar_init(&bars->drain, 1);
    bars->abort = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&tm_s);
    tc::prefetch_tmap(&tm_t);
    tc::prefetch_tmap(&tm_ds);
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
    if (lane == 0) {  // ------------------------------------------------------------- TMA
      uint32_t issued = 0, last_par = 0;
      tc::mbar_expect_tx(&bars->kv_full, 2 * BK * DH * 2);
      for (int ch = 0; ch < L::NCH; ++ch) {
        tc::tma_load_2d(smem + L::KT_OFF + ch * L::CHUNK, &tm_t, &bars->kv_full,
                        p.kcol0 + g * DH + ch * 64, row0 + kb * BK);
        tc::tma_load_2d(smem + L::KS_OFF + ch * L::CHUNK, &tm_s, &bars->kv_full,
                        p.kcol0 + g * DH + ch * 64, row0 + kb * BK);
      }
      for (int it = 0; it < n_it; ++it) {
        const int st = it % STAGES;
        const uint32_t ph = (it / STAGES) & 1;
        const int h = g * r + it / per_head, i = kb + it % per_head;
        if (!tc::mbar_wait(&bars->ld_empty[st], ph ^ 1, abort, p.status)) break;
        uint8_t* sbase = smem + L::ST_OFF + st * L::ST_STRIDE;
        tc::mbar_expect_tx(&bars->ld_full[st], L::ST_BYTES);
        for (int ch = 0; ch < L::NCH; ++ch) {
          tc::tma_load_2d(sbase + L::ST_QT + ch * L::CHUNK, &tm_t, &bars->ld_full[st],
                          p.qcol0 + h * DH + ch * 64, row0 + i * BQ);
          tc::tma_load_2d(sbase + L::ST_QS + ch * L::CHUNK, &tm_s, &bars->ld_full[st],
                          p.qcol0 + h * DH + ch * 64, row0 + i * BQ);
        }
        const int64_t lrow = ((int64_t)b * p.Hq + h) * p.lse_pitch + i * BQ;
        if (in_bounds(lrow + BQ - 1, (int64_t)p.B * p.Hq * p.lse_pitch, p.status)) {
          tc::bulk_load(sbase + L::ST_LT, p.lse2_t + lrow, BQ * 4, &bars->ld_full[st]);
          tc::bulk_load(sbase + L::ST_LS, p.lse2_s + lrow, BQ * 4, &bars->ld_full[st]);
        }
        issued |= 1u << st;
        last_par = (last_par & ~(1u << st)) | (ph << st);
      }
      if (*abort) {
        drain_wait(&bars->kv_full, 0);
        for (int st = 0; st < STAGES; ++st)
          if (issued & (1u << st)) drain_wait(&bars->ld_full[st], (last_par >> st) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {  // ---------------------------------------------------------------- UMMA
      constexpr uint32_t ID_S = tc::idesc_f16(false, BK, BQ);
      bool ok = tc::mbar_wait(&bars->kv_full, 0, abort, p.status);
      const uint64_t kt = tc::sdesc_kmajor_sw128(tc::smem_u32(smem + L::KT_OFF));
      const uint64_t ks = tc::sdesc_kmajor_sw128(tc::smem_u32(smem + L::KS_OFF));
      for (int j = 0; ok && j < n_it; ++j) {
        const int st = j % STAGES, bf = j & 1;
        // the stage has landed and the elementwise warps have read block j - 2's scores
        ok = tc::mbar_wait(&bars->ld_full[st], (j / STAGES) & 1, abort, p.status) &&
             (j < 2 || tc::mbar_wait(&bars->s_free[bf], ((j >> 1) - 1) & 1, abort, p.status));
        if (!ok) break;
        tc::fence_after_sync();
        const uint32_t sb = tc::smem_u32(smem + L::ST_OFF + st * L::ST_STRIDE);
        const uint64_t bt = tc::sdesc_kmajor_sw128(sb + L::ST_QT);
        const uint64_t bs = tc::sdesc_kmajor_sw128(sb + L::ST_QS);
#pragma unroll
        for (int k = 0; k < DH / 16; ++k) {
          const uint32_t o = (k >> 2) * L::CHUNK + (k & 3) * 32;
          tc::umma_f16(tmem + 256 * bf, tc::sdesc_advance(kt, o), tc::sdesc_advance(bt, o), ID_S,
                       k > 0 ? 1u : 0u);
        }
#pragma unroll
        for (int k = 0; k < DH / 16; ++k) {
          const uint32_t o = (k >> 2) * L::CHUNK + (k & 3) * 32;
          tc::umma_f16(tmem + 256 * bf + 128, tc::sdesc_advance(ks, o), tc::sdesc_advance(bs, o),
                       ID_S, k > 0 ? 1u : 0u);
        }
        tc::umma_commit(&bars->s_full[bf]);
        tc::umma_commit(&bars->ld_empty[st]);
      }
      tc::umma_commit(&bars->drain);
      drain_wait(&bars->drain, 0);
    }
  } else if (warp == 2 + DKDV_EW) {
    if (lane == 0) {  // ------------------------------------------------- P^T tiles to global
      for (int it = 0; it < n_it; ++it) {
        if (!tc::mbar_wait(&bars->dss_full, it & 1, abort, p.status)) break;
        const int h = g * r + it / per_head, i = kb + it % per_head;
        const int64_t tile = ((int64_t)b * p.Hq + h) * p.npairs + (int64_t)i * (i + 1) / 2 + kb;
        tc::tma_store_2d(&tm_ds, smem + L::DSS_OFF, 0, (int32_t)(tile * BK));
        tc::tma_store_2d(&tm_ds, smem + L::DSS_OFF + L::CHUNK, 64, (int32_t)(tile * BK));
        tc::bulk_commit_group();
        tc::bulk_wait_group_read<0>();
        tc::mbar_arrive(&bars->dss_free);
      }
      tc::bulk_wait_group<0>();
    }
  } else {  // ------------------------------------ elementwise: 16 key rows x 64 queries per warp
    const int quarter = warp & 3;
    const int idx = (warp - 2) >> 2;
    const int half = idx & 1;
    const int chalf = idx >> 1;
    const int cq = lane & 3;
    const int rA = quarter * 32 + half * 16 + (lane >> 2);
    const int keyA = kb * BK + rA, keyB = keyA + 8;
    const uint32_t lane16 = (uint32_t)(quarter * 32 + half * 16) << 16;
    float2 acc = make_float2(0.f, 0.f);  // sum of P (s_t - s_s) in raw score units (times scale later)
    double rows = 0.0;                   // key-block-0 CTAs, warp 2: sum of lse2_s - lse2_t
    for (int it = 0; it < n_it; ++it) {
      const int st = it % STAGES, bf = it & 1;
      const int i = kb + it % per_head;
      const float* sbase = reinterpret_cast<const float*>(smem + L::ST_OFF + st * L::ST_STRIDE);
      const float* lt = sbase + L::ST_LT / 4;
      const float* ls = sbase + L::ST_LS / 4;
      if (!tc::mbar_wait(&bars->ld_full[st], (it / STAGES) & 1, abort, p.status) ||
          !tc::mbar_wait(&bars->s_full[bf], (it >> 1) & 1, abort, p.status))
        break;
      tc::fence_after_sync();
      uint32_t rt[32], rs[32];
      __syncwarp();
      tc::tmem_ld_16x256b_x8(tmem + lane16 + 256 * bf + 64 * chalf, rt);
      tc::tmem_ld_16x256b_x8(tmem + lane16 + 256 * bf + 128 + 64 * chalf, rs);
      tc::tmem_ld_wait();
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->s_free[bf]);  // the products of block it + 2 may start
      const int qc0 = i * BQ + 64 * chalf + 2 * cq;
      const bool full = i > kb && i * BQ + BQ <= p.T;
      const float2 sl2 = make_float2(p.sl2, p.sl2);
      uint32_t pw[16];
#pragma unroll
      for (int n = 0; n < 8; ++n) {
        const float2 l2 = *reinterpret_cast<const float2*>(lt + 64 * chalf + 8 * n + 2 * cq);
        const float2 nl = make_float2(tc::neg_bits(l2.x), tc::neg_bits(l2.y));
        const float2 ta = make_float2(__uint_as_float(rt[4 * n]), __uint_as_float(rt[4 * n + 1]));
        const float2 tb = make_float2(__uint_as_float(rt[4 * n + 2]), __uint_as_float(rt[4 * n + 3]));
        const float2 sa = make_float2(__uint_as_float(rs[4 * n]), __uint_as_float(rs[4 * n + 1]));
        const float2 sb = make_float2(__uint_as_float(rs[4 * n + 2]), __uint_as_float(rs[4 * n + 3]));
        const float2 ea = tc::fma2(ta, sl2, nl), eb = tc::fma2(tb, sl2, nl);
        float pa[2] = {tc::fast_exp2(ea.x), tc::fast_exp2(ea.y)};
        float pb[2] = {tc::fast_exp2(eb.x), tc::fast_exp2(eb.y)};
        if (!full) {
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const int q = qc0 + 8 * n + e;
            if (q >= p.T || q < keyA) pa[e] = 0.f;
            if (q >= p.T || q < keyB) pb[e] = 0.f;
          }
        }
        acc = tc::fma2(make_float2(pa[0], pa[1]), tc::sub2(ta, sa), acc);
        acc = tc::fma2(make_float2(pb[0], pb[1]), tc::sub2(tb, sb), acc);
        pw[2 * n] = tc::pack_half2(pa[0], pa[1]);
        pw[2 * n + 1] = tc::pack_half2(pb[0], pb[1]);
      }
      if (kb == 0 && warp == 2) {  // lse^S - lse^T of the block's query rows (each row once)
        float t = 0.f;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int qi = lane * 4 + e;
          if (i * BQ + qi < p.T) t += ls[qi] - lt[qi];
        }
        rows += t;
      }
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->ld_empty[st]);  // this warp has read the lse rows
      if (it > 0 && !tc::mbar_wait(&bars->dss_free, (it - 1) & 1, abort, p.status)) break;
      {
        uint8_t* hb = smem + L::DSS_OFF + chalf * L::CHUNK;
#pragma unroll
        for (int n = 0; n < 8; ++n) {
          *reinterpret_cast<uint32_t*>(hb + rA * 128 + ((n ^ (rA & 7)) << 4) + cq * 4) = pw[2 * n];
          *reinterpret_cast<uint32_t*>(hb + (rA + 8) * 128 + ((n ^ ((rA + 8) & 7)) << 4) + cq * 4) =
              pw[2 * n + 1];
        }
      }
      tc::fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->dss_full);
    }
    // The CTA's partial: the warps' sums in a fixed order (natural units).
    float v = acc.x + acc.y;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) rows += __shfl_xor_sync(0xffffffffu, rows, o);
    if (lane == 0) bars->red[warp - 2] = (double)v * p.scale + rows * (double)kLn2;
    tc::named_bar_sync(1, DKDV_EW * 32);
    if (threadIdx.x == 64) {
      double t = 0.0;
      for (int w = 0; w < DKDV_EW; ++w) t += bars->red[w];
      p.part[blockIdx.x] = t;
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

// ================================================================================ dQ
// dQ = scale * dS K from the dS^T tiles the dK/dV kernel stored: no recomputation of S, P or dP.
// Persistent: one CTA per SM takes (128 query rows, query head, sequence) tiles (sched_tile,
// most key blocks first); for each key block kb <= qb one stage holds the dS^T tile (128 keys x 128
// queries: the MN-major A operand of dS K) and K_kb (128 keys x d_h: the MN-major B operand), and
// eight M128 N = d_h K16 UMMAs accumulate into one of two dQ buffers in TMEM.
//   warp 0      TMA: dS^T and K tiles, 3-stage ring
//   warp 1      TMEM owner, UMMA issuer (one thread)
//   warps 2..9  epilogue of the previous tile (its dQ buffer): transpose of RoPE, staged transposed
//               in shared memory, stored as dQKV^T columns with coalesced 16-byte stores
constexpr int DQ_THREADS = 320;

template <int DH>
struct DqLayout {
  static constexpr int BQ = 128, BK = 128, STAGES = 3;
  static constexpr int CHUNK = 128 * 128;       // 64 columns of a 128-row fp16 tile
  static constexpr int DS_TILE = 128 * 128 * 2;  // dS^T: 128 keys x 128 queries
  static constexpr int K_TILE = 128 * DH * 2;    // 128 keys x d_h
  static constexpr int STAGE = DS_TILE + K_TILE;
  static constexpr int STG_OFF = STAGES * STAGE;  // epilogue staging: d_h x 128 bf16
  static constexpr int BAR_OFF = STG_OFF + DH * 128 * 2;
  static constexpr int USED = BAR_OFF + 256;      // base alignment checked in the kernel
  static constexpr int SMEM = USED > 118 * 1024 ? USED : 118 * 1024;
  static constexpr uint32_t DQ_STRIDE = 128;      // TMEM columns between the two dQ buffers
  static_assert(USED <= 227 * 1024, "shared memory budget");
};

struct DqBars {
  uint64_t full[3], empty[3], o_full[2], o_empty[2], drain;
  uint32_t tmem_base;
  int abort;
  int stop;  // the epilogue warps' common decision to leave (a snapshot of abort)
};

struct DqTile {
  int qb, h, b;
};
// Tile n: grouped by (sequence, KV group), so that all tiles which read the K blocks of one KV head
// run close together (K read from HBM once); inside a group query blocks from the last (most keys)
// to the first, the query heads of the group next to each other.
__device__ __forceinline__ DqTile dq_tile(int n, int nqb, int Hq, int Hkv) {
  const int r = Hq / Hkv;
  const int per_group = r * nqb;
  const int grp = n / per_group, rem = n - grp * per_group;
  const int g = grp % Hkv, b = grp / Hkv;
  return DqTile{nqb - 1 - rem / r, g * r + rem % r, b};
}

template <int DH>
__global__ void __launch_bounds__(DQ_THREADS, 1)
    attn_bwd_dq_tc_kernel(const __grid_constant__ CUtensorMap tm_ds,
                          const __grid_constant__ CUtensorMap tm_kv, const BwdParams p) {
  using L = DqLayout<DH>;
  constexpr int BQ = L::BQ, BK = L::BK, NST = L::STAGES;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if (tc::smem_u32(smem_raw) & 1023u) {  // the swizzled TMA tiles need a 1024-byte aligned base
    if (threadIdx.x == 0) report(p.status, JAB_ERR_INTERNAL);
    return;
  }
  uint8_t* smem = smem_raw;
  DqBars* bars = reinterpret_cast<DqBars*>(smem + L::BAR_OFF);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &bars->abort;

  const int nqb = (p.T + BQ - 1) / BQ;
  const int n_tiles = nqb * p.Hq * p.B;
  auto n_kb_of = [&](const DqTile& tl) { return (min(tl.qb * BQ + BQ, p.T) + BK - 1) / BK; };

  if (threadIdx.x == 0) {
    for (int i = 0; i < NST; ++i) {
      tc::mbar_init(&bars->full[i], 1);
      tc::mbar_init(&bars->empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&bars->o_full[i], 1);
      tc::mbar_init(&bars->o_empty[i], EW_WARPS);
    }
    tc::mbar_init(&bars->drain, 1);
    bars->abort = 0;
    bars->stop = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&tm_ds);
    tc::prefetch_tmap(&tm_kv);
  }
  if (warp == 1) {
    tc::tmem_alloc(&bars->tmem_base, 256);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = bars->tmem_base;

  if (warp == 0) {
    if (lane == 0) {  // ---------------------------------------------------------------- TMA
      uint32_t J = 0, iss = 0, par = 0;
      bool ok = true;
      for (int it = 0, tile = sched_tile(0, gridDim.x, blockIdx.x); ok && tile < n_tiles;
           tile = sched_tile(++it, gridDim.x, blockIdx.x)) {
        const DqTile tl = dq_tile(tile, nqb, p.Hq, p.Hkv);
        const int g = tl.h / (p.Hq / p.Hkv), nkb = n_kb_of(tl);
        const int64_t pair0 = ((int64_t)tl.b * p.Hq + tl.h) * p.npairs + (int64_t)tl.qb * (tl.qb + 1) / 2;
        for (int kb = 0; kb < nkb; ++kb, ++J) {
          const int st = J % NST;
          const uint32_t ph = (J / NST) & 1;
          if (!tc::mbar_wait(&bars->empty[st], ph ^ 1, abort, p.status)) { ok = false; break; }
          uint8_t* sb = smem + st * L::STAGE;
          tc::mbar_expect_tx(&bars->full[st], L::STAGE);
          const int32_t y = (int32_t)((pair0 + kb) * BK);
          tc::tma_load_2d(sb, &tm_ds, &bars->full[st], 0, y);
          tc::tma_load_2d(sb + L::CHUNK, &tm_ds, &bars->full[st], 64, y);
          for (int ch = 0; ch < DH / 64; ++ch)
            tc::tma_load_2d(sb + L::DS_TILE + ch * L::CHUNK, &tm_kv, &bars->full[st],
                            p.kcol0 + g * DH + ch * 64, tl.b * p.T + kb * BK);
          iss |= 1u << st;
          par = (par & ~(1u << st)) | (ph << st);
        }
      }
      if (*abort)
        for (int st = 0; st < NST; ++st)
          if (iss & (1u << st)) drain_wait(&bars->full[st], (par >> st) & 1);
    }
  } else if (warp == 1) {
    if (lane == 0) {  // ---------------------------------------------------------------- UMMA
      // A = dS (M = queries, K = keys) and B = K (N = d_h, K = keys) are both MN-major tiles
      constexpr uint32_t ID_Q = tc::idesc_f16(false, BQ, DH) | (1u << 15) | (1u << 16);
      uint32_t J = 0;
      bool ok = true;
      int n = 0;
      for (int it = 0, tile = sched_tile(0, gridDim.x, blockIdx.x); ok && tile < n_tiles;
           tile = sched_tile(++it, gridDim.x, blockIdx.x), ++n) {
        const DqTile tl = dq_tile(tile, nqb, p.Hq, p.Hkv);
        const int nkb = n_kb_of(tl), ob = n & 1;
        // the buffer's previous tile (n - 2) must have been read out by the epilogue
        if (n >= 2 && !tc::mbar_wait(&bars->o_empty[ob], ((n >> 1) - 1) & 1, abort, p.status)) break;
        for (int kb = 0; kb < nkb; ++kb, ++J) {
          const int st = J % NST;
          if (!tc::mbar_wait(&bars->full[st], (J / NST) & 1, abort, p.status)) { ok = false; break; }
          tc::fence_after_sync();
          const uint32_t sb = tc::smem_u32(smem + st * L::STAGE);
          const uint64_t ad = tc::sdesc_mnmajor_sw128(sb, L::CHUNK, 1024);
          const uint64_t bd = tc::sdesc_mnmajor_sw128(sb + L::DS_TILE, L::CHUNK, 1024);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            tc::umma_f16(tmem + ob * L::DQ_STRIDE, tc::sdesc_advance(ad, k * 16 * 128),
                         tc::sdesc_advance(bd, k * 16 * 128), ID_Q, (kb > 0 || k > 0) ? 1u : 0u);
          tc::umma_commit(&bars->empty[st]);
        }
        if (!ok) break;
        tc::umma_commit(&bars->o_full[ob]);
      }
      tc::umma_commit(&bars->drain);
      drain_wait(&bars->drain, 0);
    }
  } else {  // ----------------------------------------------------- epilogue, 16 rows per warp
    const int quarter = warp & 3;
    const int half = (warp - 2) >> 2;
    const int ra = quarter * 32 + half * 16 + (lane >> 2);  // 16x256b rows of this thread
    const uint32_t lane16 = (uint32_t)(quarter * 32 + half * 16) << 16;
    bf16_t* stage = reinterpret_cast<bf16_t*>(smem + L::STG_OFF);
    int n = 0;
    for (int it = 0, tile = sched_tile(0, gridDim.x, blockIdx.x); tile < n_tiles;
         tile = sched_tile(++it, gridDim.x, blockIdx.x), ++n) {
      const DqTile tl = dq_tile(tile, nqb, p.Hq, p.Hkv);
      const int ob = n & 1, q0 = tl.qb * BQ;
      const bool have = tc::mbar_wait(&bars->o_full[ob], (n >> 1) & 1, abort, p.status);
      if (have) {
        tc::fence_after_sync();
        const int ta = q0 + ra, tb = ta + 8;
        stage_grad_16<DH>(tmem + lane16 + ob * L::DQ_STRIDE, p.scale, p.use_rope != 0,
                          ta < p.T ? ta : 0, tb < p.T ? tb : 0, p.cos_t, p.sin_t, stage, ra);
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&bars->o_empty[ob]);  // the dQ buffer is free again
      }
      tc::named_bar_sync(1, EW_WARPS * 32);  // every epilogue warp reaches this once per tile
      if (have)
        store_tile<DH>(stage, p.dqkvt + (int64_t)(p.qcol0 + tl.h * DH) * p.ldt, p.ldt,
                       (int64_t)tl.b * p.T + q0, min(BQ, p.T - q0), threadIdx.x - 64,
                       EW_WARPS * 32, p.dqkvt, (int64_t)(p.Hq + 2 * p.Hkv) * DH * p.ldt, p.status);
      // One snapshot of the abort flag between the two barriers, so that all epilogue warps leave
      // together (a warp left behind would wait on the named barrier of the next tile).
      if (threadIdx.x == 64) reinterpret_cast<volatile int*>(&bars->stop)[0] = *abort;
      tc::named_bar_sync(1, EW_WARPS * 32);  // the staging tile is read before it is rewritten
      if (reinterpret_cast<volatile int*>(&bars->stop)[0]) break;
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  if (warp == 1) {
    __syncwarp();
    tc::tmem_dealloc(tmem, 256);
  }
}

// ================================================================================ host
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

bool tmap_rows(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <typename K>
cudaError_t set_smem(K kernel, int bytes, bool& done) {
  if (done) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done = true;
  return e;
}

template <int DH>
cudaError_t launch_bwd(const AttnLaunch& L, const BwdParams& p, bool kl) {
  const int64_t N = (int64_t)L.B * L.T;
  // dS^T tiles as a 2-D fp16 tensor of 128-query rows, one 128-row block per (sequence, head,
  // query block, key block)
  const uint64_t ds_rows = (uint64_t)L.B * L.Hq * p.npairs * 128;
  CUtensorMap kv128, do128, ds128;
  if (!tmap_rows(&kv128, L.qkv, L.ldq, N, 128) ||
      !tmap_rows(&do128, L.d_o, (uint64_t)L.Hq * DH, N, 128) ||
      !tmap_rows(&ds128, L.ds, 128, ds_rows, 128) || ds_rows >= (1ull << 31))
    return cudaErrorInvalidValue;
  static bool a1 = false, a2 = false, a3 = false;
  cudaError_t e = set_smem(attn_bwd_dkdv_tc_kernel<DH, false>, DkdvLayout<DH>::SMEM, a1);
  if (e != cudaSuccess) return e;
  e = set_smem(attn_bwd_dkdv_tc_kernel<DH, true>, DkdvLayout<DH>::SMEM, a3);
  if (e != cudaSuccess) return e;
  e = set_smem(attn_bwd_dq_tc_kernel<DH>, DqLayout<DH>::SMEM, a2);
  if (e != cudaSuccess) return e;
  const int64_t n_dkdv = (int64_t)L.Hkv * L.B * ((L.T + 127) / 128);
  if (n_dkdv >= (1ll << 31)) return cudaErrorInvalidValue;
  const dim3 g1((unsigned)n_dkdv);
  if (kl)
    attn_bwd_dkdv_tc_kernel<DH, true><<<g1, DKDV_THREADS, DkdvLayout<DH>::SMEM, L.stream>>>(
        kv128, do128, ds128, p);
  else
    attn_bwd_dkdv_tc_kernel<DH, false><<<g1, DKDV_THREADS, DkdvLayout<DH>::SMEM, L.stream>>>(
        kv128, do128, ds128, p);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t dq_tiles = (int64_t)((L.T + 127) / 128) * L.Hq * L.B;
  const unsigned g2 = (unsigned)std::min<int64_t>(dq_tiles, sms > 0 ? sms : 1);
  attn_bwd_dq_tc_kernel<DH><<<g2, DQ_THREADS, DqLayout<DH>::SMEM, L.stream>>>(ds128, kv128, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_attn_bwd_tc(const AttnLaunch& L, const float* cos_t, const float* sin_t,
                               int use_rope, void* dqkvt, const float* kl_ab) {
  BwdParams p{};
  p.T = L.T;
  p.B = L.B;
  p.Hq = L.Hq;
  p.Hkv = L.Hkv;
  p.lse_pitch = L.lse_pitch;
  p.qcol0 = 0;
  p.kcol0 = L.Hq * L.dh;
  p.vcol0 = (L.Hq + L.Hkv) * L.dh;
  p.ldt = L.ldt;
  const int nq = (L.T + 127) / 128;
  p.npairs = nq * (nq + 1) / 2;
  p.scale = L.scale;
  p.sl2 = L.scale * kLog2e;
  p.a_mse = kl_ab ? kl_ab[0] : 1.f;
  p.b_kl = kl_ab ? kl_ab[1] : 0.f;
  p.lse = L.lse;
  p.dvec = L.dvec;
  p.cos_t = cos_t;
  p.sin_t = sin_t;
  p.use_rope = use_rope;
  p.dqkvt = static_cast<bf16_t*>(dqkvt);
  p.status = L.status;
  if ((reinterpret_cast<uintptr_t>(L.lse) & 15u) || (reinterpret_cast<uintptr_t>(L.dvec) & 15u) ||
      (L.lse_pitch % 128) != 0 || L.ds == nullptr || (reinterpret_cast<uintptr_t>(L.ds) & 15u))
    return cudaErrorInvalidValue;
  return L.dh == 128 ? launch_bwd<128>(L, p, kl_ab != nullptr)
                     : launch_bwd<64>(L, p, kl_ab != nullptr);
}

namespace {
template <int DH>
cudaError_t launch_tp(const CUtensorMap& ms, const CUtensorMap& mt, const CUtensorMap& md,
                      const TpParams& p, cudaStream_t st) {
  static bool attr = false;
  cudaError_t e = set_smem(attn_teacher_p_tc_kernel<DH>, TpLayout<DH>::SMEM, attr);
  if (e != cudaSuccess) return e;
  const int64_t n = (int64_t)p.Hkv * p.B * ((p.T + 127) / 128);
  if (n >= (1ll << 31)) return cudaErrorInvalidValue;
  attn_teacher_p_tc_kernel<DH><<<(unsigned)n, TP_THREADS, TpLayout<DH>::SMEM, st>>>(ms, mt, md, p);
  return cudaGetLastError();
}
}  // namespace

cudaError_t launch_attn_teacher_p_tc(const void* qkv_s, int64_t ldq_s, const void* qkv_t,
                                     int64_t ldq_t, int B, int T, int Hq, int Hkv, int dh,
                                     float scale, const float* lse2_t, const float* lse2_s,
                                     int lse_pitch, void* ds, double* part, int* status,
                                     cudaStream_t st) {
  const int64_t N = (int64_t)B * T;
  const int nq = (T + 127) / 128;
  TpParams p{};
  p.T = T;
  p.B = B;
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.lse_pitch = lse_pitch;
  p.npairs = nq * (nq + 1) / 2;
  p.qcol0 = 0;
  p.kcol0 = Hq * dh;
  p.scale = scale;
  p.sl2 = scale * kLog2e;
  p.lse2_t = lse2_t;
  p.lse2_s = lse2_s;
  p.part = part;
  p.status = status;
  if ((reinterpret_cast<uintptr_t>(lse2_t) & 15u) || (reinterpret_cast<uintptr_t>(lse2_s) & 15u) ||
      (lse_pitch % 128) != 0 || ds == nullptr || (reinterpret_cast<uintptr_t>(ds) & 15u) ||
      part == nullptr || (dh != 64 && dh != 128))
    return cudaErrorInvalidValue;
  const uint64_t ds_rows = (uint64_t)B * Hq * p.npairs * 128;
  CUtensorMap ms, mt, md;
  if (!tmap_rows(&ms, qkv_s, ldq_s, N, 128) || !tmap_rows(&mt, qkv_t, ldq_t, N, 128) ||
      !tmap_rows(&md, ds, 128, ds_rows, 128) || ds_rows >= (1ull << 31))
    return cudaErrorInvalidValue;
  return dh == 128 ? launch_tp<128>(ms, mt, md, p, st) : launch_tp<64>(ms, mt, md, p, st);
}

}  // namespace jab
