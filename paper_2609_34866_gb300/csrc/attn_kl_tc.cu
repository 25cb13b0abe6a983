// Tensor-core (tcgen05) KL attention-map term of L_JAB (Eq. 3, second term), sm_103a.
//
// For every query row i of every (candidate, sequence, query head), with the teacher's map P (float
// weights) and the student's map Q (quantised weights) over the causally visible keys j:
//
//     KL_i = sum_j P_ij (log P_ij - log Q_ij)
//          = sum_j P_ij (s^T_ij - s^S_ij) + lse^S_i - lse^T_i          (s = scaled scores)
//
// One CTA = 128 query rows of one (candidate, sequence, head); keys in blocks of 128. Both score
// blocks come from TS-form UMMAs whose A operand (the 128 query rows, teacher or student) was
// copied into tensor memory once:
//   S^S_j = Q^S K^S_j^T,  S^T_j = Q^T K^T_j^T            M128 N128 K = d_h
// The elementwise warps keep two online softmaxes in the log2 domain (running maxima m, sums l,
// lazy rescaling when a maximum grows by more than 2^8) and a = sum_j p^T_j (y^T_j - y^S_j) with
// p^T_j = 2^(y^T_j - m^T) and y = s log2(e). The row result is formed from differences only,
//     KL_i / ln 2 = a / l^T + (m^S - m^T) + log2(l^S / l^T),
// so no absolute log-sum-exp (of the size of the scores) is ever subtracted from another: the
// terms are of the size of the score perturbation and the KL, which is second order in it, keeps
// its relative precision.
//   warp 0      TMA: Q^S and Q^T once, then K^S_j and K^T_j (2-stage ring)
//   warp 1      TMEM owner, tcgen05.cp of Q^S / Q^T, UMMA issuer (one thread)
//   warps 2..9  elementwise, 16x256b TMEM shape: four threads share a row (32 of its 128 keys
//               each), two rows per thread
// Outputs: per-row KL (optional) and one fp64 partial per tile, summed in fixed order afterwards.
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
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kRescaleLog2 = 8.f;

template <int DH>
struct KlLayout {
  static constexpr int TILE = 128 * DH * 2;  // 128 rows of fp16
  static constexpr int CHUNK = 128 * 128;    // 64 columns of a 128-row tile (128-byte swizzle)
  static constexpr int QS_OFF = 0, QT_OFF = TILE;
  static constexpr int K_OFF = 2 * TILE;     // stage st: K^S at K_OFF + 2 st TILE, K^T after it
  static constexpr int STAGES = 2;
  static constexpr int BAR_OFF = K_OFF + STAGES * 2 * TILE;
  static constexpr int USED = BAR_OFF + 256 + 1024;
  static constexpr int SMEM = USED > 118 * 1024 ? USED : 118 * 1024;
  static constexpr uint32_t SS_COL = 0, ST_COL = 128, QS_COL = 256, QT_COL = 256 + DH / 2;
  static_assert(QT_COL + DH / 2 <= 512, "TMEM budget");
  static_assert(USED <= 227 * 1024, "shared memory budget");
};

struct KlBars {
  uint64_t q_full, k_full[2], k_empty[2], s_full, s_empty, drain;
  uint32_t tmem_base;
  int abort;
  double red[EW_WARPS];
};

struct KlParams {
  int T, B, C, Hq, Hkv, D, nqb, nP;
  float sl2;           // softmax scale * log2(e)
  double* part;        // [C, B, Hq, nP]  sum of KL_i over the tile's rows
  float* kl_rows;      // [C, B, Hq, T] or null
  int* status;
};

__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = tc::globaltimer();
  while (!tc::mbar_test(bar, parity))
    if (tc::globaltimer() - t0 > tc::kWaitLimitNs) break;
}

// Row maxima of one score block: rows A (x[h][4n + 0, 1]) and B (x[h][4n + 2, 3]) of this thread,
// combined over the four threads that share each row.
__device__ __forceinline__ void row_max(const float (&x)[2][32], float& ma, float& mb) {
  ma = x[0][0];
  mb = x[0][2];
#pragma unroll
  for (int h = 0; h < 2; ++h)
#pragma unroll
    for (int n = 0; n < 8; ++n) {
      ma = tc::fmax3(ma, x[h][4 * n], x[h][4 * n + 1]);
      mb = tc::fmax3(mb, x[h][4 * n + 2], x[h][4 * n + 3]);
    }
  ma = fmaxf(ma, __shfl_xor_sync(0xffffffffu, ma, 1));
  mb = fmaxf(mb, __shfl_xor_sync(0xffffffffu, mb, 1));
  ma = fmaxf(ma, __shfl_xor_sync(0xffffffffu, ma, 2));
  mb = fmaxf(mb, __shfl_xor_sync(0xffffffffu, mb, 2));
}

// Running state of one row: maxima (log2 domain), sums of 2^(y - m) and a.
struct RowState {
  float mt, ms, lt, ls, a;
};

// Moves the running maxima to the block maxima (raw scores bt, bs) when they grow by more than
// 2^8, rescaling the sums accordingly. The same decision is taken by the four threads of a row.
__device__ __forceinline__ void advance_max(RowState& r, float bt, float bs, float sl2) {
  const float nt = fmaxf(r.mt, bt * sl2), ns = fmaxf(r.ms, bs * sl2);
  if (nt > r.mt + kRescaleLog2) {
    const float al = tc::fast_exp2(r.mt - nt);  // 0 for the first block (r.mt = -inf)
    r.lt *= al;
    r.a *= al;
    r.mt = nt;
  }
  if (ns > r.ms + kRescaleLog2) {
    r.ls *= tc::fast_exp2(r.ms - ns);
    r.ms = ns;
  }
}

template <int DH>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    attn_kl_tc_kernel(const __grid_constant__ CUtensorMap tm_s,
                      const __grid_constant__ CUtensorMap tm_t, const KlParams p) {
  using L = KlLayout<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  KlBars* bars = reinterpret_cast<KlBars*>(smem + L::BAR_OFF);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &bars->abort;

  // CTA order: grouped by (sequence x candidate, KV group), so that the CTAs which stream the K blocks
  // of one KV head run close together (read from HBM about once); inside a group query blocks from
  // the last (most keys) to the first, the query heads of the group next to each other.
  const int ratio = p.Hq / p.Hkv;
  const int per_group = ratio * p.nqb;
  const int grp = (int)blockIdx.x / per_group, rem = (int)blockIdx.x - grp * per_group;
  const int qb = p.nqb - 1 - rem / ratio;
  const int g = grp % p.Hkv;
  const int h = g * ratio + rem % ratio;
  const int b = (grp / p.Hkv) % p.B, c = (grp / p.Hkv) / p.B;
  const int q0 = qb * BQ;
  const int nkb = min(qb + 1, (p.T + BK - 1) / BK);
  const int row0 = b * p.T;

  if (threadIdx.x == 0) {
    tc::mbar_init(&bars->q_full, 1);
    for (int i = 0; i < L::STAGES; ++i) {
      tc::mbar_init(&bars->k_full[i], 1);
      tc::mbar_init(&bars->k_empty[i], 1);
    }
    tc::mbar_init(&bars->s_full, 1);
    tc::mbar_init(&bars->s_empty, EW_WARPS);
    tc::mbar_init(&bars->drain, 1);
    bars->abort = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&tm_s);
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
      const int qs_col = c * p.D + h * DH, qt_col = h * DH;
      const int ks_col = c * p.D + (p.Hq + g) * DH, kt_col = (p.Hq + g) * DH;
      uint32_t issued = 0, last_par = 0;
      tc::mbar_expect_tx(&bars->q_full, 2 * L::TILE);
      for (int ch = 0; ch < DH / 64; ++ch) {
        tc::tma_load_2d(smem + L::QS_OFF + ch * L::CHUNK, &tm_s, &bars->q_full, qs_col + ch * 64,
                        row0 + q0);
        tc::tma_load_2d(smem + L::QT_OFF + ch * L::CHUNK, &tm_t, &bars->q_full, qt_col + ch * 64,
                        row0 + q0);
      }
      for (int j = 0; j < nkb; ++j) {
        const int st = j & 1;
        const uint32_t ph = (uint32_t)(j >> 1) & 1u;
        if (!tc::mbar_wait(&bars->k_empty[st], ph ^ 1, abort, p.status)) break;
        uint8_t* ks = smem + L::K_OFF + st * 2 * L::TILE;
        tc::mbar_expect_tx(&bars->k_full[st], 2 * L::TILE);
        for (int ch = 0; ch < DH / 64; ++ch) {
          tc::tma_load_2d(ks + ch * L::CHUNK, &tm_s, &bars->k_full[st], ks_col + ch * 64,
                          row0 + j * BK);
          tc::tma_load_2d(ks + L::TILE + ch * L::CHUNK, &tm_t, &bars->k_full[st], kt_col + ch * 64,
                          row0 + j * BK);
        }
        issued |= 1u << st;
        last_par = (last_par & ~(1u << st)) | (ph << st);
      }
      if (*abort) {
        drain_wait(&bars->q_full, 0);
        for (int st = 0; st < L::STAGES; ++st)
          if (issued & (1u << st)) drain_wait(&bars->k_full[st], (last_par >> st) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {  // ---------------------------------------------------------------- UMMA
      constexpr uint32_t ID_S = tc::idesc_f16(false, BQ, BK);
      bool ok = tc::mbar_wait(&bars->q_full, 0, abort, p.status);
      if (ok) {
        tc::fence_after_sync();
        const uint32_t qs = tc::smem_u32(smem + L::QS_OFF), qt = tc::smem_u32(smem + L::QT_OFF);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint32_t off = (kk >> 2) * L::CHUNK + (kk & 3) * 32;
          tc::tmem_cp_128x256b(tmem + L::QS_COL + kk * 8, tc::sdesc_kmajor_sw128(qs + off));
          tc::tmem_cp_128x256b(tmem + L::QT_COL + kk * 8, tc::sdesc_kmajor_sw128(qt + off));
        }
      }
      for (int j = 0; ok && j < nkb; ++j) {
        const int st = j & 1;
        if (!tc::mbar_wait(&bars->k_full[st], (j >> 1) & 1, abort, p.status) ||
            !tc::mbar_wait(&bars->s_empty, (j & 1) ^ 1, abort, p.status)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        const uint64_t kd_s =
            tc::sdesc_kmajor_sw128(tc::smem_u32(smem + L::K_OFF + st * 2 * L::TILE));
        const uint64_t kd_t =
            tc::sdesc_kmajor_sw128(tc::smem_u32(smem + L::K_OFF + st * 2 * L::TILE + L::TILE));
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint32_t off = (kk >> 2) * L::CHUNK + (kk & 3) * 32;
          tc::umma_f16_ts(tmem + L::SS_COL, tmem + L::QS_COL + kk * 8, tc::sdesc_advance(kd_s, off),
                          ID_S, kk > 0 ? 1u : 0u);
          tc::umma_f16_ts(tmem + L::ST_COL, tmem + L::QT_COL + kk * 8, tc::sdesc_advance(kd_t, off),
                          ID_S, kk > 0 ? 1u : 0u);
        }
        tc::umma_commit(&bars->s_full);
        tc::umma_commit(&bars->k_empty[st]);
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
    const float2 sl2 = make_float2(p.sl2, p.sl2);
    RowState ra{-INFINITY, -INFINITY, 0.f, 0.f, 0.f}, rb{-INFINITY, -INFINITY, 0.f, 0.f, 0.f};
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      if (!tc::mbar_wait(&bars->s_full, j & 1, abort, p.status)) {
        ok = false;
        break;
      }
      tc::fence_after_sync();
      // xs / xt[hh][4n + e]: e < 2 row A, key 128 j + 64 hh + 8n + 2 cq + e; e = 2, 3 row B.
      float xs[2][32], xt[2][32];
      {
        uint32_t r0[32], r1[32], r2[32], r3[32];
        __syncwarp();
        tc::tmem_ld_16x256b_x8(tmem + lane16 + L::SS_COL, r0);
        tc::tmem_ld_16x256b_x8(tmem + lane16 + L::SS_COL + 64, r1);
        tc::tmem_ld_16x256b_x8(tmem + lane16 + L::ST_COL, r2);
        tc::tmem_ld_16x256b_x8(tmem + lane16 + L::ST_COL + 64, r3);
        tc::tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          xs[0][i] = __uint_as_float(r0[i]);
          xs[1][i] = __uint_as_float(r1[i]);
          xt[0][i] = __uint_as_float(r2[i]);
          xt[1][i] = __uint_as_float(r3[i]);
        }
      }
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->s_empty);  // the next block's scores may overwrite
      const int k0 = j * BK + 2 * cq;
      const bool masked = j * BK + BK - 1 > q0 || j * BK + BK > p.T;  // diagonal or ragged block
      if (masked) {
#pragma unroll
        for (int hh = 0; hh < 2; ++hh)
#pragma unroll
          for (int n = 0; n < 8; ++n)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int key = k0 + 64 * hh + 8 * n + e;
              if (key > tA || key >= p.T) xs[hh][4 * n + e] = xt[hh][4 * n + e] = -INFINITY;
              if (key > tB || key >= p.T) xs[hh][4 * n + 2 + e] = xt[hh][4 * n + 2 + e] = -INFINITY;
            }
      }
      float btA, btB, bsA, bsB;
      row_max(xt, btA, btB);
      row_max(xs, bsA, bsB);
      advance_max(ra, btA, bsA, p.sl2);
      advance_max(rb, btB, bsB, p.sl2);
      const float2 nmtA = make_float2(tc::neg_bits(ra.mt), tc::neg_bits(ra.mt));
      const float2 nmsA = make_float2(tc::neg_bits(ra.ms), tc::neg_bits(ra.ms));
      const float2 nmtB = make_float2(tc::neg_bits(rb.mt), tc::neg_bits(rb.mt));
      const float2 nmsB = make_float2(tc::neg_bits(rb.ms), tc::neg_bits(rb.ms));
      float2 ltA = make_float2(0.f, 0.f), lsA = ltA, aA = ltA, ltB = ltA, lsB = ltA, aB = ltA;
#pragma unroll
      for (int hh = 0; hh < 2; ++hh)
#pragma unroll
        for (int n = 0; n < 8; ++n) {
          const float2 tA2 = make_float2(xt[hh][4 * n], xt[hh][4 * n + 1]);
          const float2 sA2 = make_float2(xs[hh][4 * n], xs[hh][4 * n + 1]);
          const float2 tB2 = make_float2(xt[hh][4 * n + 2], xt[hh][4 * n + 3]);
          const float2 sB2 = make_float2(xs[hh][4 * n + 2], xs[hh][4 * n + 3]);
          const float2 etA = tc::fma2(tA2, sl2, nmtA), esA = tc::fma2(sA2, sl2, nmsA);
          const float2 etB = tc::fma2(tB2, sl2, nmtB), esB = tc::fma2(sB2, sl2, nmsB);
          const float2 ptA = make_float2(tc::fast_exp2(etA.x), tc::fast_exp2(etA.y));
          const float2 psA = make_float2(tc::fast_exp2(esA.x), tc::fast_exp2(esA.y));
          const float2 ptB = make_float2(tc::fast_exp2(etB.x), tc::fast_exp2(etB.y));
          const float2 psB = make_float2(tc::fast_exp2(esB.x), tc::fast_exp2(esB.y));
          float2 dA = tc::mul2(tc::sub2(tA2, sA2), sl2), dB = tc::mul2(tc::sub2(tB2, sB2), sl2);
          if (masked) {  // masked keys: -inf - (-inf) is NaN; their weight p^T is 0
            dA = make_float2(fmaxf(dA.x, -1e30f), fmaxf(dA.y, -1e30f));
            dB = make_float2(fmaxf(dB.x, -1e30f), fmaxf(dB.y, -1e30f));
          }
          ltA = tc::add2(ltA, ptA);
          lsA = tc::add2(lsA, psA);
          aA = tc::fma2(ptA, dA, aA);
          ltB = tc::add2(ltB, ptB);
          lsB = tc::add2(lsB, psB);
          aB = tc::fma2(ptB, dB, aB);
        }
      ra.lt += ltA.x + ltA.y;
      ra.ls += lsA.x + lsA.y;
      ra.a += aA.x + aA.y;
      rb.lt += ltB.x + ltB.y;
      rb.ls += lsB.x + lsB.y;
      rb.a += aB.x + aB.y;
    }
    // Row results: sums over the four threads of each row, then the difference form above.
    double acc = 0.0;
    if (ok) {
#pragma unroll
      for (int o = 1; o <= 2; o <<= 1) {
        ra.lt += __shfl_xor_sync(0xffffffffu, ra.lt, o);
        ra.ls += __shfl_xor_sync(0xffffffffu, ra.ls, o);
        ra.a += __shfl_xor_sync(0xffffffffu, ra.a, o);
        rb.lt += __shfl_xor_sync(0xffffffffu, rb.lt, o);
        rb.ls += __shfl_xor_sync(0xffffffffu, rb.ls, o);
        rb.a += __shfl_xor_sync(0xffffffffu, rb.a, o);
      }
      const float klA =
          kLn2 * (__fdiv_rn(ra.a, ra.lt) + (ra.ms - ra.mt) + log2f(__fdiv_rn(ra.ls, ra.lt)));
      const float klB =
          kLn2 * (__fdiv_rn(rb.a, rb.lt) + (rb.ms - rb.mt) + log2f(__fdiv_rn(rb.ls, rb.lt)));
      if (cq == 0) {
        const int64_t rbase = (((int64_t)c * p.B + b) * p.Hq + h) * p.T;
        const int64_t ext_r = (int64_t)p.C * p.B * p.Hq * p.T;
        if (tA < p.T) {
          acc += (double)klA;
          if (p.kl_rows && in_bounds(rbase + tA, ext_r, p.status)) p.kl_rows[rbase + tA] = klA;
        }
        if (tB < p.T) {
          acc += (double)klB;
          if (p.kl_rows && in_bounds(rbase + tB, ext_r, p.status)) p.kl_rows[rbase + tB] = klB;
        }
      }
    }
    acc = warp_sum(acc);
    if (lane == 0) bars->red[warp - 2] = acc;
    tc::named_bar_sync(1, EW_WARPS * 32);  // every elementwise warp reaches this exactly once
    if (warp == 2 && lane == 0 && ok) {
      double tot = 0.0;
      for (int w = 0; w < EW_WARPS; ++w) tot += bars->red[w];
      const int64_t pi = (((int64_t)c * p.B + b) * p.Hq + h) * p.nP + qb;
      if (in_bounds(pi, (int64_t)p.C * p.B * p.Hq * p.nP, p.status)) p.part[pi] = tot;
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
cudaError_t launch_kl(const CUtensorMap& ts, const CUtensorMap& tt, const KlParams& p,
                      cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(attn_kl_tc_kernel<DH>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         KlLayout<DH>::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int64_t n = (int64_t)p.Hq * p.B * p.C * p.nqb;
  if (n >= (1ll << 31)) return cudaErrorInvalidValue;
  const dim3 grid((unsigned)n);
  attn_kl_tc_kernel<DH><<<grid, NUM_THREADS, KlLayout<DH>::SMEM, st>>>(ts, tt, p);
  return cudaGetLastError();
}

}  // namespace

int attn_kl_tc_rows() { return BQ; }

cudaError_t launch_attn_kl_tc(const void* qkv_s, int64_t ldq, const void* qkv_t, int B, int T,
                              int C, int Hq, int Hkv, int dh, float scale, double* part, int nP,
                              float* kl_rows, int* status, cudaStream_t st) {
  const int D = (Hq + 2 * Hkv) * dh;
  const int64_t N = (int64_t)B * T;
  CUtensorMap ts, tt;
  if (!tmap_fp16(&ts, qkv_s, (uint64_t)ldq, (uint64_t)N) ||
      !tmap_fp16(&tt, qkv_t, (uint64_t)D, (uint64_t)N))
    return cudaErrorInvalidValue;
  KlParams p{};
  p.T = T;
  p.B = B;
  p.C = C;
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.D = D;
  p.nqb = (T + BQ - 1) / BQ;
  p.nP = nP;
  p.sl2 = scale * kLog2e;
  p.part = part;
  p.kl_rows = kl_rows;
  p.status = status;
  if (p.nqb > nP) return cudaErrorInvalidValue;
  return dh == 128 ? launch_kl<128>(ts, tt, p, st) : launch_kl<64>(ts, tt, p, st);
}

}  // namespace jab
