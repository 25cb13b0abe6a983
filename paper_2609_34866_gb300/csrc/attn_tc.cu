// Tensor-core (tcgen05) causal GQA flash attention with the L_JAB epilogue, sm_103a.
//
// One persistent kernel (below) for every GQA ratio: a tile is 128 query rows, either 64 rows of
// two query heads of one KV group stacked (even ratio: both heads read every K/V tile) or 128 rows
// of one head. Per mode the epilogue writes
//     mode 0 (teacher)  A_ref = O (fp32), lse, partial ||A||^2
//     mode 1 (loss)     partial SSE = sum (O - A_ref)^2                     (Eq. 3)
//     mode 2 (loss+bwd) also dO = O - A_ref (fp16), lse in log2 units, D = rowsum(dO * O)
// The SSE partials are per (candidate, sequence, head, tile rows), fp64, reduced in fixed order.
#include <cudaTypedefs.h>

#include <algorithm>

#include "kernels.h"
#include "tc.cuh"

namespace jab {
namespace {

constexpr int BQ = 128;          // query rows of a tile
constexpr int EW_WARPS = 8;      // softmax warps
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kRescaleLog2 = 8.f;  // rescale O only when the row max grows by more than 2^8

struct FwdParams {
  int T, B, C, Hq, Hkv, D, nqb, nP, lse_pitch;
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

// ============================================================================ attention kernel
// Persistent: one CTA per SM takes tiles in the order of sched_tile. With two heads per tile (HPT =
// 2) a tile is 64 query rows of two query heads of one KV group (GQA: both read the same K and V)
// stacked into the 128 rows of every UMMA: TMEM lane r < 64 is row q0 + r of head h0, lane 64 + r
// is row q0 + r of head h0 + 1. With one head per tile (HPT = 1, any GQA ratio) lane r is row
// q0 + r of head h0.
// Keys come in blocks of 128 so that both products are M128 N128 UMMAs with the A operand in
// tensor memory (TS form), the shape that runs the tensor pipe at full rate on sm_103a:
//   S_j = Q K_j^T     A = Q (TMEM, copied from the TMA-loaded smem tile by tcgen05.cp), B = K_j
//   O  += P_j V_j     A = P_j (TMEM, fp16 pairs written by the softmax threads), B = V_j (smem,
//                     MN-major)
// TMEM columns: S at 0 (128 columns; the softmax reads a block out at once, after which S_{j+1}
// may overwrite it), O double-buffered by tile parity at 128 / 128 + DH, Q (DH / 2 columns) and P
// (64 columns) after them. With two O buffers the epilogue of tile i runs on its own warps while the
// softmax warps already work on tile i + 1.
//   warp 0       TMA: Q tile, K ring (3 stages: a K load is issued once S two blocks back has
//                completed and must land before S of the block after next)
//   warp 1       TMEM owner, tcgen05.cp of Q, UMMA issuer (one thread): S, and for d_h = 64 also
//                P V; for d_h = 128 warp 15 issues P V (two issuers, so that S of the next block
//                is not held back behind the issue of P V, and vice versa)
//   warps 2..9   softmax: warp (quarter q, half h) owns the 16 rows at lanes 32 q + 16 h; with the
//                16x256b TMEM shape four threads share a row (32 of its 128 scores each, two rows per
//                thread), so row maxima and sums need only warp shuffles. Lazy rescaling as in the
//                single-head kernel. At the end of a tile the row statistics go to shared memory.
//   warp 10      TMA: V ring (2 stages), so that K loads never queue behind a V stage that is busy
//   warps 11..14 epilogue, one TMEM lane quarter each (32x32b shape, one row per thread, 32 columns
//                at a time): O is staged through shared memory so that A_ref loads and dO / A
//                stores are coalesced; per-mode outputs and the SSE partials. Each thread
//                prefetches its row of the next tile's A_ref into L2 a whole tile ahead.
constexpr int SQ = 64, SKB = 128, SK_ST = 3, SV_ST = 2;
// d_h = 128: S and P V are issued by two threads (warp 1 and PV_WARP), so that S of the next block
// never waits behind the issue of the current P V. d_h = 64: one issuer (measured faster there).
template <int DH> struct Issue {
  static constexpr bool kSplit = DH == 128;
  static constexpr int kThreads = kSplit ? 512 : 480;
};
constexpr int PV_WARP = 15;
constexpr int EPI_WARPS = 4, EPI_WARP0 = 11;

struct StackBars {
  uint64_t q_full, q_empty, k_full[SK_ST], k_empty[SK_ST], v_full[SV_ST], v_empty[SV_ST];
  uint64_t s_full, s_empty, p_full, pv_done, o_full[2], o_empty[2], st_full[2], st_empty[2];
  uint64_t drain, drain_pv;
  uint32_t tmem_base;
  int abort;
  double red[2][EPI_WARPS];         // [tile parity][epilogue warp]
  float row_m[2][128], row_l[2][128];  // [tile parity][stacked row]: running max (log2), sum
};

template <int DH>
struct StackLayout {
  static constexpr int CHUNK = 128 * 128;  // 64 columns of a 128-row tile (128-byte swizzle)
  static constexpr int TILE = 128 * DH * 2;
  static constexpr int Q_OFF = 0;
  static constexpr int K_OFF = Q_OFF + TILE;
  static constexpr int V_OFF = K_OFF + SK_ST * TILE;
  static constexpr int EPI_OFF = V_OFF + SV_ST * TILE;  // per epilogue warp: 32 x 32 fp32
  static constexpr int BAR_OFF = EPI_OFF + EPI_WARPS * 4096;
  static constexpr int USED = BAR_OFF + (int)sizeof(StackBars) + 1024;
  static constexpr int SMEM = USED > 118 * 1024 ? USED : 118 * 1024;
  static constexpr uint32_t S_COL = 0, O_COL = SKB, Q_COL = SKB + 2 * DH,
                            P_COL = SKB + 2 * DH + DH / 2;
  static_assert(P_COL + SKB / 2 <= 512, "TMEM budget");
};

struct StackTile {
  int hu, bc, qb, nkb;  // head unit (HPT consecutive query heads), sequence x candidate, row block
};

// Tile k: grouped by (sequence x candidate, KV group), so that the tiles which stream the K and V
// blocks of one KV head run close together (K and V read from HBM about once); inside a group query
// blocks from the last (most key blocks) to the first, the head units of the group next to each
// other. rph = query rows per head in a tile; units (query heads / HPT) is a multiple of Hkv.
__device__ __forceinline__ StackTile stack_tile(int k, int units, int Hkv, int nqb, int T, int rph) {
  const int upg = units / Hkv;  // head units per KV group
  const int per_group = upg * nqb;
  const int grp = k / per_group, rem = k - grp * per_group;
  StackTile t;
  t.hu = (grp % Hkv) * upg + rem % upg;
  t.bc = grp / Hkv;
  t.qb = nqb - 1 - rem / upg;
  t.nkb = (min((t.qb + 1) * rph, T) + SKB - 1) / SKB;
  return t;
}

// HPT = query heads per tile: 2 stacks 64 rows of two heads of one KV group (even GQA ratio), 1
// takes 128 rows of one head (any ratio, e.g. GPT-2's separate heads).
template <int DH, int MODE, int HPT>
__global__ void __launch_bounds__(Issue<DH>::kThreads, 1)
    attn_fwd_pair_kernel(const __grid_constant__ CUtensorMap tm_q,
                         const __grid_constant__ CUtensorMap tm_kv, const FwdParams p) {
  using L = StackLayout<DH>;
  constexpr int RPH = 128 / HPT;  // query rows of each head in a tile
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  StackBars* bars = reinterpret_cast<StackBars*>(smem + L::BAR_OFF);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &bars->abort;
  const int units = p.Hq / HPT, BC = p.B * p.C;
  const int nqb = (p.T + RPH - 1) / RPH;
  const int ntiles = units * BC * nqb;
  const int ratio = p.Hq / p.Hkv;

  if (threadIdx.x == 0) {
    tc::mbar_init(&bars->q_full, 1);
    tc::mbar_init(&bars->q_empty, 1);
    for (int i = 0; i < SK_ST; ++i) {
      tc::mbar_init(&bars->k_full[i], 1);
      tc::mbar_init(&bars->k_empty[i], 1);
    }
    for (int i = 0; i < SV_ST; ++i) {
      tc::mbar_init(&bars->v_full[i], 1);
      tc::mbar_init(&bars->v_empty[i], 1);
    }
    tc::mbar_init(&bars->s_full, 1);
    tc::mbar_init(&bars->s_empty, EW_WARPS);
    tc::mbar_init(&bars->p_full, EW_WARPS);
    tc::mbar_init(&bars->pv_done, 1);
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&bars->o_full[i], 1);
      tc::mbar_init(&bars->o_empty[i], EPI_WARPS);
      tc::mbar_init(&bars->st_full[i], EW_WARPS);
      tc::mbar_init(&bars->st_empty[i], EPI_WARPS);
    }
    tc::mbar_init(&bars->drain, 1);
    tc::mbar_init(&bars->drain_pv, 1);
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

  if (warp == 0 || warp == 10) {
    if (lane == 0) {  // ------------------------------------------------ TMA: Q and K (warp 0), V (10)
      const bool is_v = warp == 10;
      int gi = 0, tc_ = 0;
      uint32_t iss = 0, par = 0, qiss = 0, qpar = 0;
      bool ok = true;
      uint64_t* full = is_v ? bars->v_full : bars->k_full;
      uint64_t* empty = is_v ? bars->v_empty : bars->k_empty;
      uint8_t* ring = smem + (is_v ? L::V_OFF : L::K_OFF);
      const int NST = is_v ? SV_ST : SK_ST;
      for (int it = 0, k = sched_tile(0, gridDim.x, blockIdx.x); ok && k < ntiles;
           k = sched_tile(++it, gridDim.x, blockIdx.x), ++tc_) {
        const StackTile tl = stack_tile(k, units, p.Hkv, nqb, p.T, RPH);
        const int b = tl.bc % p.B, c = tl.bc / p.B, h0 = HPT * tl.hu, g = h0 / ratio;
        const int row0 = b * p.T, q0 = tl.qb * RPH;
        const int col = c * p.D + (is_v ? p.Hq + p.Hkv + g : p.Hq + g) * DH;
        if (!is_v) {
          if (!tc::mbar_wait(&bars->q_empty, (tc_ & 1) ^ 1, abort, p.status)) break;
          tc::mbar_expect_tx(&bars->q_full, L::TILE);
          for (int ch = 0; ch < DH / 64; ++ch)
            for (int hd = 0; hd < HPT; ++hd)
              tc::tma_load_2d(smem + L::Q_OFF + ch * L::CHUNK + hd * RPH * 128, &tm_q, &bars->q_full,
                              c * p.D + (h0 + hd) * DH + ch * 64, row0 + q0);
          qiss = 1;
          qpar = tc_ & 1;
        }
        for (int j = 0; j < tl.nkb; ++j, ++gi) {
          const int st = gi % NST;
          const uint32_t ph = (gi / NST) & 1;
          if (!tc::mbar_wait(&empty[st], ph ^ 1, abort, p.status)) { ok = false; break; }
          tc::mbar_expect_tx(&full[st], L::TILE);
          for (int ch = 0; ch < DH / 64; ++ch)
            tc::tma_load_2d(ring + st * L::TILE + ch * L::CHUNK, &tm_kv, &full[st], col + ch * 64,
                            row0 + j * SKB);
          iss |= 1u << st;
          par = (par & ~(1u << st)) | (ph << st);
        }
      }
      if (*abort) {
        if (qiss) drain_wait(&bars->q_full, qpar);
        for (int st = 0; st < NST; ++st)
          if (iss & (1u << st)) drain_wait(&full[st], (par >> st) & 1);
      }
    }
  } else if (warp == 1 || (Issue<DH>::kSplit && warp == PV_WARP)) {
    if (lane == 0) {  // ------------------------------------------ UMMA: S (warp 1), P V (PV_WARP)
      constexpr uint32_t ID_S = tc::idesc_f16(false, 128, SKB);
      constexpr uint32_t ID_PV = tc::idesc_f16(false, 128, DH) | (1u << 16);  // B = V, MN-major
      int g0 = 0, tc_ = 0;
      bool ok = true;
      // S of global block gg, once the softmax has read S_{gg-1} out of tensor memory.
      auto issue_s = [&](int gg) -> bool {
        const int ks = gg % SK_ST;
        if (!tc::mbar_wait(&bars->k_full[ks], (gg / SK_ST) & 1, abort, p.status)) return false;
        if (!tc::mbar_wait(&bars->s_empty, (gg & 1) ^ 1, abort, p.status)) return false;
        tc::fence_after_sync();
        const uint64_t kd = tc::sdesc_kmajor_sw128(tc::smem_u32(smem + L::K_OFF + ks * L::TILE));
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk)
          tc::umma_f16_ts(tmem + L::S_COL, tmem + L::Q_COL + kk * 8,
                          tc::sdesc_advance(kd, (kk >> 2) * L::CHUNK + (kk & 3) * 32), ID_S,
                          kk > 0 ? 1u : 0u);
        tc::umma_commit(&bars->s_full);
        tc::umma_commit(&bars->k_empty[ks]);
        return true;
      };
      // P V of global block gg into the O buffer of tile tc_; the tile's first one waits until the
      // epilogue has read that buffer's previous tile out.
      auto issue_pv = [&](int gg, bool first) -> bool {
        const int vs = gg % SV_ST, ob = tc_ & 1;
        if (!tc::mbar_wait(&bars->v_full[vs], (gg / SV_ST) & 1, abort, p.status)) return false;
        if (!tc::mbar_wait(&bars->p_full, gg & 1, abort, p.status)) return false;
        if (first && tc_ >= 2 &&
            !tc::mbar_wait(&bars->o_empty[ob], ((tc_ >> 1) - 1) & 1, abort, p.status))
          return false;
        tc::fence_after_sync();
        const uint64_t vd =
            tc::sdesc_mnmajor_sw128(tc::smem_u32(smem + L::V_OFF + vs * L::TILE), L::CHUNK, 1024);
#pragma unroll
        for (int k = 0; k < SKB / 16; ++k)
          tc::umma_f16_ts(tmem + L::O_COL + ob * DH, tmem + L::P_COL + k * 8,
                          tc::sdesc_advance(vd, k * 16 * 128), ID_PV, (!first || k > 0) ? 1u : 0u);
        tc::umma_commit(&bars->pv_done);
        tc::umma_commit(&bars->v_empty[vs]);
        return true;
      };
      // Q of tile t into TMEM (its TMA load landed; the previous Q is no longer read).
      auto load_q = [&](int t) -> bool {
        if (!tc::mbar_wait(&bars->q_full, t & 1, abort, p.status)) return false;
        tc::fence_after_sync();
        const uint32_t q_base = tc::smem_u32(smem + L::Q_OFF);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk)
          tc::tmem_cp_128x256b(tmem + L::Q_COL + kk * 8,
                               tc::sdesc_kmajor_sw128(q_base + (kk >> 2) * L::CHUNK + (kk & 3) * 32));
        tc::umma_commit(&bars->q_empty);
        return true;
      };
      // S runs one block ahead of P V, across tile boundaries too: the next tile's Q and first S
      // are issued before this tile's last P V, so the softmax finds S ready when it starts the
      // next tile. The new Q may replace the old one once the softmax has read this tile's last S
      // (that S has then completed).
      int it = 0, k = sched_tile(0, gridDim.x, blockIdx.x);
      if (warp == 1) {
        if (k < ntiles) ok = load_q(0) && issue_s(0);
        while (ok && k < ntiles) {
          const StackTile tl = stack_tile(k, units, p.Hkv, nqb, p.T, RPH);
          const int kn = sched_tile(it + 1, gridDim.x, blockIdx.x);
          for (int j = 0; ok && j < tl.nkb; ++j) {
            const int gg = g0 + j;
            if (j + 1 < tl.nkb) {
              ok = issue_s(gg + 1);
            } else if (kn < ntiles) {
              ok = tc::mbar_wait(&bars->s_empty, gg & 1, abort, p.status) && load_q(tc_ + 1) &&
                   issue_s(gg + 1);
            }
            if (!Issue<DH>::kSplit) ok = ok && issue_pv(gg, j == 0);
          }
          if (!ok) break;
          if (!Issue<DH>::kSplit) tc::umma_commit(&bars->o_full[tc_ & 1]);
          g0 += tl.nkb;
          ++tc_;
          k = kn;
          ++it;
        }
      } else {
        while (ok && k < ntiles) {
          const StackTile tl = stack_tile(k, units, p.Hkv, nqb, p.T, RPH);
          for (int j = 0; ok && j < tl.nkb; ++j) ok = issue_pv(g0 + j, j == 0);
          if (!ok) break;
          tc::umma_commit(&bars->o_full[tc_ & 1]);
          g0 += tl.nkb;
          ++tc_;
          k = sched_tile(++it, gridDim.x, blockIdx.x);
        }
      }
      uint64_t* dr = warp == 1 ? &bars->drain : &bars->drain_pv;
      tc::umma_commit(dr);
      drain_wait(dr, 0);
    }
  } else if (warp < EPI_WARP0) {  // ------------------------------------------------------ softmax
    const int quarter = warp & 3;
    const int half = (warp - 2) >> 2;
    const int cq = lane & 3;                                   // column pair within each 8 columns
    const int rA = quarter * 32 + half * 16 + (lane >> 2);     // stacked rows of this thread
    const int rB = rA + 8;
    const uint32_t lane16 = (uint32_t)(quarter * 32 + half * 16) << 16;
    int g = 0, tc_ = 0;
    for (int it = 0, k = sched_tile(0, gridDim.x, blockIdx.x); k < ntiles;
         k = sched_tile(++it, gridDim.x, blockIdx.x), ++tc_) {
      if (*abort) break;
      const StackTile tl = stack_tile(k, units, p.Hkv, nqb, p.T, RPH);
      const int q0 = tl.qb * RPH;
      const int tA = q0 + (rA & (RPH - 1)), tB = q0 + (rB & (RPH - 1));
      const uint32_t o_col = L::O_COL + (tc_ & 1) * DH;
      float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;
      bool ok = true;
      for (int j = 0; j < tl.nkb; ++j, ++g) {
        if (!tc::mbar_wait(&bars->s_full, g & 1, abort, p.status)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        // x[0]: columns 0..63, x[1]: 64..127; x[h][4n + e] for e < 2 is row A, column
        // 64 h + 8n + 2 cq + e; e = 2, 3 the same columns of row B.
        float x[2][32];
        {
          uint32_t r0[32], r1[32];
          __syncwarp();
          tc::tmem_ld_16x256b_x8(tmem + lane16 + L::S_COL, r0);
          tc::tmem_ld_16x256b_x8(tmem + lane16 + L::S_COL + 64, r1);
          tc::tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            x[0][i] = __uint_as_float(r0[i]);
            x[1][i] = __uint_as_float(r1[i]);
          }
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&bars->s_empty);  // S_{g+1} may overwrite the columns
        const int k0 = j * SKB + 2 * cq;
        if (j * SKB + SKB - 1 > q0 || j * SKB + SKB > p.T) {  // diagonal or ragged block: mask
#pragma unroll
          for (int hh = 0; hh < 2; ++hh)
#pragma unroll
            for (int n = 0; n < 8; ++n)
#pragma unroll
              for (int e = 0; e < 2; ++e) {
                const int key = k0 + 64 * hh + 8 * n + e;
                if (key > tA || key >= p.T) x[hh][4 * n + e] = -INFINITY;
                if (key > tB || key >= p.T) x[hh][4 * n + 2 + e] = -INFINITY;
              }
        }
        float mxA = x[0][0], mxB = x[0][2];
#pragma unroll
        for (int hh = 0; hh < 2; ++hh)
#pragma unroll
          for (int n = 0; n < 8; ++n) {
            mxA = tc::fmax3(mxA, x[hh][4 * n], x[hh][4 * n + 1]);
            mxB = tc::fmax3(mxB, x[hh][4 * n + 2], x[hh][4 * n + 3]);
          }
        mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, 1));
        mxB = fmaxf(mxB, __shfl_xor_sync(0xffffffffu, mxB, 1));
        mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, 2));
        mxB = fmaxf(mxB, __shfl_xor_sync(0xffffffffu, mxB, 2));
        // Scores are raw (unscaled) here; the softmax scale times log2(e) is applied in the exponent.
        const float mnA = fmaxf(mA, mxA * p.sl2), mnB = fmaxf(mB, mxB * p.sl2);
        const bool rsA = mnA > mA + kRescaleLog2, rsB = mnB > mB + kRescaleLog2;
        const float muA = rsA ? mnA : mA, muB = rsB ? mnB : mB;
        const float alA = rsA ? tc::fast_exp2(mA - mnA) : 1.f;
        const float alB = rsB ? tc::fast_exp2(mB - mnB) : 1.f;
        // Packed FP32 pairs (two columns of one row) keep the tensor pipe at speed meanwhile.
        const float2 sl2 = make_float2(p.sl2, p.sl2);
        const float2 nmA = make_float2(tc::neg_bits(muA), tc::neg_bits(muA));
        const float2 nmB = make_float2(tc::neg_bits(muB), tc::neg_bits(muB));
        float2 sA = make_float2(0.f, 0.f), sB = make_float2(0.f, 0.f);
#pragma unroll
        for (int hh = 0; hh < 2; ++hh)
#pragma unroll
          for (int n = 0; n < 8; ++n) {
            const float2 ea = tc::fma2(make_float2(x[hh][4 * n], x[hh][4 * n + 1]), sl2, nmA);
            const float2 eb = tc::fma2(make_float2(x[hh][4 * n + 2], x[hh][4 * n + 3]), sl2, nmB);
            x[hh][4 * n] = tc::fast_exp2(ea.x);
            x[hh][4 * n + 1] = tc::fast_exp2(ea.y);
            x[hh][4 * n + 2] = tc::fast_exp2(eb.x);
            x[hh][4 * n + 3] = tc::fast_exp2(eb.y);
            sA = tc::add2(sA, make_float2(x[hh][4 * n], x[hh][4 * n + 1]));
            sB = tc::add2(sB, make_float2(x[hh][4 * n + 2], x[hh][4 * n + 3]));
          }
        lA = lA * alA + (sA.x + sA.y);  // this thread's share of row A; summed over the 4 at the end
        lB = lB * alB + (sB.x + sB.y);
        mA = muA;
        mB = muB;
        uint32_t pw[32];  // P words: pw[2n] row A, pw[2n + 1] row B, column 4n + cq of P
#pragma unroll
        for (int hh = 0; hh < 2; ++hh)
#pragma unroll
          for (int n = 0; n < 8; ++n) {
            pw[2 * (8 * hh + n)] = tc::pack_half2(x[hh][4 * n], x[hh][4 * n + 1]);
            pw[2 * (8 * hh + n) + 1] = tc::pack_half2(x[hh][4 * n + 2], x[hh][4 * n + 3]);
          }
        // P_{g-1} V_{g-1} (and so every earlier P V) must have completed before P is overwritten
        // or O is rescaled.
        if (g > 0 && !tc::mbar_wait(&bars->pv_done, (g - 1) & 1, abort, p.status)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        if (j > 0 && __any_sync(0xffffffffu, rsA || rsB)) {
#pragma unroll 1
          for (int ch = 0; ch < DH / 64; ++ch) {
            uint32_t r[32];
            const uint32_t col = o_col + ch * 64;
            __syncwarp();
            tc::tmem_ld_16x256b_x8(tmem + lane16 + col, r);
            tc::tmem_ld_wait();
            const float2 a2 = make_float2(alA, alA), b2 = make_float2(alB, alB);
#pragma unroll
            for (int n = 0; n < 8; ++n) {
              const float2 ra = tc::mul2(make_float2(__uint_as_float(r[4 * n]), __uint_as_float(r[4 * n + 1])), a2);
              const float2 rb = tc::mul2(make_float2(__uint_as_float(r[4 * n + 2]), __uint_as_float(r[4 * n + 3])), b2);
              r[4 * n] = __float_as_uint(ra.x);
              r[4 * n + 1] = __float_as_uint(ra.y);
              r[4 * n + 2] = __float_as_uint(rb.x);
              r[4 * n + 3] = __float_as_uint(rb.y);
            }
            tc::tmem_st_16x256b_x8(tmem + lane16 + col, r);
          }
        }
        __syncwarp();
        tc::tmem_st_16x128b_x16(tmem + lane16 + L::P_COL, pw);
        tc::tmem_st_wait();
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&bars->p_full);
      }
      // Row statistics for the epilogue warps (the buffer of this tile parity was last read by the
      // epilogue of tile tc_ - 2).
      lA += __shfl_xor_sync(0xffffffffu, lA, 1);
      lB += __shfl_xor_sync(0xffffffffu, lB, 1);
      lA += __shfl_xor_sync(0xffffffffu, lA, 2);
      lB += __shfl_xor_sync(0xffffffffu, lB, 2);
      const int sbf = tc_ & 1;
      if (!ok || (tc_ >= 2 &&
                  !tc::mbar_wait(&bars->st_empty[sbf], ((tc_ >> 1) - 1) & 1, abort, p.status)))
        break;
      if (cq == 0) {
        bars->row_m[sbf][rA] = mA;
        bars->row_l[sbf][rA] = lA;
        bars->row_m[sbf][rB] = mB;
        bars->row_l[sbf][rB] = lB;
      }
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->st_full[sbf]);
    }
  } else if (warp < EPI_WARP0 + EPI_WARPS) {  // ------------------------------------- epilogue
    // Coalesced pass: the warp's 32 rows x 32 columns of O go through shared memory; lane l then
    // handles 16 bytes of rows 4 i + l / 8 (i < 8), eight lanes per 128-byte row segment. In mode 2
    // each lane accumulates its share of D = rowsum(dO * O) for its rows in this layout and the
    // eight lanes of a row add them at the end of the tile (no second pass through the slots).
    const int quarter = warp & 3;
    const int ew = warp - EPI_WARP0;
    const int row = quarter * 32 + lane;  // stacked row = TMEM lane
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    float* stg = reinterpret_cast<float*>(smem + L::EPI_OFF + ew * 4096);
    const int rbase = quarter * 32;
    const int c4 = lane & 7;
    int tc_ = 0;
    uint32_t range_bits = 0;  // mode 2: an fp16 dO value out of range (inf) or NaN
    const int64_t ext_a = (int64_t)p.B * p.T * p.Hq * DH;         // A_ref, A, dO elements
    const int64_t ext_p = (int64_t)p.C * p.B * p.Hq * p.nP;       // loss partials
    // A_ref row segment (DH fp32) of this thread's stacked row of tile k into L2, one line at a time
    auto prefetch_aref = [&](int k) {
      const StackTile tn = stack_tile(k, units, p.Hkv, nqb, p.T, RPH);
      const int tt = tn.qb * RPH + (row & (RPH - 1));
      if (tt >= p.T) return;
      const float* src = p.a_ref + ((int64_t)(tn.bc % p.B) * p.T + tt) * (int64_t)(p.Hq * DH) +
                         (HPT * tn.hu + row / RPH) * DH;
#pragma unroll
      for (int l = 0; l < DH / 32; ++l) tc::prefetch_line_l2(src + 32 * l);
    };
    for (int it = 0, k = sched_tile(0, gridDim.x, blockIdx.x); k < ntiles;
         k = sched_tile(++it, gridDim.x, blockIdx.x), ++tc_) {
      if (*abort) break;
      const StackTile tl = stack_tile(k, units, p.Hkv, nqb, p.T, RPH);
      const int b = tl.bc % p.B, c = tl.bc / p.B;
      const int h = HPT * tl.hu + row / RPH;
      const int q0 = tl.qb * RPH;
      const int t = q0 + (row & (RPH - 1));
      const int row0 = b * p.T;
      if (MODE != 0) {  // A_ref of this tile (the first one) and of the next, a whole tile ahead
        if (it == 0) prefetch_aref(k);
        const int kn = sched_tile(it + 1, gridDim.x, blockIdx.x);
        if (kn < ntiles) prefetch_aref(kn);
      }
      const int ob = tc_ & 1;
      const uint32_t ph = (tc_ >> 1) & 1;
      double acc = 0.0;
      const bool have = tc::mbar_wait(&bars->st_full[ob], ph, abort, p.status) &&
                        tc::mbar_wait(&bars->o_full[ob], ph, abort, p.status);
      if (have) {
        const float m = bars->row_m[ob][row], lt = bars->row_l[ob][row];
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&bars->st_empty[ob]);
        tc::fence_after_sync();
        const float inv_l = __fdiv_rn(1.f, lt);
        float2 sq = make_float2(0.f, 0.f);  // packed partial sum of squares
        float dpart[8];                     // mode 2: this lane's share of D for rows 4 i + lane / 8
#pragma unroll
        for (int i = 0; i < 8; ++i) dpart[i] = 0.f;
        const float2 il2 = make_float2(inv_l, inv_l);
        // A_ref rows of this lane in the coalesced layout (loading them a chunk ahead costs more in
        // register spills than it hides)
        float4 av[8];
        auto load_aref = [&](int ch, float4 (&dst)[8]) {
          const int col = h * DH + ch * 32 + c4 * 4;
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int tt = q0 + ((rbase + 4 * i + (lane >> 3)) & (RPH - 1));
            const int64_t aoff = ((int64_t)row0 + tt) * (int64_t)(p.Hq * DH) + col;
            if (tt < p.T && in_bounds(aoff + 3, ext_a, p.status))
              dst[i] = __ldg(reinterpret_cast<const float4*>(p.a_ref + aoff));
          }
        };
#pragma unroll 1
        for (int ch = 0; ch < DH / 32; ++ch) {
          const int col = h * DH + ch * 32 + c4 * 4;
          if (MODE != 0) load_aref(ch, av);
          {
            uint32_t r[32];
            __syncwarp();
            tc::tmem_ld32(tmem + lane_base + L::O_COL + ob * DH + ch * 32, r);
            tc::tmem_ld_wait();
            if (ch == DH / 32 - 1) {  // O of this buffer is read out: the next-but-one tile may use it
              tc::fence_before_sync();
              __syncwarp();
              if (lane == 0) tc::mbar_arrive(&bars->o_empty[ob]);
            }
#pragma unroll
            for (int v = 0; v < 8; ++v) {
              const float2 lo = tc::mul2(make_float2(__uint_as_float(r[4 * v]), __uint_as_float(r[4 * v + 1])), il2);
              const float2 hi = tc::mul2(make_float2(__uint_as_float(r[4 * v + 2]), __uint_as_float(r[4 * v + 3])), il2);
              *reinterpret_cast<float4*>(stg + lane * 32 + ((v ^ (lane & 7)) << 2)) =
                  make_float4(lo.x, lo.y, hi.x, hi.y);
            }
          }
          __syncwarp();
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int rr = 4 * i + (lane >> 3);
            const float4 ov = *reinterpret_cast<const float4*>(stg + rr * 32 + ((c4 ^ (rr & 7)) << 2));
            const int tt = q0 + ((rbase + rr) & (RPH - 1));
            if (tt >= p.T) continue;
            const int64_t off = ((int64_t)row0 + tt) * (int64_t)(p.Hq * DH) + col;
            if (!in_bounds(off + 3, ext_a, p.status)) continue;
            if (MODE == 0) {
              *reinterpret_cast<float4*>(p.a_out + off) = ov;
              const float2 v01 = make_float2(ov.x, ov.y), v23 = make_float2(ov.z, ov.w);
              sq = tc::fma2(v23, v23, tc::fma2(v01, v01, sq));
            } else {
              const float4 a = av[i];
              const float2 e01 = tc::sub2(make_float2(ov.x, ov.y), make_float2(a.x, a.y));
              const float2 e23 = tc::sub2(make_float2(ov.z, ov.w), make_float2(a.z, a.w));
              sq = tc::fma2(e23, e23, tc::fma2(e01, e01, sq));
              if (MODE == 2) {
                const __half2 a01 = __floats2half2_rn(e01.x, e01.y), a23 = __floats2half2_rn(e23.x, e23.y);
                uint2 u;
                u.x = *reinterpret_cast<const uint32_t*>(&a01);
                u.y = *reinterpret_cast<const uint32_t*>(&a23);
                *reinterpret_cast<uint2*>(p.d_o + off) = u;
                range_bits |= half2_exp_all_ones(u.x) | half2_exp_all_ones(u.y);
                // D = rowsum(dO * O) with dO as stored (fp16-rounded)
                const float2 f01 = __half22float2(a01), f23 = __half22float2(a23);
                const float2 d2 = tc::fma2(f23, make_float2(ov.z, ov.w),
                                           tc::mul2(f01, make_float2(ov.x, ov.y)));
                dpart[i] += d2.x + d2.y;
              }
            }
          }
          __syncwarp();  // the staging slots are rewritten by the next chunk
        }
        if (MODE == 2) {  // the eight lanes of a row (lane / 8 equal) add their shares, fixed tree
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            float v = dpart[i];
            v += __shfl_xor_sync(0xffffffffu, v, 1);
            v += __shfl_xor_sync(0xffffffffu, v, 2);
            v += __shfl_xor_sync(0xffffffffu, v, 4);
            const int rr = 4 * i + (lane >> 3);
            const int tt = q0 + ((rbase + rr) & (RPH - 1));
            const int64_t li = ((int64_t)b * p.Hq + h) * p.lse_pitch + tt;
            if ((lane & 7) == 0 && tt < p.T && in_bounds(li, (int64_t)p.B * p.Hq * p.lse_pitch, p.status))
              p.dvec[li] = v;
          }
        }
        if (MODE != 1 && p.lse != nullptr && t < p.T &&
            in_bounds(((int64_t)b * p.Hq + h) * p.lse_pitch + t, (int64_t)p.B * p.Hq * p.lse_pitch,
                      p.status)) {
          const int64_t li = ((int64_t)b * p.Hq + h) * p.lse_pitch + t;
          p.lse[li] = MODE == 2 ? m + log2f(lt) : (m + log2f(lt)) * kLn2;  // mode 2: log2 units
        }
        acc = (double)sq.x + (double)sq.y;
      }
      acc = warp_sum(acc);
      double* red = bars->red[tc_ & 1];  // alternate by tile
      if (lane == 0) red[ew] = acc;
      tc::named_bar_sync(2, EPI_WARPS * 32);  // every epilogue warp reaches this once per tile
      if (HPT == 2 && lane == 0 && (quarter & 1) == 0 && have) {
        // head hd = row >> 6 has lane quarters 2 hd and 2 hd + 1; quarter q is epilogue warp (q + 1) & 3
        const int hd = row >> 6;
        const double v = red[(2 * hd + 1) & 3] + red[(2 * hd + 2) & 3];
        const int64_t pi = (((int64_t)c * p.B + b) * p.Hq + h) * p.nP + tl.qb;
        if (in_bounds(pi, ext_p, p.status)) p.part[pi] = v;
      }
      if (HPT == 1 && lane == 0 && quarter == 0 && have) {  // one head: all four lane quarters
        const int64_t pi = (((int64_t)c * p.B + b) * p.Hq + h) * p.nP + tl.qb;
        if (in_bounds(pi, ext_p, p.status)) p.part[pi] = ((red[0] + red[1]) + red[2]) + red[3];
      }
      if (!have) break;
    }
    if (MODE == 2 && range_bits) report(p.status, JAB_ERR_RANGE);
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

template <int DH, int MODE, int HPT>
cudaError_t launch_fwd_pair(const CUtensorMap& tq, const CUtensorMap& tkv, const FwdParams& p,
                            int grid, cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(attn_fwd_pair_kernel<DH, MODE, HPT>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         StackLayout<DH>::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  attn_fwd_pair_kernel<DH, MODE, HPT><<<grid, Issue<DH>::kThreads, StackLayout<DH>::SMEM, st>>>(tq,
                                                                                      tkv, p);
  return cudaGetLastError();
}

}  // namespace

int attn_fwd_tc_rows(int Hq, int Hkv) { return (Hq / Hkv) % 2 == 0 ? SQ : BQ; }

cudaError_t launch_attn_fwd_tc(const AttnLaunch& L, int mode) {
  auto fn = encode_fn();
  if (fn == nullptr) return cudaErrorNotSupported;
  const int64_t N = (int64_t)L.B * L.T;
  cuuint64_t dims[2] = {(cuuint64_t)L.ldq, (cuuint64_t)N};
  cuuint64_t strides[1] = {(cuuint64_t)L.ldq * 2};
  cuuint32_t estr[2] = {1, 1};
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
  p.C = L.C;
  // Two heads of one KV group share every K/V tile when the GQA ratio is even (64 rows of each
  // stacked into a tile); otherwise a tile is 128 rows of one head. Same kernel either way.
  const bool pair = (L.Hq / L.Hkv) % 2 == 0;
  const int rph = pair ? SQ : BQ;
  CUtensorMap tq, tkv;
  cuuint32_t box_q[2] = {64, (cuuint32_t)rph};
  cuuint32_t box_kv[2] = {64, (cuuint32_t)SKB};
  if (fn(&tq, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(L.qkv), dims, strides, box_q,
         estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS ||
      fn(&tkv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(L.qkv), dims, strides, box_kv,
         estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 1;
  }
  const int64_t ntiles = (int64_t)(L.Hq / (pair ? 2 : 1)) * L.B * L.C * ((L.T + rph - 1) / rph);
  const int grid = (int)std::min<int64_t>(ntiles, sms);
#define JAB_FWD2(DH_, M_, H_) return launch_fwd_pair<DH_, M_, H_>(tq, tkv, p, grid, L.stream)
  if (pair) {
    if (L.dh == 128) {
      if (mode == 0) JAB_FWD2(128, 0, 2);
      if (mode == 1) JAB_FWD2(128, 1, 2);
      JAB_FWD2(128, 2, 2);
    }
    if (mode == 0) JAB_FWD2(64, 0, 2);
    if (mode == 1) JAB_FWD2(64, 1, 2);
    JAB_FWD2(64, 2, 2);
  }
  if (L.dh == 128) {
    if (mode == 0) JAB_FWD2(128, 0, 1);
    if (mode == 1) JAB_FWD2(128, 1, 1);
    JAB_FWD2(128, 2, 1);
  }
  if (mode == 0) JAB_FWD2(64, 0, 1);
  if (mode == 1) JAB_FWD2(64, 1, 1);
  JAB_FWD2(64, 2, 1);
#undef JAB_FWD2
}

}  // namespace jab
