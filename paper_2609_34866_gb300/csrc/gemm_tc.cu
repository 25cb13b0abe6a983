// Tensor-core (tcgen05) GEMMs of the L_JAB path on sm_103a.
//
//   C[m, n] = sum_k A[m, k] B[n, k]        A K-major 16-bit, fp32 accumulation in TMEM; B K-major
//                                          (stored [n][k]) or MN-major (stored [k][n])
//
// Persistent, warp-specialised kernel on CTA pairs (clusters of two CTAs on two SMs, cta_group::2):
// a pair computes a 256 x 256 tile with M256 N256 K16 UMMAs issued by its even CTA; each CTA holds
// 128 rows of A, half of the B tile and 128 lanes of the accumulator (details above the kernel).
//   warp 0      TMA producer: the CTA's 128x64 A tile and 128x64 half of B per stage, 6-stage ring
//   warp 1      TMEM owner (512 columns, allocated by the pair) and, in the even CTA, UMMA issuer
//   warps 2..5  epilogue: tcgen05.ld of the CTA's 128 x 256 fp32 accumulator, one lane per thread
// Two accumulators (2 x 256 TMEM columns) let the epilogue of one tile overlap the next mainloop.
//
// Epilogues:
//   projection  [Q|K|V] = X w_hat^T: rotate-half RoPE on the Q and K heads (partner column +-d_h/2
//               lives in the same thread's row), fp16 store.
//   wgrad       G = dQKV^T X (K = tokens, split-K): ds[o, g] += coef * sum_{i in g} G[o,i] r[o,i]
//               with the LSQ factor r of Eq. 13 recomputed from w and s; G is never stored. X is
//               read as it is stored, [tokens, features], as the MN-major B operand (two 64-feature
//               TMA boxes per CTA and stage), so no transposed copy of X is needed.
//   store       coef * dQKV^T X as fp32 dW (STE weight gradient) and / or its squared norm; with a
//               split K the partial tiles are added into a zeroed dW with vector atomics and the
//               norm is reduced from dW afterwards in fixed order.
#include <cudaTypedefs.h>

#include "kernels.h"
#include "tc.cuh"

namespace jab {
namespace {

constexpr int BM = 128, BN = 256, BK = 64;  // BM: rows of one CTA (an epilogue's 128 TMEM lanes)
constexpr int A_BYTES = BM * BK * 2;
constexpr int NUM_THREADS = 192;
constexpr uint32_t TMEM_COLS = 2 * BN;

enum EpiKind { kEpiRope = 0, kEpiLsq = 1, kEpiStore = 2 };

struct GemmParams {
  int64_t M;
  int Nn, K;
  int num_m, num_n, splits, k_blocks, group_m;
  int* status;
  // projection epilogue
  half_t* C;
  int D, n_rot, dh, T;
  const float* cos_t;
  const float* sin_t;
  // LSQ epilogue
  const bf16_t* w;
  const float* s;
  int d, G, bits;
  float coef;
  float* ds;
  float* dspart;  // fp32 [splits, M, d/G]: each unit's partial, summed over the splits in order
  // weight-gradient store epilogue (a split K adds partial tiles into a zeroed dw)
  float* dw;
};

__device__ __forceinline__ void decode_unit(const GemmParams& p, int unit, int& mb, int& nb,
                                            int& ks) {
  const int tiles = p.num_m * p.num_n;
  ks = unit / tiles;
  const int t = unit - ks * tiles;
  const int span = p.group_m * p.num_n;
  const int grp = t / span;
  const int first_m = grp * p.group_m;
  const int gm = min(p.group_m, p.num_m - first_m);
  const int local = t - grp * span;
  mb = first_m + local % gm;
  nb = local / gm;
}

__device__ __forceinline__ void k_range(const GemmParams& p, int ks, int& kb0, int& kb1) {
  kb0 = (int)((int64_t)p.k_blocks * ks / p.splits);
  kb1 = (int)((int64_t)p.k_blocks * (ks + 1) / p.splits);
}

// Waits for a barrier phase while draining at exit: time-bounded, ignores the abort flag.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = tc::globaltimer();
  while (!tc::mbar_test(bar, parity)) {
    if (tc::globaltimer() - t0 > tc::kWaitLimitNs) break;
  }
}

__device__ __forceinline__ void epi_rope(const GemmParams& p, uint32_t taddr, int mb, int nb,
                                         int row) {
  const int64_t m = (int64_t)mb * BM + row;
  const bool row_ok = m < p.M;
  const int t = row_ok ? (int)(m % p.T) : 0;
  const int half = p.dh >> 1;
#pragma unroll 1
  for (int pr = 0; pr < BN / 64; ++pr) {
    const int c1 = (p.dh == 128) ? (pr >> 1) * 4 + (pr & 1) : pr * 2;
    const int c2 = c1 + half / 32;
    const int col1 = nb * BN + c1 * 32;
    if (col1 >= p.Nn) continue;  // uniform over the warp
    uint32_t ra[32], rb[32];
    __syncwarp();  // tcgen05.ld is warp-collective (.sync.aligned)
    tc::tmem_ld32(taddr + c1 * 32, ra);
    tc::tmem_ld32(taddr + c2 * 32, rb);
    tc::tmem_ld_wait();
    float a[32], b[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      a[i] = __uint_as_float(ra[i]);
      b[i] = __uint_as_float(rb[i]);
    }
    const int o = col1 % p.D;
    if (p.n_rot > 0 && o < p.n_rot &&
        in_bounds((int64_t)t * half + o % p.dh + 31, (int64_t)p.T * half, p.status)) {
      const int jj0 = o % p.dh;
      const float4* cp = reinterpret_cast<const float4*>(p.cos_t + (int64_t)t * half + jj0);
      const float4* sp = reinterpret_cast<const float4*>(p.sin_t + (int64_t)t * half + jj0);
      // Packed FP32 pairs: this epilogue overlaps the next tile's UMMAs, which scalar FP32
      // instructions at a high rate slow down.
#pragma unroll
      for (int v = 0; v < 8; ++v) {
        const float4 c4 = __ldg(cp + v), s4 = __ldg(sp + v);
#pragma unroll
        for (int e = 0; e < 4; e += 2) {
          const int i = v * 4 + e;
          const float2 cs = e ? make_float2(c4.z, c4.w) : make_float2(c4.x, c4.y);
          const float2 sn = e ? make_float2(s4.z, s4.w) : make_float2(s4.x, s4.y);
          const float2 nsn = make_float2(tc::neg_bits(sn.x), tc::neg_bits(sn.y));
          const float2 x1 = make_float2(a[i], a[i + 1]), x2 = make_float2(b[i], b[i + 1]);
          const float2 ra = tc::fma2(x2, nsn, tc::mul2(x1, cs));  // x1 cos - x2 sin
          const float2 rb = tc::fma2(x1, sn, tc::mul2(x2, cs));   // x2 cos + x1 sin
          a[i] = ra.x;
          a[i + 1] = ra.y;
          b[i] = rb.x;
          b[i + 1] = rb.y;
        }
      }
    }
    if (row_ok && in_bounds(m * p.Nn + col1 + half + 31, p.M * (int64_t)p.Nn, p.status)) {
      uint4* d1 = reinterpret_cast<uint4*>(p.C + m * p.Nn + col1);
      uint4* d2 = reinterpret_cast<uint4*>(p.C + m * p.Nn + col1 + half);
      uint32_t inf_bits = 0;  // a half with all exponent bits set: inf (out of fp16 range) or NaN
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        uint4 u1, u2;
        __half2* h1 = reinterpret_cast<__half2*>(&u1);
        __half2* h2 = reinterpret_cast<__half2*>(&u2);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          h1[e] = __floats2half2_rn(a[v * 8 + 2 * e], a[v * 8 + 2 * e + 1]);
          h2[e] = __floats2half2_rn(b[v * 8 + 2 * e], b[v * 8 + 2 * e + 1]);
        }
        inf_bits |= half2_exp_all_ones(u1.x) | half2_exp_all_ones(u1.y) |
                    half2_exp_all_ones(u1.z) | half2_exp_all_ones(u1.w) |
                    half2_exp_all_ones(u2.x) | half2_exp_all_ones(u2.y) |
                    half2_exp_all_ones(u2.z) | half2_exp_all_ones(u2.w);
        d1[v] = u1;
        d2[v] = u2;
      }
      if (inf_bits) report(p.status, JAB_ERR_RANGE);
    }
  }
}

// STE weight gradient (App. B: d w_hat / d w = 1, so dL/dW = dL/dw_hat = coef * dQKV^T X): the
// tile times coef stored as fp32 rows of dw (with a split K each unit's partial tile is added with
// vector atomics). Packed FP32 pairs, as this runs beside the next tile's UMMAs.
__device__ __forceinline__ void epi_store(const GemmParams& p, uint32_t taddr, int mb, int nb,
                                          int row) {
  const int64_t o = (int64_t)mb * BM + row;  // M = D is a multiple of 128: every row is valid
  const float2 c2 = make_float2(p.coef, p.coef);
#pragma unroll 1
  for (int c = 0; c < BN / 32; ++c) {
    const int i0 = nb * BN + c * 32;
    if (i0 >= p.Nn) break;  // uniform over the warp
    uint32_t r[32];
    __syncwarp();
    tc::tmem_ld32(taddr + c * 32, r);
    tc::tmem_ld_wait();
    float g[32];
#pragma unroll
    for (int i = 0; i < 32; i += 2) {
      const float2 v = tc::mul2(make_float2(__uint_as_float(r[i]), __uint_as_float(r[i + 1])), c2);
      g[i] = v.x;
      g[i + 1] = v.y;
    }
    if (p.dw != nullptr && in_bounds(o * p.Nn + i0 + 31, p.M * (int64_t)p.Nn, p.status)) {
      float4* d = reinterpret_cast<float4*>(p.dw + o * p.Nn + i0);
      if (p.splits > 1) {  // a K range: add the partial tile into the zeroed dw
#pragma unroll
        for (int v = 0; v < 8; ++v)
          atomicAdd(d + v, make_float4(g[4 * v], g[4 * v + 1], g[4 * v + 2], g[4 * v + 3]));
      } else {
#pragma unroll
        for (int v = 0; v < 8; ++v) d[v] = make_float4(g[4 * v], g[4 * v + 1], g[4 * v + 2], g[4 * v + 3]);
      }
    }
  }
}

__device__ __forceinline__ void epi_lsq(const GemmParams& p, uint32_t taddr, int mb, int nb,
                                        int ks, int row) {
  const int o = mb * BM + row;  // M = D is a multiple of 128: every row is valid
  const int qmax = qmax_of(p.bits);
  const int ng = p.d / p.G;
  // one value per (split, row, group): this unit's tile covers whole groups (BN is a multiple of G)
  float* part_out = p.dspart + ((int64_t)ks * p.M + o) * ng;
  const int64_t part_extent = (int64_t)p.splits * p.M * ng;
  float part = 0.f;
  int cur = -1;
#pragma unroll 1
  for (int c = 0; c < BN / 32; ++c) {
    const int i0 = nb * BN + c * 32;
    if (i0 >= p.Nn) break;  // uniform over the warp
    uint32_t r[32];
    __syncwarp();
    tc::tmem_ld32(taddr + c * 32, r);
    tc::tmem_ld_wait();
    const int g = i0 / p.G;
    float acc = 0.f;
    if (in_bounds((int64_t)o * p.d + i0 + 31, (int64_t)p.M * p.d, p.status) &&
        in_bounds((int64_t)o * ng + g, (int64_t)p.M * ng, p.status)) {
      const float sc = __ldg(p.s + (int64_t)o * ng + g);
      const uint4* wp = reinterpret_cast<const uint4*>(p.w + (int64_t)o * p.d + i0);
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        const uint4 u = __ldg(wp + v);
        const bf16_t* wb = reinterpret_cast<const bf16_t*>(&u);
#pragma unroll
        for (int e = 0; e < 8; ++e)
          acc = fmaf(__uint_as_float(r[v * 8 + e]), lsq_factor(__bfloat162float(wb[e]), sc, qmax),
                     acc);
      }
    }
    if (g != cur) {
      if (cur >= 0 && in_bounds(((int64_t)ks * p.M + o) * ng + cur, part_extent, p.status))
        part_out[cur] = p.coef * part;
      part = 0.f;
      cur = g;
    }
    part += acc;
  }
  if (cur >= 0 && in_bounds(((int64_t)ks * p.M + o) * ng + cur, part_extent, p.status))
    part_out[cur] = p.coef * part;
}

// ------------------------------------------------------------------ CTA-pair variant (cta_group::2)
// Two CTAs of a cluster on two SMs share one 256 x 256 tile: CTA r holds rows 128 r .. 128 r + 127
// of A and rows 128 r .. of the B tile (the N half it loads), and its 128 accumulator lanes. One
// M256 N256 K16 UMMA per 16-deep K step, issued by the even CTA, reads A and B from both CTAs' shared
// memory. Each SM then stages 16 KB of A and 16 KB of B per K block instead of the 16 + 32 KB of a
// one-CTA 128 x 256 tile, so six stages fit where four did and the operand loads have 1.7x the
// look-ahead (the one-CTA layout was bound by it: three stages instead of four cost it 10-26 %).
//   warp 0      TMA producer (both CTAs): its rows of A and its half of B, completion counted on the
//               even CTA's stage barrier, which expects both CTAs' bytes
//   warp 1      TMEM owner (both CTAs, allocated collectively); UMMA issuer (even CTA, one thread);
//               each stage's commit releases the stage in both CTAs, each tile's commit wakes both
//               CTAs' epilogues
//   warps 2..5  epilogue (both CTAs): this CTA's 128 rows, as in the single-CTA kernel; the
//               accumulator is free again once all eight epilogue warps of the pair have arrived on
//               the even CTA's barrier
constexpr int STAGES2 = 6;
constexpr int BM2 = 2 * BM;                 // rows of A per pair tile
constexpr int B2_ROWS = BN / 2;             // rows (K-major) or columns (MN-major) of B per CTA
constexpr int B2_BYTES = B2_ROWS * BK * 2;  // 16 KB
constexpr int STAGE2_BYTES = A_BYTES + B2_BYTES;
constexpr int SMEM2_BYTES = STAGES2 * STAGE2_BYTES + 1024 + 256;

struct Bars2 {
  uint64_t full[STAGES2], empty[STAGES2], tfull[2], tempty[2], drain;
  uint32_t tmem_base;
  int abort;
};
static_assert(STAGES2 * STAGE2_BYTES + (int)sizeof(Bars2) <= SMEM2_BYTES - 1024, "shared memory");

template <int EPI, bool BF16, bool B_MN>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm2_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  Bars2* bars = reinterpret_cast<Bars2*>(smem + STAGES2 * STAGE2_BYTES);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = tc::cluster_ctarank();  // 0: issues the pair's UMMAs
  const bool leader = rank == 0;
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  const int total = p.num_m * p.num_n * p.splits;  // num_m counts 256-row blocks here
  volatile int* abort = &bars->abort;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES2; ++s) {
      tc::mbar_init(&bars->full[s], 1);
      tc::mbar_init(&bars->empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      tc::mbar_init(&bars->tfull[a], 1);
      tc::mbar_init(&bars->tempty[a], 2 * 4);  // the epilogue warps of both CTAs
    }
    tc::mbar_init(&bars->drain, 1);
    bars->abort = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&tmA);
    tc::prefetch_tmap(&tmB);
  }
  if (warp == 1) {
    tc::tmem_alloc2(&bars->tmem_base, TMEM_COLS);
    tc::tmem_relinquish2();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  // both CTAs' barriers are initialised and their tensor memory allocated before any signal crosses
  tc::cluster_sync();
  const uint32_t tmem = bars->tmem_base;
  const uint32_t full_lead = tc::mapa_shared(tc::smem_u32(&bars->full[0]), 0);
  const uint32_t tempty_lead = tc::mapa_shared(tc::smem_u32(&bars->tempty[0]), 0);

  if (warp == 0) {
    if (lane == 0) {  // ---------------- TMA producer
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0, last_parity = 0;  // per-stage bitmasks for the exit drain (even CTA)
      for (int unit = pair; unit < total && !*abort; unit += npairs) {
        int mb, nb, ks, kb0, kb1;
        decode_unit(p, unit, mb, nb, ks);
        k_range(p, ks, kb0, kb1);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!tc::mbar_wait(&bars->empty[stage], phase ^ 1, abort, p.status)) break;
          uint8_t* sa = smem + stage * STAGE2_BYTES;
          const uint32_t bar = full_lead + stage * 8;
          if (leader) tc::mbar_expect_tx(&bars->full[stage], 2 * STAGE2_BYTES);
          tc::tma_load_2d_pair(sa, &tmA, bar, kb * BK, mb * BM2 + (int)rank * BM);
          if (B_MN)  // B stored [k][n]: this CTA's two boxes of BK rows x 64 columns
            for (int c = 0; c < B2_ROWS / 64; ++c)
              tc::tma_load_2d_pair(sa + A_BYTES + c * (BK * 128), &tmB, bar,
                                   nb * BN + (int)rank * B2_ROWS + c * 64, kb * BK);
          else
            tc::tma_load_2d_pair(sa + A_BYTES, &tmB, bar, kb * BK, nb * BN + (int)rank * B2_ROWS);
          issued |= 1u << stage;
          last_parity = (last_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES2) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (*abort && leader)  // let every issued copy of the pair land before shared memory goes
        for (int s = 0; s < STAGES2; ++s)
          if (issued & (1u << s)) drain_wait(&bars->full[s], (last_parity >> s) & 1);
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {  // ---------------- UMMA issuer of the pair
      constexpr uint32_t IDESC = tc::idesc_f16(BF16, BM2, BN) | (B_MN ? (1u << 16) : 0u);
      int stage = 0, it = 0;
      uint32_t phase = 0;
      for (int unit = pair; unit < total && !*abort; unit += npairs, ++it) {
        int mb, nb, ks, kb0, kb1;
        decode_unit(p, unit, mb, nb, ks);
        k_range(p, ks, kb0, kb1);
        const int acc = it & 1;
        const uint32_t aphase = (it >> 1) & 1;
        if (!tc::mbar_wait_cluster(&bars->tempty[acc], aphase ^ 1, abort, p.status)) break;
        tc::fence_after_sync();
        const uint32_t d_tmem = tmem + acc * BN;
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!tc::mbar_wait(&bars->full[stage], phase, abort, p.status)) {
            ok = false;
            break;
          }
          tc::fence_after_sync();
          const uint32_t a0 = tc::smem_u32(smem + stage * STAGE2_BYTES);
          const uint32_t b0 = a0 + A_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            tc::umma2_f16(d_tmem, tc::sdesc_kmajor_sw128(a0 + k * 32),
                          B_MN ? tc::sdesc_mnmajor_sw128(b0 + k * 16 * 128, BK * 128, 1024)
                               : tc::sdesc_kmajor_sw128(b0 + k * 32),
                          IDESC, (kb > kb0 || k > 0) ? 1u : 0u);
          tc::umma2_commit_mc(&bars->empty[stage], 0x3);
          if (++stage == STAGES2) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        tc::umma2_commit_mc(&bars->tfull[acc], 0x3);
      }
      tc::umma2_commit_mc(&bars->drain, 0x1);  // every UMMA of the pair has completed once this flips
      drain_wait(&bars->drain, 0);
    }
  } else {  // ---------------- epilogue warps 2..5 (both CTAs)
    const int q = warp & 3;
    const int row = q * 32 + lane;
    int it = 0;
    for (int unit = pair; unit < total && !*abort; unit += npairs, ++it) {
      int mb, nb, ks;
      decode_unit(p, unit, mb, nb, ks);
      const int acc = it & 1;
      const uint32_t aphase = (it >> 1) & 1;
      if (!tc::mbar_wait(&bars->tfull[acc], aphase, abort, p.status)) break;
      tc::fence_after_sync();
      const uint32_t taddr = tmem + ((uint32_t)(q * 32) << 16) + acc * BN;
      const int mb128 = 2 * mb + (int)rank;  // this CTA's 128-row block
      if (EPI == kEpiRope)
        epi_rope(p, taddr, mb128, nb, row);  // masks rows past M itself
      else if ((int64_t)mb128 * BM < p.M) {  // M is a multiple of 128: whole halves are valid or not
        if (EPI == kEpiLsq)
          epi_lsq(p, taddr, mb128, nb, ks, row);
        else
          epi_store(p, taddr, mb128, nb, row);
      }
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) {
        if (leader)
          tc::mbar_arrive(&bars->tempty[acc]);
        else
          tc::mbar_arrive_cluster(tempty_lead + acc * 8);
      }
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  // the pair's UMMAs have completed (the issuer drained) and no arrival is in flight to the other
  // CTA before either frees its tensor memory or exits
  tc::cluster_sync();
  tc::fence_after_sync();
  if (warp == 1) {
    __syncwarp();
    tc::tmem_dealloc2(tmem, TMEM_COLS);
  }
}

// ------------------------------------------------------------------ host side
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

// Row-major [outer, inner] 16-bit matrix with row pitch `pitch` elements; box = box_outer rows of
// 64 elements (128 B, the swizzle span).
bool make_tmap(CUtensorMap* m, const void* base, bool bf16, uint64_t inner, uint64_t outer,
               uint64_t pitch, uint32_t box_outer) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15u) || (pitch * 2) % 16) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {pitch * 2};
  cuuint32_t box[2] = {(cuuint32_t)BK, box_outer};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2,
            const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

// CTA-pair launch: clusters of two, one pair per two SMs (as many pairs as fit at once).
template <int EPI, bool BF16, bool B_MN>
cudaError_t launch_gemm2(const CUtensorMap& ta, const CUtensorMap& tb, GemmParams& p,
                         cudaStream_t st) {
  auto kern = gemm2_tc_kernel<EPI, BF16, B_MN>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM2_BYTES);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = 2;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  cfg.blockDim = dim3(NUM_THREADS);
  cfg.dynamicSmemBytes = SMEM2_BYTES;
  cfg.stream = st;
  const int sms = sm_count();
  // The pairs that fit at once depend only on the kernel and the device: asked once, so that a
  // launch makes no occupancy query (a launch-bound loop pays for every host call).
  static int clusters = 0;
  if (clusters < 1) {
    cfg.gridDim = dim3((unsigned)(sms / 2 * 2));
    if (cudaOccupancyMaxActiveClusters(&clusters, kern, &cfg) != cudaSuccess || clusters < 1)
      clusters = sms / 2;
  }
  const int64_t total = (int64_t)p.num_m * p.num_n * p.splits;
  const int pairs = (int)std::min<int64_t>(total, std::min(clusters, sms / 2));
  cfg.gridDim = dim3((unsigned)(2 * pairs));
  return cudaLaunchKernelEx(&cfg, kern, ta, tb, p);
}

}  // namespace

cudaError_t launch_proj_gemm_tc(const void* A, const void* Bw, void* C, int64_t M, int Nn, int K,
                                int D, int n_rot, int dh, int T, const float* cos_t,
                                const float* sin_t, int* status, cudaStream_t st) {
  CUtensorMap ta, tb;
  if (!make_tmap(&ta, A, false, K, M, K, BM) || !make_tmap(&tb, Bw, false, K, Nn, K, B2_ROWS))
    return cudaErrorInvalidValue;
  GemmParams p{};
  p.M = M;
  p.Nn = Nn;
  p.K = K;
  p.num_m = (int)((M + BM2 - 1) / BM2);  // 256-row blocks: CTA pairs
  p.num_n = (Nn + BN - 1) / BN;
  p.splits = 1;
  p.k_blocks = K / BK;
  p.group_m = 16;  // 16 pair rows = 4096 rows of X and all of W in L2 while the N tiles pass
  p.status = status;
  p.C = static_cast<half_t*>(C);
  p.D = D;
  p.n_rot = n_rot;
  p.dh = dh;
  p.T = T;
  p.cos_t = cos_t;
  p.sin_t = sin_t;
  return launch_gemm2<kEpiRope, false, false>(ta, tb, p, st);
}

// Split K so that the units (tile x K range) fill whole waves of the persistent grid: the makespan
// in k-blocks is ceil(tiles * s / sms) * (k_blocks / s + kFill), kFill standing for a unit's pipeline
// fill and drain. (768 tiles on 152 SMs without a split leave 8 SMs a sixth full-K unit while the
// others idle.) Each unit keeps at least 16 k-blocks; near-ties go to fewer splits (fewer atomics
// and unit boundaries).
int choose_splits(int tiles, int k_blocks, int sms) {
  constexpr double kFill = 8.0;
  int splits = 1;
  double best = (double)((tiles + sms - 1) / sms) * ((double)k_blocks + kFill);
  for (int s = 2; s <= 32 && k_blocks / s >= 16; ++s) {
    const double t = (double)(((int64_t)tiles * s + sms - 1) / sms) * ((double)k_blocks / s + kFill);
    if (t < best * 0.995) {
      best = t;
      splits = s;
    }
  }
  return splits;
}

cudaError_t launch_wgrad_lsq_tc(const void* dqkvt, int64_t ldt, const void* x, const void* w,
                                const float* s, int64_t N, int D, int d, int G, int bits,
                                float coef, float* ds, float* dspart, int* status, cudaStream_t st) {
  CUtensorMap ta, tb;
  if (!make_tmap(&ta, dqkvt, true, N, D, ldt, BM) || !make_tmap(&tb, x, true, d, N, d, BK))
    return cudaErrorInvalidValue;
  GemmParams p{};
  p.M = D;
  p.Nn = d;
  p.K = (int)std::min<int64_t>(N, INT32_MAX);
  p.num_m = (D + BM2 - 1) / BM2;  // 256-row blocks: CTA pairs
  p.num_n = (d + BN - 1) / BN;
  p.k_blocks = (int)((N + BK - 1) / BK);
  p.splits = choose_splits(p.num_m * p.num_n, p.k_blocks, sm_count() / 2);
  p.group_m = 8;
  p.status = status;
  p.w = static_cast<const bf16_t*>(w);
  p.s = s;
  p.d = d;
  p.G = G;
  p.bits = bits;
  p.coef = coef;
  p.ds = ds;
  p.dspart = dspart;
  // every (split, row, group) partial is written once; the splits are summed in order: the scale
  // gradient is bit-identical between calls
  cudaError_t e = launch_gemm2<kEpiLsq, true, true>(ta, tb, p, st);
  if (e != cudaSuccess) return e;
  return launch_split_sum(dspart, p.splits, (int64_t)D * (d / G), ds, st);
}

cudaError_t launch_wgrad_store_tc(const void* dqkvt, int64_t ldt, const void* x, int64_t N, int D,
                                  int d, float coef, float* dw, double* sqnorm, float* scratch,
                                  double* red, bool deterministic, int* status, cudaStream_t st) {
  CUtensorMap ta, tb;
  if (!make_tmap(&ta, dqkvt, true, N, D, ldt, BM) || !make_tmap(&tb, x, true, d, N, d, BK))
    return cudaErrorInvalidValue;
  GemmParams p{};
  p.M = D;
  p.Nn = d;
  p.K = (int)std::min<int64_t>(N, INT32_MAX);
  p.num_m = (D + BM2 - 1) / BM2;  // 256-row blocks: CTA pairs
  p.num_n = (d + BN - 1) / BN;
  p.k_blocks = (int)((N + BK - 1) / BK);
  p.group_m = 8;
  p.status = status;
  p.coef = coef;
  // dW goes to the caller's buffer, or to the scratch when only the norm is asked for. A split K
  // adds the partial tiles into a zeroed dW with atomics (the last bits depend on their order);
  // the deterministic mode keeps one unit per tile.
  const int64_t n_w = (int64_t)D * d;
  float* target = dw != nullptr ? dw : scratch;
  p.splits = deterministic ? 1 : choose_splits(p.num_m * p.num_n, p.k_blocks, sm_count() / 2);
  p.dw = target;
  cudaError_t e;
  if (p.splits > 1) {
    e = cudaMemsetAsync(target, 0, (size_t)n_w * sizeof(float), st);
    if (e != cudaSuccess) return e;
  }
  e = launch_gemm2<kEpiStore, true, true>(ta, tb, p, st);
  if (e != cudaSuccess || sqnorm == nullptr) return e;
  return launch_sumsq(target, n_w, red, sqnorm, st);  // fixed order
}

}  // namespace jab
