// Layout of the caller-provided workspace (host-side arithmetic only).
#pragma once

#include <stddef.h>
#include <stdint.h>

#include "../../include/jab.h"

namespace jab {

constexpr int kPartRows = 64;  // query rows per loss partial (one partial per (c, b, h, 64 rows))
constexpr int kRedBlocks = 1024;  // blocks of a grid-stride reduction over the weights
constexpr int kMaxSplits = 32;    // K splits of the weight-gradient GEMMs at most

struct Workspace {
  // byte offsets into ws; SIZE_MAX when absent
  size_t x16;      // fp16 [N, d]            X converted for the fp16 tensor-core path
  size_t w16;      // fp16 [C, D, d]         w_hat per candidate (or W for the teacher)
  size_t qkv;      // fp16 [N, C*D]          projected, RoPE-rotated Q|K|V for every candidate
  size_t rope;     // fp32 [2, T, d_h/2]     cos then sin
  size_t part;     // fp64 [C, B, Hq, nP]    per-tile partial sums (SSE or ||A||^2)
  size_t status;   // int32 [4]              reserved
  size_t scal;     // fp64 [2, C]            per-candidate scalars (MSE and KL terms)
  size_t red;      // fp64 [C, kRedBlocks]   per-block partial sums of the quantisation error
  // backward only
  size_t d_o;      // fp16 [N, Hq*d_h]       e = A_hat - A_ref (dL/dA_hat up to 2/n)
  size_t lse;      // fp32 [B, Hq, Tp]       student log-sum-exp in log2 units (Tp = T rounded to 128)
  size_t dvec;     // fp32 [B, Hq, Tp]       rowsum(dO * O)
  size_t dqkvt;    // bf16 [D, ldt]          dL/d[Q|K|V] (pre-RoPE), transposed
  size_t ds;       // fp16 [B, Hq, nq (nq + 1) / 2, 128, 128]   dS^T tile of every (query block,
                   //                        key block <= query block) pair, nq = ceil(T / 128)
  size_t gpart;    // fp32 [kMaxSplits, D, d/G]  scale-gradient partial of every K split (summed in order)
  size_t dwscr;    // fp32 [D, d]            dW when only its squared norm is asked for
  size_t lse_t;    // fp32 [B, Hq, Tp]       teacher log-sum-exp in log2 units (KL term's gradient)
  size_t klpart;   // fp64 [Hkv, B, nq]      KL partial sum of every teacher-probability CTA
  int64_t ldt;     // row pitch (elements) of dqkvt: N rounded up to 64
  int64_t tp;      // row pitch (elements) of lse and dvec: T rounded up to 128
  size_t total;
};

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

inline int64_t block_rows(const jab_block_desc* d) {
  return (int64_t)(d->n_q_heads + 2 * d->n_kv_heads) * d->head_dim;
}

inline Workspace plan_workspace(const jab_block_desc* d, int64_t B, int64_t T, int64_t C,
                                bool bwd) {
  Workspace w;
  const int64_t N = B * T, D = block_rows(d), dm = d->d_model, dh = d->head_dim;
  const int64_t nP = (T + kPartRows - 1) / kPartRows;
  w.ldt = (N + 63) / 64 * 64;
  w.tp = (T + 127) / 128 * 128;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  w.status = take(64);
  w.x16 = take((size_t)N * dm * 2);
  w.w16 = take((size_t)C * D * dm * 2);
  w.qkv = take((size_t)N * C * D * 2);
  w.rope = take((size_t)2 * T * (dh / 2) * 4);
  w.part = take((size_t)C * B * d->n_q_heads * nP * 8);
  w.scal = take((size_t)2 * C * 8);
  w.red = take((size_t)C * kRedBlocks * 8);
  if (bwd) {
    w.d_o = take((size_t)N * d->n_q_heads * dh * 2);
    w.lse = take((size_t)B * d->n_q_heads * w.tp * 4);
    w.dvec = take((size_t)B * d->n_q_heads * w.tp * 4);
    w.dqkvt = take((size_t)D * w.ldt * 2);
    const int64_t nq = (T + 127) / 128;
    w.ds = take((size_t)B * d->n_q_heads * (nq * (nq + 1) / 2) * 128 * 128 * 2);
    w.gpart = take((size_t)kMaxSplits * D * (dm / d->group_size) * 4);
    w.dwscr = take((size_t)D * dm * 4);
    w.lse_t = take((size_t)B * d->n_q_heads * w.tp * 4);
    w.klpart = take((size_t)d->n_kv_heads * B * nq * 8);
  } else {
    w.d_o = w.lse = w.dvec = w.dqkvt = w.ds = w.gpart = w.dwscr = w.lse_t = w.klpart = SIZE_MAX;
  }
  w.total = off;
  return w;
}

}  // namespace jab
