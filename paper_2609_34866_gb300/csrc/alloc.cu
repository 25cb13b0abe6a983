// Bit-width allocation over layers (Section 2.4, Eq. 7; App. B "Allocators"): host code only, no
// device memory and no CUDA call. It consumes a score table Omega[layer][width] (direct L_JAB from
// jab_loss_forward, or the C1 / C2 scores of Eq. 6) and solves
//   min sum_i Omega_i(b_i)   s.t.   sum_i n_i b_i <= avg_bits * sum_i n_i   (cost of Eq. 8)
// by the greedy walk of App. B: every layer starts at its highest width; while over budget, the
// one-step downgrade with the least score increase per bit saved is applied; then, while one fits,
// the one-step upgrade with the largest score decrease per bit is applied. The Pareto variant runs
// the same walk over each layer's non-dominated (cost, score) points only. Ties go to the lowest
// layer index; ratios are compared in double precision.
#include <cmath>
#include <cstdint>
#include <vector>

#include "../../include/jab.h"

namespace {

struct LayerPath {
  std::vector<int> k;  // indices into the width list, increasing cost
  int pos;             // current position in k
};

}  // namespace

extern "C" jab_status jab_allocate_bits(const double* omega_host, const int32_t* widths_host,
                                        const int64_t* n_weights_host, int32_t L,
                                        int32_t n_widths, double avg_bits, int32_t method,
                                        int32_t* bits_out_host) {
  if (!omega_host || !widths_host || !n_weights_host || !bits_out_host || L < 1 || n_widths < 1 ||
      (method != 0 && method != 1) || !std::isfinite(avg_bits))
    return JAB_ERR_INVALID_ARG;
  for (int k = 0; k < n_widths; ++k)
    if (widths_host[k] < 1 || (k > 0 && widths_host[k] <= widths_host[k - 1]))
      return JAB_ERR_INVALID_ARG;
  int64_t n_total = 0;
  for (int i = 0; i < L; ++i) {
    if (n_weights_host[i] < 1) return JAB_ERR_INVALID_ARG;
    n_total += n_weights_host[i];
    for (int k = 0; k < n_widths; ++k)
      if (!std::isfinite(omega_host[(int64_t)i * n_widths + k])) return JAB_ERR_INVALID_ARG;
  }
  const double budget = avg_bits * (double)n_total;
  auto om = [&](int i, int k) { return omega_host[(int64_t)i * n_widths + k]; };

  std::vector<LayerPath> path(L);
  for (int i = 0; i < L; ++i) {
    if (method == 0) {
      for (int k = 0; k < n_widths; ++k) path[i].k.push_back(k);
    } else {  // keep a point only if every cheaper point scores strictly worse
      for (int k = 0; k < n_widths; ++k)
        if (path[i].k.empty() || om(i, k) < om(i, path[i].k.back())) path[i].k.push_back(k);
    }
    path[i].pos = (int)path[i].k.size() - 1;
  }
  auto width = [&](int i, int p) { return (int64_t)widths_host[path[i].k[p]]; };
  auto score = [&](int i, int p) { return om(i, path[i].k[p]); };

  int64_t cheapest = 0, cost = 0;
  for (int i = 0; i < L; ++i) {
    cheapest += n_weights_host[i] * width(i, 0);
    cost += n_weights_host[i] * width(i, path[i].pos);
  }
  if ((double)cheapest > budget) return JAB_ERR_INVALID_ARG;

  while ((double)cost > budget) {  // downgrades
    int pick = -1;
    double best = 0.0;
    for (int i = 0; i < L; ++i) {
      const int p = path[i].pos;
      if (p == 0) continue;
      const int64_t dc = n_weights_host[i] * (width(i, p) - width(i, p - 1));
      const double r = (score(i, p - 1) - score(i, p)) / (double)dc;
      if (pick < 0 || r < best) {
        best = r;
        pick = i;
      }
    }
    if (pick < 0) return JAB_ERR_INVALID_ARG;  // unreachable: the cheapest allocation fits
    const int p = path[pick].pos;
    cost -= n_weights_host[pick] * (width(pick, p) - width(pick, p - 1));
    path[pick].pos = p - 1;
  }
  for (;;) {  // leftovers: upgrades that fit and lower the total score
    int pick = -1;
    double best = 0.0;
    for (int i = 0; i < L; ++i) {
      const int p = path[i].pos;
      if (p + 1 == (int)path[i].k.size()) continue;
      const int64_t dc = n_weights_host[i] * (width(i, p + 1) - width(i, p));
      const double gain = score(i, p) - score(i, p + 1);
      if ((double)(cost + dc) > budget || !(gain > 0.0)) continue;
      const double r = gain / (double)dc;
      if (pick < 0 || r > best) {
        best = r;
        pick = i;
      }
    }
    if (pick < 0) break;
    const int p = path[pick].pos;
    cost += n_weights_host[pick] * (width(pick, p + 1) - width(pick, p));
    path[pick].pos = p + 1;
  }
  for (int i = 0; i < L; ++i) bits_out_host[i] = (int32_t)width(i, path[i].pos);
  return JAB_OK;
}
