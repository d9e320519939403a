// Error-aware layer budget allocation (CompressKV Sec. 3.4, Eq. 4; Sec. 4
// fixes m = 32 and M = 3 * B_per_layer).  Host only.
//
// The offline per-layer error scores e_l are normalised (Eq. 4), every layer
// gets the minimum m, and the remaining R = B_total - L*m is shared in
// proportion to the normalised errors with no layer above M: a layer whose
// share would pass M - m is capped there and the others share the rest again
// (water filling).  The real shares are rounded so that the budgets add up
// to B_total exactly: floors first, then +1 to the largest fractional parts,
// ties to the lower layer index.  All arithmetic is IEEE double in layer
// order (this file is compiled without floating-point contraction), so the
// result is reproducible bit for bit on any host.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <vector>

#include "compresskv.h"

namespace {

// Eq. 4: e~_l = e_l / sum_k e_k; equal weights when every error is zero.
std::vector<double> normalise(const double* e, int n) {
  double total = 0.0;
  for (int l = 0; l < n; ++l) total += e[l];
  std::vector<double> w(n);
  for (int l = 0; l < n; ++l) w[l] = total == 0.0 ? 1.0 / n : e[l] / total;
  return w;
}

// Real shares x_l, sum x_l = amount, x_l <= room, proportional to w among the
// layers below room.
std::vector<double> water_fill(const std::vector<double>& w, double amount, double room) {
  const int n = static_cast<int>(w.size());
  std::vector<double> share(n, 0.0), give(n, 0.0);
  std::vector<char> free_(n, 1);
  double left = amount;
  for (int round = 0; round < n; ++round) {
    double w_free = 0.0;
    int n_free = 0;
    for (int l = 0; l < n; ++l) {
      if (free_[l]) {
        w_free += w[l];
        ++n_free;
      }
    }
    if (n_free == 0) break;
    bool any_over = false;
    for (int l = 0; l < n; ++l) {
      give[l] = 0.0;
      if (free_[l]) {
        give[l] = w_free > 0.0 ? left * w[l] / w_free : left / n_free;
        any_over = any_over || give[l] > room;
      }
    }
    if (!any_over) {
      for (int l = 0; l < n; ++l)
        if (free_[l]) share[l] = give[l];
      break;
    }
    for (int l = 0; l < n; ++l) {
      if (free_[l] && give[l] > room) {
        share[l] = room;
        left -= room;
        free_[l] = 0;
      }
    }
  }
  return share;
}

}  // namespace

extern "C" int compresskv_allocate_layer_budgets(const double* layer_errors, int32_t n_layers,
                                                 int64_t total_budget, int32_t min_budget,
                                                 int32_t max_budget, int32_t* budgets) {
  if (!layer_errors || !budgets || n_layers < 1) return CKV_ERR_INVALID_ARG;
  for (int l = 0; l < n_layers; ++l)
    if (!(layer_errors[l] >= 0.0) || std::isinf(layer_errors[l])) return CKV_ERR_INVALID_ARG;
  const int64_t L = n_layers;
  const int64_t m = min_budget;
  const int64_t M = max_budget > 0 ? max_budget : (3 * total_budget) / L;
  if (m < 0 || M < m || L * m > total_budget || total_budget > L * M || M > INT32_MAX)
    return CKV_ERR_BUDGET;
  const int64_t rest = total_budget - L * m;
  const int64_t room = M - m;
  const std::vector<double> w = normalise(layer_errors, n_layers);
  const std::vector<double> share =
      water_fill(w, static_cast<double>(rest), static_cast<double>(room));
  std::vector<int64_t> base(n_layers);
  std::vector<double> frac(n_layers);
  int64_t sum = 0;
  for (int l = 0; l < n_layers; ++l) {
    base[l] = std::min(static_cast<int64_t>(std::floor(share[l])), room);
    frac[l] = share[l] - static_cast<double>(base[l]);
    sum += base[l];
  }
  int64_t missing = rest - sum;
  std::vector<int> order;
  if (missing > 0) {
    for (int l = 0; l < n_layers; ++l)
      if (base[l] < room) order.push_back(l);
    std::stable_sort(order.begin(), order.end(),
                     [&](int a, int b) { return frac[a] > frac[b]; });  // ties: lower index
    for (int i = 0; i < static_cast<int>(order.size()) && missing > 0; ++i, --missing)
      ++base[order[i]];
  } else if (missing < 0) {
    for (int l = n_layers - 1; l >= 0; --l)
      if (base[l] > 0) order.push_back(l);
    std::stable_sort(order.begin(), order.end(),
                     [&](int a, int b) { return frac[a] < frac[b]; });  // ties: higher index
    for (int i = 0; i < static_cast<int>(order.size()) && missing < 0; ++i, ++missing)
      --base[order[i]];
  }
  for (int l = 0; l < n_layers; ++l) budgets[l] = static_cast<int32_t>(m + base[l]);
  return CKV_OK;
}
