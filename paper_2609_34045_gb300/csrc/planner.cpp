// Block placement over a ring (host code): Algorithm 1 (Partition), head placement by
// rotation, the admission tiers, the evaluation's baseline divisions and the per-device block
// limit.  See include/kafila_plan.h for the contract of each entry point.
#include <algorithm>
#include <cmath>
#include <limits>
#include <vector>

#include "../../include/kafila_plan.h"

namespace {

// The cost of n blocks on device i, written once so that the candidates and every test against
// a bound evaluate the same expression (a candidate is then never rejected by rounding).
inline double cost(double fixed, double per, int n) { return fixed + static_cast<double>(n) * per; }

// The largest n in [0, cap] with cost(fixed, per, n) <= tau (cost is increasing in n).
int most_blocks_within(double fixed, double per, double tau, int cap) {
  if (cap <= 0 || cost(fixed, per, 0) > tau) return 0;
  double q = std::floor((tau - fixed) / per);
  int n = q >= static_cast<double>(cap) ? cap : (q < 0.0 ? 0 : static_cast<int>(q));
  while (n < cap && cost(fixed, per, n + 1) <= tau) ++n;
  while (n > 0 && cost(fixed, per, n) > tau) --n;
  return n;
}

// The Feasible pass of Algorithm 1 for bound tau: left to right, each device takes as many blocks
// as the bound and its limit allow while leaving one for every device after it.
bool feasible(int k, int m, const double *fixed, const double *per, const int *lim, double tau, int *n) {
  int left = k;
  for (int i = 0; i < m; ++i) {
    if (fixed[i] > tau) return false;
    const int ni = std::min(most_blocks_within(fixed[i], per[i], tau, lim[i]), left - (m - 1 - i));
    if (ni < 1) return false;
    n[i] = ni;
    left -= ni;
  }
  return left == 0;
}

int partition_impl(int k, int m, const double *fixed, const double *per, const int *lim, int *n_out,
                   double *tau_out) {
  // the bottleneck of any division is fixed(i) + n per(i) for some device i and count n
  std::vector<double> cand;
  for (int i = 0; i < m; ++i)
    for (int n = 1; n <= std::min(k, lim[i]); ++n) cand.push_back(cost(fixed[i], per[i], n));
  std::sort(cand.begin(), cand.end());
  std::vector<int> n(m);
  // smallest feasible candidate (feasibility is monotone in the bound)
  size_t lo = 0, hi = cand.size();
  while (lo < hi) {
    const size_t mid = lo + (hi - lo) / 2;
    if (feasible(k, m, fixed, per, lim, cand[mid], n.data()))
      hi = mid;
    else
      lo = mid + 1;
  }
  if (lo == cand.size()) return KFL_ERR_INFEASIBLE;
  feasible(k, m, fixed, per, lim, cand[lo], n_out);
  *tau_out = cand[lo];
  return KFL_OK;
}

bool is_finite(double x) { return std::isfinite(x); }

}  // namespace

extern "C" int kfl_partition(int k, int m, const double *fixed, const double *per, const int *lim, int *n_out,
                             double *tau_out) {
  if (k < 1 || m < 1 || !fixed || !per || !lim || !n_out || !tau_out) return KFL_ERR_ARG;
  for (int i = 0; i < m; ++i)
    if (!is_finite(fixed[i]) || !is_finite(per[i]) || per[i] <= 0.0 || lim[i] < 0) return KFL_ERR_ARG;
  if (m > k) return KFL_ERR_INFEASIBLE;
  return partition_impl(k, m, fixed, per, lim, n_out, tau_out);
}

extern "C" int kfl_divide(int k, int m, const double *weight, int *n_out) {
  if (m < 1 || k < m || !n_out) return KFL_ERR_ARG;
  if (!weight) {
    for (int i = 0; i < m; ++i) n_out[i] = k / m + (i < k % m ? 1 : 0);
    return KFL_OK;
  }
  double total = 0.0;
  for (int i = 0; i < m; ++i) {
    if (!is_finite(weight[i]) || weight[i] <= 0.0) return KFL_ERR_ARG;
    total += weight[i];
  }
  // largest remainder: the floors of the exact shares, then one more block to each of the
  // largest remainders (the lower index first on ties)
  std::vector<double> rem(m);
  int given = 0;
  for (int i = 0; i < m; ++i) {
    const double share = static_cast<double>(k) * weight[i] / total;
    n_out[i] = static_cast<int>(std::floor(share));
    rem[i] = share - n_out[i];
    given += n_out[i];
  }
  std::vector<int> order(m);
  for (int i = 0; i < m; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return rem[a] > rem[b]; });
  for (int j = 0; given < k; ++j, ++given) ++n_out[order[j % m]];
  // every member of a ring holds a block
  for (int i = 0; i < m; ++i) {
    if (n_out[i] > 0) continue;
    int big = 0;
    for (int j = 1; j < m; ++j)
      if (n_out[j] > n_out[big]) big = j;
    --n_out[big];
    ++n_out[i];
  }
  return KFL_OK;
}

extern "C" int kfl_plan_ring(int k, int m, const kfl_plan_device *dev, int anchor, double beta_block,
                             double beta_head, double mu, int *n_out, kfl_plan *plan) {
  if (k < 1 || m < 1 || !dev || !n_out || !plan || anchor < 0 || anchor >= m || !(mu >= 0.0 && mu < 1.0))
    return KFL_ERR_ARG;
  for (int i = 0; i < m; ++i)
    if (dev[i].lim_body < 0 || dev[i].lim_head < 0) return KFL_ERR_ARG;
  plan->head = anchor;
  plan->tau = 0.0;
  plan->tau_anchor = std::numeric_limits<double>::infinity();
  plan->undersized = -1;
  bool all_bw = true, all_tp = true;
  for (int i = 0; i < m; ++i) {
    all_bw = all_bw && dev[i].bw > 0.0 && is_finite(dev[i].bw) && is_finite(dev[i].o);
    all_tp = all_tp && dev[i].throughput > 0.0 && is_finite(dev[i].throughput);
  }
  std::vector<double> fixed(m), per(m);
  std::vector<int> lim(m), n(m);
  // the fixed-order problem with device r as head, devices taken around the ring from r
  auto solve = [&](int r, bool priced, double *tau) {
    for (int j = 0; j < m; ++j) {
      const int d = (r + j) % m;
      const bool head = j == 0;
      if (priced) {
        fixed[j] = dev[d].o + (head ? beta_head / dev[d].bw : 0.0);
        per[j] = beta_block / dev[d].bw;
      } else {
        fixed[j] = 0.0;
        per[j] = 1.0 / dev[d].throughput;
      }
      lim[j] = head ? dev[d].lim_head : dev[d].lim_body;
    }
    if (m > k) return KFL_ERR_INFEASIBLE;
    return partition_impl(k, m, fixed.data(), per.data(), lim.data(), n.data(), tau);
  };
  auto unrotate = [&](int r) {
    for (int j = 0; j < m; ++j) n_out[(r + j) % m] = n[j];
  };
  if (all_bw) {
    if (!(beta_block > 0.0) || !(beta_head >= 0.0) || !is_finite(beta_block) || !is_finite(beta_head)) return KFL_ERR_ARG;
    plan->tier = 1;
    // every rotation is one exact solve; the anchor keeps the head unless another rotation's
    // bottleneck is below tau_anchor (1 - mu)
    std::vector<double> taus(m, std::numeric_limits<double>::infinity());
    for (int r = 0; r < m; ++r) {
      double t;
      if (solve(r, true, &t) == KFL_OK) taus[r] = t;
    }
    plan->tau_anchor = taus[anchor];
    int best = -1;
    for (int j = 0; j < m; ++j) {
      const int r = (anchor + j) % m;
      if (std::isfinite(taus[r]) && (best < 0 || taus[r] < taus[best])) best = r;
    }
    if (best < 0) return KFL_ERR_INFEASIBLE;
    const int head = taus[best] < taus[anchor] * (1.0 - mu) ? best : anchor;
    double t;
    solve(head, true, &t);
    unrotate(head);
    plan->head = head;
    plan->tau = t;
    return KFL_OK;
  }
  if (all_tp) {
    plan->tier = 2;
    double t;
    const int rc = solve(anchor, false, &t);
    if (rc != KFL_OK) return rc;
    unrotate(anchor);
    plan->tau = t;
    return KFL_OK;
  }
  plan->tier = 3;
  if (m > k) return KFL_ERR_INFEASIBLE;
  std::vector<double> w(m);
  for (int j = 0; j < m; ++j) w[j] = dev[(anchor + j) % m].working_set;
  const int rc = kfl_divide(k, m, w.data(), n.data());
  if (rc != KFL_OK) return rc;
  unrotate(anchor);
  // admission: the least informed division has not looked at the limits
  for (int j = 0; j < m; ++j) {
    const int d = (anchor + j) % m;
    if (n_out[d] > (j == 0 ? dev[d].lim_head : dev[d].lim_body)) {
      plan->undersized = d;
      return KFL_ERR_INFEASIBLE;
    }
  }
  return KFL_OK;
}

extern "C" int kfl_block_limit(const kfl_model_cfg *cfg, size_t room_bytes, int is_head, int *lim_out) {
  if (!cfg || !lim_out) return KFL_ERR_ARG;
  const int flags = is_head ? KFL_IS_HEAD : 0;
  auto bytes = [&](int n, size_t *out) {
    if (n == 0 && !flags) {
      *out = 0;
      return KFL_OK;
    }
    return kfl_stage_memory_bytes(cfg, 0, n, flags, out);
  };
  size_t b = 0;
  int rc = bytes(0, &b);
  if (rc != KFL_OK) return rc;
  if (b > room_bytes) {
    *lim_out = 0;
    return KFL_OK;
  }
  // stage memory grows with the block count: the largest n that fits
  int lo = 0, hi = cfg->n_layers_total;
  while (lo < hi) {
    const int mid = lo + (hi - lo + 1) / 2;
    rc = bytes(mid, &b);
    if (rc != KFL_OK) return rc;
    if (b <= room_bytes)
      lo = mid;
    else
      hi = mid - 1;
  }
  *lim_out = lo;
  return KFL_OK;
}
