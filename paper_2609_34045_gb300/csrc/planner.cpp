// Block placement over a ring (host code): the exact fixed-order division of Section V-B, head
// placement by rotation, the admission tiers, the evaluation's baseline divisions and the per-device block
// limit.  See include/kafila_plan.h for the contract of each entry point.
#include <algorithm>
#include <cmath>
#include <functional>
#include <limits>
#include <queue>
#include <utility>
#include <vector>

#include "../../include/kafila_plan.h"

namespace {

// The cost of n blocks on device i (Eq. 2), written once so that every cost compared or returned
// is the same expression.
inline double cost(double fixed, double per, int n) { return fixed + static_cast<double>(n) * per; }

// Fixed-order chain division (Section V-B, "Block placement"): k contiguous blocks over devices
// 0..m-1 in ring order, device i holding 1 <= n_i <= lim(i) blocks at cost(i, n_i), minimizing
// the largest cost.  Which blocks a device holds does not change its cost, only how many, so any
// counts within the limits that sum to k are a valid chain.
//
// Every device starts with its one obligatory block; the other k - m are handed out one at a
// time, each to the device whose cost after taking it is lowest (the lower ring index on ties).
// A device's successive costs never decrease, so the handed-out blocks are the k - m cheapest
// increments that any division could take, and the resulting maximum is the smallest any
// division reaches.  The bottleneck is the maximum of costs of the returned division itself,
// evaluated with the same expression as every other cost, so it is exactly attained.
int partition_impl(int k, int m, const double *fixed, const double *per, const int *lim, int *n_out,
                   double *tau_out) {
  if (m > k) return KFL_ERR_INFEASIBLE;
  long long room = 0;
  for (int i = 0; i < m; ++i) {
    if (lim[i] < 1) return KFL_ERR_INFEASIBLE;
    room += std::min(lim[i], k);
  }
  if (room < k) return KFL_ERR_INFEASIBLE;
  using Next = std::pair<double, int>;  // (cost with one more block, device)
  std::priority_queue<Next, std::vector<Next>, std::greater<Next>> next;
  double tau = -std::numeric_limits<double>::infinity();
  for (int i = 0; i < m; ++i) {
    n_out[i] = 1;
    tau = std::max(tau, cost(fixed[i], per[i], 1));
    if (lim[i] > 1) next.push({cost(fixed[i], per[i], 2), i});
  }
  for (int given = m; given < k; ++given) {
    const Next t = next.top();
    next.pop();
    const int i = t.second;
    ++n_out[i];
    tau = std::max(tau, t.first);
    if (n_out[i] < lim[i]) next.push({cost(fixed[i], per[i], n_out[i] + 1), i});
  }
  *tau_out = tau;
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
