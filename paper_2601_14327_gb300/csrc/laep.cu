// LAEP host algorithms (the pruning decision and the expert rearrangement).
//
// Sec. 3.2 Eq. 1-2 and Appendix Algorithm 1 decide which experts a layer keeps
// from the per-expert token numbers (ETN); Sec. 3.4.3 sets the layer-adaptive
// alpha; Appendix Algorithm 2 places experts on n_g groups (devices) so that
// their token loads balance. All of this runs on the host on E <= a few
// hundred numbers per layer.
#include <algorithm>
#include <limits>
#include <numeric>
#include <vector>

#include "common.cuh"

namespace {

// Expert ids in ascending load order; equal loads keep the id order.
std::vector<int> ascending(const int32_t *counts, int E) {
  std::vector<int> order(E);
  std::iota(order.begin(), order.end(), 0);
  std::stable_sort(order.begin(), order.end(),
                   [&](int a, int b) { return counts[a] < counts[b]; });
  return order;
}

}  // namespace

extern "C" {

// LAEP pruning decision (Sec. 3.2 Eq. 1-2, Algorithm 1 with one histogram).
int laep_prune_mask(const int32_t *counts_host, int E, int64_t S, int k, double alpha,
                    double beta, int prune_count, uint8_t *active_mask_host, int *n_pruned) {
  if (!counts_host || !active_mask_host)
    return moe::set_error(MOE_ERR_ARG, "laep_prune_mask: null pointer");
  if (E <= 0 || k <= 0 || k > E || S < 0)
    return moe::set_error(MOE_ERR_ARG, "laep_prune_mask: bad sizes E=%d k=%d S=%lld", E, k,
                          (long long)S);
  for (int e = 0; e < E; ++e)
    if (counts_host[e] < 0) return moe::set_error(MOE_ERR_ARG, "laep_prune_mask: negative count");
  // Ascending load order; equal loads keep index order (lower index first).
  std::vector<int> order(E);
  std::iota(order.begin(), order.end(), 0);
  std::stable_sort(order.begin(), order.end(),
                   [&](int a, int b) { return counts_host[a] < counts_host[b]; });
  for (int e = 0; e < E; ++e) active_mask_host[e] = 1;
  const int max_prune = E - k;  // routing needs k live experts
  int pruned = 0;
  if (prune_count >= 0) {
    pruned = std::min(prune_count, max_prune);
    for (int r = 0; r < pruned; ++r) active_mask_host[order[r]] = 0;
  } else {
    // Thresholds of Algorithm 1: cumulative < S*topK*beta, individual < S*topK*alpha/E.
    const double beta_thr = double(S) * double(k) * beta;
    const double alpha_thr = double(S) * double(k) * alpha / double(E);
    int64_t running = 0;
    for (int r = 0; r < E; ++r) {
      const int e = order[r];
      running += counts_host[e];
      if (double(running) < beta_thr && double(counts_host[e]) < alpha_thr && pruned < max_prune) {
        active_mask_host[e] = 0;
        ++pruned;
      }
    }
  }
  if (n_pruned) *n_pruned = pruned;
  return MOE_OK;
}

double laep_layer_alpha(int L, int layer, double alpha_edge, double alpha_middle) {
  if (L <= 0 || layer < 0 || layer >= L) return alpha_middle;
  const int n6 = L / 6;  // first and last sixth of the layers
  return (layer < n6 || layer >= L - n6) ? alpha_edge : alpha_middle;
}

// Algorithm 1 with an ETN history of ITER iterations x L layers.
int laep_prune_layers(const int32_t *etn_host, int iters, int L, int E, int64_t S, int k,
                      const double *alpha_host, double beta, uint8_t *mask_host,
                      int32_t *n_pruned_host) {
  if (!etn_host || !alpha_host || !mask_host)
    return moe::set_error(MOE_ERR_ARG, "laep_prune_layers: null pointer");
  if (iters <= 0 || L <= 0 || E <= 0 || k <= 0 || k > E || S < 0)
    return moe::set_error(MOE_ERR_ARG, "laep_prune_layers: bad sizes");
  for (int64_t i = 0; i < int64_t(iters) * L * E; ++i)
    if (etn_host[i] < 0) return moe::set_error(MOE_ERR_ARG, "laep_prune_layers: negative count");
  std::vector<int64_t> marker(size_t(L) * E, 0), total(size_t(L) * E, 0), exp_dis(L, 0);
  for (int it = 0; it < iters; ++it) {
    for (int l = 0; l < L; ++l) {
      const int32_t *c = etn_host + (size_t(it) * L + l) * E;
      const double beta_thr = double(S) * double(k) * beta;
      const double alpha_thr = double(S) * double(k) * alpha_host[l] / double(E);
      int64_t running = 0;  // restarts for every (iteration, layer)
      for (int e : ascending(c, E)) {
        running += c[e];
        if (double(running) < beta_thr && double(c[e]) < alpha_thr) {
          ++exp_dis[l];
          ++marker[size_t(l) * E + e];
        }
      }
      for (int e = 0; e < E; ++e) total[size_t(l) * E + e] += c[e];
    }
  }
  for (int l = 0; l < L; ++l) {
    const int64_t *m = &marker[size_t(l) * E];
    const int64_t *tl = &total[size_t(l) * E];
    int64_t flagged = 0;
    for (int e = 0; e < E; ++e) flagged += m[e] > 0;
    // mean flagged count over the iterations, rounded half up
    int64_t n = (2 * exp_dis[l] + iters) / (2 * int64_t(iters));
    n = std::min<int64_t>({n, int64_t(E - k), flagged});
    std::vector<int> order(E);
    std::iota(order.begin(), order.end(), 0);
    std::sort(order.begin(), order.end(), [&](int a, int b) {
      if (m[a] != m[b]) return m[a] > m[b];
      if (tl[a] != tl[b]) return tl[a] < tl[b];
      return a < b;
    });
    uint8_t *mask = mask_host + size_t(l) * E;
    for (int e = 0; e < E; ++e) mask[e] = 1;
    for (int64_t r = 0; r < n; ++r) mask[order[r]] = 0;
    if (n_pruned_host) n_pruned_host[l] = int32_t(n);
  }
  return MOE_OK;
}

// Algorithm 2: greedy placement of n experts into n_groups groups.
int laep_rearrange(const int64_t *load_host, int n, int n_groups, int32_t *order_host,
                   int32_t *group_of_host, int64_t *group_load_host) {
  if (!load_host || !order_host || n <= 0 || n_groups <= 0 || n_groups > n)
    return moe::set_error(MOE_ERR_ARG, "laep_rearrange: bad arguments");
  const int cap = (n + n_groups - 1) / n_groups;  // == n / n_groups when it divides
  std::vector<int> desc(n);
  std::iota(desc.begin(), desc.end(), 0);
  std::stable_sort(desc.begin(), desc.end(),
                   [&](int a, int b) { return load_host[a] > load_host[b]; });
  std::vector<std::vector<int>> members(n_groups);
  std::vector<int64_t> sums(n_groups, 0);
  std::vector<bool> full(n_groups, false);
  for (int e : desc) {
    while (true) {
      int g = -1;
      for (int q = 0; q < n_groups; ++q)  // smallest sum among groups not marked full
        if (!full[q] && (g < 0 || sums[q] < sums[g])) g = q;
      if (g < 0) return moe::set_error(MOE_ERR_INVARIANT, "laep_rearrange: no group has room");
      if (int(members[g].size()) < cap) {
        members[g].push_back(e);
        sums[g] += load_host[e];
        break;
      }
      full[g] = true;
    }
  }
  int pos = 0;
  for (int g = 0; g < n_groups; ++g)
    for (int e : members[g]) {
      order_host[pos++] = e;
      if (group_of_host) group_of_host[e] = g;
    }
  if (group_load_host)
    for (int g = 0; g < n_groups; ++g) group_load_host[g] = sums[g];
  return MOE_OK;
}

}  // extern "C"
