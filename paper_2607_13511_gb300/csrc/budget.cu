// Rank and storage budgets from the energy trace (host code).
//
// The method is greedy with sequential deflation (§2.3, §2.4): a run at inner rank k1 (a block boundary) is the
// first k1 components of any run at a larger rank on the same matrix, so one run at the largest rank gives the
// energy E(k) at every block boundary. Two uses follow: the smallest rank (hence mu = k / min(m, n)) that reaches a
// target energy, which is how equal-energy comparisons across methods are set up (§3), and the allocation of ranks
// across the matrices of a model under one storage budget (§5).
#include <cmath>
#include <vector>

#include <algorithm>

#include "externd.h"

extern "C" {

int externd_block_boundaries(int64_t m, int64_t n, double mu, int block, int64_t* ranks, int64_t* count) {
  if (count == nullptr) return EXTERND_EINVAL;
  int64_t k;
  int b;
  int st = externd_rank(m, n, mu, &k);
  if (st != EXTERND_OK) return st;
  st = externd_block_width(m, n, block, &b);
  if (st != EXTERND_OK) return st;
  const int64_t nb = (k + b - 1) / b;
  if (ranks != nullptr) {
    if (*count < nb) return EXTERND_EINVAL;
    for (int64_t i = 0; i < nb; ++i) ranks[i] = std::min<int64_t>((i + 1) * b, k);
  }
  *count = nb;
  return EXTERND_OK;
}

int externd_rank_for_energy(int64_t m, int64_t n, double mu, int block, const double* trace, int64_t ntrace,
                            double target, int64_t* k) {
  if (trace == nullptr || k == nullptr || !std::isfinite(target)) return EXTERND_EINVAL;
  int64_t nb = 0;
  int st = externd_block_boundaries(m, n, mu, block, nullptr, &nb);
  if (st != EXTERND_OK) return st;
  if (ntrace != nb) return EXTERND_EINVAL;
  std::vector<int64_t> ranks(nb);
  st = externd_block_boundaries(m, n, mu, block, ranks.data(), &nb);
  if (st != EXTERND_OK) return st;
  *k = 0;
  for (int64_t i = 0; i < nb; ++i)
    if (trace[i] >= target) {
      *k = ranks[i];
      break;
    }
  return EXTERND_OK;
}

int externd_allocate_ranks(int64_t nmat, const int64_t* npts, const int64_t* ks, const double* energies,
                           const double* costs, const double* weights, double budget, int64_t* chosen) {
  if (nmat < 1 || npts == nullptr || ks == nullptr || energies == nullptr || costs == nullptr ||
      chosen == nullptr || !std::isfinite(budget))
    return EXTERND_EINVAL;
  std::vector<int64_t> off(nmat + 1, 0);
  for (int64_t j = 0; j < nmat; ++j) {
    if (npts[j] < 0 || !(costs[j] > 0) || !std::isfinite(costs[j])) return EXTERND_EINVAL;
    if (weights != nullptr && (!(weights[j] >= 0) || !std::isfinite(weights[j]))) return EXTERND_EINVAL;
    off[j + 1] = off[j] + npts[j];
    for (int64_t i = off[j]; i < off[j + 1]; ++i)
      if (!std::isfinite(energies[i]) || ks[i] <= (i == off[j] ? 0 : ks[i - 1])) return EXTERND_EINVAL;
  }
  // Greedy: repeatedly take the next block of the matrix with the largest weighted energy gain per unit of
  // storage that still fits (ties to the lower matrix index); optimal when every curve is concave in k.
  std::vector<int64_t> taken(nmat, 0);
  double spent = 0.0;
  for (;;) {
    int64_t best_j = -1;
    double best = 0.0;
    for (int64_t j = 0; j < nmat; ++j) {
      if (taken[j] >= npts[j]) continue;
      const int64_t i = off[j] + taken[j];
      const int64_t k_prev = taken[j] == 0 ? 0 : ks[i - 1];
      const double e_prev = taken[j] == 0 ? 0.0 : energies[i - 1];
      const double cost = costs[j] * (double)(ks[i] - k_prev);
      if (spent + cost > budget + 1e-12) continue;
      const double gain = (weights == nullptr ? 1.0 : weights[j]) * (energies[i] - e_prev) / cost;
      if (best_j < 0 || gain > best) {
        best = gain;
        best_j = j;
      }
    }
    if (best_j < 0) break;
    const int64_t i = off[best_j] + taken[best_j];
    spent += costs[best_j] * (double)(ks[i] - (taken[best_j] == 0 ? 0 : ks[i - 1]));
    ++taken[best_j];
  }
  for (int64_t j = 0; j < nmat; ++j) chosen[j] = taken[j] == 0 ? 0 : ks[off[j] + taken[j] - 1];
  return EXTERND_OK;
}

}  // extern "C"
