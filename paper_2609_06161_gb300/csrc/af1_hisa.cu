// af1_hisa.cu — the budget arithmetic of AF1's Hierarchical Shapley
// Allocation (Sec. 3.2) as host functions of given Shapley scores: the
// temperature softmax of layer scores into layer budgets (Eq.
// hisa_layer_budget), the module-level MAD normalisation (Eq. hisa_mad_norm),
// logistic map, Soft-OR fusion and size-aware density allocation (Eq.
// hisa_module_budget), and the budget-to-rank conversion of App. "Budget-to-
// rank conversion". Estimating the Shapley scores themselves needs a model
// and calibration data and is not part of this library.
#include <stdint.h>

#include <algorithm>
#include <cmath>
#include <string>
#include <vector>

#include "af1.h"
#include "af1_internal.h"

namespace {

double median(std::vector<double> v) {
  std::sort(v.begin(), v.end());
  const size_t k = v.size();
  return (k % 2) ? v[k / 2] : 0.5 * (v[k / 2 - 1] + v[k / 2]);
}

bool all_finite(const double* v, int64_t n) {
  for (int64_t i = 0; i < n; ++i)
    if (!std::isfinite(v[i])) return false;
  return true;
}

// (phi_i - median) / (1.4826 MAD + eps).
std::vector<double> mad_z(const double* phi, int64_t n, double eps) {
  std::vector<double> v(phi, phi + n);
  const double med = median(v);
  std::vector<double> dev(n);
  for (int64_t i = 0; i < n; ++i) dev[i] = std::fabs(phi[i] - med);
  const double mad = median(dev);
  std::vector<double> z(n);
  for (int64_t i = 0; i < n; ++i) z[i] = (phi[i] - med) / (1.4826 * mad + eps);
  return z;
}

}  // namespace

extern "C" {

int af1_hisa_layer_budgets(const double* phi, int64_t L, double B_total, double tau, double* B_out) {
  if (phi == nullptr || B_out == nullptr || L <= 0 || !(tau > 0.0) || !std::isfinite(B_total) || !all_finite(phi, L))
    return af1::set_error(AF1_ERR_INVALID_ARG, "af1_hisa_layer_budgets: need L > 0 finite scores, tau > 0");
  double top = phi[0] / tau;
  for (int64_t l = 1; l < L; ++l) top = std::max(top, phi[l] / tau);
  double tot = 0.0;
  for (int64_t l = 0; l < L; ++l) tot += std::exp(phi[l] / tau - top);
  for (int64_t l = 0; l < L; ++l) B_out[l] = B_total * std::exp(phi[l] / tau - top) / tot;
  return AF1_OK;
}

int af1_hisa_module_budgets(const double* phi_dir, const double* phi_mag, const int64_t* params, int64_t N,
                            double B_l, double alpha, double eps, double* b_out) {
  if (phi_dir == nullptr || phi_mag == nullptr || params == nullptr || b_out == nullptr || N <= 0 ||
      !std::isfinite(B_l) || !std::isfinite(alpha) || !(eps >= 0.0) || !all_finite(phi_dir, N) ||
      !all_finite(phi_mag, N))
    return af1::set_error(AF1_ERR_INVALID_ARG, "af1_hisa_module_budgets: invalid arguments");
  for (int64_t i = 0; i < N; ++i)
    if (params[i] <= 0) return af1::set_error(AF1_ERR_INVALID_ARG, "af1_hisa_module_budgets: parameter counts must be > 0");
  const std::vector<double> zd = mad_z(phi_dir, N, eps), zm = mad_z(phi_mag, N, eps);
  std::vector<double> w(N);
  double total = 0.0, den = 0.0;
  for (int64_t i = 0; i < N; ++i) {
    const double pd = 1.0 / (1.0 + std::exp(-zd[i]));
    const double pm = 1.0 / (1.0 + std::exp(-zm[i]));
    const double v = 1.0 - (1.0 - pd) * (1.0 - pm);  // Soft-OR of the two failure modes
    w[i] = std::pow(v / (double)params[i] + eps, alpha);
    total += (double)params[i];
    den += (double)params[i] * w[i];
  }
  if (!(den > 0.0)) return af1::set_error(AF1_ERR_INVALID_ARG, "af1_hisa_module_budgets: degenerate densities");
  for (int64_t i = 0; i < N; ++i) b_out[i] = B_l * total * w[i] / den;
  return AF1_OK;
}

int af1_budget_to_rank(double b, int64_t m, int64_t n, int64_t* r_out) {
  if (r_out == nullptr || m <= 0 || n <= 0 || !(b >= 0.0) || !std::isfinite(b))
    return af1::set_error(AF1_ERR_INVALID_ARG, "af1_budget_to_rank: need b >= 0 finite, m, n > 0");
  const double r = std::floor(b * (double)m * (double)n / (double)(m + n) + 0.5);
  *r_out = (int64_t)std::min(std::max(r, 1.0), (double)af1::kMaxCols);
  return AF1_OK;
}

}  // extern "C"
