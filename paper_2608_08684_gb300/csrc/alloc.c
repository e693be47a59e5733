/*
 * Host budget allocator: Sec. 4.4 and Algorithm 1 "Budget Allocation" of the
 * RippleKV paper (Eqs. 9-12, constrained by Eq. 5), and the calibration
 * average that produces its input profile (Sec. 4.3, Eq. 8).
 *
 * Compiled with -ffp-contract=off: every product and sum is rounded on its
 * own, so the result does not depend on whether the host has fused
 * multiply-add (the GPU machines are aarch64, where the compiler would otherwise
 * contract a*b+c).
 */
#include <math.h>
#include <stdlib.h>

#include "ripple.h"

int32_t ripple_keep_count(int64_t budget, int32_t seq_len, int32_t window) {
  if (seq_len < 1 || window < 1 || window > seq_len || budget < 0) return -1;
  int64_t n = budget > window ? budget : window;
  return (int32_t)(n < seq_len ? n : seq_len);
}

/* Eq. 11's clip: identity when clipping is disabled. */
static double clip_weight(double x, int clip, double lo, double hi) {
  if (!clip) return x;
  if (x < lo) x = lo;
  if (x > hi) x = hi;
  return x;
}

ripple_status ripple_alloc_budgets(const double *sens_host, int32_t n_layers, double ratio,
                                   double gamma, int64_t global_budget,
                                   int64_t *budgets_host) {
  if (sens_host == NULL || budgets_host == NULL || n_layers < 1) return RIPPLE_EINVAL;
  if (!isfinite(ratio) || ratio < 1.0) return RIPPLE_EINVAL;
  if (isnan(gamma) || (gamma > 0.0 && gamma < 1.0)) return RIPPLE_EINVAL;
  if (global_budget < 0) return RIPPLE_EINVAL;
  for (int32_t l = 0; l < n_layers; ++l)
    if (!isfinite(sens_host[l])) return RIPPLE_EINVAL;

  const int n = n_layers;
  double *w = (double *)malloc(sizeof(double) * (size_t)n * 2);
  if (w == NULL) return RIPPLE_ENOMEM;
  double *frac = w + n;

  /* Eq. 9: min-max normalisation; identical sensitivities give s_hat = 0. */
  double s_min = sens_host[0], s_max = sens_host[0];
  for (int l = 0; l < n; ++l) {
    if (sens_host[l] < s_min) s_min = sens_host[l];
    if (sens_host[l] > s_max) s_max = sens_host[l];
  }
  const int constant = (s_max == s_min);
  const double span = s_max - s_min;

  /* Eq. 10: w~_l = exp(log r * s_hat_l); Eq. 11: clip, then mean one. */
  const double log_r = log(ratio);
  const int clip = (gamma > 0.0 && isfinite(gamma));
  const double lo = clip ? 1.0 / gamma : 0.0;
  double total = 0.0;
  for (int l = 0; l < n; ++l) {
    const double s_hat = constant ? 0.0 : (sens_host[l] - s_min) / span;
    const double c = clip_weight(exp(log_r * s_hat), clip, lo, gamma);
    w[l] = c;
    total += c;
  }
  const double mean = total / (double)n;
  for (int l = 0; l < n; ++l) w[l] = w[l] / mean;

  /* Eq. 12 with Eq. 5: floor of each quota, then largest remainders. */
  const double avg = (double)global_budget / (double)n;
  int64_t assigned = 0;
  for (int l = 0; l < n; ++l) {
    const double quota = avg * w[l];
    const double base = floor(quota);
    frac[l] = quota - base;
    budgets_host[l] = (int64_t)base;
    assigned += budgets_host[l];
  }
  int64_t left = global_budget - assigned;
  /* Rank of layer l among fractional parts: larger first, ties to lower index. */
  for (int l = 0; l < n && left > 0; ++l) {
    int64_t rank = 0;
    for (int j = 0; j < n; ++j)
      if (frac[j] > frac[l] || (frac[j] == frac[l] && j < l)) ++rank;
    if (rank < left) budgets_host[l] += 1;
  }
  free(w);
  return RIPPLE_OK;
}

/* Eq. 8: s_l = (1/N) sum_i d_{i,l}, accumulated in example order. */
ripple_status ripple_sensitivity_profile(const double *d_host, int32_t n_examples,
                                         int32_t n_layers, double *s_host) {
  if (d_host == NULL || s_host == NULL || n_examples < 1 || n_layers < 1) return RIPPLE_EINVAL;
  const size_t total = (size_t)n_examples * (size_t)n_layers;
  for (size_t j = 0; j < total; ++j)
    if (!isfinite(d_host[j])) return RIPPLE_EINVAL;
  for (int32_t l = 0; l < n_layers; ++l) {
    double acc = 0.0;
    for (int32_t i = 0; i < n_examples; ++i) acc += d_host[(size_t)i * n_layers + l];
    s_host[l] = acc / (double)n_examples;
  }
  return RIPPLE_OK;
}

const char *ripple_status_string(int32_t status) {
  switch (status) {
    case RIPPLE_OK: return "ok";
    case RIPPLE_EINVAL: return "invalid argument";
    case RIPPLE_EWORKSPACE: return "workspace too small";
    case RIPPLE_EFULL: return "cache full";
    case RIPPLE_ECUDA: return "CUDA error";
    case RIPPLE_ETIMEOUT: return "in-kernel wait timed out";
    case RIPPLE_EBOUNDS: return "index out of range";
    case RIPPLE_ENOMEM: return "host allocation failed";
    default: return "unknown status";
  }
}
