// Timestep-dependent expert capacity (arXiv 2604.01622, Sec. 4.2 and Table 1; the
// normalized Gaussian of the appendix "Scheduler Definitions and FLOPs Equivalence").
// Host code: turns per-sequence masking ratios into the per-group capacities k_g that
// ec_ctx_create / ec_ctx_set_capacity take.
#include <cmath>
#include <cstdint>

#include "../../include/ecmoe.h"

namespace {

double normalized_gaussian(double r, double sigma) {
  const double inv = 1.0 / (2.0 * sigma * sigma);
  const double g_r = std::exp(-(r - 0.5) * (r - 0.5) * inv);
  const double g_0 = std::exp(-0.25 * inv);   // g(0) = g(1)
  return (g_r - g_0) / (1.0 - g_0);
}

// Scheduler value s(r) in [0, 1]; NAN for an unknown scheduler.
double schedule_value(int32_t sched, double r, double sigma) {
  const double pi = 3.14159265358979323846;
  switch (sched) {
    case EC_SCHED_STATIC: return 0.5;
    case EC_SCHED_LINEAR: return r;
    case EC_SCHED_LINEAR_REV: return 1.0 - r;
    case EC_SCHED_COSINE: return 0.5 - 0.5 * std::cos(pi * r);
    case EC_SCHED_COSINE_REV: return 0.5 + 0.5 * std::cos(pi * r);
    case EC_SCHED_GAUSSIAN: return normalized_gaussian(r, sigma);
    case EC_SCHED_GAUSSIAN_REV: return 1.0 - normalized_gaussian(r, sigma);
  }
  return NAN;
}

}  // namespace

extern "C" ec_status ec_capacity_schedule(int32_t scheduler, double k_min, double k_max,
                                          double sigma, int32_t E, int32_t G,
                                          const int32_t* group_off, const double* r,
                                          int32_t* k_g) {
  if (!group_off || !r || !k_g) return EC_ERR_INVALID_ARG;
  if (scheduler < EC_SCHED_STATIC || scheduler > EC_SCHED_GAUSSIAN_REV) return EC_ERR_INVALID_ARG;
  if (!(k_min >= 0.0) || !(k_max >= k_min) || !std::isfinite(k_max)) return EC_ERR_INVALID_ARG;
  if ((scheduler == EC_SCHED_GAUSSIAN || scheduler == EC_SCHED_GAUSSIAN_REV) && !(sigma > 0.0))
    return EC_ERR_INVALID_ARG;
  if (E <= 0 || G <= 0) return EC_ERR_SHAPE;
  for (int32_t g = 0; g < G; ++g) {
    if (group_off[g + 1] < group_off[g]) return EC_ERR_SHAPE;
    if (!(r[g] >= 0.0 && r[g] <= 1.0)) return EC_ERR_INVALID_ARG;
  }
  for (int32_t g = 0; g < G; ++g) {
    double k = k_min + (k_max - k_min) * schedule_value(scheduler, r[g], sigma);
    k = k < k_min ? k_min : (k > k_max ? k_max : k);            // clamp(., k_min, k_max)
    const int64_t L = (int64_t)group_off[g + 1] - group_off[g];
    // per-sequence capacity: the share of k L / E token-expert pairs each expert takes
    int64_t c = (int64_t)std::floor(k * (double)L / (double)E + 0.5);
    c = c < 0 ? 0 : (c > L ? L : c);
    k_g[g] = (int32_t)c;
  }
  return EC_OK;
}
