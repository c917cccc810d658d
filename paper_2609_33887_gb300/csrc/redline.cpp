// Redline selection on the host (Sec. 3.2 steps (ii)-(iv) and the appendices
// on the exact binomial p-value, Holm, fixed sequence and deployment): counts
// of reference-relative violations, exact binomial p-values, the multiple
// test, deployment, budget sweeps and calibration-size quantities.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <numeric>
#include <vector>

#include "redline.h"

namespace {

constexpr double kHalfLog2Pi = 0.91893853320467274178;  // log(sqrt(2 pi))

// ---------------------------------------------------------------------------
// Binomial probabilities by Loader's saddle-point expansion (C. Loader, "Fast
// and accurate computation of binomial probabilities", 2000):
//   b(k; n, p) = sqrt(n / (2 pi k (n - k)))
//                * exp(S(n) - S(k) - S(n - k) - D(k, n p) - D(n - k, n q))
// with S(x) = log x! - log(sqrt(2 pi x) (x / e)^x), the error of Stirling's
// formula, and D(x, M) = x log(x / M) + M - x, the deviance of x from M. Both
// pieces stay small or are computed without cancellation, so the result keeps
// a relative error of a few ulps where log-gamma differences would lose
// log10(n) digits.
// ---------------------------------------------------------------------------

// S(x) for a positive integer x.
double stirling_error(double x) {
  if (x <= 15.0) {
    // x! is exact in double up to 15! (about 1.3e12)
    double f = 1.0;
    for (int i = 2; i <= static_cast<int>(x); ++i) f *= i;
    return std::log(f) - (x + 0.5) * std::log(x) + x - kHalfLog2Pi;
  }
  // Stirling series sum_k B_2k / (2k (2k - 1) x^(2k - 1)); the Bernoulli
  // numbers B_2..B_10 give 1/12, -1/360, 1/1260, -1/1680, 1/1188, and the next
  // term is below 1e-16 of S(x) for x > 15.
  const double x2 = x * x;
  return (1.0 / 12 - (1.0 / 360 - (1.0 / 1260 - (1.0 / 1680 - (1.0 / 1188) / x2) / x2) / x2) / x2) / x;
}

// D(x, M) = x log(x / M) + M - x for x >= 0, M > 0.
double deviance(double x, double M) {
  if (std::fabs(x - M) < 0.1 * (x + M)) {
    // with v = (x - M) / (x + M): log(x / M) = 2 (v + v^3/3 + v^5/5 + ...), so
    // D = (x - M) v + 2 x (v^3/3 + v^5/5 + ...), free of cancellation
    const double v = (x - M) / (x + M);
    const double v2 = v * v;
    double s = (x - M) * v;
    double e = 2.0 * x * v;
    for (int j = 1; j < 200; ++j) {
      e *= v2;
      const double s1 = s + e / (2 * j + 1);
      if (s1 == s) break;
      s = s1;
    }
    return s;
  }
  return x * std::log(x / M) + M - x;
}

// log b(k; n, p) for 0 <= k <= n, 0 < p < 1, q = 1 - p.
double log_pmf(int64_t k, int64_t n, double p, double q) {
  if (k == 0) return static_cast<double>(n) * std::log1p(-p);
  if (k == n) return static_cast<double>(n) * std::log(p);
  const double N = static_cast<double>(n), K = static_cast<double>(k), R = static_cast<double>(n - k);
  const double e = stirling_error(N) - stirling_error(K) - stirling_error(R) - deviance(K, N * p) - deviance(R, N * q);
  return e + 0.5 * std::log(N / (K * R)) - kHalfLog2Pi;
}

// Pr[Bin(n, p) <= k]. Sums the shorter tail starting from its largest term:
// below the mean the terms fall geometrically towards 0, above it towards n,
// so each sum stops once a term no longer moves it.
double binom_cdf(int64_t k, int64_t n, double p) {
  if (k < 0) return 0.0;
  if (k >= n) return 1.0;
  if (p <= 0.0) return 1.0;
  if (p >= 1.0) return 0.0;
  const double q = 1.0 - p;
  const double mean = static_cast<double>(n) * p;
  if (static_cast<double>(k) <= mean) {
    // b(j - 1) / b(j) = j q / ((n - j + 1) p) <= 1 for j <= k <= n p
    const double lead = log_pmf(k, n, p, q);
    double t = 1.0, s = 1.0;
    for (int64_t j = k; j > 0; --j) {
      t *= static_cast<double>(j) * q / (static_cast<double>(n - j + 1) * p);
      s += t;
      if (t <= s * 1e-17) break;
    }
    return std::exp(lead) * s;
  }
  // b(j + 1) / b(j) = (n - j) p / ((j + 1) q) < 1 for j > n p - q
  const double lead = log_pmf(k + 1, n, p, q);
  double t = 1.0, s = 1.0;
  for (int64_t j = k + 1; j < n; ++j) {
    t *= static_cast<double>(n - j) * p / (static_cast<double>(j + 1) * q);
    s += t;
    if (t <= s * 1e-17) break;
  }
  return 1.0 - std::exp(lead) * s;
}

bool prob_ok(double x) { return x >= 0.0 && x <= 1.0; }  // false for NaN

// Largest c with Pr[Bin(n, alpha) <= c] <= level, -1 if none. The CDF rises
// with c, so bisect between c = -1 (CDF 0) and c = n (CDF 1).
int64_t critical_count(int64_t n, double alpha, double level) {
  if (level >= 1.0) return n;
  int64_t lo = -1, hi = n;  // cdf(lo) <= level < cdf(hi)
  while (hi - lo > 1) {
    const int64_t mid = lo + (hi - lo) / 2;
    if (binom_cdf(mid, n, alpha) <= level)
      lo = mid;
    else
      hi = mid;
  }
  return lo;
}

bool better(double a, double b, int32_t higher_is_better) { return higher_is_better ? a > b : a < b; }

int check_grid(const bd_redline_grid* g) {
  if (g == nullptr || g->violations == nullptr || g->cost == nullptr) return BD_ERR_NULL;
  if (g->m < 1 || g->m > 65536 || g->n < 0 || g->n > 1000000000LL) return BD_ERR_SHAPE;
  if (g->ref_index < 0 || g->ref_index >= g->m) return BD_ERR_SHAPE;
  for (int32_t i = 0; i < g->m; ++i) {
    if (g->violations[i] < 0 || g->violations[i] > g->n) return BD_ERR_SHAPE;
    if (!std::isfinite(g->cost[i])) return BD_ERR_ARG;
  }
  return BD_OK;
}

int check_rule(const bd_redline_rule* r, int32_t m) {
  if (r == nullptr) return BD_ERR_NULL;
  if (!(r->delta > 0.0 && r->delta <= 1.0)) return BD_ERR_ARG;
  if (r->procedure == BD_REDLINE_FIXED_SEQUENCE) {
    if (r->order == nullptr) return BD_ERR_NULL;
    std::vector<char> seen(static_cast<size_t>(m), 0);
    for (int32_t i = 0; i < m; ++i) {
      const int32_t o = r->order[i];
      if (o < 0 || o >= m || seen[o]) return BD_ERR_ARG;
      seen[o] = 1;
    }
  } else if (r->procedure != BD_REDLINE_HOLM && r->procedure != BD_REDLINE_BONFERRONI) {
    return BD_ERR_ARG;
  }
  return BD_OK;
}

// Step (iii) on checked arguments.
void run_test(const double* p, int32_t m, const bd_redline_rule& r, uint8_t* valid) {
  std::fill(valid, valid + m, uint8_t{0});
  if (r.procedure == BD_REDLINE_HOLM) {
    std::vector<int32_t> idx(static_cast<size_t>(m));
    std::iota(idx.begin(), idx.end(), 0);
    std::stable_sort(idx.begin(), idx.end(), [&](int32_t a, int32_t b) { return p[a] < p[b]; });
    for (int32_t i = 0; i < m; ++i) {  // rank i + 1
      if (p[idx[i]] <= r.delta / static_cast<double>(m - i))
        valid[idx[i]] = 1;
      else
        break;
    }
  } else if (r.procedure == BD_REDLINE_BONFERRONI) {
    const double t = r.delta / static_cast<double>(m);
    for (int32_t i = 0; i < m; ++i) valid[i] = p[i] <= t ? 1 : 0;
  } else {
    for (int32_t i = 0; i < m; ++i) {
      const int32_t c = r.order[i];
      if (p[c] <= r.delta)
        valid[c] = 1;
      else
        break;
    }
  }
}

int32_t run_deploy(const uint8_t* valid, const double* cost, int32_t m, int32_t hib, int32_t ref) {
  int32_t best = -1;
  for (int32_t i = 0; i < m; ++i)
    if (valid[i] && (best < 0 || better(cost[i], cost[best], hib))) best = i;
  return best < 0 ? ref : best;
}

}  // namespace

extern "C" {

int bd_binom_cdf(int64_t k, int64_t n, double p, double* out) {
  if (out == nullptr) return BD_ERR_NULL;
  if (n < 0) return BD_ERR_SHAPE;
  if (!prob_ok(p)) return BD_ERR_ARG;
  *out = binom_cdf(k, n, p);
  return BD_OK;
}

int bd_redline_violations(const uint8_t* outcomes, int64_t n, int32_t m, int64_t ld, int32_t ref_index,
                          int64_t* violations) {
  if (violations == nullptr || (outcomes == nullptr && n > 0)) return BD_ERR_NULL;
  if (n < 0 || m < 1 || ld < m || ref_index < 0 || ref_index >= m) return BD_ERR_SHAPE;
  std::fill(violations, violations + m, int64_t{0});
  for (int64_t i = 0; i < n; ++i) {
    const uint8_t* row = outcomes + i * ld;
    if (row[ref_index] == 0) continue;
    for (int32_t j = 0; j < m; ++j) violations[j] += row[j] == 0 ? 1 : 0;
  }
  return BD_OK;
}

int bd_redline_pvalues(const int64_t* violations, int32_t m, int64_t n, double alpha, double* p) {
  if (violations == nullptr || p == nullptr) return BD_ERR_NULL;
  if (m < 1 || n < 0) return BD_ERR_SHAPE;
  if (!prob_ok(alpha)) return BD_ERR_ARG;
  for (int32_t i = 0; i < m; ++i)
    if (violations[i] < 0 || violations[i] > n) return BD_ERR_SHAPE;
  for (int32_t i = 0; i < m; ++i) p[i] = binom_cdf(violations[i], n, alpha);
  return BD_OK;
}

int bd_redline_test(const double* p, int32_t m, const bd_redline_rule* rule, uint8_t* valid) {
  if (p == nullptr || valid == nullptr) return BD_ERR_NULL;
  if (m < 1) return BD_ERR_SHAPE;
  if (const int st = check_rule(rule, m)) return st;
  for (int32_t i = 0; i < m; ++i)
    if (std::isnan(p[i])) return BD_ERR_ARG;
  run_test(p, m, *rule, valid);
  return BD_OK;
}

int bd_redline_deploy(const uint8_t* valid, const double* cost, int32_t m, int32_t higher_is_better,
                      int32_t ref_index, int32_t* deployed) {
  if (valid == nullptr || cost == nullptr || deployed == nullptr) return BD_ERR_NULL;
  if (m < 1 || ref_index < 0 || ref_index >= m) return BD_ERR_SHAPE;
  for (int32_t i = 0; i < m; ++i)
    if (std::isnan(cost[i])) return BD_ERR_ARG;
  *deployed = run_deploy(valid, cost, m, higher_is_better, ref_index);
  return BD_OK;
}

int bd_redline_select(const bd_redline_grid* grid, double alpha, const bd_redline_rule* rule, double* p,
                      uint8_t* valid, int32_t* deployed) {
  if (deployed == nullptr) return BD_ERR_NULL;
  if (const int st = check_grid(grid)) return st;
  if (const int st = check_rule(rule, grid->m)) return st;
  if (!prob_ok(alpha)) return BD_ERR_ARG;
  const int32_t m = grid->m;
  std::vector<double> pv(static_cast<size_t>(m));
  std::vector<uint8_t> ok(static_cast<size_t>(m));
  for (int32_t i = 0; i < m; ++i) pv[i] = binom_cdf(grid->violations[i], grid->n, alpha);
  run_test(pv.data(), m, *rule, ok.data());
  if (p != nullptr) std::copy(pv.begin(), pv.end(), p);
  if (valid != nullptr) std::copy(ok.begin(), ok.end(), valid);
  *deployed = run_deploy(ok.data(), grid->cost, m, grid->higher_is_better, grid->ref_index);
  return BD_OK;
}

int bd_redline_sweep(const bd_redline_grid* grid, const double* alphas, int32_t n_alpha, const bd_redline_rule* rule,
                     int32_t* deployed, int32_t* n_valid, int32_t* first_gain) {
  if (deployed == nullptr || (alphas == nullptr && n_alpha > 0)) return BD_ERR_NULL;
  if (n_alpha < 0) return BD_ERR_SHAPE;
  if (const int st = check_grid(grid)) return st;
  if (const int st = check_rule(rule, grid->m)) return st;
  for (int32_t a = 0; a < n_alpha; ++a)
    if (!prob_ok(alphas[a])) return BD_ERR_ARG;
  const int32_t m = grid->m;
  std::vector<double> pv(static_cast<size_t>(m));
  std::vector<uint8_t> ok(static_cast<size_t>(m));
  int32_t gain = -1;
  for (int32_t a = 0; a < n_alpha; ++a) {
    for (int32_t i = 0; i < m; ++i) pv[i] = binom_cdf(grid->violations[i], grid->n, alphas[a]);
    run_test(pv.data(), m, *rule, ok.data());
    const int32_t d = run_deploy(ok.data(), grid->cost, m, grid->higher_is_better, grid->ref_index);
    deployed[a] = d;
    if (n_valid != nullptr) n_valid[a] = static_cast<int32_t>(std::count(ok.begin(), ok.end(), uint8_t{1}));
    if (gain < 0 && better(grid->cost[d], grid->cost[grid->ref_index], grid->higher_is_better)) gain = a;
  }
  if (first_gain != nullptr) *first_gain = gain;
  return BD_OK;
}

int bd_redline_critical_count(int64_t n, double alpha, double level, int64_t* c) {
  if (c == nullptr) return BD_ERR_NULL;
  if (n < 0) return BD_ERR_SHAPE;
  if (!prob_ok(alpha) || !prob_ok(level)) return BD_ERR_ARG;
  *c = critical_count(n, alpha, level);
  return BD_OK;
}

int bd_redline_power(int64_t n, double risk, double alpha, double level, double* power) {
  if (power == nullptr) return BD_ERR_NULL;
  if (n < 0) return BD_ERR_SHAPE;
  if (!prob_ok(alpha) || !prob_ok(level) || !prob_ok(risk)) return BD_ERR_ARG;
  const int64_t c = critical_count(n, alpha, level);
  *power = c >= 0 ? binom_cdf(c, n, risk) : 0.0;
  return BD_OK;
}

int bd_redline_min_calibration(double risk, double alpha, double level, double target, int64_t n_max, int64_t* n0) {
  if (n0 == nullptr) return BD_ERR_NULL;
  if (n_max < 1 || n_max > 10000000LL) return BD_ERR_SHAPE;
  if (!prob_ok(alpha) || !prob_ok(level) || !prob_ok(risk) || !prob_ok(target)) return BD_ERR_ARG;
  // Walk n down from n_max. The critical count never grows as n falls (the
  // CDF at a fixed count rises as n falls), so c(n - 1) is found from c(n)
  // by stepping down.
  int64_t c = critical_count(n_max, alpha, level);
  for (int64_t n = n_max; n >= 1; --n) {
    if (n < n_max) {
      if (c > n) c = n;
      while (c >= 0 && binom_cdf(c, n, alpha) > level) --c;
    }
    const double pw = c >= 0 ? binom_cdf(c, n, risk) : 0.0;
    if (pw < target) {
      *n0 = n == n_max ? -1 : n + 1;
      return BD_OK;
    }
  }
  *n0 = 1;
  return BD_OK;
}

int bd_redline_tpf(const int32_t* counts, int32_t steps, int32_t T, int64_t ld, int32_t n_seq, double* tpf) {
  if (tpf == nullptr || (counts == nullptr && steps > 0)) return BD_ERR_NULL;
  if (steps < 0 || T < 1 || ld < T || n_seq < 1) return BD_ERR_SHAPE;
  std::vector<int64_t> sum(static_cast<size_t>(T), 0);
  for (int32_t s = 0; s < steps; ++s)
    for (int32_t t = 0; t < T; ++t) {
      const int32_t v = counts[s * ld + t];
      if (v < 0) return BD_ERR_ARG;
      sum[t] += v;
    }
  for (int32_t t = 0; t < T; ++t)
    tpf[t] = steps == 0 ? 0.0 : static_cast<double>(sum[t]) / (static_cast<double>(steps) * n_seq);
  return BD_OK;
}

}  // extern "C"
