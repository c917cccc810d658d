/*
 * redline: choosing the serving configuration to deploy from calibration
 * outcomes, with a finite-sample bound on its reference-relative risk.
 *
 * The commit step of bdcommit.h scores a whole grid of accept thresholds per
 * forward; these entry points turn the calibration record of such a grid into
 * the configuration that is deployed (Sec. 3.2, "Redline in four steps"):
 *   (i)   a grid of m configurations that includes the reference, n
 *         calibration prompts, a risk budget alpha and a failure probability
 *         delta;
 *   (ii)  for every configuration, V = the number of prompts the reference
 *         answers correctly and the configuration does not (the empirical
 *         form of the joint risk of Eq. 1), and the exact one-sided binomial
 *         p-value p = Pr[Bin(n, alpha) <= V] for H0: R > alpha (appendix on
 *         the exact binomial p-value);
 *   (iii) a multiple test at family-wise level delta: Holm's step-down
 *         (primary), Bonferroni (its conservative floor) or the fixed-sequence
 *         walk (secondary) (appendices on Holm and on fixed sequence);
 *   (iv)  deployment of the valid configuration with the best cost, the
 *         highest TPF or the least memory, or of the reference when none is
 *         valid (deployment appendix).
 * Plus the calibration-size quantities of the paper's sample-size table and
 * the cost input that the commit step's per-threshold counts provide.
 *
 * Everything here runs on the host, in double precision, synchronously; no
 * entry point touches the GPU, allocates device memory or keeps state between
 * calls. All pointers are host pointers owned by the caller, read (const) or
 * written only within the sizes given. Return value: 0 (BD_OK) or a negative
 * bd_status of bdcommit.h; a rejected call writes no output.
 *
 * Numerics. p-values are computed from one binomial probability evaluated
 * with Loader's saddle-point expansion (C. Loader, "Fast and accurate
 * computation of binomial probabilities", 2000) and a ratio recurrence over
 * the shorter tail; relative error below 1e-12 wherever the value is a normal
 * double. Decisions compare those doubles with delta / k in double precision.
 */
#ifndef REDLINE_H
#define REDLINE_H

#include <stdint.h>

#include "bdcommit.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Multiple-testing procedures of step (iii). */
typedef enum {
  BD_REDLINE_HOLM = 0,          /* sort p ascending; reject while p_(i) <= delta / (m - i + 1); stop at the first failure */
  BD_REDLINE_BONFERRONI = 1,    /* reject every p <= delta / m */
  BD_REDLINE_FIXED_SEQUENCE = 2 /* walk `order`, reject while p <= delta; stop at the first failure */
} bd_redline_procedure;

/* One calibration grid.
 *   m           configurations, 1 <= m <= 65536, the reference included
 *   n           calibration prompts, 0 <= n <= 1e9
 *   violations  [m] V of each configuration, 0 <= V <= n (V of the reference is 0
 *               when it comes from bd_redline_violations)
 *   cost        [m] finite cost measure: TPF or accepted tokens per target
 *               forward (higher_is_better = 1), or weight memory (0)
 *   ref_index   the reference configuration, 0 <= ref_index < m */
typedef struct {
  int32_t m;
  int64_t n;
  const int64_t* violations;
  const double* cost;
  int32_t ref_index;
  int32_t higher_is_better;
} bd_redline_grid;

/* The test of step (iii).
 *   delta      family-wise error level, 0 < delta <= 1 (0.10 in the paper)
 *   procedure  a bd_redline_procedure
 *   order      [m] permutation of 0..m-1 giving the fixed-sequence walk (fixed
 *              in advance, independent of the calibration outcomes); ignored
 *              (may be NULL) for the other procedures */
typedef struct {
  double delta;
  int32_t procedure;
  const int32_t* order;
} bd_redline_rule;

/* Pr[Bin(n, p) <= k]: 0 for k < 0, 1 for k >= n. n >= 0, 0 <= p <= 1.
 * BD_ERR_NULL without `out`; BD_ERR_SHAPE for n < 0; BD_ERR_ARG for p outside
 * [0, 1] or NaN. */
int bd_binom_cdf(int64_t k, int64_t n, double p, double* out);

/* Step (ii), counting (Eq. 1): violations[lam] = #{i : outcomes[i*ld + ref_index]
 * != 0 and outcomes[i*ld + lam] == 0} for the prompt-major correctness matrix
 * outcomes [n][ld] (bytes, nonzero = correct), lam < m <= ld.
 * BD_ERR_NULL for NULL pointers (outcomes may be NULL when n == 0);
 * BD_ERR_SHAPE for n < 0, m < 1, ld < m or ref_index outside [0, m). */
int bd_redline_violations(const uint8_t* outcomes, int64_t n, int32_t m, int64_t ld, int32_t ref_index,
                          int64_t* violations);

/* Step (ii), p-values: p[lam] = Pr[Bin(n, alpha) <= violations[lam]].
 * BD_ERR_SHAPE for m < 1, n < 0 or a count outside [0, n]; BD_ERR_ARG for alpha
 * outside [0, 1] or NaN. */
int bd_redline_pvalues(const int64_t* violations, int32_t m, int64_t n, double alpha, double* p);

/* Step (iii): valid[lam] = 1 when H0 of lam is rejected, else 0.
 * BD_ERR_SHAPE for m < 1; BD_ERR_ARG for delta outside (0, 1], a NaN p-value,
 * an unknown procedure, or (fixed sequence) an order that is not a
 * permutation of 0..m-1; BD_ERR_NULL when fixed sequence gets no order. */
int bd_redline_test(const double* p, int32_t m, const bd_redline_rule* rule, uint8_t* valid);

/* Step (iv): the valid configuration with the best cost (ties: the lowest
 * index), or ref_index when none is valid.
 * BD_ERR_SHAPE for m < 1 or ref_index outside [0, m); BD_ERR_ARG for a NaN cost. */
int bd_redline_deploy(const uint8_t* valid, const double* cost, int32_t m, int32_t higher_is_better,
                      int32_t ref_index, int32_t* deployed);

/* Steps (ii)-(iv) at one budget. p [m] and valid [m] may be NULL when not wanted;
 * *deployed receives the deployed configuration. */
int bd_redline_select(const bd_redline_grid* grid, double alpha, const bd_redline_rule* rule, double* p,
                      uint8_t* valid, int32_t* deployed);

/* Steps (ii)-(iv) at every budget alphas[0..n_alpha-1] (any order).
 *   deployed    [n_alpha] deployed configuration per budget
 *   n_valid     [n_alpha] number of valid configurations per budget, or NULL
 *   first_gain  index of the first budget, in the given order, whose deployed
 *               configuration has a strictly better cost than the reference,
 *               -1 if none; with ascending budgets this is the smallest budget
 *               with a gain of the error-levels appendix. May be NULL.
 * BD_ERR_SHAPE for n_alpha < 0. */
int bd_redline_sweep(const bd_redline_grid* grid, const double* alphas, int32_t n_alpha, const bd_redline_rule* rule,
                     int32_t* deployed, int32_t* n_valid, int32_t* first_gain);

/* Calibration size (sample-size table (b)): the largest count c with
 * Pr[Bin(n, alpha) <= c] <= level, or -1 when even c = 0 fails; c / n is the
 * largest empirical risk that passes a test at that level.
 * BD_ERR_SHAPE for n < 0; BD_ERR_ARG for alpha or level outside [0, 1]. */
int bd_redline_critical_count(int64_t n, double alpha, double level, int64_t* c);

/* Power of the exact test (sample-size table (a)): the probability that a
 * configuration of true joint risk `risk` passes a test at `level`,
 * Pr[Bin(n, risk) <= c] with c = bd_redline_critical_count(n, alpha, level)
 * (0 when c = -1). Same argument errors, plus BD_ERR_ARG for risk outside [0, 1]. */
int bd_redline_power(int64_t n, double risk, double alpha, double level, double* power);

/* Prompts needed (sample-size table (a)): the smallest n0 in [1, n_max] such
 * that the power is at least `target` at every n in [n0, n_max]; -1 when the
 * power at n_max is below the target. The power is not monotone in n (the
 * critical count moves in integer steps), which is why every n up to n_max is
 * checked.
 * BD_ERR_SHAPE for n_max < 1 or n_max > 10,000,000; BD_ERR_ARG as above and
 * for target outside [0, 1]. */
int bd_redline_min_calibration(double risk, double alpha, double level, double target, int64_t n_max, int64_t* n0);

/* Cost input from the commit step: tokens committed per forward and per
 * sequence at each accept threshold,
 *   tpf[t] = sum_s counts[s * ld + t] / (steps * n_seq),
 * for the per-threshold counts (bd_exec.out_counts) of `steps` forwards over
 * n_seq sequences, copied to host memory. 0 when steps == 0.
 * BD_ERR_SHAPE for steps < 0, T < 1, ld < T or n_seq < 1; BD_ERR_ARG for a
 * negative count. */
int bd_redline_tpf(const int32_t* counts, int32_t steps, int32_t T, int64_t ld, int32_t n_seq, double* tpf);

#ifdef __cplusplus
}
#endif

#endif /* REDLINE_H */
