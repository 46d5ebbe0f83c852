/*
 * sforacle.h - CPU oracle for frontier accounting (TEST INFRASTRUCTURE).
 *
 * A plain, slow, literal restatement of the paper's definitions, used only to
 * check the CUDA path: the test suite, the package smoke check and the timed
 * CPU baseline of the benchmark call it; no product code path may.  It shares
 * no code, header, table or helper with the CUDA library.
 *
 * Conventions: d is int64 nanoseconds laid out [T][R][S] row-major; stages and
 * ranks are 0-based; every count and sum is an exact integer; the only
 * floating point is the fp64 share/gain quotient (one IEEE division of two
 * converted int64 values).
 *
 * Return codes: 0 ok, 1 a negative duration, 2 a value out of range
 * (a duration or a rank-local prefix >= 2^47 ns, or a wall time outside
 * [0, 2^47)), 3 bad arguments.
 */
#ifndef SFORACLE_H
#define SFORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SFO_OK 0
#define SFO_NEGATIVE 1
#define SFO_RANGE 2
#define SFO_BADARG 3

/* label bits */
#define SFO_L_FRONTIER_ACCOUNTING (1u << 0)
#define SFO_L_DIRECT_EXPOSURE (1u << 1)
#define SFO_L_SYNC_WAIT_DEPENDENT (1u << 2)
#define SFO_L_CO_CRITICAL (1u << 3)
#define SFO_L_ROLE_AWARE_NEEDED (1u << 4)
#define SFO_L_TELEMETRY_LIMITED (1u << 5)
#define SFO_L_RAW_ONLY (1u << 6)

typedef struct sfo_ratio { int64_t num, den; } sfo_ratio;

typedef struct sfo_config {
  sfo_ratio gamma_A, gamma_G, eta_A, eta_G, tau_C, eta_Q, gamma_switch, gamma_elig, closure_max,
      overlap_max;
  int64_t denom_floor_ns;
  int32_t max_missing_ranks;
  uint32_t model_fit_mask;
} sfo_config;

/* Sec. 3 Eq. 1: prefix, max-prefix frontier, increments, lowest attaining rank.
   F, ties nullable; a, lead, mk may be null too. */
int sfo_frontier(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t* F, int64_t* a,
                 int32_t* lead, int32_t* ties, int64_t* mk);

/* Sec. 3 Eq. 2 numerators and denominators, per-(stage, rank) credit of each
   increment to its lead rank, lead counts and the per-step leading stage.
   Window of global step g is floor(g / W); row i of the outputs is global
   window floor(t0 / W) + i.  Outputs are overwritten (not accumulated). */
int sfo_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W, int64_t* X,
                int64_t* D, int64_t* E, int32_t* C, uint8_t* step_lead);

/* Top-k suspects: stages by X, (stage, rank) pairs by E; value-0 entries are
   not suspects and pad with -1.  top_pair is [nW][k][2] = (stage, rank). */
int sfo_topk(const int64_t* X, const int64_t* E, int64_t nW, int64_t S, int64_t R, int32_t k,
             int32_t* top_stage, int64_t* top_stage_value, int32_t* top_pair, int64_t* top_pair_value);

/* Sec. 4: per-rank window lower median of each stage (baseline b~). Windows
   start at step 0 of d; the last may be short. m is [nW][R][S]. */
int sfo_window_median(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W, int64_t* m);

/* Sec. 4 Eq. 4 numerator, literally: for every step, replace stage s by
   min(d, m) on every rank, recompute the frontier, accumulate F_S - F'_S. */
int sfo_direct_gain(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W, const int64_t* m,
                    int64_t* Y);

/* Whole labeler (Sec. 4, App. A-C under the stated readings).  role [R],
   missing [nW], wall [T][R] are nullable; other_stage < 0 means none.
   Per-window outputs; every pointer except cfg and labels is nullable. */
int sfo_label_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W,
                      const int32_t* role, const int32_t* missing, const int64_t* wall,
                      int32_t other_stage, const sfo_config* cfg, uint32_t* labels,
                      uint32_t* route_mask, uint32_t* amb_mask, double* share, double* gain,
                      int64_t* X, int64_t* D, int64_t* Y, int64_t* m, int32_t* n_confident,
                      int32_t* n_switch);

/* Routing baselines the paper compares against (Sec. 3 per-stage max and
   average; Sec. 6 routing table), per window and stage:
     M    = sum_t max_r d[t,r,s]                      (per-stage max)
     SUM  = sum_t sum_r d[t,r,s], as 128 bits (lo,hi)  (per-stage average x R)
     SLOW = sum_t d[t,r*_t,s], r*_t the lowest rank with the largest total
            (slowest-rank breakdown)
     RANK0= sum_t d[t,0,s]                            (rank-0 local total)
   Windows as in sfo_windows (t0, W).  Outputs overwritten; each nullable. */
int sfo_baselines(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W, int64_t* M,
                  uint64_t* SUM, int64_t* SLOW, int64_t* RANK0);

/* Localization evidence of Sec. 4, per step and stage: the lag
     L[t,s] = F[t,s] - median_r P[t,r,s]   (lower median over ranks),
   its increment dL[t,s] = L[t,s] - L[t,s-1] (L[t,-1] = 0), and the
   max-minus-second-max gap G[t,s] = F[t,s] - (second largest P[t,r,s], a tie
   at the top counting as the second; with R = 1 the gap is 0).
   Outputs [T][S], each nullable. */
int sfo_rank_lag(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t* L, int64_t* dL, int64_t* G);

/* Raw rank spread of the Sec. 6 routing table, per window and stage:
   sum_t (max_r d[t,r,s] - median_r d[t,r,s]), lower median over ranks. */
int sfo_raw_spread(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W, int64_t* SPREAD);

/* The lag evidence of Sec. 4 per window (windows as in sfo_windows):
   LW [nW][S] = sum over the window's steps of L[t,s], GW [nW][S] = sum of
   G[t,s] (the window's delta-lag sums are LW[w][s] - LW[w][s-1]).  Outputs
   overwritten; each nullable. */
int sfo_rank_lag_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W, int64_t* LW,
                         int64_t* GW);

void sfo_config_default(sfo_config* cfg);

/* Frontier within role groups (App. A role check: no global frontier across
   incompatible roles; Sec. 3 Eq. 1 applied inside each group).  group [R]
   gives each rank's group in [0, G).  For every group g and step t:
     F_g[t,s] = max of P[t,r,s] over the ranks r of g (0 for a group with no rank),
     a_g[t,s] = F_g[t,s] - F_g[t,s-1] with F_g[t,-1] = 0.
   Per window (t0, W as in sfo_windows): Xg [G][nW][S] = sum of a_g over the
   window's steps, Dg [G][nW] = sum of F_g[t,S-1].  Outputs overwritten. */
int sfo_group_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, const int32_t* group, int64_t G,
                      int64_t t0, int64_t W, int64_t* Xg, int64_t* Dg);

/* Reporting groups aggregated after the frontier (Sec. 3, accumulation
   expansion): Y [nW][K] = sum of X[w][s] over the stages s with
   stage_group[s] = k, stage_group [S] in [0, K). */
int sfo_stage_group_sum(const int64_t* X, int64_t nW, int64_t S, const int32_t* stage_group, int64_t K,
                        int64_t* Y);

#ifdef __cplusplus
}
#endif
#endif
