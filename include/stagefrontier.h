/*
 * stagefrontier.h - C ABI of libstagefrontier, synchronization-aware frontier
 * accounting over a telemetry tensor of per-(step, rank, stage) durations,
 * computed by CUDA kernels for sm_103a (GB300).
 *
 * Problem statement (Sec. 3, Eq. 1-2): for step t, rank r and ordered stage s
 * let d[t,r,s] >= 0 be the measured duration.  The rank-local prefix is
 * P[t,r,s] = sum_{j<=s} d[t,r,j], the frontier F[t,s] = max_r P[t,r,s] with
 * F[t,-1] = 0, the increment a[t,s] = F[t,s] - F[t,s-1] >= 0 and the exposed
 * makespan F[t,S-1] = sum_s a[t,s] (Theorem 1).  A window of steps has stage
 * share A_s = sum_t a[t,s] / sum_t F[t,S-1].
 *
 * Conventions shared by every entry point
 *   - d is int64 nanoseconds, row-major [T][R][S], contiguous, 16-byte aligned
 *     (else SF_EINVAL_ALIGN).  Stages and ranks are 0-based.
 *   - Every data pointer is a DEVICE pointer owned by the caller unless the
 *     argument says "host".  The library never allocates device memory, never
 *     frees, and never synchronizes: work is enqueued on `stream` and the call
 *     returns.  Output buffers must not alias inputs.
 *   - Host-detectable errors (shapes, null required pointers, alignment,
 *     configuration) return a negative sf_status before anything is enqueued.
 *   - Errors found on the device (invalid durations, a bounded wait that ran
 *     out) are OR-ed into the caller's device word `*status` (nullable; the
 *     caller zeroes it and reads it after its own synchronization).  When a
 *     status bit is set, the outputs of that call are unspecified.
 *   - Supported shapes: 1 <= T, 1 <= R <= 65536, 1 <= S <= 32,
 *     1 <= W <= 65536 (window length in steps), 1 <= k <= 32.
 *   - Valid durations satisfy 0 <= d < 2^47 and every rank total
 *     P[t,r,S-1] < 2^47 ns (about 39 hours per step); anything else sets
 *     SF_ST_NEGATIVE or SF_ST_RANGE.  All sums over a window then fit int64.
 *   - Ties: the lead rank of (t,s) is the LOWEST rank attaining F[t,s] (how
 *     many ranks attain it is reported by sf_frontier_ties); the leading stage
 *     of a step is the lowest stage with the largest increment.
 *   - Integer outputs are exact and deterministic (integer atomics commute);
 *     fp64 outputs are one IEEE division of two int64 values.
 */
#ifndef STAGEFRONTIER_H
#define STAGEFRONTIER_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum sf_status {
  SF_OK = 0,
  SF_EINVAL = -1,        /* bad shape, null required pointer or bad configuration */
  SF_EINVAL_ALIGN = -2,  /* a pointer is not aligned as documented */
  SF_EUNSUPPORTED = -3,  /* shape outside the supported limits */
  SF_ECUDA = -4,         /* a CUDA runtime call (launch, attribute, driver entry) failed */
  SF_EWORKSPACE = -5     /* workspace pointer null or smaller than required */
} sf_status;

/* device status bits */
#define SF_ST_NEGATIVE 1u /* some duration (or wall time) was negative */
#define SF_ST_RANGE 2u    /* some duration, rank total or wall time was >= 2^47 */
#define SF_ST_TIMEOUT 4u  /* a bounded device-side wait gave up; outputs incomplete */
#define SF_ST_INDEX 8u    /* an index input (a rank's group id) was out of range; that rank was skipped */

/* Label bits (Sec. 4 Tab. core labels, App. B, App. C).  RAW_ONLY marks a
   window whose denominator is below the floor: raw advances, no shares. */
#define SF_LABEL_FRONTIER_ACCOUNTING (1u << 0)
#define SF_LABEL_DIRECT_EXPOSURE (1u << 1)
#define SF_LABEL_SYNC_WAIT_DEPENDENT (1u << 2)
#define SF_LABEL_CO_CRITICAL (1u << 3)
#define SF_LABEL_ROLE_AWARE_NEEDED (1u << 4)
#define SF_LABEL_TELEMETRY_LIMITED (1u << 5)
#define SF_LABEL_RAW_ONLY (1u << 6)

/* step_lead byte written by sf_direct_gain: low 5 bits = leading stage,
   bit 7 = the step is a confident unique leader (Sec. 4). */
#define SF_STEP_CONFIDENT 0x80u

/* Human-readable name of a status code (host string, never null). */
const char* sf_status_str(int code);

/* Number of windows a call covering global steps [t0, t0+T) touches:
   floor((t0+T-1)/W) - floor(t0/W) + 1.  Returns 0 on bad arguments. */
int64_t sf_num_windows(int64_t t0, int64_t T, int64_t W);

/* Kernels this library has launched since it was loaded (all entry points). */
uint64_t sf_launch_count(void);

/* Self-test of the device-side bounded waits every pipelined kernel uses: a
   one-CTA kernel waits on a barrier phase that never completes, gives up after
   limit_ns (0 < limit_ns <= 2 s) and ORs SF_ST_TIMEOUT into *status (device,
   required).  The kernel then exits normally; nothing faults or traps. */
sf_status sf_selftest_bounded_wait(uint64_t limit_ns, uint32_t* status, cudaStream_t stream);

/*
 * sf_frontier - Sec. 3 Eq. 1 on every step.
 *   d         [T][R][S] durations (device, 16-byte aligned).
 *   a         [T][S] increments a[t,s] (device, nullable).
 *   lead      [T][S] lowest rank attaining F[t,s] (device, nullable).
 *   makespan  [T] exposed makespan F[t,S-1] (device, nullable).
 *   status    device error word (nullable).
 * At least one output must be non-null.
 */
sf_status sf_frontier(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t* a, int32_t* lead,
                      int64_t* makespan, uint32_t* status, cudaStream_t stream);

/*
 * sf_frontier_ties - the size of the lead rank's tie set, among the
 * localization evidence of Sec. 4 (the "latest-rank tie set"; Fig. 1 has a
 * real tie at the backward boundary): ties[t,s] = #{r : P[t,r,s] = F[t,s]},
 * the number of ranks whose prefix reaches the frontier.  1 marks a unique
 * lead rank; more, a tie that sf_frontier resolved to the lowest rank.
 *   d       [T][R][S] durations (device, 16-byte aligned).
 *   a       [T][S] increments from sf_frontier on the same d (device, 8-byte
 *           aligned); F[t,s] is rebuilt as their prefix over s.
 *   ties    [T][S] int32 (device, 4-byte aligned, caller-owned).
 *   status  device error word (nullable): SF_ST_NEGATIVE / SF_ST_RANGE as in
 *           sf_frontier.
 * Reads d once more (one CTA per step range).  Errors: SF_EINVAL (null d, a
 * or ties, bad shape), SF_EINVAL_ALIGN.
 */
sf_status sf_frontier_ties(const int64_t* d, int64_t T, int64_t R, int64_t S, const int64_t* a, int32_t* ties,
                           uint32_t* status, cudaStream_t stream);

/*
 * sf_window_aggregate - Eq. 2 numerators and denominators plus per-(stage,
 * rank) credit, fused into the frontier pass.  Global step g = t0 + t belongs
 * to window floor(g / W); output row i is global window floor(t0 / W) + i,
 * i < sf_num_windows(t0, T, W).  A chunked caller passes the same buffers
 * with successive t0 and accumulate = 1 so windows that straddle chunks sum
 * correctly.
 *   X         [nW][S]    sum_t a[t,s]                            (device, required)
 *   D         [nW]       sum_t F[t,S-1]                          (device, required)
 *   E         [nW][S][R] sum of a[t,s] over steps whose lead rank is r (device, nullable)
 *   C         [nW][S][R] number of steps whose lead rank at s is r (device, nullable)
 *   step_lead [T]        leading stage argmax_s a[t,s]           (device, nullable)
 *   accumulate 0: the call first zeroes X, D, E, C; 1: adds to their contents.
 */
sf_status sf_window_aggregate(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0,
                              int64_t W, int64_t* X, int64_t* D, int64_t* E, int32_t* C,
                              uint8_t* step_lead, int32_t accumulate, uint32_t* status,
                              cudaStream_t stream);

/*
 * sf_window_baselines - the routing baselines the paper compares frontier
 * accounting against (Sec. 3 per-stage max and average, Props 1-2; Sec. 6
 * routing table), per window and stage, in one pass over d:
 *   M     [nW][S]    sum_t max_r d[t,r,s]                  (per-stage max)
 *   SUM   [nW][S][2] sum_t sum_r d[t,r,s] as a 128-bit (lo, hi) pair
 *                    (per-stage average times R; exact)
 *   SLOW  [nW][S]    sum_t d[t,r*,s], r* the step's slowest rank (largest total,
 *                    lowest rank on ties): the slowest-rank breakdown
 *   RANK0 [nW][S]    sum_t d[t,0,s]                          (rank-0 local total)
 * Windows, t0 and accumulate as in sf_window_aggregate; all outputs device,
 * required.
 */
sf_status sf_window_baselines(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W,
                              int64_t* M, uint64_t* SUM, int64_t* SLOW, int64_t* RANK0,
                              int32_t accumulate, uint32_t* status, cudaStream_t stream);

/*
 * sf_rank_lag - localization evidence of Sec. 4 per step and stage:
 *   L  [T][S] lag F[t,s] - median_r P[t,r,s] (lower median over ranks),
 *   dL [T][S] its increment L[t,s] - L[t,s-1] (L[t,-1] = 0),
 *   G  [T][S] max-minus-second-max gap F[t,s] - (second largest P[t,r,s]; a
 *             tie at the top counts as the second, so ties give 0; R = 1 gives 0).
 * Outputs device, nullable (at least one).  workspace: device, 256-byte
 * aligned, at least one step's scratch; sf_rank_workspace_size(T, R, S)
 * bytes (about 40 MB, so that the scratch stays in L2) processes the steps
 * in the fewest chunks that still fit L2.  The workspace is overwritten and
 * may be reused as soon as the call's work on `stream` is done.
 */
sf_status sf_rank_lag(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t* L, int64_t* dL, int64_t* G,
                      void* workspace, size_t workspace_bytes, uint32_t* status, cudaStream_t stream);

/*
 * sf_raw_spread - the raw rank spread of the Sec. 6 routing table, per window
 * and stage: sum_t (max_r d[t,r,s] - median_r d[t,r,s]), lower median over
 * ranks.  spread [nW][S] device; windows, t0 and accumulate as in
 * sf_window_aggregate; workspace as in sf_rank_lag.
 */
sf_status sf_raw_spread(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W,
                        int64_t* spread, int32_t accumulate, void* workspace, size_t workspace_bytes,
                        uint32_t* status, cudaStream_t stream);

/*
 * sf_rank_lag_windows - the same evidence as window evidence: per window and
 * stage, Lw = sum_t L[t,s] and Gw = sum_t G[t,s] (the window's delta-lag sums
 * are Lw[w][s] - Lw[w][s-1]).  Lw, Gw [nW][S] device, nullable (at least
 * one); windows, t0 and accumulate as in sf_window_aggregate; workspace as in
 * sf_rank_lag.
 */
sf_status sf_rank_lag_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W,
                              int64_t* Lw, int64_t* Gw, int32_t accumulate, void* workspace, size_t workspace_bytes,
                              uint32_t* status, cudaStream_t stream);

/* Suggested workspace bytes for sf_rank_lag, sf_rank_lag_windows and sf_raw_spread (0 for a bad shape). */
size_t sf_rank_workspace_size(int64_t T, int64_t R, int64_t S);

/*
 * sf_group_aggregate - the frontier taken within role groups.  The App. A
 * contract check forbids one global frontier across ranks whose roles
 * differ (the labeler then emits role_aware_needed); with a rank -> group
 * map the frontier of Sec. 3 Eq. 1 is taken inside each group instead:
 *   F_g[t,s] = max of P[t,r,s] over the ranks r of group g (0 if g has none),
 *   a_g[t,s] = F_g[t,s] - F_g[t,s-1], F_g[t,-1] = 0,
 *   Xg [nW][G][S] sum_t a_g[t,s],  Dg [nW][G] sum_t F_g[t,S-1]   (device, required)
 * group [R] int32 device: each rank's group in [0, G); a rank whose id is
 * outside that range is left out and SF_ST_INDEX is set.  1 <= G <= 4096,
 * G*S <= 4096.  Windows, t0 and accumulate as in sf_window_aggregate.  The
 * group Xg[:, g, :], Dg[:, g] feed sf_label_gates like X, D.
 */
sf_status sf_group_aggregate(const int64_t* d, int64_t T, int64_t R, int64_t S, const int32_t* group, int64_t G,
                             int64_t t0, int64_t W, int64_t* Xg, int64_t* Dg, int32_t accumulate, uint32_t* status,
                             cudaStream_t stream);

/*
 * sf_stage_group_sum - reporting groups aggregated after the frontier
 * (Sec. 3: with gradient accumulation the ordered stage list is expanded by
 * accumulation index before the frontier, and semantic groups such as
 * "forward" or "backward" are summed only afterwards):
 *   Y [nW][K] = sum of X[w][s] over the stages s with stage_group[s] = k.
 * X [nW][S] device; stage_group [S] HOST array, values in [0, K), 1 <= K <= 32;
 * Y device, overwritten.  nW = 0 is a no-op.
 */
sf_status sf_stage_group_sum(const int64_t* X, int64_t nW, int64_t S, const int32_t* stage_group, int64_t K,
                             int64_t* Y, cudaStream_t stream);

/*
 * sf_gathered_to_steps - rank-major ingest.  The window-boundary gather of
 * Sec. 5 leaves each window's telemetry as one [R][n][S] block (each rank's
 * [n, S] buffer, in rank order).  This converts ceil(T / N) such blocks,
 * stored one after another (block b holds steps b*N .. min(T, (b+1)*N) - 1,
 * so only the last may be short), into the [T][R][S] layout every other
 * entry point reads.  src and dst device, 16-byte aligned, not overlapping.
 */
sf_status sf_gathered_to_steps(const int64_t* src, int64_t T, int64_t R, int64_t S, int64_t N, int64_t* dst,
                               cudaStream_t stream);

/*
 * sf_topk_suspects - per window, the k stages with the largest X (Sec. 4
 * routing uses the top two shares) and the k (stage, rank) pairs with the
 * largest lead-rank credit E.  Order: value descending, then lower stage,
 * then lower rank.  Entries with value 0 are not suspects; unused slots hold
 * -1 (values 0).
 *   X [nW][S], E [nW][S][R] (device; E nullable when no pair output is asked)
 *   top_stage [nW][k], top_stage_value [nW][k] (device, nullable)
 *   top_pair [nW][k][2] = (stage, rank), top_pair_value [nW][k] (device, nullable)
 */
sf_status sf_topk_suspects(const int64_t* X, const int64_t* E, int64_t nW, int64_t S, int64_t R,
                           int32_t k, int32_t* top_stage, int64_t* top_stage_value,
                           int32_t* top_pair, int64_t* top_pair_value, cudaStream_t stream);

/* Labeler thresholds as exact rationals num/den (0 <= num <= 2^31,
   0 < den <= 2^31).  Defaults (App. C): gamma_A 2/5, gamma_G 1/10,
   eta_A = eta_G 1/20, tau_C 4/5, closure_max 1/20, overlap_max 1/100,
   max_missing_ranks 0, model_fit_mask 0 (W_s = 0).  eta_Q, gamma_switch and
   gamma_elig have no published value: 1/20, 1/4, 1/2.  denom_floor_ns 1. */
typedef struct sf_ratio {
  int64_t num, den;
} sf_ratio;

typedef struct sf_label_config {
  sf_ratio gamma_A, gamma_G, eta_A, eta_G, tau_C, eta_Q, gamma_switch, gamma_elig, closure_max,
      overlap_max;
  int64_t denom_floor_ns;
  int32_t max_missing_ranks;
  uint32_t model_fit_mask; /* bit s set: workload semantics support sync-wait dependence (W_s = 1) */
} sf_label_config;

/* Fill *cfg (host) with the defaults above. */
void sf_label_config_default(sf_label_config* cfg);

/*
 * sf_window_median - the per-rank window baseline of Sec. 4 (Eq. 4): for each
 * window w (steps [wW, min((w+1)W, T)) of d, starting at d's first step), rank
 * r and stage s, the LOWER median of {d[t,r,s]}: element floor((n-1)/2) of the
 * ascending order, n the window's step count.
 *   m  [nW][R][S] (device), nW = ceil(T / W).
 */
sf_status sf_window_median(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W,
                           int64_t* m, uint32_t* status, cudaStream_t stream);

/*
 * sf_direct_gain - the evidence pass of the labeler (Sec. 4): per window the
 * Eq. 2 numerators X and denominator D, optionally the lead-rank credit E and
 * lead counts C exactly as sf_window_aggregate defines them (so one pass over
 * d serves both), the Eq. 4 numerators
 * Y[w,s] = sum_t (F[t,S-1] - F'[t,S-1]) where F' replaces stage s by the
 * clipped baseline min(d, m) on every rank, the per-step leading stage with its
 * confidence (unique leader whose margin over the runner-up is
 * >= eta_Q * F[t,S-1], F > 0), and telemetry-quality sums (App. A).
 *   m          [nW][R][S] from sf_window_median (device).
 *   wall       [T][R] step wall times (device, nullable).
 *   other_stage index of the residual stage, or -1.
 *   X [nW][S], Y [nW][S], D [nW] (device, required; overwritten).
 *   E [nW][S][R] int64, C [nW][S][R] int32 (device, nullable; overwritten).
 *   step_lead  [T] leading stage | SF_STEP_CONFIDENT (device, required).
 *   quality    [nW][6] uint64 (device, nullable; overwritten): 128-bit sums
 *              (lo, hi) of the closure residual, the overlap error and the wall
 *              time.  With wall: residual max(0,e), overlap max(0,-e),
 *              e = wall - sum_{s != other} d.  Without wall but with
 *              other_stage: residual d[other], wall = the rank total.
 */
sf_status sf_direct_gain(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W,
                         const int64_t* m, const int64_t* wall, int32_t other_stage,
                         sf_ratio eta_Q, int64_t* X, int64_t* Y, int64_t* D, int64_t* E, int32_t* C,
                         uint8_t* step_lead, uint64_t* quality, uint32_t* status, cudaStream_t stream);

/*
 * sf_label_gates - App. C gates per window from the evidence above: shares
 * A = X/D and gains G = Y/D (fp64), routing candidate set (shortest prefix of
 * stages by X descending reaching tau_C * D), ambiguity set E_amb = C_A u C_G
 * (stages whose X, resp. Y, is strictly within eta * D of the top), leader
 * switches between consecutive confident steps, and the label bitmask.
 *   role    [R] rank role ids (device, nullable): more than one distinct value
 *           sets ROLE_AWARE_NEEDED.
 *   missing [nW] missing-rank count per window (device, nullable).
 *   quality from sf_direct_gain (device, nullable).
 *   cfg     host pointer.
 *   labels, route_mask, amb_mask [nW] (device, required); share, gain [nW][S]
 *   (device, nullable); n_confident, n_switch [nW] int32 (device, nullable).
 */
sf_status sf_label_gates(int64_t T, int64_t R, int64_t S, int64_t W, const int64_t* X,
                         const int64_t* Y, const int64_t* D, const uint8_t* step_lead,
                         const uint64_t* quality, const int32_t* role, const int32_t* missing,
                         const sf_label_config* cfg, uint32_t* labels, uint32_t* route_mask,
                         uint32_t* amb_mask, double* share, double* gain, int32_t* n_confident,
                         int32_t* n_switch, cudaStream_t stream);

/* Workspace bytes sf_label_windows needs for (T, R, S, W); 0 on bad arguments. */
size_t sf_label_windows_workspace_size(int64_t T, int64_t R, int64_t S, int64_t W);

/*
 * sf_label_windows - the whole labeler: sf_window_median, sf_direct_gain and
 * sf_label_gates in sequence on `stream`, with intermediates (medians, X, Y,
 * D, step leaders, quality sums) in the caller's device `workspace`
 * (>= sf_label_windows_workspace_size bytes, 256-byte aligned).
 *   X, Y [nW][S], D [nW] (device, nullable): copies of the evidence.
 */
sf_status sf_label_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W,
                           const int32_t* role, const int32_t* missing, const int64_t* wall,
                           int32_t other_stage, const sf_label_config* cfg, void* workspace,
                           size_t workspace_bytes, uint32_t* labels, uint32_t* route_mask,
                           uint32_t* amb_mask, double* share, double* gain, int64_t* X,
                           int64_t* Y, int64_t* D, uint32_t* status, cudaStream_t stream);

/*
 * sf_stream_windows - the whole hot path over a tensor that lives in HOST
 * memory: the steps are cut into chunks of chunk_steps steps (a multiple of
 * W, so every chunk holds whole windows); each chunk is copied host->device on
 * `copy_stream` into one of two device staging buffers and then, on
 * `stream`, gets sf_window_median, sf_direct_gain (with lead-rank credit when
 * E/C are given), sf_topk_suspects and sf_label_gates, its windows written to
 * the output rows they belong to.  The copy of the next chunk overlaps the
 * computation of the current one when h_d is page-locked and the two streams
 * differ.  This is the chunked streaming of the largest workload
 * (Sec. 5's window-boundary delivery of rank vectors, here host to GPU).
 *   h_d        [T][R][S] host, 16-byte aligned (page-locked for overlap).
 *   staging    device, >= sf_stream_windows_staging_size(T, R, S, chunk_steps)
 *              bytes, 16-byte aligned: two chunk buffers.
 *   workspace  device, >= sf_label_windows_workspace_size(min(chunk_steps, T),
 *              R, S, W) bytes: one chunk's medians and step leaders.
 *   outputs (device) indexed by global window: X, Y [nW][S], D [nW] required;
 *   E [nW][S][R], C [nW][S][R], top_stage, top_pair [nW][k][2],
 *   top_pair_value [nW][k], share, gain [nW][S] nullable; labels, route_mask,
 *   amb_mask [nW] required.  No telemetry-quality or role inputs.
 * The call creates and releases four CUDA events; it allocates no memory.
 * Returns when everything is enqueued.
 */
sf_status sf_stream_windows(const int64_t* h_d, int64_t T, int64_t R, int64_t S, int64_t W, int32_t k,
                            int64_t chunk_steps, const sf_label_config* cfg, int64_t* staging,
                            size_t staging_bytes, void* workspace, size_t workspace_bytes, int64_t* X,
                            int64_t* Y, int64_t* D, int64_t* E, int32_t* C, int32_t* top_stage,
                            int32_t* top_pair, int64_t* top_pair_value, uint32_t* labels,
                            uint32_t* route_mask, uint32_t* amb_mask, double* share, double* gain,
                            uint32_t* status, cudaStream_t stream, cudaStream_t copy_stream);

/* Device staging bytes sf_stream_windows needs; 0 on bad arguments. */
size_t sf_stream_windows_staging_size(int64_t T, int64_t R, int64_t S, int64_t chunk_steps);

/*
 * sf_stream_gathered_windows - sf_stream_windows over telemetry as the
 * window-boundary gather delivers it (Sec. 5): h_g holds the windows'
 * [R][n][S] blocks one after another (window w's block at element w*W*R*S,
 * the last window possibly short), in host memory.  Each chunk is copied as
 * is, converted on the device (sf_gathered_to_steps) into a third staging
 * buffer, and then takes the same path.  Arguments and outputs as in
 * sf_stream_windows; staging >= sf_stream_gathered_staging_size(...) bytes.
 */
sf_status sf_stream_gathered_windows(const int64_t* h_g, int64_t T, int64_t R, int64_t S, int64_t W, int32_t k,
                                     int64_t chunk_steps, const sf_label_config* cfg, int64_t* staging,
                                     size_t staging_bytes, void* workspace, size_t workspace_bytes, int64_t* X,
                                     int64_t* Y, int64_t* D, int64_t* E, int32_t* C, int32_t* top_stage,
                                     int32_t* top_pair, int64_t* top_pair_value, uint32_t* labels,
                                     uint32_t* route_mask, uint32_t* amb_mask, double* share, double* gain,
                                     uint32_t* status, cudaStream_t stream, cudaStream_t copy_stream);
size_t sf_stream_gathered_staging_size(int64_t T, int64_t R, int64_t S, int64_t chunk_steps);

/*
 * sf_label_windows_noalloc - sf_label_windows for callers that cannot
 * allocate device memory.  The paper has no counterpart; this is a
 * deployment variant of the labeler above.  It exists because an always-on
 * monitor runs inside someone else's training job: the framework's caching
 * allocator owns the device memory there, and a cudaMalloc issued from the
 * monitoring hook can block on or synchronize the device (stalling the very
 * step it measures) and carve memory out of that pool; a side-car with a
 * fixed memory budget may have no allocator to call at all.
 *
 * Scratch: one static device array of SF_STATIC_SCRATCH_BYTES (16 MiB) in
 * this library, held by every GPU that loads the library until the process
 * exits.  A problem whose sf_label_windows_workspace_size exceeds it returns
 * SF_EWORKSPACE before anything is enqueued.  The call allocates nothing and
 * frees nothing.
 *
 * Set-up: the first call on each device looks up the array's device address
 * (cudaGetSymbolAddress) with that device current, and caches it; make that
 * first call before any stream capture.  The cached address belongs to the
 * device's current primary context: after cudaDeviceReset (or any other
 * reset of that context) the module is loaded afresh and the array may move,
 * so do not call this entry point again in a process that has reset the
 * device.
 *
 * Sharing: all calls on a device use the same array, and it keeps whatever
 * the last call left there.  Each call zeroes the parts it accumulates into,
 * so calls ordered on one stream are independent; calls that can overlap on
 * the GPU (other streams without an ordering event, concurrent host threads)
 * race on the array and corrupt each other's results.
 *
 * Arguments, outputs and errors are those of sf_label_windows, without the
 * workspace pair.
 */
#define SF_STATIC_SCRATCH_BYTES (16u * 1024u * 1024u)

sf_status sf_label_windows_noalloc(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W,
                                   const int32_t* role, const int32_t* missing, const int64_t* wall,
                                   int32_t other_stage, const sf_label_config* cfg, uint32_t* labels,
                                   uint32_t* route_mask, uint32_t* amb_mask, double* share,
                                   double* gain, int64_t* X, int64_t* Y, int64_t* D,
                                   uint32_t* status, cudaStream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* STAGEFRONTIER_H */
