/*
 * sfgen.c - seeded synthetic telemetry for the frontier-accounting workloads.
 *
 * This module produces INPUTS only: int64 nanosecond stage durations
 * d[t][r][s] that imitate the per-(step, rank, stage) CPU wall-clock spans a
 * synchronous data-parallel trainer records (Sec. 3, "ordered, non-overlapping
 * stage spans"; the paper's DDP/FSDP runs are replaced by this simulation).
 * It holds none of the accounting method: no frontier, no increments, no
 * window statistics.  Both the CPU oracle and the CUDA path consume its output.
 *
 * Simulation of one step (each step is independent, so any thread count gives
 * identical bytes):
 *   - every rank keeps a local clock c[r] starting at 0;
 *   - intrinsic work x[t][r][s] = llround(median[s] * exp(sigma * z)),
 *     z ~ N(0,1) from a counter-based hash of (seed, t, r, s);
 *   - faults (stalls, heavy-tailed jitter, node slowdowns) modify x;
 *   - a non-sync stage records d = x and advances c[r] += x;
 *   - a sync stage models a blocking collective: the group is released when
 *     the last rank arrives (release = latest clock), so each rank records
 *     d = (release - c[r]) + x and leaves at release + x.
 *
 * Random numbers: SplitMix64 finaliser chained over the key words, top 53
 * bits as a double in [0,1).  Box-Muller for normals, inverse CDF for Pareto.
 * Build with -ffp-contract=off so x86-64 and aarch64 hosts agree.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define SFGEN_MAX_S 64

/* purposes of the hash streams */
enum { P_NORMAL_A = 1, P_NORMAL_B = 2, P_PARETO_SEL = 3, P_PARETO_VAL = 4 };

typedef struct sfgen_stall {      /* add `delta` ns to x on (rank, stage) for steps [t_begin, t_end) */
  int64_t t_begin, t_end, rank, stage, delta;
} sfgen_stall;

typedef struct sfgen_params {
  int64_t R, S;
  double median_ns[SFGEN_MAX_S];
  double sigma;
  uint64_t sync_mask;            /* bit s set: stage s is a sync point */
  uint64_t seed;
  /* additive stalls */
  int32_t n_stalls;
  const sfgen_stall* stalls;
  /* heavy-tailed jitter: with probability pareto_p a (t, r) cell has all its
     intrinsic x multiplied by Pareto(alpha, x_m = 1) = (1-u)^(-1/alpha) */
  double pareto_p, pareto_alpha;
  /* node slowdown: ranks [node_r0, node_r1) x steps [node_t0, node_t1) get x += x / node_div */
  int64_t node_r0, node_r1, node_t0, node_t1, node_div;
} sfgen_params;

static inline uint64_t mix64(uint64_t z) {
  z += 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

static inline uint64_t hash5(uint64_t seed, uint64_t purpose, uint64_t a, uint64_t b, uint64_t c) {
  uint64_t h = mix64(seed ^ mix64(purpose));
  h = mix64(h ^ a);
  h = mix64(h ^ (b + 0x632BE59BD9B4E019ull));
  h = mix64(h ^ (c + 0x8CB92BA72F3D8DD7ull));
  return h;
}

static inline double u01(uint64_t h) { return (double)(h >> 11) * (1.0 / 9007199254740992.0); }

/* Public: one uniform in [0,1) for host-side seeded choices (fault positions). */
double sfgen_uniform(uint64_t seed, uint64_t purpose, uint64_t a, uint64_t b, uint64_t c) {
  return u01(hash5(seed, purpose, a, b, c));
}

static inline double normal_at(uint64_t seed, int64_t t, int64_t r, int64_t s) {
  double u1 = u01(hash5(seed, P_NORMAL_A, (uint64_t)t, (uint64_t)r, (uint64_t)s));
  double u2 = u01(hash5(seed, P_NORMAL_B, (uint64_t)t, (uint64_t)r, (uint64_t)s));
  double rad = sqrt(-2.0 * log(1.0 - u1));
  return rad * cos(6.283185307179586 * u2);
}

static void fill_step(const sfgen_params* p, int64_t t, int64_t* out, int64_t* clk) {
  const int64_t R = p->R, S = p->S;
  for (int64_t r = 0; r < R; ++r) clk[r] = 0;
  /* heavy-tail multipliers for this step, one per rank (1.0 when not selected) */
  for (int64_t s = 0; s < S; ++s) {
    int is_sync = (int)((p->sync_mask >> s) & 1ull);
    int64_t release = 0;
    if (is_sync) {
      for (int64_t r = 0; r < R; ++r) release = clk[r] > release ? clk[r] : release;
    }
    for (int64_t r = 0; r < R; ++r) {
      double mult = exp(p->sigma * normal_at(p->seed, t, r, s));
      if (p->pareto_p > 0.0) {
        double sel = u01(hash5(p->seed, P_PARETO_SEL, (uint64_t)t, (uint64_t)r, 0));
        if (sel < p->pareto_p) {
          double u = u01(hash5(p->seed, P_PARETO_VAL, (uint64_t)t, (uint64_t)r, 0));
          mult *= pow(1.0 - u, -1.0 / p->pareto_alpha);
        }
      }
      int64_t x = llround(p->median_ns[s] * mult);
      if (p->node_div > 0 && r >= p->node_r0 && r < p->node_r1 && t >= p->node_t0 && t < p->node_t1)
        x += x / p->node_div;
      for (int32_t i = 0; i < p->n_stalls; ++i) {
        const sfgen_stall* st = &p->stalls[i];
        if (st->rank == r && st->stage == s && t >= st->t_begin && t < st->t_end) x += st->delta;
      }
      int64_t* cell = out + r * S + s;
      if (is_sync) {
        *cell = (release - clk[r]) + x;
        clk[r] = release + x;
      } else {
        *cell = x;
        clk[r] += x;
      }
    }
  }
}

typedef struct job {
  const sfgen_params* p;
  int64_t t0, tb, te;
  int64_t* out;
  int rc;
} job;

static void* run_job(void* arg) {
  job* j = (job*)arg;
  int64_t* clk = (int64_t*)malloc(sizeof(int64_t) * (size_t)j->p->R);
  if (!clk) { j->rc = -2; return NULL; }
  const int64_t RS = j->p->R * j->p->S;
  for (int64_t t = j->tb; t < j->te; ++t) fill_step(j->p, j->t0 + t, j->out + t * RS, clk);
  free(clk);
  j->rc = 0;
  return NULL;
}

/*
 * Fill out[0 .. nsteps) with steps t0 .. t0+nsteps-1 (global step indices
 * feed the hash, so a chunked fill equals a whole fill).  Returns 0 on success.
 */
int sfgen_fill(const sfgen_params* p, int64_t t0, int64_t nsteps, int64_t* out, int nthreads) {
  if (!p || !out || p->R <= 0 || p->S <= 0 || p->S > SFGEN_MAX_S || nsteps < 0) return -1;
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  if (nsteps < nthreads) nthreads = (int)(nsteps > 0 ? nsteps : 1);
  job jobs[256];
  pthread_t th[256];
  for (int i = 0; i < nthreads; ++i) {
    jobs[i].p = p;
    jobs[i].t0 = t0;
    jobs[i].tb = nsteps * i / nthreads;
    jobs[i].te = nsteps * (i + 1) / nthreads;
    jobs[i].out = out;
    jobs[i].rc = -3;
  }
  for (int i = 1; i < nthreads; ++i)
    if (pthread_create(&th[i], NULL, run_job, &jobs[i]) != 0) { jobs[i].rc = -4; th[i] = 0; }
  run_job(&jobs[0]);
  int rc = jobs[0].rc;
  for (int i = 1; i < nthreads; ++i) {
    if (jobs[i].rc != -4) pthread_join(th[i], NULL);
    if (jobs[i].rc != 0) rc = jobs[i].rc;
  }
  return rc;
}

/* Step wall times w[t][r] for the telemetry-quality inputs: the rank's
   recorded total plus a seeded closure residual of up to `resid_frac` of it
   (negative residual = overlapping spans).  Inputs only. */
int sfgen_wall(const int64_t* d, int64_t nsteps, int64_t R, int64_t S, int64_t t0, uint64_t seed,
               double resid_frac, int64_t* wall) {
  if (!d || !wall || R <= 0 || S <= 0 || nsteps < 0) return -1;
  for (int64_t t = 0; t < nsteps; ++t)
    for (int64_t r = 0; r < R; ++r) {
      int64_t tot = 0;
      for (int64_t s = 0; s < S; ++s) tot += d[(t * R + r) * S + s];
      double u = u01(hash5(seed, 7, (uint64_t)(t0 + t), (uint64_t)r, 0));
      wall[t * R + r] = tot + llround((2.0 * u - 1.0) * resid_frac * (double)tot);
    }
  return 0;
}
