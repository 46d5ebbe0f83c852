/*
 * sforacle.c - CPU oracle for frontier accounting (TEST INFRASTRUCTURE ONLY;
 * see sforacle.h).  Each function evaluates the paper's definition with
 * plain loops in the order the paper states it.  Nothing here is blocked,
 * fused or reordered for speed.
 *
 * Readings where the paper is silent (documented with the design):
 *   - lead rank: lowest rank attaining the frontier;
 *   - window median: lower median, element floor((n-1)/2) of the sorted column;
 *   - gain baseline: per-rank window median, clipped b = min(d, m);
 *   - tie sets C_A, C_G: stages strictly within eta * D of the top numerator;
 *   - routing set: shortest prefix of stages by (X desc, s asc) whose
 *     cumulative X reaches tau_C * D;
 *   - step confidence: unique leading stage whose margin over the runner-up
 *     is >= eta_Q * F_S with F_S > 0; switches counted between consecutive
 *     confident steps of a window.
 */
#include "sforacle.h"

#include <stdlib.h>
#include <string.h>

#define LIMIT47 ((int64_t)1 << 47)

typedef __int128 i128;

void sfo_config_default(sfo_config* c) {
  /* App. C default gates; eta_Q, gamma_switch, gamma_elig have no published
     value and take 1/20, 1/4, 1/2. */
  c->gamma_A = (sfo_ratio){2, 5};
  c->gamma_G = (sfo_ratio){1, 10};
  c->eta_A = (sfo_ratio){1, 20};
  c->eta_G = (sfo_ratio){1, 20};
  c->tau_C = (sfo_ratio){4, 5};
  c->eta_Q = (sfo_ratio){1, 20};
  c->gamma_switch = (sfo_ratio){1, 4};
  c->gamma_elig = (sfo_ratio){1, 2};
  c->closure_max = (sfo_ratio){1, 20};
  c->overlap_max = (sfo_ratio){1, 100};
  c->denom_floor_ns = 1;
  c->max_missing_ranks = 0;
  c->model_fit_mask = 0;
}

static int check_shape(int64_t T, int64_t R, int64_t S) {
  return T >= 1 && R >= 1 && R <= 65536 && S >= 1 && S <= 32;
}

/* Frontier of one step (Eq. 1).  P holds R prefixes. */
static int step_frontier(const int64_t* dt, int64_t R, int64_t S, int64_t* P, int64_t* F,
                         int64_t* a, int32_t* lead, int32_t* ties, int64_t* mk) {
  for (int64_t r = 0; r < R; ++r) P[r] = 0;
  int64_t F_prev = 0; /* F_{t,0} = 0 */
  for (int64_t s = 0; s < S; ++s) {
    for (int64_t r = 0; r < R; ++r) {
      int64_t v = dt[r * S + s];
      if (v < 0) return SFO_NEGATIVE;
      if (v >= LIMIT47) return SFO_RANGE;
      P[r] += v; /* P_{t,r,s} = sum_{j<=s} d_{t,r,j} */
    }
    int64_t Fs = P[0];
    for (int64_t r = 1; r < R; ++r)
      if (P[r] > Fs) Fs = P[r]; /* F_{t,s} = max_r P_{t,r,s} */
    int32_t ld = -1, nt = 0;
    for (int64_t r = 0; r < R; ++r)
      if (P[r] == Fs) {
        if (ld < 0) ld = (int32_t)r; /* lowest rank attaining the frontier */
        ++nt;
      }
    if (F) F[s] = Fs;
    if (a) a[s] = Fs - F_prev; /* a_{t,s} = F_{t,s} - F_{t,s-1} */
    if (lead) lead[s] = ld;
    if (ties) ties[s] = nt;
    F_prev = Fs;
  }
  for (int64_t r = 0; r < R; ++r)
    if (P[r] >= LIMIT47) return SFO_RANGE;
  if (mk) *mk = F_prev; /* makespan F_{t,S} */
  return SFO_OK;
}

int sfo_frontier(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t* F, int64_t* a,
                 int32_t* lead, int32_t* ties, int64_t* mk) {
  if (!d || !check_shape(T, R, S)) return SFO_BADARG;
  int64_t* P = (int64_t*)malloc(sizeof(int64_t) * (size_t)R);
  if (!P) return SFO_BADARG;
  int rc = SFO_OK;
  for (int64_t t = 0; t < T && rc == SFO_OK; ++t)
    rc = step_frontier(d + t * R * S, R, S, P, F ? F + t * S : NULL, a ? a + t * S : NULL,
                       lead ? lead + t * S : NULL, ties ? ties + t * S : NULL, mk ? mk + t : NULL);
  free(P);
  return rc;
}

static int64_t floordiv(int64_t a, int64_t b) { return a / b; /* a >= 0 here */ }

int sfo_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W, int64_t* X,
                int64_t* D, int64_t* E, int32_t* C, uint8_t* step_lead) {
  if (!d || !check_shape(T, R, S) || W < 1 || W > 65536 || t0 < 0 || !X || !D) return SFO_BADARG;
  int64_t w_first = floordiv(t0, W);
  int64_t nW = floordiv(t0 + T - 1, W) - w_first + 1;
  memset(X, 0, sizeof(int64_t) * (size_t)(nW * S));
  memset(D, 0, sizeof(int64_t) * (size_t)nW);
  if (E) memset(E, 0, sizeof(int64_t) * (size_t)(nW * S * R));
  if (C) memset(C, 0, sizeof(int32_t) * (size_t)(nW * S * R));
  int64_t* P = (int64_t*)malloc(sizeof(int64_t) * (size_t)R);
  int64_t* a = (int64_t*)malloc(sizeof(int64_t) * (size_t)S);
  int32_t* lead = (int32_t*)malloc(sizeof(int32_t) * (size_t)S);
  int rc = (P && a && lead) ? SFO_OK : SFO_BADARG;
  for (int64_t t = 0; t < T && rc == SFO_OK; ++t) {
    int64_t mk = 0;
    rc = step_frontier(d + t * R * S, R, S, P, NULL, a, lead, NULL, &mk);
    if (rc != SFO_OK) break;
    int64_t w = floordiv(t0 + t, W) - w_first;
    D[w] += mk;                                   /* sum_t F_{t,S} */
    int64_t best = 0;
    for (int64_t s = 0; s < S; ++s) {
      X[w * S + s] += a[s];                       /* sum_t a_{t,s} */
      if (E) E[(w * S + s) * R + lead[s]] += a[s]; /* credit to the lead rank */
      if (C) C[(w * S + s) * R + lead[s]] += 1;
      if (a[s] > a[best]) best = s;               /* leading stage, lowest s on ties */
    }
    if (step_lead) step_lead[t] = (uint8_t)best;
  }
  free(P);
  free(a);
  free(lead);
  return rc;
}

typedef struct entry { int64_t value; int64_t index; } entry;

static int cmp_entry(const void* pa, const void* pb) {
  const entry* x = (const entry*)pa;
  const entry* y = (const entry*)pb;
  if (x->value != y->value) return x->value > y->value ? -1 : 1; /* value descending */
  return x->index < y->index ? -1 : (x->index > y->index ? 1 : 0); /* index ascending */
}

int sfo_topk(const int64_t* X, const int64_t* E, int64_t nW, int64_t S, int64_t R, int32_t k,
             int32_t* top_stage, int64_t* top_stage_value, int32_t* top_pair, int64_t* top_pair_value) {
  if (!X || nW < 1 || S < 1 || S > 32 || R < 1 || R > 65536 || k < 1 || k > 32) return SFO_BADARG;
  entry* buf = (entry*)malloc(sizeof(entry) * (size_t)(S * R));
  if (!buf) return SFO_BADARG;
  for (int64_t w = 0; w < nW; ++w) {
    for (int64_t s = 0; s < S; ++s) buf[s] = (entry){X[w * S + s], s};
    qsort(buf, (size_t)S, sizeof(entry), cmp_entry);
    for (int32_t i = 0; i < k; ++i) {
      int ok = i < S && buf[i].value > 0;
      if (top_stage) top_stage[w * k + i] = ok ? (int32_t)buf[i].index : -1;
      if (top_stage_value) top_stage_value[w * k + i] = ok ? buf[i].value : 0;
    }
    if (E && (top_pair || top_pair_value)) {
      for (int64_t j = 0; j < S * R; ++j) buf[j] = (entry){E[w * S * R + j], j}; /* j = s*R + r */
      qsort(buf, (size_t)(S * R), sizeof(entry), cmp_entry);
      for (int32_t i = 0; i < k; ++i) {
        int ok = i < S * R && buf[i].value > 0;
        if (top_pair) {
          top_pair[(w * k + i) * 2 + 0] = ok ? (int32_t)(buf[i].index / R) : -1;
          top_pair[(w * k + i) * 2 + 1] = ok ? (int32_t)(buf[i].index % R) : -1;
        }
        if (top_pair_value) top_pair_value[w * k + i] = ok ? buf[i].value : 0;
      }
    }
  }
  free(buf);
  return SFO_OK;
}

static int cmp_i64(const void* pa, const void* pb) {
  int64_t x = *(const int64_t*)pa, y = *(const int64_t*)pb;
  return x < y ? -1 : (x > y ? 1 : 0);
}

int sfo_window_median(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W, int64_t* m) {
  if (!d || !m || !check_shape(T, R, S) || W < 1 || W > 65536) return SFO_BADARG;
  int64_t nW = (T + W - 1) / W;
  int64_t* col = (int64_t*)malloc(sizeof(int64_t) * (size_t)W);
  if (!col) return SFO_BADARG;
  for (int64_t w = 0; w < nW; ++w) {
    int64_t tb = w * W, te = tb + W < T ? tb + W : T, n = te - tb;
    for (int64_t r = 0; r < R; ++r)
      for (int64_t s = 0; s < S; ++s) {
        for (int64_t t = tb; t < te; ++t) col[t - tb] = d[(t * R + r) * S + s];
        qsort(col, (size_t)n, sizeof(int64_t), cmp_i64);
        m[(w * R + r) * S + s] = col[(n - 1) / 2]; /* lower median */
      }
  }
  free(col);
  return SFO_OK;
}

int sfo_direct_gain(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W, const int64_t* m,
                    int64_t* Y) {
  if (!d || !m || !Y || !check_shape(T, R, S) || W < 1 || W > 65536) return SFO_BADARG;
  int64_t nW = (T + W - 1) / W;
  int64_t* P = (int64_t*)malloc(sizeof(int64_t) * (size_t)R);
  int64_t* step = (int64_t*)malloc(sizeof(int64_t) * (size_t)(R * S));
  int rc = (P && step) ? SFO_OK : SFO_BADARG;
  memset(Y, 0, sizeof(int64_t) * (size_t)(nW * S));
  for (int64_t t = 0; t < T && rc == SFO_OK; ++t) {
    int64_t w = t / W;
    const int64_t* dt = d + t * R * S;
    int64_t FS = 0;
    rc = step_frontier(dt, R, S, P, NULL, NULL, NULL, NULL, &FS);
    for (int64_t s = 0; s < S && rc == SFO_OK; ++s) {
      /* replace stage s by the clipped baseline b = min(d, m) on every rank */
      memcpy(step, dt, sizeof(int64_t) * (size_t)(R * S));
      for (int64_t r = 0; r < R; ++r) {
        int64_t base = m[(w * R + r) * S + s];
        if (base < step[r * S + s]) step[r * S + s] = base;
      }
      int64_t FSp = 0;
      rc = step_frontier(step, R, S, P, NULL, NULL, NULL, NULL, &FSp);
      Y[w * S + s] += FS - FSp; /* numerator of G_s */
    }
  }
  free(P);
  free(step);
  return rc;
}

/* exact "lhs * r.den CMP r.num * rhs" helpers */
static int gt_ratio(i128 lhs, sfo_ratio r, i128 rhs) { return lhs * r.den > (i128)r.num * rhs; }
static int lt_ratio(i128 lhs, sfo_ratio r, i128 rhs) { return lhs * r.den < (i128)r.num * rhs; }
static int ge_ratio(i128 lhs, sfo_ratio r, i128 rhs) { return lhs * r.den >= (i128)r.num * rhs; }

static int valid_ratio(sfo_ratio r) {
  return r.den > 0 && r.den <= ((int64_t)1 << 31) && r.num >= 0 && r.num <= ((int64_t)1 << 31);
}

int sfo_label_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t W,
                      const int32_t* role, const int32_t* missing, const int64_t* wall,
                      int32_t other_stage, const sfo_config* cfg, uint32_t* labels,
                      uint32_t* route_mask, uint32_t* amb_mask, double* share, double* gain,
                      int64_t* Xo, int64_t* Do, int64_t* Yo, int64_t* mo, int32_t* n_confident,
                      int32_t* n_switch) {
  if (!d || !cfg || !labels || !check_shape(T, R, S) || W < 1 || W > 65536) return SFO_BADARG;
  if (other_stage >= S) return SFO_BADARG;
  const sfo_ratio* rs[] = {&cfg->gamma_A, &cfg->gamma_G, &cfg->eta_A, &cfg->eta_G, &cfg->tau_C,
                           &cfg->eta_Q, &cfg->gamma_switch, &cfg->gamma_elig, &cfg->closure_max,
                           &cfg->overlap_max};
  for (int i = 0; i < 10; ++i)
    if (!valid_ratio(*rs[i])) return SFO_BADARG;
  const int64_t nW = (T + W - 1) / W;
  int64_t* X = (int64_t*)calloc((size_t)(nW * S), sizeof(int64_t));
  int64_t* D = (int64_t*)calloc((size_t)nW, sizeof(int64_t));
  int64_t* Y = (int64_t*)calloc((size_t)(nW * S), sizeof(int64_t));
  int64_t* m = (int64_t*)malloc(sizeof(int64_t) * (size_t)(nW * R * S));
  int64_t* F = (int64_t*)malloc(sizeof(int64_t) * (size_t)S);
  int64_t* a = (int64_t*)malloc(sizeof(int64_t) * (size_t)S);
  int64_t* P = (int64_t*)malloc(sizeof(int64_t) * (size_t)R);
  int rc = (X && D && Y && m && F && a && P) ? SFO_OK : SFO_BADARG;

  /* step 1: windows' frontier numerators/denominator (Eq. 2) */
  if (rc == SFO_OK) rc = sfo_windows(d, T, R, S, 0, W, X, D, NULL, NULL, NULL);
  /* step 2: per-rank window medians and the clipped-gain numerators (Eq. 4) */
  if (rc == SFO_OK) rc = sfo_window_median(d, T, R, S, W, m);
  if (rc == SFO_OK) rc = sfo_direct_gain(d, T, R, S, W, m, Y);

  int role_mixed = 0;
  if (role)
    for (int64_t r = 1; r < R; ++r)
      if (role[r] != role[0]) role_mixed = 1;

  for (int64_t w = 0; w < nW && rc == SFO_OK; ++w) {
    const int64_t tb = w * W, te = tb + W < T ? tb + W : T, n = te - tb;
    const int64_t* Xw = X + w * S;
    const int64_t* Yw = Y + w * S;
    const int64_t Dw = D[w];

    /* step 3: leader-switch evidence between confident unique leaders (Sec. 4) */
    int32_t e = 0, sw = 0, last = -1;
    for (int64_t t = tb; t < te; ++t) {
      int64_t FS = 0;
      rc = step_frontier(d + t * R * S, R, S, P, F, a, NULL, NULL, &FS);
      if (rc != SFO_OK) break;
      int64_t best = 0;
      for (int64_t s = 1; s < S; ++s)
        if (a[s] > a[best]) best = s;
      int64_t second = 0;
      for (int64_t s = 0; s < S; ++s)
        if (s != best && a[s] > second) second = a[s];
      int confident = FS > 0 && ge_ratio((i128)(a[best] - second), cfg->eta_Q, (i128)FS);
      if (confident) {
        if (last >= 0 && last != (int32_t)best) ++sw;
        last = (int32_t)best;
        ++e;
      }
    }
    if (rc != SFO_OK) break;
    int high_switch = e >= 2 && ge_ratio((i128)e, cfg->gamma_elig, (i128)n) &&
                      gt_ratio((i128)sw, cfg->gamma_switch, (i128)(e - 1));

    /* step 4: telemetry quality (App. A closure and overlap shares; App. C gates) */
    int tel = 0;
    if (missing && missing[w] > cfg->max_missing_ranks) tel = 1;
    if (wall || other_stage >= 0) {
      i128 res = 0, ovl = 0, wsum = 0;
      for (int64_t t = tb; t < te; ++t)
        for (int64_t r = 0; r < R; ++r) {
          const int64_t* row = d + (t * R + r) * S;
          int64_t tot = 0, other = 0;
          for (int64_t s = 0; s < S; ++s) tot += row[s];
          if (other_stage >= 0) other = row[other_stage];
          if (wall) {
            int64_t wv = wall[t * R + r];
            if (wv < 0) { rc = SFO_NEGATIVE; break; }
            if (wv >= LIMIT47) { rc = SFO_RANGE; break; }
            int64_t err = wv - (tot - other); /* e = w - sum_{s != other} d */
            if (err > 0) res += err;
            else ovl += -err;
            wsum += wv;
          } else {
            res += other; /* recorded residual stage, step total as wall time */
            wsum += tot;
          }
        }
      if (rc != SFO_OK) break;
      if (gt_ratio(res, cfg->closure_max, wsum)) tel = 1;
      if (gt_ratio(ovl, cfg->overlap_max, wsum)) tel = 1;
    }
    /* below the denominator floor (and always at D = 0) only raw advances are emitted */
    int raw_only = Dw < cfg->denom_floor_ns || Dw == 0;
    if (raw_only) tel = 1;

    uint32_t lab = SFO_L_FRONTIER_ACCOUNTING, route = 0, amb = 0;
    if (tel) lab |= SFO_L_TELEMETRY_LIMITED;
    if (role_mixed) lab |= SFO_L_ROLE_AWARE_NEEDED;
    if (raw_only) {
      lab |= SFO_L_RAW_ONLY;
    } else {
      int64_t s1 = 0, g1 = 0;
      for (int64_t s = 1; s < S; ++s) {
        if (Xw[s] > Xw[s1]) s1 = s;
        if (Yw[s] > Yw[g1]) g1 = s;
      }
      int nA = 0, nG = 0;
      for (int64_t s = 0; s < S; ++s) {
        if (lt_ratio((i128)(Xw[s1] - Xw[s]), cfg->eta_A, (i128)Dw)) { amb |= 1u << s; ++nA; }
        if (lt_ratio((i128)(Yw[g1] - Yw[s]), cfg->eta_G, (i128)Dw)) { amb |= 1u << s; ++nG; }
      }
      /* routing candidate set: shortest leading-share prefix reaching tau_C */
      int8_t used[32] = {0};
      i128 cum = 0;
      for (int64_t i = 0; i < S; ++i) {
        int64_t pick = -1;
        for (int64_t s = 0; s < S; ++s)
          if (!used[s] && (pick < 0 || Xw[s] > Xw[pick])) pick = s;
        used[pick] = 1;
        route |= 1u << pick;
        cum += Xw[pick];
        if (ge_ratio(cum, cfg->tau_C, (i128)Dw)) break;
      }
      int hiA = gt_ratio((i128)Xw[s1], cfg->gamma_A, (i128)Dw);
      int loG = lt_ratio((i128)Yw[s1], cfg->gamma_G, (i128)Dw);
      int W1 = (int)((cfg->model_fit_mask >> s1) & 1u);
      int gain_tie = nG >= 2 && ge_ratio((i128)Yw[g1], cfg->gamma_G, (i128)Dw);
      if (hiA && loG) lab |= W1 ? SFO_L_SYNC_WAIT_DEPENDENT : SFO_L_CO_CRITICAL;
      if (hiA && !loG) lab |= SFO_L_DIRECT_EXPOSURE;
      if (nA >= 2 || gain_tie || high_switch) {
        /* near ties and switching leaders downgrade a strong label */
        lab |= SFO_L_CO_CRITICAL;
        lab &= ~(SFO_L_DIRECT_EXPOSURE | SFO_L_SYNC_WAIT_DEPENDENT);
      }
      if (tel || role_mixed) lab &= ~(SFO_L_DIRECT_EXPOSURE | SFO_L_SYNC_WAIT_DEPENDENT);
    }
    labels[w] = lab;
    if (route_mask) route_mask[w] = route;
    if (amb_mask) amb_mask[w] = amb;
    for (int64_t s = 0; s < S; ++s) {
      if (share) share[w * S + s] = raw_only ? 0.0 : (double)Xw[s] / (double)Dw; /* A_s, Eq. 2 */
      if (gain) gain[w * S + s] = raw_only ? 0.0 : (double)Yw[s] / (double)Dw;   /* G_s, Eq. 4 */
    }
    if (n_confident) n_confident[w] = e;
    if (n_switch) n_switch[w] = sw;
  }
  if (rc == SFO_OK) {
    if (Xo) memcpy(Xo, X, sizeof(int64_t) * (size_t)(nW * S));
    if (Do) memcpy(Do, D, sizeof(int64_t) * (size_t)nW);
    if (Yo) memcpy(Yo, Y, sizeof(int64_t) * (size_t)(nW * S));
    if (mo) memcpy(mo, m, sizeof(int64_t) * (size_t)(nW * R * S));
  }
  free(X);
  free(D);
  free(Y);
  free(m);
  free(F);
  free(a);
  free(P);
  return rc;
}

int sfo_baselines(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W, int64_t* M,
                  uint64_t* SUM, int64_t* SLOW, int64_t* RANK0) {
  if (!d || !check_shape(T, R, S) || W < 1 || W > 65536 || t0 < 0) return SFO_BADARG;
  int64_t w_first = t0 / W;
  int64_t nW = (t0 + T - 1) / W - w_first + 1;
  if (M) memset(M, 0, sizeof(int64_t) * (size_t)(nW * S));
  if (SUM) memset(SUM, 0, sizeof(uint64_t) * (size_t)(nW * S * 2));
  if (SLOW) memset(SLOW, 0, sizeof(int64_t) * (size_t)(nW * S));
  if (RANK0) memset(RANK0, 0, sizeof(int64_t) * (size_t)(nW * S));
  for (int64_t t = 0; t < T; ++t) {
    const int64_t* dt = d + t * R * S;
    int64_t w = (t0 + t) / W - w_first;
    /* the slowest rank: largest total, lowest rank on ties */
    int64_t slow = 0, best = -1;
    for (int64_t r = 0; r < R; ++r) {
      int64_t tot = 0;
      for (int64_t s = 0; s < S; ++s) {
        int64_t v = dt[r * S + s];
        if (v < 0) return SFO_NEGATIVE;
        if (v >= LIMIT47) return SFO_RANGE;
        tot += v;
      }
      if (tot >= LIMIT47) return SFO_RANGE;
      if (tot > best) { best = tot; slow = r; }
    }
    for (int64_t s = 0; s < S; ++s) {
      int64_t mx = dt[s];
      unsigned __int128 sum = 0;
      for (int64_t r = 0; r < R; ++r) {
        if (dt[r * S + s] > mx) mx = dt[r * S + s];
        sum += (unsigned __int128)dt[r * S + s];
      }
      if (M) M[w * S + s] += mx;
      if (SUM) {
        unsigned __int128 acc = ((unsigned __int128)SUM[(w * S + s) * 2 + 1] << 64) | SUM[(w * S + s) * 2];
        acc += sum;
        SUM[(w * S + s) * 2] = (uint64_t)acc;
        SUM[(w * S + s) * 2 + 1] = (uint64_t)(acc >> 64);
      }
      if (SLOW) SLOW[w * S + s] += dt[slow * S + s];
      if (RANK0) RANK0[w * S + s] += dt[s];
    }
  }
  return SFO_OK;
}

int sfo_rank_lag(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t* L, int64_t* dL, int64_t* G) {
  if (!d || !check_shape(T, R, S)) return SFO_BADARG;
  int64_t* P = (int64_t*)malloc(sizeof(int64_t) * (size_t)R);
  int64_t* col = (int64_t*)malloc(sizeof(int64_t) * (size_t)R);
  int rc = (P && col) ? SFO_OK : SFO_BADARG;
  for (int64_t t = 0; t < T && rc == SFO_OK; ++t) {
    for (int64_t r = 0; r < R; ++r) P[r] = 0;
    int64_t prev = 0;
    for (int64_t s = 0; s < S; ++s) {
      for (int64_t r = 0; r < R; ++r) {
        int64_t v = d[(t * R + r) * S + s];
        if (v < 0) { rc = SFO_NEGATIVE; break; }
        if (v >= LIMIT47) { rc = SFO_RANGE; break; }
        P[r] += v;
        col[r] = P[r];
      }
      if (rc != SFO_OK) break;
      qsort(col, (size_t)R, sizeof(int64_t), cmp_i64);
      const int64_t F = col[R - 1];                      /* F[t,s] = max_r P */
      const int64_t med = col[(R - 1) / 2];              /* lower median over ranks */
      const int64_t second = R >= 2 ? col[R - 2] : F;    /* second largest, ties counted */
      const int64_t lag = F - med;
      if (L) L[t * S + s] = lag;
      if (dL) dL[t * S + s] = lag - prev;
      if (G) G[t * S + s] = F - second;
      prev = lag;
    }
    for (int64_t r = 0; r < R && rc == SFO_OK; ++r)
      if (P[r] >= LIMIT47) rc = SFO_RANGE;
  }
  free(P);
  free(col);
  return rc;
}

int sfo_raw_spread(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W, int64_t* SPREAD) {
  if (!d || !SPREAD || !check_shape(T, R, S) || W < 1 || W > 65536 || t0 < 0) return SFO_BADARG;
  const int64_t w_first = t0 / W, nW = (t0 + T - 1) / W - w_first + 1;
  memset(SPREAD, 0, sizeof(int64_t) * (size_t)(nW * S));
  int64_t* col = (int64_t*)malloc(sizeof(int64_t) * (size_t)R);
  if (!col) return SFO_BADARG;
  int rc = SFO_OK;
  for (int64_t t = 0; t < T && rc == SFO_OK; ++t) {
    const int64_t w = (t0 + t) / W - w_first;
    for (int64_t s = 0; s < S; ++s) {
      for (int64_t r = 0; r < R; ++r) {
        col[r] = d[(t * R + r) * S + s];
        if (col[r] < 0) rc = SFO_NEGATIVE;
        else if (col[r] >= LIMIT47) rc = SFO_RANGE;
      }
      qsort(col, (size_t)R, sizeof(int64_t), cmp_i64);
      SPREAD[w * S + s] += col[R - 1] - col[(R - 1) / 2]; /* max minus lower median over ranks */
    }
  }
  free(col);
  return rc;
}

int sfo_group_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, const int32_t* group, int64_t G,
                      int64_t t0, int64_t W, int64_t* Xg, int64_t* Dg) {
  if (!d || !group || !check_shape(T, R, S) || G < 1 || G > 65536 || W < 1 || W > 65536 || t0 < 0 || !Xg ||
      !Dg)
    return SFO_BADARG;
  for (int64_t r = 0; r < R; ++r)
    if (group[r] < 0 || group[r] >= G) return SFO_BADARG;
  int64_t w_first = floordiv(t0, W);
  int64_t nW = floordiv(t0 + T - 1, W) - w_first + 1;
  memset(Xg, 0, sizeof(int64_t) * (size_t)(G * nW * S));
  memset(Dg, 0, sizeof(int64_t) * (size_t)(G * nW));
  int64_t* P = (int64_t*)malloc(sizeof(int64_t) * (size_t)R);
  int64_t* Fg = (int64_t*)malloc(sizeof(int64_t) * (size_t)G);     /* F_g[t,s] at the current s */
  int64_t* Fprev = (int64_t*)malloc(sizeof(int64_t) * (size_t)G);  /* F_g[t,s-1] */
  int rc = (P && Fg && Fprev) ? SFO_OK : SFO_BADARG;
  for (int64_t t = 0; t < T && rc == SFO_OK; ++t) {
    const int64_t* dt = d + t * R * S;
    int64_t w = floordiv(t0 + t, W) - w_first;
    for (int64_t r = 0; r < R; ++r) P[r] = 0;
    for (int64_t g = 0; g < G; ++g) Fprev[g] = 0;
    for (int64_t s = 0; s < S && rc == SFO_OK; ++s) {
      for (int64_t g = 0; g < G; ++g) Fg[g] = 0;
      for (int64_t r = 0; r < R; ++r) {
        int64_t v = dt[r * S + s];
        if (v < 0) { rc = SFO_NEGATIVE; break; }
        if (v >= LIMIT47) { rc = SFO_RANGE; break; }
        P[r] += v;
        if (P[r] > Fg[group[r]]) Fg[group[r]] = P[r]; /* max over the group's ranks */
      }
      for (int64_t g = 0; g < G && rc == SFO_OK; ++g) {
        Xg[(g * nW + w) * S + s] += Fg[g] - Fprev[g]; /* a_g[t,s] */
        Fprev[g] = Fg[g];
      }
    }
    for (int64_t r = 0; r < R && rc == SFO_OK; ++r)
      if (P[r] >= LIMIT47) rc = SFO_RANGE;
    for (int64_t g = 0; g < G && rc == SFO_OK; ++g) Dg[g * nW + w] += Fprev[g]; /* F_g[t,S-1] */
  }
  free(P);
  free(Fg);
  free(Fprev);
  return rc;
}

int sfo_stage_group_sum(const int64_t* X, int64_t nW, int64_t S, const int32_t* stage_group, int64_t K,
                        int64_t* Y) {
  if (!X || !stage_group || !Y || nW < 0 || S < 1 || S > 32 || K < 1 || K > 32) return SFO_BADARG;
  for (int64_t s = 0; s < S; ++s)
    if (stage_group[s] < 0 || stage_group[s] >= K) return SFO_BADARG;
  memset(Y, 0, sizeof(int64_t) * (size_t)(nW * K));
  for (int64_t w = 0; w < nW; ++w)
    for (int64_t s = 0; s < S; ++s) Y[w * K + stage_group[s]] += X[w * S + s];
  return SFO_OK;
}

int sfo_rank_lag_windows(const int64_t* d, int64_t T, int64_t R, int64_t S, int64_t t0, int64_t W, int64_t* LW,
                         int64_t* GW) {
  if (!d || !check_shape(T, R, S) || W < 1 || W > 65536 || t0 < 0) return SFO_BADARG;
  const int64_t w_first = t0 / W, nW = (t0 + T - 1) / W - w_first + 1;
  int64_t* L = (int64_t*)malloc(sizeof(int64_t) * (size_t)(T * S));
  int64_t* G = (int64_t*)malloc(sizeof(int64_t) * (size_t)(T * S));
  int rc = (L && G) ? sfo_rank_lag(d, T, R, S, L, NULL, G) : SFO_BADARG;
  if (LW) memset(LW, 0, sizeof(int64_t) * (size_t)(nW * S));
  if (GW) memset(GW, 0, sizeof(int64_t) * (size_t)(nW * S));
  for (int64_t t = 0; t < T && rc == SFO_OK; ++t) {
    const int64_t w = (t0 + t) / W - w_first;
    for (int64_t s = 0; s < S; ++s) {
      if (LW) LW[w * S + s] += L[t * S + s]; /* sum_t L[t,s] */
      if (GW) GW[w * S + s] += G[t * S + s]; /* sum_t G[t,s] */
    }
  }
  free(L);
  free(G);
  return rc;
}
