/*
 * oracle.c -- plain, slow, fp64 CPU oracle for the STRIDE scoring path
 * (arXiv 2609.14636).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or
 * call this file: only tests/, __graft_entry__.smoke() and bench.py's CPU
 * baseline leg use it.  It shares no code, header, table or constant with the
 * CUDA library; the two meet only in the seeded input generators.
 *
 * Every function below writes out the paper's definition directly, in fp64,
 * with no blocking, fusion or reordering beyond what the definition states:
 *
 *   oracle_row_logprobs   log pi(y_t) for student and teacher (the log-softmax
 *                         implied by pi in Eq. 1 and Eq. 4), the per-token
 *                         reward r_t of Eq. 1 reported as d_t = -r_t
 *                         (the per-token KL estimate of Sec. 3.2).
 *   oracle_scan_batch     per-turn mean teacher log-prob l_k (Eq. 4); the
 *                         early-stop rule of Eq. 5 with the prefix-buffer
 *                         offset (Sec. 4.1, "Synergy with the prefix buffer":
 *                         the sum runs over newly generated turns only); the
 *                         token-level variant used for math (Sec. 5.5).
 *                         Also the token-level OPD loss of Eq. 2 on the
 *                         retained tokens (Algorithm 1: the loss covers the
 *                         tokens kept, including the triggering turn), per
 *                         turn and per trajectory, and the within-turn
 *                         relative-position decile profile of d and log pi_T
 *                         (Observation 1, Sec. 3.2).
 *   oracle_step_update    the same rules applied online, one generated token
 *                         per rollout per call (Algorithm 1, inner turn loop).
 *   oracle_select_restart quality gate l_k > alpha (Sec. 4.2, step 1), the
 *                         longest correct prefix K_max and the weakest correct
 *                         turn k* of Eq. 6 (Algorithm 1, K_max / k* / K0).
 *
 * Readings where the paper is silent: sums are strict "< lambda" and
 * "> alpha"; turns are 0-based, so the returned k* equals K0 (the number of
 * reused turns); ties in Eq. 6 go to the lowest index; K_max = 0 gives
 * k* = 0; an empty turn is an error; a row whose logits are all -inf has
 * LSE = -inf and NaN log-probs; an out-of-range token gives NaN for its row
 * and an error return.
 *
 * Parity pins: see tests/test_oracle_pins.py (closed forms, brute force in
 * arbitrary precision, invariants, hand-worked cases in tests/golden/).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_DTYPE_BF16 0
#define ORACLE_DTYPE_F32 1
#define ORACLE_MODE_TURN_MEAN 0
#define ORACLE_MODE_TOKEN_SUM 1

#define ORACLE_OK 0
#define ORACLE_ERR_ARG 1
#define ORACLE_ERR_TOKEN 2
#define ORACLE_ERR_EMPTY_TURN 3

/* bf16 is the upper 16 bits of an IEEE-754 binary32. */
static double bf16_bits_to_double(uint16_t h) {
  uint32_t u = ((uint32_t)h) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

static double logit_at(const void* base, int dtype, int64_t ld, int64_t r, int64_t j) {
  if (dtype == ORACLE_DTYPE_BF16) {
    const uint16_t* p = (const uint16_t*)base;
    return bf16_bits_to_double(p[r * ld + j]);
  } else {
    const float* p = (const float*)base;
    return (double)p[r * ld + j];
  }
}

/* log sum_j exp(x_j), computed as m + log sum_j exp(x_j - m) with m = max_j x_j.
 * NaN entries are skipped by the max (a comparison with NaN is false) but
 * reach the sum, so a NaN anywhere gives NaN.  All -inf gives -inf. */
static double row_lse(const void* base, int dtype, int64_t ld, int64_t V, int64_t r) {
  double m = -INFINITY;
  for (int64_t j = 0; j < V; ++j) {
    double x = logit_at(base, dtype, ld, r, j);
    if (x > m) m = x;
  }
  if (m == -INFINITY) {
    /* every entry is -inf (or NaN): sum of exp is 0, unless a NaN is present */
    for (int64_t j = 0; j < V; ++j) {
      double x = logit_at(base, dtype, ld, r, j);
      if (x != x) return NAN;
    }
    return -INFINITY;
  }
  double s = 0.0;
  for (int64_t j = 0; j < V; ++j) s += exp(logit_at(base, dtype, ld, r, j) - m);
  return m + log(s);
}

typedef struct {
  const void* S;
  const void* T;
  int dtype;
  int64_t ld, V;
  const int32_t* tokens;
  int64_t r0, r1;
  double *logp_s, *logp_t, *d, *lse_s, *lse_t, *x_s, *x_t;
  int bad_token;
} rows_job;

static void* rows_worker(void* arg) {
  rows_job* jb = (rows_job*)arg;
  for (int64_t r = jb->r0; r < jb->r1; ++r) {
    int32_t y = jb->tokens[r];
    double ls = jb->S ? row_lse(jb->S, jb->dtype, jb->ld, jb->V, r) : NAN;
    double lt = row_lse(jb->T, jb->dtype, jb->ld, jb->V, r);
    double xs = NAN, xt = NAN, ps = NAN, pt = NAN;
    if (y >= 0 && (int64_t)y < jb->V) {
      xs = jb->S ? logit_at(jb->S, jb->dtype, jb->ld, r, y) : NAN;
      xt = logit_at(jb->T, jb->dtype, jb->ld, r, y);
      ps = xs - ls; /* log pi_S(y_t) */
      pt = xt - lt; /* log pi_T(y_t) */
    } else {
      jb->bad_token = 1;
    }
    if (jb->logp_s) jb->logp_s[r] = ps;
    if (jb->logp_t) jb->logp_t[r] = pt;
    if (jb->d) jb->d[r] = ps - pt; /* d_t = -r_t (Eq. 1) */
    if (jb->lse_s) jb->lse_s[r] = ls;
    if (jb->lse_t) jb->lse_t[r] = lt;
    if (jb->x_s) jb->x_s[r] = xs;
    if (jb->x_t) jb->x_t[r] = xt;
  }
  return NULL;
}

/* Per-row log-probabilities of the sampled token under student S and teacher T.
 * S, T: [rows, ld] row-major, dtype bf16 (raw uint16 bits) or fp32.
 * S may be NULL (teacher only: student outputs are NaN).
 * Any output pointer may be NULL.  Rows are split across nthreads threads;
 * each row is computed independently, so the thread count does not change
 * any result. */
int oracle_row_logprobs(const void* S, const void* T, int dtype, int64_t ld, int64_t V,
                        const int32_t* tokens, int64_t rows, double* logp_s, double* logp_t,
                        double* d, double* lse_s, double* lse_t, double* x_s, double* x_t,
                        int nthreads) {
  if (!T || !tokens || V < 1 || ld < V || rows < 0) return ORACLE_ERR_ARG;
  if (dtype != ORACLE_DTYPE_BF16 && dtype != ORACLE_DTYPE_F32) return ORACLE_ERR_ARG;
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 1024) nthreads = 1024;
  if ((int64_t)nthreads > rows) nthreads = rows > 0 ? (int)rows : 1;
  rows_job* jobs = (rows_job*)calloc((size_t)nthreads, sizeof(rows_job));
  pthread_t* th = (pthread_t*)calloc((size_t)nthreads, sizeof(pthread_t));
  if (!jobs || !th) {
    free(jobs);
    free(th);
    return ORACLE_ERR_ARG;
  }
  for (int i = 0; i < nthreads; ++i) {
    rows_job* jb = &jobs[i];
    jb->S = S;
    jb->T = T;
    jb->dtype = dtype;
    jb->ld = ld;
    jb->V = V;
    jb->tokens = tokens;
    jb->r0 = rows * i / nthreads;
    jb->r1 = rows * (i + 1) / nthreads;
    jb->logp_s = logp_s;
    jb->logp_t = logp_t;
    jb->d = d;
    jb->lse_s = lse_s;
    jb->lse_t = lse_t;
    jb->x_s = x_s;
    jb->x_t = x_t;
  }
  int started = 0;
  for (int i = 1; i < nthreads; ++i) {
    if (pthread_create(&th[i], NULL, rows_worker, &jobs[i]) != 0) break;
    started = i;
  }
  rows_worker(&jobs[0]);
  for (int i = 1; i <= started; ++i) pthread_join(th[i], NULL);
  for (int i = started + 1; i < nthreads; ++i) rows_worker(&jobs[i]); /* threads that failed to start */
  int bad = 0;
  for (int i = 0; i < nthreads; ++i) bad |= jobs[i].bad_token;
  free(jobs);
  free(th);
  return bad ? ORACLE_ERR_TOKEN : ORACLE_OK;
}

/* Batch scan over ragged trajectories.
 *
 * Layout: rows are trajectory-major; trajectory i owns rows
 * [traj_row_off[i], traj_row_off[i+1]) and turns [traj_turn_off[i],
 * traj_turn_off[i+1]); turn k owns rows [turn_row_off[k], turn_row_off[k+1]).
 * Row indices are relative to traj_row_off[0] for the per-row arrays.
 *
 * TURN_MEAN (Eq. 4, Eq. 5 with the prefix-buffer offset):
 *   l_k = (1/n_k) sum_{i in turn k} logp_T(i);  S_K = cum_in + sum_{k<=K} l_k;
 *   stop at the first turn K with S_K < lambda; the stopping turn is kept,
 *   and stop_row is its last row.
 * TOKEN_SUM (Sec. 5.5):  C_t = cum_in + sum_{i<=t} logp_T(i); stop at the first
 *   token t with C_t < lambda; that token is kept.
 * Turns after the stop are still summarised (they are reported, not scored
 * differently); only the first crossing is recorded.
 *
 * OPD loss (Eq. 2, r_t = logp_T - logp_S held constant): the per-token term
 * -logp_S(t) * r_t = logp_S(t) * d(t).  turn_sum_l is its sum over each turn;
 * traj_loss / traj_loss_tokens sum it over the retained tokens: every token
 * of the turns up to and including the stopping turn (TURN_MEAN), every token
 * up to and including the stopping token (TOKEN_SUM), all tokens if the rule
 * never fires (Algorithm 1, loss on the retained tokens).
 *
 * Within-turn profile (Observation 1): token i (0-based) of a turn of n_k
 * tokens falls in decile floor(10 i / n_k); profile[3j+0] += d, profile[3j+1]
 * += logp_T, profile[3j+2] += 1 for its decile j.  The profile is added to
 * (not cleared).
 *
 * Outputs (each may be NULL): per turn sum_t, sum_d, sum_l, mean (fp64), n,
 * cum after the turn; per trajectory final cum, stop_turn (trajectory-local,
 * -1 none), stop_row (trajectory-local token position, -1 none), retained
 * loss and token count; per row row_cum = running token sum (TOKEN_SUM) or
 * the turn-end running sum at turn-end rows and NaN elsewhere (TURN_MEAN);
 * profile [30].  logp_s may be NULL when the loss outputs are not wanted. */
int oracle_scan_batch(const double* logp_t, const double* d, const double* logp_s,
                      const int64_t* traj_row_off, const int64_t* turn_row_off,
                      const int32_t* traj_turn_off, int32_t n_traj, int mode, const double* lambda,
                      const double* cum_in, double* turn_sum_t, double* turn_sum_d,
                      double* turn_sum_l, double* turn_mean, int64_t* turn_n, double* turn_cum,
                      double* traj_cum, int32_t* stop_turn, int64_t* stop_row, double* traj_loss,
                      int64_t* traj_loss_tokens, double* row_cum, double* profile) {
  if (!logp_t || !traj_row_off || !turn_row_off || !traj_turn_off || !lambda || n_traj < 0)
    return ORACLE_ERR_ARG;
  if (mode != ORACLE_MODE_TURN_MEAN && mode != ORACLE_MODE_TOKEN_SUM) return ORACLE_ERR_ARG;
  const int64_t base = traj_row_off[0];
  for (int32_t i = 0; i < n_traj; ++i) {
    int32_t k0 = traj_turn_off[i], k1 = traj_turn_off[i + 1];
    if (k1 < k0) return ORACLE_ERR_ARG;
    if (turn_row_off[k0] != traj_row_off[i] || turn_row_off[k1] != traj_row_off[i + 1])
      return ORACLE_ERR_ARG;
    double cum = cum_in ? cum_in[i] : 0.0;
    int32_t st_turn = -1;
    int64_t st_row = -1;
    double loss = 0.0;
    int64_t loss_n = 0;
    for (int32_t k = k0; k < k1; ++k) {
      int64_t a = turn_row_off[k], b = turn_row_off[k + 1];
      if (b <= a) return ORACLE_ERR_EMPTY_TURN; /* Eq. 4 needs n_k >= 1 */
      int64_t n = b - a;
      /* a turn (TURN_MEAN) or a token (TOKEN_SUM) is retained when the rule
       * has not fired before it */
      int turn_retained = (st_turn < 0);
      double s_t = 0.0, s_d = 0.0, s_l = 0.0;
      for (int64_t r = a; r < b; ++r) {
        double lt = logp_t[r - base];
        double dd = d ? d[r - base] : 0.0;
        double term = logp_s ? logp_s[r - base] * dd : 0.0; /* -logp_S * r_t (Eq. 2) */
        s_t += lt;
        s_d += dd;
        s_l += term;
        if (profile) {
          int64_t j = (10 * (r - a)) / n;
          profile[3 * j + 0] += dd;
          profile[3 * j + 1] += lt;
          profile[3 * j + 2] += 1.0;
        }
        if (mode == ORACLE_MODE_TOKEN_SUM) {
          if (st_row < 0) {
            loss += term;
            loss_n += 1;
          }
          cum += lt;
          if (row_cum) row_cum[r - base] = cum;
          if (st_row < 0 && cum < lambda[i]) {
            st_row = r - traj_row_off[i];
            st_turn = k - k0;
          }
        } else {
          if (turn_retained) {
            loss += term;
            loss_n += 1;
          }
          if (row_cum) row_cum[r - base] = NAN;
        }
      }
      double mean = s_t / (double)n; /* Eq. 4 */
      if (mode == ORACLE_MODE_TURN_MEAN) {
        cum += mean; /* Eq. 5 left-hand side, over new turns only */
        if (row_cum) row_cum[b - 1 - base] = cum;
        if (st_turn < 0 && cum < lambda[i]) {
          st_turn = k - k0;
          st_row = (b - 1) - traj_row_off[i];
        }
      }
      if (turn_sum_t) turn_sum_t[k] = s_t;
      if (turn_sum_d) turn_sum_d[k] = s_d;
      if (turn_sum_l) turn_sum_l[k] = s_l;
      if (turn_mean) turn_mean[k] = mean;
      if (turn_n) turn_n[k] = n;
      if (turn_cum) turn_cum[k] = cum;
    }
    if (traj_cum) traj_cum[i] = cum;
    if (stop_turn) stop_turn[i] = st_turn;
    if (stop_row) stop_row[i] = st_row;
    if (traj_loss) traj_loss[i] = loss;
    if (traj_loss_tokens) traj_loss_tokens[i] = loss_n;
  }
  return ORACLE_OK;
}

/* Per-rollout state carried between decode steps (the oracle's own layout). */
typedef struct {
  double cum;        /* running sum (Eq. 5 left-hand side, or token sum) */
  double turn_sum_t; /* open turn: sum of logp_T */
  double turn_sum_d; /* open turn: sum of d */
  double turn_sum_l; /* open turn: sum of the OPD-loss terms logp_S * d */
  double loss;       /* OPD loss (Eq. 2) over the tokens scored, all retained */
  int64_t rows_seen; /* tokens scored so far (= retained tokens) */
  int64_t stop_row;  /* token position of the first crossing, -1 none */
  int32_t stop_turn; /* turn of the first crossing, -1 none */
  int32_t turn_tokens;
  int32_t turn_idx;
  int32_t stopped;
} oracle_rollout;

/* One decode step (Algorithm 1, inner loop, one token per rollout).
 * For rollout b: if it has stopped, nothing is read or changed and its
 * outputs are NaN.  Otherwise logp_s/logp_t/d of its token are taken from
 * the inputs (computed by oracle_row_logprobs), the open turn accumulates,
 * TOKEN_SUM tests the running sum at every token, and when turn_end[b] is set
 * the turn closes: l = sum_t / n (Eq. 4), TURN_MEAN adds l to the running sum
 * and tests it (Eq. 5).  A closed turn's stats are reported in the turn_*
 * outputs (turn_n = 0 when no turn closed at this step).  Every scored token
 * is retained (a stopped rollout scores nothing more), so its OPD-loss term
 * logp_S * d (Eq. 2) is added to the rollout's loss. */
int oracle_step_update(const double* logp_s, const double* logp_t, const uint8_t* turn_end,
                       int32_t B, int mode, const double* lambda, oracle_rollout* st,
                       double* out_logp_s, double* out_logp_t, double* out_d, uint8_t* stopped_now,
                       double* turn_sum_t, double* turn_sum_d, double* turn_sum_l, double* turn_mean,
                       int32_t* turn_n, double* turn_cum) {
  if (!logp_s || !logp_t || !turn_end || !lambda || !st || B < 0) return ORACLE_ERR_ARG;
  for (int32_t b = 0; b < B; ++b) {
    oracle_rollout* s = &st[b];
    if (stopped_now) stopped_now[b] = 0;
    if (turn_n) turn_n[b] = 0;
    if (turn_sum_t) turn_sum_t[b] = 0.0;
    if (turn_sum_d) turn_sum_d[b] = 0.0;
    if (turn_sum_l) turn_sum_l[b] = 0.0;
    if (turn_mean) turn_mean[b] = 0.0;
    if (turn_cum) turn_cum[b] = 0.0;
    if (s->stopped) {
      if (out_logp_s) out_logp_s[b] = NAN;
      if (out_logp_t) out_logp_t[b] = NAN;
      if (out_d) out_d[b] = NAN;
      continue;
    }
    double ps = logp_s[b], pt = logp_t[b], dd = ps - pt;
    if (out_logp_s) out_logp_s[b] = ps;
    if (out_logp_t) out_logp_t[b] = pt;
    if (out_d) out_d[b] = dd;
    s->turn_sum_t += pt;
    s->turn_sum_d += dd;
    s->turn_sum_l += ps * dd;
    s->loss += ps * dd;
    s->turn_tokens += 1;
    int64_t pos = s->rows_seen;
    s->rows_seen += 1;
    if (mode == ORACLE_MODE_TOKEN_SUM) {
      s->cum += pt;
      if (s->cum < lambda[b]) {
        s->stopped = 1;
        s->stop_row = pos;
        s->stop_turn = s->turn_idx;
        if (stopped_now) stopped_now[b] = 1;
      }
    }
    if (turn_end[b]) {
      double mean = s->turn_sum_t / (double)s->turn_tokens; /* Eq. 4 */
      if (mode == ORACLE_MODE_TURN_MEAN) {
        s->cum += mean; /* Eq. 5 */
        if (s->cum < lambda[b]) {
          s->stopped = 1;
          s->stop_row = pos;
          s->stop_turn = s->turn_idx;
          if (stopped_now) stopped_now[b] = 1;
        }
      }
      if (turn_n) turn_n[b] = s->turn_tokens;
      if (turn_sum_t) turn_sum_t[b] = s->turn_sum_t;
      if (turn_sum_d) turn_sum_d[b] = s->turn_sum_d;
      if (turn_sum_l) turn_sum_l[b] = s->turn_sum_l;
      if (turn_mean) turn_mean[b] = mean;
      if (turn_cum) turn_cum[b] = s->cum;
      s->turn_idx += 1;
      s->turn_tokens = 0;
      s->turn_sum_t = 0.0;
      s->turn_sum_d = 0.0;
      s->turn_sum_l = 0.0;
    }
  }
  return ORACLE_OK;
}

/* Restart choice from a stored record of per-turn means (Sec. 4.2 steps 1-2,
 * Eq. 6, Algorithm 1):
 *   correct_k = (mask == NULL or mask[k] != 0) and (l_k > alpha), k < n_turns;
 *   K_max     = largest K with correct_k for every k < K;
 *   k*        = argmin_{0 <= k < K_max} l_k, lowest index on ties;
 *   K_max = 0 gives k* = 0 (no reusable prefix, restart from scratch).
 * The 0-based k* is K0, the number of turns reused as context.  All compares
 * are in fp32, the precision of the stored record. */
int oracle_select_restart(const float* mean, const int32_t* n_turns, const uint8_t* mask,
                          float alpha, int32_t N, int32_t T_max, int32_t* k_star, int32_t* k_max) {
  if (!mean || !n_turns || !k_star || !k_max || N < 0 || T_max < 0) return ORACLE_ERR_ARG;
  for (int32_t i = 0; i < N; ++i) {
    int32_t nt = n_turns[i];
    if (nt < 0 || nt > T_max) return ORACLE_ERR_ARG;
    const float* l = mean + (int64_t)i * T_max;
    const uint8_t* m = mask ? mask + (int64_t)i * T_max : NULL;
    int32_t K = 0;
    while (K < nt && (m == NULL || m[K] != 0) && (l[K] > alpha)) ++K;
    int32_t best = 0;
    for (int32_t k = 1; k < K; ++k)
      if (l[k] < l[best]) best = k;
    k_max[i] = K;
    k_star[i] = best;
  }
  return ORACLE_OK;
}

/* Prefix buffer update (Algorithm 1: "record this trajectory's {l_k} to
 * H(x)"; Sec. 4.2 step 3, prefix reuse).  Trajectory i belongs to task
 * task[i] and reused the first k0[i] turns of that task's stored record as
 * context, so its own record is those k0[i] stored turns followed by the
 * means of its newly generated turns (turn_mean over its turns
 * traj_turn_off[i] .. traj_turn_off[i+1]-1, stored in fp32), truncated to
 * T_max turns.  k0[i] is clamped to the stored record's length.  Each task
 * may appear at most once per call.  mean: [n_tasks, T_max]; n_turns:
 * [n_tasks]. */
int oracle_buffer_record(float* mean, int32_t* n_turns, int32_t n_tasks, int32_t T_max,
                         const int32_t* task, const int32_t* k0, const float* turn_mean,
                         const int32_t* traj_turn_off, int32_t n_traj) {
  if (!mean || !n_turns || !task || !turn_mean || !traj_turn_off || n_traj < 0 || T_max < 0)
    return ORACLE_ERR_ARG;
  for (int32_t i = 0; i < n_traj; ++i) {
    int32_t x = task[i];
    if (x < 0 || x >= n_tasks) return ORACLE_ERR_ARG;
    int32_t keep = k0 ? k0[i] : 0;
    if (keep < 0) keep = 0;
    if (keep > n_turns[x]) keep = n_turns[x];
    int32_t len = keep;
    for (int32_t k = traj_turn_off[i]; k < traj_turn_off[i + 1] && len < T_max; ++k)
      mean[(int64_t)x * T_max + len++] = turn_mean[k];
    n_turns[x] = len;
  }
  return ORACLE_OK;
}

int oracle_rollout_size(void) { return (int)sizeof(oracle_rollout); }
