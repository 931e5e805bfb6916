/*
 * CommitKV CPU oracle — TEST INFRASTRUCTURE ONLY.
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline /
 * reference legs may load or call this code.  It shares no code with the
 * CUDA library and never runs on the product path.
 *
 * Plain, slow, fp64 restatement of the page deletion effect of
 * "CommitKV: Lifecycle-Aware KV Cache Compression via Commit Transitions
 * for Multi-Turn Agents" (arXiv 2608.07855), Section 3.2:
 *
 *   attention of one head at query position p over the resident tokens i
 *   with p_i <= p (the causal condition written under the sums of Eq. 6):
 *       s_i = scale * <q_p, k_i>,  a_pi = softmax_i(s_i),  o_p = sum_i a_pi v_i
 *   deletion of an event page E and renormalisation (Eq. 6):
 *       o_p^{\E} = (o_p - sum_{i in E, p_i <= p} a_pi v_i)
 *                  / (1 - sum_{i in E, p_i <= p} a_pi)
 *   window effect (Eq. 7):
 *       R_h(E; Q) = max_{p in Q} ||o_p - o_p^{\E}||_2 / ||o_p||_2,
 *       R(E; Q)   = max_h R_h(E; Q)
 *   set effect (Eq. 11): the same with every token of a page set A deleted
 *   at once; greedy joint test (Eq. 11 and the inner loop of Algorithm 1):
 *   accept E iff R(D u {E}) <= tau_joint, scanning all candidates in order.
 *
 * Two independent ways of computing an effect are provided:
 *   "explicit": the deleted tokens are removed from the softmax, which is
 *               recomputed from scratch (the definition of o^{\E});
 *   "closed":   Eq. 6 evaluated from the one unmasked softmax.
 * Tests pin each against the other and against a pure-Python brute force.
 *
 * Readings where the paper is silent (all shared with the GPU library's
 * documentation, not with its code):
 *   - h ranges over query heads; query head h reads KV head h / (Hq / H).
 *   - several layers are aggregated by the same max as heads; a layer mask
 *     selects which layers take part (all by default).
 *   - degenerate cases, applied in this order per query row:
 *       (1) no deleted token is visible to p            -> r = 0
 *       (2) every visible token is deleted (1 - s = 0)  -> r = +inf
 *       (3) ||o_p|| = 0: r = 0 if o_p^{\E} = o_p, else +inf
 *     a row that sees no token at all has o_p = 0 and falls under (1).
 *   - scale = 1/sqrt(d) unless given.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
  int32_t M, H, Hq, d, S, W, P;
  const double *K, *V;                  /* [M][H][S][d] */
  const int32_t *pos;                   /* [S] absolute positions */
  const double *Q;                      /* [M][Hq][W][d] probe queries */
  const int32_t *qpos;                  /* [W] absolute query positions */
  const int32_t *page_start, *page_len; /* [P] resident-index spans */
  const uint8_t *layer_mask;            /* [M] or NULL = every layer */
  double scale;
} okv_problem;

#define OKV_INF (1.0 / 0.0)

static int layer_on(const okv_problem *pb, int l) { return !pb->layer_mask || pb->layer_mask[l]; }

static const double *kv_row(const okv_problem *pb, const double *base, int l, int kvh, int i) {
  return base + (((size_t)l * pb->H + kvh) * pb->S + i) * pb->d;
}

static const double *q_row(const okv_problem *pb, int l, int h, int w) {
  return pb->Q + (((size_t)l * pb->Hq + h) * pb->W + w) * pb->d;
}

static double dot(const double *a, const double *b, int d) {
  double s = 0.0;
  for (int c = 0; c < d; ++c) s += a[c] * b[c];
  return s;
}

/* Softmax attention output over the tokens i with vis[i] && !drop[i].
 * s[] holds the scaled scores.  Returns the number of tokens used; o is
 * zeroed when none is used. */
static int attend(const okv_problem *pb, int l, int kvh, const double *s, const uint8_t *vis,
                  const uint8_t *drop, double *o) {
  int d = pb->d, n = 0;
  double m = -OKV_INF;
  for (int i = 0; i < pb->S; ++i)
    if (vis[i] && !(drop && drop[i])) {
      if (s[i] > m) m = s[i];
      ++n;
    }
  for (int c = 0; c < d; ++c) o[c] = 0.0;
  if (n == 0) return 0;
  double l_sum = 0.0;
  for (int i = 0; i < pb->S; ++i)
    if (vis[i] && !(drop && drop[i])) {
      double e = exp(s[i] - m);
      l_sum += e;
      const double *v = kv_row(pb, pb->V, l, kvh, i);
      for (int c = 0; c < d; ++c) o[c] += e * v[c];
    }
  for (int c = 0; c < d; ++c) o[c] /= l_sum;
  return n;
}

/* Relative change ||o - o2|| / ||o|| with rule (3). */
static double rel_change(const double *o, const double *o2, int d) {
  double num = 0.0, den = 0.0;
  for (int c = 0; c < d; ++c) {
    double t = o[c] - o2[c];
    num += t * t;
    den += o[c] * o[c];
  }
  if (den == 0.0) return num == 0.0 ? 0.0 : OKV_INF;
  return sqrt(num) / sqrt(den);
}

/* ------------------------------------------------------------------ */
/* per-(layer, query head) work split over threads                      */

typedef struct {
  const okv_problem *pb;
  int mode;          /* 0 explicit, 1 closed form */
  double *R_head;    /* [M][Hq][P] */
  int unit_begin, unit_end;
  int status;
} effects_job;

static void score_row(const okv_problem *pb, int l, int h, int w, double *s, uint8_t *vis) {
  int g = pb->Hq / pb->H, kvh = h / g;
  const double *q = q_row(pb, l, h, w);
  for (int i = 0; i < pb->S; ++i) {
    vis[i] = pb->pos[i] <= pb->qpos[w];
    s[i] = vis[i] ? pb->scale * dot(q, kv_row(pb, pb->K, l, kvh, i), pb->d) : 0.0;
  }
}

static void *effects_worker(void *arg) {
  effects_job *jb = (effects_job *)arg;
  const okv_problem *pb = jb->pb;
  int d = pb->d, S = pb->S, P = pb->P, g = pb->Hq / pb->H;
  double *s = malloc(sizeof(double) * (S > 0 ? S : 1));
  uint8_t *vis = malloc(S > 0 ? S : 1);
  uint8_t *drop = calloc(S > 0 ? S : 1, 1);
  double *o = malloc(sizeof(double) * d), *o2 = malloc(sizeof(double) * d);
  if (!s || !vis || !drop || !o || !o2) {
    jb->status = -1;
    goto done;
  }
  for (int unit = jb->unit_begin; unit < jb->unit_end; ++unit) {
    int l = unit / pb->Hq, h = unit % pb->Hq, kvh = h / g;
    double *Rh = jb->R_head + (size_t)unit * P;
    for (int E = 0; E < P; ++E) Rh[E] = 0.0;
    if (!layer_on(pb, l)) continue;
    for (int w = 0; w < pb->W; ++w) {
      score_row(pb, l, h, w, s, vis);
      int n_vis = attend(pb, l, kvh, s, vis, NULL, o);
      /* closed form needs the unmasked weights a_i = e_i / l */
      double m = -OKV_INF, l_sum = 0.0;
      if (jb->mode == 1 && n_vis > 0) {
        for (int i = 0; i < S; ++i)
          if (vis[i] && s[i] > m) m = s[i];
        for (int i = 0; i < S; ++i)
          if (vis[i]) l_sum += exp(s[i] - m);
      }
      for (int E = 0; E < P; ++E) {
        int b = pb->page_start[E], e = b + pb->page_len[E];
        int n_del = 0;
        for (int i = b; i < e; ++i) n_del += vis[i];
        double r;
        if (n_del == 0) {
          r = 0.0; /* rule (1) */
        } else if (n_del == n_vis) {
          r = OKV_INF; /* rule (2) */
        } else if (jb->mode == 0) {
          for (int i = b; i < e; ++i) drop[i] = 1;
          attend(pb, l, kvh, s, vis, drop, o2);
          for (int i = b; i < e; ++i) drop[i] = 0;
          r = rel_change(o, o2, d);
        } else {
          /* Eq. 6: o^{\E} = (o - sum_E a v) / (1 - sum_E a) */
          double sa = 0.0;
          for (int c = 0; c < d; ++c) o2[c] = 0.0;
          for (int i = b; i < e; ++i)
            if (vis[i]) {
              double a = exp(s[i] - m) / l_sum;
              sa += a;
              const double *v = kv_row(pb, pb->V, l, kvh, i);
              for (int c = 0; c < d; ++c) o2[c] += a * v[c];
            }
          for (int c = 0; c < d; ++c) o2[c] = (o[c] - o2[c]) / (1.0 - sa);
          r = rel_change(o, o2, d);
        }
        if (r > Rh[E]) Rh[E] = r; /* Eq. 7: max over the window */
      }
    }
  }
done:
  free(s);
  free(vis);
  free(drop);
  free(o);
  free(o2);
  return NULL;
}

static int check_problem(const okv_problem *pb) {
  if (!pb || pb->M < 1 || pb->H < 1 || pb->Hq < pb->H || pb->Hq % pb->H || pb->d < 1 || pb->S < 0 ||
      pb->W < 0 || pb->P < 0)
    return -1;
  for (int E = 0; E < pb->P; ++E) {
    if (pb->page_len[E] < 0 || pb->page_start[E] < 0 || pb->page_start[E] + pb->page_len[E] > pb->S)
      return -1;
  }
  return 0;
}

static int run_units(const okv_problem *pb, int mode, double *R_head, int nthreads) {
  int units = pb->M * pb->Hq;
  if (nthreads < 1) nthreads = 1;
  if (nthreads > units) nthreads = units;
  if (nthreads > 256) nthreads = 256;
  pthread_t th[256];
  effects_job jobs[256];
  int created[256];
  int per = (units + nthreads - 1) / nthreads;
  for (int t = 0; t < nthreads; ++t) {
    jobs[t].pb = pb;
    jobs[t].mode = mode;
    jobs[t].R_head = R_head;
    jobs[t].unit_begin = t * per;
    jobs[t].unit_end = (t + 1) * per < units ? (t + 1) * per : units;
    jobs[t].status = 0;
    created[t] = nthreads > 1 && pthread_create(&th[t], NULL, effects_worker, &jobs[t]) == 0;
    if (!created[t]) effects_worker(&jobs[t]);
  }
  int st = 0;
  for (int t = 0; t < nthreads; ++t) {
    if (created[t]) pthread_join(th[t], NULL);
    st |= jobs[t].status;
  }
  return st;
}

/* Per-(layer, query head, page) window effect R_h(E; Q) by explicit
 * deletion and recomputation.  R_head is [M][Hq][P]; entries of layers
 * outside the mask are 0.  Returns 0 on success. */
int okv_effects_explicit(const okv_problem *pb, double *R_head, int nthreads) {
  if (check_problem(pb)) return -1;
  return run_units(pb, 0, R_head, nthreads);
}

/* The same through the closed form of Eq. 6. */
int okv_effects_closed(const okv_problem *pb, double *R_head, int nthreads) {
  if (check_problem(pb)) return -1;
  return run_units(pb, 1, R_head, nthreads);
}

/* ------------------------------------------------------------------ */
/* per-row softmax statistics: m = max scaled score, l = sum exp(s - m),  */
/* o = normalised output, n = number of visible tokens.                  */

typedef struct {
  const okv_problem *pb;
  double *m, *l, *o;
  int32_t *n;
  int row_begin, row_end;
} stats_job;

static void *stats_worker(void *arg) {
  stats_job *jb = (stats_job *)arg;
  const okv_problem *pb = jb->pb;
  int S = pb->S, g = pb->Hq / pb->H;
  double *s = malloc(sizeof(double) * (S > 0 ? S : 1));
  uint8_t *vis = malloc(S > 0 ? S : 1);
  for (int row = jb->row_begin; row < jb->row_end; ++row) {
    int w = row % pb->W, h = (row / pb->W) % pb->Hq, l = row / (pb->W * pb->Hq);
    score_row(pb, l, h, w, s, vis);
    double m = -OKV_INF, ls = 0.0;
    for (int i = 0; i < S; ++i)
      if (vis[i] && s[i] > m) m = s[i];
    for (int i = 0; i < S; ++i)
      if (vis[i]) ls += exp(s[i] - m);
    jb->m[row] = m;
    jb->l[row] = ls;
    jb->n[row] = attend(pb, l, h / g, s, vis, NULL, jb->o + (size_t)row * pb->d);
  }
  free(s);
  free(vis);
  return NULL;
}

/* Row order is (layer, query head, window position).  Every layer is
 * computed regardless of the mask. */
int okv_row_stats(const okv_problem *pb, double *m, double *l, double *o, int32_t *n, int nthreads) {
  if (check_problem(pb)) return -1;
  int rows = pb->M * pb->Hq * pb->W;
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  if (nthreads > rows) nthreads = rows > 0 ? rows : 1;
  pthread_t th[256];
  stats_job jobs[256];
  int created[256];
  int per = (rows + nthreads - 1) / nthreads;
  for (int t = 0; t < nthreads; ++t) {
    jobs[t] = (stats_job){pb, m, l, o, n, t * per, (t + 1) * per < rows ? (t + 1) * per : rows};
    created[t] = nthreads > 1 && pthread_create(&th[t], NULL, stats_worker, &jobs[t]) == 0;
    if (!created[t]) stats_worker(&jobs[t]);
  }
  for (int t = 0; t < nthreads; ++t)
    if (created[t]) pthread_join(th[t], NULL);
  return 0;
}

/* ------------------------------------------------------------------ */
/* set effects and the greedy joint test                                */

typedef struct {
  const okv_problem *pb;
  const uint8_t *drop; /* [S] tokens deleted together */
  double *R_unit;      /* [M][Hq] max over the window */
  int unit_begin, unit_end;
} set_job;

static void *set_worker(void *arg) {
  set_job *jb = (set_job *)arg;
  const okv_problem *pb = jb->pb;
  int S = pb->S, d = pb->d, g = pb->Hq / pb->H;
  double *s = malloc(sizeof(double) * (S > 0 ? S : 1));
  uint8_t *vis = malloc(S > 0 ? S : 1);
  double *o = malloc(sizeof(double) * d), *o2 = malloc(sizeof(double) * d);
  for (int unit = jb->unit_begin; unit < jb->unit_end; ++unit) {
    int l = unit / pb->Hq, h = unit % pb->Hq;
    double R = 0.0;
    if (layer_on(pb, l)) {
      for (int w = 0; w < pb->W; ++w) {
        score_row(pb, l, h, w, s, vis);
        int n_vis = attend(pb, l, h / g, s, vis, NULL, o);
        int n_del = 0;
        for (int i = 0; i < S; ++i) n_del += vis[i] && jb->drop[i];
        double r;
        if (n_del == 0)
          r = 0.0;
        else if (n_del == n_vis)
          r = OKV_INF;
        else {
          attend(pb, l, h / g, s, vis, jb->drop, o2);
          r = rel_change(o, o2, d);
        }
        if (r > R) R = r;
      }
    }
    jb->R_unit[unit] = R;
  }
  free(s);
  free(vis);
  free(o);
  free(o2);
  return NULL;
}

/* R(A) for the deletion set given as a token mask, by explicit deletion.
 * R_unit (optional, [M][Hq]) receives the per-head maxima. */
double okv_set_effect_explicit(const okv_problem *pb, const uint8_t *drop, double *R_unit, int nthreads) {
  if (check_problem(pb)) return -1.0;
  int units = pb->M * pb->Hq;
  double *buf = R_unit ? R_unit : malloc(sizeof(double) * units);
  if (nthreads < 1) nthreads = 1;
  if (nthreads > units) nthreads = units;
  if (nthreads > 256) nthreads = 256;
  pthread_t th[256];
  set_job jobs[256];
  int created[256];
  int per = (units + nthreads - 1) / nthreads;
  for (int t = 0; t < nthreads; ++t) {
    jobs[t] = (set_job){pb, drop, buf, t * per, (t + 1) * per < units ? (t + 1) * per : units};
    created[t] = nthreads > 1 && pthread_create(&th[t], NULL, set_worker, &jobs[t]) == 0;
    if (!created[t]) set_worker(&jobs[t]);
  }
  for (int t = 0; t < nthreads; ++t)
    if (created[t]) pthread_join(th[t], NULL);
  double R = 0.0;
  for (int u = 0; u < units; ++u)
    if (buf[u] > R) R = buf[u];
  if (!R_unit) free(buf);
  return R;
}

/* Greedy joint test by explicit deletion of D u {E} at every step.
 * accepted[P] is set to 1 for accepted pages (others untouched: the
 * caller zeroes it); step_R[j] = R(D u {cand[j]}). */
int okv_greedy_explicit(const okv_problem *pb, const int32_t *cand, int n_cand, double tau,
                        uint8_t *accepted, double *step_R, int nthreads) {
  if (check_problem(pb)) return -1;
  uint8_t *drop = calloc(pb->S > 0 ? pb->S : 1, 1);
  uint8_t *trial = malloc(pb->S > 0 ? pb->S : 1);
  for (int j = 0; j < n_cand; ++j) {
    int E = cand[j];
    if (E < 0 || E >= pb->P) {
      free(drop);
      free(trial);
      return -1;
    }
    memcpy(trial, drop, pb->S);
    for (int i = pb->page_start[E]; i < pb->page_start[E] + pb->page_len[E]; ++i) trial[i] = 1;
    double R = okv_set_effect_explicit(pb, trial, NULL, nthreads);
    step_R[j] = R;
    if (R <= tau) {
      accepted[E] = 1;
      memcpy(drop, trial, pb->S);
    }
  }
  free(drop);
  free(trial);
  return 0;
}

/* Greedy joint test through Eq. 6 with the deleted page set treated as one
 * deletion set: per row the sums over D u {E} are the sums over D plus the
 * sums over E (the pages are disjoint).  Needs the row statistics from
 * okv_row_stats (m, l, o, n).  Rows are split over threads per step. */
typedef struct {
  const okv_problem *pb;
  const double *m, *l, *o;
  const int32_t *n;
  double *uA, *sA; /* [rows][d], [rows] */
  int32_t *nA;     /* [rows] */
  int E;
  int commit; /* 0: evaluate, 1: add E into the accepted sums */
  double R;
  int row_begin, row_end;
} greedy_job;

static void *greedy_worker(void *arg) {
  greedy_job *jb = (greedy_job *)arg;
  const okv_problem *pb = jb->pb;
  int d = pb->d, g = pb->Hq / pb->H;
  double *u = malloc(sizeof(double) * d), *o2 = malloc(sizeof(double) * d);
  int b = pb->page_start[jb->E], e = b + pb->page_len[jb->E];
  double Rmax = 0.0;
  for (int row = jb->row_begin; row < jb->row_end; ++row) {
    int w = row % pb->W, h = (row / pb->W) % pb->Hq, l = row / (pb->W * pb->Hq);
    if (!layer_on(pb, l)) continue;
    const double *q = q_row(pb, l, h, w);
    const double *o = jb->o + (size_t)row * d;
    double *uA = jb->uA + (size_t)row * d;
    double s = jb->sA[row];
    int n_del = jb->nA[row];
    for (int c = 0; c < d; ++c) u[c] = uA[c];
    for (int i = b; i < e; ++i) {
      if (pb->pos[i] > pb->qpos[w]) continue;
      double a = exp(pb->scale * dot(q, kv_row(pb, pb->K, l, h / g, i), d) - jb->m[row]) / jb->l[row];
      const double *v = kv_row(pb, pb->V, l, h / g, i);
      for (int c = 0; c < d; ++c) u[c] += a * v[c];
      s += a;
      ++n_del;
    }
    if (jb->commit) {
      for (int c = 0; c < d; ++c) uA[c] = u[c];
      jb->sA[row] = s;
      jb->nA[row] = n_del;
      continue;
    }
    double r;
    if (n_del == 0)
      r = 0.0;
    else if (n_del == jb->n[row])
      r = OKV_INF;
    else {
      for (int c = 0; c < d; ++c) o2[c] = (o[c] - u[c]) / (1.0 - s);
      r = rel_change(o, o2, d);
    }
    if (r > Rmax) Rmax = r;
  }
  jb->R = Rmax;
  free(u);
  free(o2);
  return NULL;
}

static double greedy_pass(greedy_job *base, int rows, int nthreads, int E, int commit) {
  pthread_t th[256];
  greedy_job jobs[256];
  int created[256];
  int per = (rows + nthreads - 1) / nthreads;
  for (int t = 0; t < nthreads; ++t) {
    jobs[t] = *base;
    jobs[t].E = E;
    jobs[t].commit = commit;
    jobs[t].row_begin = t * per;
    jobs[t].row_end = (t + 1) * per < rows ? (t + 1) * per : rows;
    created[t] = nthreads > 1 && pthread_create(&th[t], NULL, greedy_worker, &jobs[t]) == 0;
    if (!created[t]) greedy_worker(&jobs[t]);
  }
  double R = 0.0;
  for (int t = 0; t < nthreads; ++t) {
    if (created[t]) pthread_join(th[t], NULL);
    if (jobs[t].R > R) R = jobs[t].R;
  }
  return R;
}

int okv_greedy_closed(const okv_problem *pb, const double *m, const double *l, const double *o,
                      const int32_t *n, const int32_t *cand, int n_cand, double tau, uint8_t *accepted,
                      double *step_R, int nthreads) {
  if (check_problem(pb)) return -1;
  int rows = pb->M * pb->Hq * pb->W;
  if (rows == 0) {
    for (int j = 0; j < n_cand; ++j) step_R[j] = 0.0;
    return 0;
  }
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  if (nthreads > rows) nthreads = rows;
  greedy_job base;
  memset(&base, 0, sizeof base);
  base.pb = pb;
  base.m = m;
  base.l = l;
  base.o = o;
  base.n = n;
  base.uA = calloc((size_t)rows * pb->d, sizeof(double));
  base.sA = calloc(rows, sizeof(double));
  base.nA = calloc(rows, sizeof(int32_t));
  if (!base.uA || !base.sA || !base.nA) return -1;
  for (int j = 0; j < n_cand; ++j) {
    int E = cand[j];
    if (E < 0 || E >= pb->P) {
      free(base.uA);
      free(base.sA);
      free(base.nA);
      return -1;
    }
    double R = greedy_pass(&base, rows, nthreads, E, 0);
    step_R[j] = R;
    if (R <= tau) {
      accepted[E] = 1;
      greedy_pass(&base, rows, nthreads, E, 1);
    }
  }
  free(base.uA);
  free(base.sA);
  free(base.nA);
  return 0;
}
