/*
 * CPU oracle of the MeanField joint-configuration scorer -- TEST INFRASTRUCTURE.
 *
 * Plain C99, fp64 arithmetic on float32 inputs.  Only tests/, the smoke check
 * and the benchmark's CPU-baseline leg may load it; the CUDA path never does.
 * It shares no code with the CUDA path.  Each function names the passage of
 * the paper (arXiv 2609.02109) it follows.  Where the paper is silent the
 * reading taken is stated inline.
 */
#include "mf_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ---------------------------------------------------------------------------
 * Problem geometry
 * ------------------------------------------------------------------------- */

static int32_t d_in_of(const orc_problem *p) { return p->d_local + 4; }

static int64_t params_per_model(const orc_problem *p) {
  int64_t din = d_in_of(p), h1 = p->hidden1, h2 = p->hidden2;
  int64_t n = h1 * din + h1;
  int64_t last = h1;
  if (h2 > 0) { n += h2 * h1 + h2; last = h2; }
  return n + 2 * last + 2;
}

static int64_t option_offset(const orc_problem *p, int32_t model) {
  int64_t off = 0;
  for (int32_t i = 0; i < model; ++i) off += p->n_options[i];
  return off;
}

/* Eq. 1: |Lambda| = prod_i |Lambda_i|. */
uint64_t orc_space_size(const orc_problem *p) {
  uint64_t n = 1;
  for (int32_t i = 0; i < p->n_models; ++i) {
    uint64_t k = (uint64_t)p->n_options[i];
    if (k == 0) return 0;
    if (n > UINT64_MAX / k) return 0;
    n *= k;
  }
  return n;
}

/* Eq. 1, enumerated as a mixed-radix number.  Reading (paper silent on the
 * order): C order, idx = sum_i o_i * prod_{j>i} K_j, the last model fastest. */
void orc_decode(const orc_problem *p, uint64_t idx, int32_t *o) {
  for (int32_t i = p->n_models - 1; i >= 0; --i) {
    uint64_t k = (uint64_t)p->n_options[i];
    o[i] = (int32_t)(idx % k);
    idx /= k;
  }
}

/* ---------------------------------------------------------------------------
 * One joint configuration: aggregate (Eq. 2 in the coupled reading),
 * per-model predictor (Eq. 6), constraints (Eq. 4) and objective (Eq. 3).
 * ------------------------------------------------------------------------- */

/* ReLU; a NaN input stays NaN (the torch.relu convention), so a NaN anywhere
 * in a predictor reaches its outputs and the candidate becomes infeasible. */
static double relu(double v) { return v < 0.0 ? 0.0 : v; }

/* Eq. 6: f_i = g_i(lambda_i, aggregate state).  g_i is an MLP (Sec. III-B);
 * at inference BatchNorm folds into the Linear layers and Dropout is the
 * identity, so the layers are Linear -> ReLU -> [Linear -> ReLU] -> Linear,
 * with an optional sigmoid on the two outputs (the paper's output unit). */
static void predictor(const orc_problem *p, int32_t model, const double *z,
                      double *thr, double *lat, double *mag) {
  const int32_t din = d_in_of(p), h1 = p->hidden1, h2 = p->hidden2;
  const float *w = p->weights + (int64_t)model * params_per_model(p);
  const float *W1 = w;
  const float *b1 = W1 + (int64_t)h1 * din;
  double a1[h1 > 0 ? h1 : 1];
  for (int32_t j = 0; j < h1; ++j) {
    double s = (double)b1[j];
    for (int32_t k = 0; k < din; ++k) s += (double)W1[(int64_t)j * din + k] * z[k];
    a1[j] = relu(s);
  }
  const float *next = b1 + h1;
  double *h = a1;
  int32_t hl = h1;
  double a2[h2 > 0 ? h2 : 1];
  if (h2 > 0) {
    const float *W2 = next;
    const float *b2 = W2 + (int64_t)h2 * h1;
    for (int32_t j = 0; j < h2; ++j) {
      double s = (double)b2[j];
      for (int32_t k = 0; k < h1; ++k) s += (double)W2[(int64_t)j * h1 + k] * a1[k];
      a2[j] = relu(s);
    }
    next = b2 + h2;
    h = a2;
    hl = h2;
  }
  const float *W3 = next;
  const float *b3 = W3 + 2 * (int64_t)hl;
  double y[2];
  for (int32_t o = 0; o < 2; ++o) {
    double s = (double)b3[o];
    double m = fabs((double)b3[o]);
    for (int32_t k = 0; k < hl; ++k) {
      s += (double)W3[(int64_t)o * hl + k] * h[k];
      m += fabs((double)W3[(int64_t)o * hl + k]) * fabs(h[k]);
    }
    if (p->out_act == 1) s = 1.0 / (1.0 + exp(-s));
    y[o] = s;
    if (mag) mag[o] = m;
  }
  *thr = y[0];
  *lat = y[1];
}

double orc_score_digits(const orc_problem *p, const int32_t *o, int32_t *feasible,
                        double *pred, double *agg) {
  const int32_t n = p->n_models, dl = p->d_local, din = d_in_of(p);
  /* Aggregate GPU state: summed SM share, VRAM and bandwidth demand of the
   * chosen options of all N models (in model order), plus N. */
  double A[4] = {0.0, 0.0, 0.0, (double)n};
  for (int32_t i = 0; i < n; ++i) {
    const float *d = p->demand + 3 * (option_offset(p, i) + o[i]);
    A[0] += (double)d[0];
    A[1] += (double)d[1];
    A[2] += (double)d[2];
  }
  double s[4];
  if (p->agg_scale) {
    for (int c = 0; c < 4; ++c) s[c] = (double)p->agg_scale[c];
  } else {
    /* Reading (paper silent on input scaling): each aggregate feature is
     * brought to about [0, 1]. */
    s[0] = 1.0 / (0.6 * n); s[1] = 1.0 / (20.0 * n); s[2] = 1.0 / (1500.0 * n); s[3] = 1.0 / 8.0;
    /* the products are formed as the float32 values the library would store */
    for (int c = 0; c < 4; ++c) s[c] = (double)(float)s[c];
  }
  if (agg) for (int c = 0; c < 4; ++c) agg[c] = A[c];

  double z[din];
  double J = 0.0, penalty = 0.0;
  int32_t sla_ok = 1;
  for (int32_t i = 0; i < n; ++i) {
    const float *x = p->local_feats + (int64_t)dl * (option_offset(p, i) + o[i]);
    for (int32_t k = 0; k < dl; ++k) z[k] = (double)x[k];
    for (int c = 0; c < 4; ++c) z[dl + c] = A[c] * s[c];
    double thr, lat;
    predictor(p, i, z, &thr, &lat, NULL);
    if (pred) { pred[2 * i] = thr; pred[2 * i + 1] = lat; }
    /* Eq. 3 first term, with the throughput-weighted objective sum_i w_i thr_i */
    J += (double)p->obj_w[i] * thr;
    if (!(lat <= (double)p->sla[i])) sla_ok = 0;
    double over = lat - (double)p->sla[i];
    penalty += over > 0.0 ? over : 0.0;
  }
  /* Eq. 4: sum_i r_i^VRAM <= R (inclusive) ... */
  int32_t feas = A[1] <= (double)p->vram_cap;
  if (p->objective == 0) {
    /* ... and every per-model SLA (latency ceiling, inclusive). */
    feas = feas && sla_ok;
  } else {
    /* soft-latency objective: the SLA enters as a linear penalty only */
    J -= (double)p->soft_penalty * penalty;
  }
  if (isnan(J)) feas = 0;
  if (feasible) *feasible = feas;
  /* Infeasible candidates receive J = -inf (Sec. II, constraints). */
  return feas ? J : -INFINITY;
}

void orc_score_list(const orc_problem *p, const uint64_t *idx, uint64_t n,
                    double *score, int32_t *feasible, double *pred, double *agg,
                    int32_t nthreads) {
  const uint64_t total = orc_space_size(p);
  const int32_t nm = p->n_models;
  (void)nthreads;
#ifdef _OPENMP
#pragma omp parallel for schedule(static) num_threads(nthreads > 0 ? nthreads : 1)
#endif
  for (int64_t t = 0; t < (int64_t)n; ++t) {
    int32_t o[64];
    int32_t f = 0;
    double J = -INFINITY;
    if (idx[t] < total) {
      orc_decode(p, idx[t], o);
      J = orc_score_digits(p, o, &f, pred ? pred + 2 * nm * t : NULL, agg ? agg + 4 * t : NULL);
    }
    score[t] = J;
    if (feasible) feasible[t] = f;
  }
}

/* Condition scale of every predictor output of one candidate: the magnitude
 * |b3_o| + sum_k |W3[o][k]| |h_k| of the terms of the final dot product, with
 * the exact last hidden layer h (before the output activation).  Rounding
 * errors of a reduced-precision evaluation scale with this sum, not with the
 * possibly cancelling output itself. */
static void pred_scale_digits(const orc_problem *p, const int32_t *o, double *scale) {
  const int32_t n = p->n_models, dl = p->d_local, din = d_in_of(p);
  double A[4] = {0.0, 0.0, 0.0, (double)n};
  for (int32_t i = 0; i < n; ++i) {
    const float *d = p->demand + 3 * (option_offset(p, i) + o[i]);
    A[0] += (double)d[0]; A[1] += (double)d[1]; A[2] += (double)d[2];
  }
  double s[4];
  if (p->agg_scale) {
    for (int c = 0; c < 4; ++c) s[c] = (double)p->agg_scale[c];
  } else {
    s[0] = 1.0 / (0.6 * n); s[1] = 1.0 / (20.0 * n); s[2] = 1.0 / (1500.0 * n); s[3] = 1.0 / 8.0;
    for (int c = 0; c < 4; ++c) s[c] = (double)(float)s[c];
  }
  double z[din];
  for (int32_t i = 0; i < n; ++i) {
    const float *x = p->local_feats + (int64_t)dl * (option_offset(p, i) + o[i]);
    for (int32_t k = 0; k < dl; ++k) z[k] = (double)x[k];
    for (int c = 0; c < 4; ++c) z[dl + c] = A[c] * s[c];
    double thr, lat;
    predictor(p, i, z, &thr, &lat, scale + 2 * i);
  }
}

void orc_pred_scale_list(const orc_problem *p, const uint64_t *idx, uint64_t n, double *scale,
                         int32_t nthreads) {
  const uint64_t total = orc_space_size(p);
  const int32_t nm = p->n_models;
  (void)nthreads;
#ifdef _OPENMP
#pragma omp parallel for schedule(static) num_threads(nthreads > 0 ? nthreads : 1)
#endif
  for (int64_t t = 0; t < (int64_t)n; ++t) {
    int32_t o[64];
    if (idx[t] < total) {
      orc_decode(p, idx[t], o);
      pred_scale_digits(p, o, scale + 2 * nm * t);
    } else {
      for (int32_t j = 0; j < 2 * nm; ++j) scale[2 * nm * t + j] = 0.0;
    }
  }
}

/* ---------------------------------------------------------------------------
 * Exhaustive search: lambda* = argmax_{lambda in Lambda} J (Sec. II), extended
 * to the top-k and the number of feasible candidates.  Total order: J
 * descending, then index ascending, so the answer does not depend on the
 * enumeration order.
 * ------------------------------------------------------------------------- */

static int precedes(double ja, uint64_t ia, double jb, uint64_t ib) {
  return ja > jb || (ja == jb && ia < ib);
}

static void topk_insert(int32_t k, uint64_t *ti, double *ts, double J, uint64_t idx) {
  if (!precedes(J, idx, ts[k - 1], ti[k - 1])) return;
  int32_t pos = k - 1;
  while (pos > 0 && precedes(J, idx, ts[pos - 1], ti[pos - 1])) {
    ts[pos] = ts[pos - 1];
    ti[pos] = ti[pos - 1];
    --pos;
  }
  ts[pos] = J;
  ti[pos] = idx;
}

void orc_exhaustive(const orc_problem *p, uint64_t lo, uint64_t hi, int32_t k,
                    uint64_t *topk_idx, double *topk_score, uint64_t *count,
                    int32_t nthreads) {
  for (int32_t j = 0; j < k; ++j) { topk_idx[j] = UINT64_MAX; topk_score[j] = -INFINITY; }
  uint64_t total_count = 0;
  const uint64_t size = orc_space_size(p);
  if (hi > size) hi = size;
  if (nthreads < 1) nthreads = 1;
#ifdef _OPENMP
#pragma omp parallel num_threads(nthreads)
#endif
  {
    uint64_t *li = (uint64_t *)malloc(sizeof(uint64_t) * (size_t)k);
    double *ls = (double *)malloc(sizeof(double) * (size_t)k);
    for (int32_t j = 0; j < k; ++j) { li[j] = UINT64_MAX; ls[j] = -INFINITY; }
    uint64_t c = 0;
    int32_t o[64];
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 4096)
#endif
    for (int64_t t = (int64_t)lo; t < (int64_t)hi; ++t) {
      int32_t f = 0;
      orc_decode(p, (uint64_t)t, o);
      double J = orc_score_digits(p, o, &f, NULL, NULL);
      if (f) {
        ++c;
        topk_insert(k, li, ls, J, (uint64_t)t);
      }
    }
#ifdef _OPENMP
#pragma omp critical
#endif
    {
      total_count += c;
      for (int32_t j = 0; j < k; ++j)
        if (li[j] != UINT64_MAX) topk_insert(k, topk_idx, topk_score, ls[j], li[j]);
    }
    free(li);
    free(ls);
  }
  *count = total_count;
}

/* ---------------------------------------------------------------------------
 * GA scheduler (Sec. IV-C): population, tournament selection, crossover,
 * mutation, elitism.  Random draws come from a counter-based SplitMix64
 * (Steele, Lea and Flood, OOPSLA 2014): output number ctr of the sequence
 * whose state starts at seed is mix(seed + (ctr + 1) * 0x9E3779B97F4A7C15).
 * ------------------------------------------------------------------------- */

uint64_t orc_splitmix64(uint64_t seed, uint64_t ctr) {
  uint64_t z = seed + (ctr + 1) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

/* Counter layout: gen (32 bits) | slot (20) | purpose (4) | j (8). */
uint64_t orc_rng(uint64_t seed, uint32_t gen, uint32_t slot, uint32_t purpose, uint32_t j) {
  uint64_t ctr = ((uint64_t)gen << 32) | ((uint64_t)(slot & 0xFFFFFu) << 12) |
                 ((uint64_t)(purpose & 0xFu) << 8) | (uint64_t)(j & 0xFFu);
  return orc_splitmix64(seed, ctr);
}

enum { GA_INIT = 0, GA_TOUR_A = 1, GA_TOUR_B = 2, GA_CROSS = 3, GA_MUT = 4, GA_MUTVAL = 5 };

/* Uniform integer in [0, k): high 32 bits scaled by k. */
static int32_t unif_int(uint64_t r, uint32_t k) {
  return (int32_t)(((r >> 32) * (uint64_t)k) >> 32);
}

void orc_ga_init(const orc_problem *p, const orc_ga_params *g, uint64_t seed, int32_t *pop) {
  const int32_t n = p->n_models;
  for (int32_t c = 0; c < g->pop; ++c)
    for (int32_t i = 0; i < n; ++i)
      pop[(int64_t)c * n + i] =
          unif_int(orc_rng(seed, 0, (uint32_t)c, GA_INIT, (uint32_t)i), (uint32_t)p->n_options[i]);
}

/* Tournament selection: draw `tournament` slots with replacement; the winner
 * has the highest fitness, the lowest slot among equals. */
static int32_t tournament(const orc_ga_params *g, const double *f, uint64_t seed,
                          uint32_t gen, uint32_t child, uint32_t purpose) {
  int32_t best = -1;
  for (int32_t t = 0; t < g->tournament; ++t) {
    int32_t s = unif_int(orc_rng(seed, gen, child, purpose, (uint32_t)t), (uint32_t)g->pop);
    if (best < 0 || f[s] > f[best] || (f[s] == f[best] && s < best)) best = s;
  }
  return best;
}

void orc_ga_step(const orc_problem *p, const orc_ga_params *g, uint64_t seed, int32_t gen,
                 const int32_t *pop, const double *fitness, int32_t *next) {
  const int32_t n = p->n_models;
  const uint32_t G = (uint32_t)gen + 1u; /* draws of the generation being produced */
  const uint32_t mut_thr = (uint32_t)floor(g->mutation_p * 16777216.0 + 0.5);
  int32_t first = 0;
  if (g->elitism) {
    /* elitism: the fittest individual (lowest slot among equals) survives unchanged */
    int32_t e = 0;
    for (int32_t c = 1; c < g->pop; ++c)
      if (fitness[c] > fitness[e]) e = c;
    memcpy(next, pop + (int64_t)e * n, sizeof(int32_t) * (size_t)n);
    first = 1;
  }
  for (int32_t c = first; c < g->pop; ++c) {
    int32_t a = tournament(g, fitness, seed, G, (uint32_t)c, GA_TOUR_A);
    int32_t b = tournament(g, fitness, seed, G, (uint32_t)c, GA_TOUR_B);
    for (int32_t i = 0; i < n; ++i) {
      /* uniform crossover: each gene from one parent with probability 1/2 */
      uint64_t rc = orc_rng(seed, G, (uint32_t)c, GA_CROSS, (uint32_t)i);
      int32_t gene = (rc >> 63) ? pop[(int64_t)b * n + i] : pop[(int64_t)a * n + i];
      /* per-gene mutation: redraw the option uniformly */
      uint64_t rm = orc_rng(seed, G, (uint32_t)c, GA_MUT, (uint32_t)i);
      if ((uint32_t)(rm >> 40) < mut_thr)
        gene = unif_int(orc_rng(seed, G, (uint32_t)c, GA_MUTVAL, (uint32_t)i),
                        (uint32_t)p->n_options[i]);
      next[(int64_t)c * n + i] = gene;
    }
  }
}

double orc_ga_run(const orc_problem *p, const orc_ga_params *g, uint64_t seed,
                  int32_t *best_genome, int32_t nthreads) {
  const int32_t n = p->n_models;
  int32_t *pop = (int32_t *)malloc(sizeof(int32_t) * (size_t)g->pop * n);
  int32_t *nxt = (int32_t *)malloc(sizeof(int32_t) * (size_t)g->pop * n);
  double *fit = (double *)malloc(sizeof(double) * (size_t)g->pop);
  (void)nthreads;
  orc_ga_init(p, g, seed, pop);
  double best = -INFINITY;
  for (int32_t gen = 0; gen < g->gens; ++gen) {
#ifdef _OPENMP
#pragma omp parallel for schedule(static) num_threads(nthreads > 0 ? nthreads : 1)
#endif
    for (int32_t c = 0; c < g->pop; ++c) fit[c] = orc_score_digits(p, pop + (int64_t)c * n, NULL, NULL, NULL);
    if (gen == g->gens - 1) {
      int32_t e = 0;
      for (int32_t c = 1; c < g->pop; ++c)
        if (fit[c] > fit[e]) e = c;
      best = fit[e];
      memcpy(best_genome, pop + (int64_t)e * n, sizeof(int32_t) * (size_t)n);
      break;
    }
    orc_ga_step(p, g, seed, gen, pop, fit, nxt);
    int32_t *t = pop; pop = nxt; nxt = t;
  }
  free(pop);
  free(nxt);
  free(fit);
  return best;
}

/* ---------------------------------------------------------------------------
 * Fixed-context mode: Sec. III-B holds the observed state s_t fixed during the
 * search, so each predictor g_i(lambda_i, s_t) depends on its own option only;
 * Eq. 3 is the utility, Eq. 4 the constraints.
 * ------------------------------------------------------------------------- */

/* The observed state fed to the predictors, scaled like the aggregate. */
static void fc_inputs(const orc_problem *p, const orc_fc *fc, double *zs) {
  const int32_t n = p->n_models;
  double s[4];
  if (p->agg_scale) {
    for (int c = 0; c < 4; ++c) s[c] = (double)p->agg_scale[c];
  } else {
    s[0] = 1.0 / (0.6 * n); s[1] = 1.0 / (20.0 * n); s[2] = 1.0 / (1500.0 * n); s[3] = 1.0 / 8.0;
    for (int c = 0; c < 4; ++c) s[c] = (double)(float)s[c];
  }
  for (int c = 0; c < 4; ++c) zs[c] = (double)fc->obs[c] * s[c];
}

/* Model i's term of Eq. 3 for option row r: returns u and sets *fhat, *f, *ok. */
static double fc_term(const orc_problem *p, const orc_fc *fc, int32_t i, int64_t r, const double *zs,
                      double *fhat_out, double *f_out, int32_t *ok_out) {
  const int32_t dl = p->d_local, din = d_in_of(p);
  double z[din];
  const float *x = p->local_feats + (int64_t)dl * r;
  for (int32_t k = 0; k < dl; ++k) z[k] = (double)x[k];
  for (int c = 0; c < 4; ++c) z[dl + c] = zs[c];
  double fhat, lat;
  predictor(p, i, z, &fhat, &lat, NULL);
  /* per-variant min-max normalisation of the raw predicted throughput */
  const double f = (fhat - (double)fc->f_min[r]) / ((double)fc->f_max[r] - (double)fc->f_min[r]);
  /* eta_i: the option's variant differs from the one in use (none in use: 0) */
  const int32_t eta = fc->prev_variant[i] >= 0 && fc->variant[r] != fc->prev_variant[i];
  const double margin = (double)fc->tau[i] + (double)fc->delta - f;
  const double u = (double)fc->omega[i] * f * (double)fc->quality[r] -
                   (double)fc->alpha * (double)eta * (double)fc->reload_cost[i] -
                   (double)fc->beta * (margin > 0.0 ? margin * margin : 0.0);
  if (fhat_out) *fhat_out = fhat;
  if (f_out) *f_out = f;
  /* the hard throughput floor f_i >= tau_i (inclusive) */
  if (ok_out) *ok_out = f >= (double)fc->tau[i];
  return u;
}

void orc_fc_local(const orc_problem *p, const orc_fc *fc, double *fhat, double *f, int32_t *ok,
                  double *u) {
  double zs[4];
  fc_inputs(p, fc, zs);
  for (int32_t i = 0; i < p->n_models; ++i)
    for (int32_t o = 0; o < p->n_options[i]; ++o) {
      const int64_t r = option_offset(p, i) + o;
      u[r] = fc_term(p, fc, i, r, zs, &fhat[r], &f[r], &ok[r]);
    }
}

double orc_fc_score_digits(const orc_problem *p, const orc_fc *fc, const int32_t *o, int32_t *feasible) {
  double zs[4];
  fc_inputs(p, fc, zs);
  double J = 0.0, vram = 0.0;
  int32_t floors = 1;
  for (int32_t i = 0; i < p->n_models; ++i) {
    const int64_t r = option_offset(p, i) + o[i];
    int32_t ok;
    J += fc_term(p, fc, i, r, zs, NULL, NULL, &ok);
    floors = floors && ok;
    vram += (double)p->demand[3 * r + 1];
  }
  int32_t feas = floors && vram <= (double)p->vram_cap;
  if (isnan(J)) feas = 0;
  if (feasible) *feasible = feas;
  return feas ? J : -INFINITY;
}

void orc_fc_exhaustive(const orc_problem *p, const orc_fc *fc, uint64_t lo, uint64_t hi, int32_t k,
                       uint64_t *topk_idx, double *topk_score, uint64_t *count, int32_t nthreads) {
  for (int32_t j = 0; j < k; ++j) { topk_idx[j] = UINT64_MAX; topk_score[j] = -INFINITY; }
  uint64_t total_count = 0;
  const uint64_t size = orc_space_size(p);
  if (hi > size) hi = size;
  if (nthreads < 1) nthreads = 1;
#ifdef _OPENMP
#pragma omp parallel num_threads(nthreads)
#endif
  {
    uint64_t *li = (uint64_t *)malloc(sizeof(uint64_t) * (size_t)k);
    double *ls = (double *)malloc(sizeof(double) * (size_t)k);
    for (int32_t j = 0; j < k; ++j) { li[j] = UINT64_MAX; ls[j] = -INFINITY; }
    uint64_t c = 0;
    int32_t o[64];
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 4096)
#endif
    for (int64_t t = (int64_t)lo; t < (int64_t)hi; ++t) {
      int32_t f = 0;
      orc_decode(p, (uint64_t)t, o);
      const double J = orc_fc_score_digits(p, fc, o, &f);
      if (f) {
        ++c;
        topk_insert(k, li, ls, J, (uint64_t)t);
      }
    }
#ifdef _OPENMP
#pragma omp critical
#endif
    {
      total_count += c;
      for (int32_t j = 0; j < k; ++j)
        if (li[j] != UINT64_MAX) topk_insert(k, topk_idx, topk_score, ls[j], li[j]);
    }
    free(li);
    free(ls);
  }
  *count = total_count;
}

uint64_t orc_vram_feasible(const orc_problem *p, uint64_t lo, uint64_t hi, uint64_t *out, uint64_t cap) {
  const uint64_t size = orc_space_size(p);
  if (hi > size) hi = size;
  uint64_t c = 0;
  int32_t o[64];
  for (uint64_t t = lo; t < hi; ++t) {
    orc_decode(p, t, o);
    double vram = 0.0;
    for (int32_t i = 0; i < p->n_models; ++i) vram += (double)p->demand[3 * (option_offset(p, i) + o[i]) + 1];
    /* Eq. 4: sum_i r_i^VRAM <= R; the others are removed when Lambda is built */
    if (vram <= (double)p->vram_cap) {
      if (c < cap) out[c] = t;
      ++c;
    }
  }
  return c;
}

/* ---------------------------------------------------------------------------
 * Eq. 3 utility on the coupled aggregate (the predictors see the candidate's own
 * summed demands, as in orc_score_digits).
 * ------------------------------------------------------------------------- */

/* Model i's term of Eq. 3 from its raw predicted throughput fhat (option row r). */
static double util_term(const orc_fc *fc, int32_t i, int64_t r, double fhat, int32_t *ok) {
  const double f = (fhat - (double)fc->f_min[r]) / ((double)fc->f_max[r] - (double)fc->f_min[r]);
  const int32_t eta = fc->prev_variant[i] >= 0 && fc->variant[r] != fc->prev_variant[i];
  const double margin = (double)fc->tau[i] + (double)fc->delta - f;
  *ok = f >= (double)fc->tau[i];
  return (double)fc->omega[i] * f * (double)fc->quality[r] -
         (double)fc->alpha * (double)eta * (double)fc->reload_cost[i] -
         (double)fc->beta * (margin > 0.0 ? margin * margin : 0.0);
}

double orc_util_score_digits(const orc_problem *p, const orc_fc *fc, const int32_t *o, int32_t *feasible,
                             double *pred, double *agg) {
  const int32_t n = p->n_models, dl = p->d_local, din = d_in_of(p);
  double A[4] = {0.0, 0.0, 0.0, (double)n};
  for (int32_t i = 0; i < n; ++i) {
    const float *d = p->demand + 3 * (option_offset(p, i) + o[i]);
    A[0] += (double)d[0];
    A[1] += (double)d[1];
    A[2] += (double)d[2];
  }
  double s[4];
  if (p->agg_scale) {
    for (int c = 0; c < 4; ++c) s[c] = (double)p->agg_scale[c];
  } else {
    s[0] = 1.0 / (0.6 * n); s[1] = 1.0 / (20.0 * n); s[2] = 1.0 / (1500.0 * n); s[3] = 1.0 / 8.0;
    for (int c = 0; c < 4; ++c) s[c] = (double)(float)s[c];
  }
  if (agg) for (int c = 0; c < 4; ++c) agg[c] = A[c];
  double z[din];
  double J = 0.0;
  int32_t floors = 1;
  for (int32_t i = 0; i < n; ++i) {
    const int64_t r = option_offset(p, i) + o[i];
    const float *x = p->local_feats + (int64_t)dl * r;
    for (int32_t k = 0; k < dl; ++k) z[k] = (double)x[k];
    for (int c = 0; c < 4; ++c) z[dl + c] = A[c] * s[c];
    double thr, lat;
    predictor(p, i, z, &thr, &lat, NULL);
    if (pred) { pred[2 * i] = thr; pred[2 * i + 1] = lat; }
    int32_t ok;
    J += util_term(fc, i, r, thr, &ok);
    floors = floors && ok;
  }
  int32_t feas = floors && A[1] <= (double)p->vram_cap;
  if (isnan(J)) feas = 0;
  if (feasible) *feasible = feas;
  return feas ? J : -INFINITY;
}

void orc_util_score_list(const orc_problem *p, const orc_fc *fc, const uint64_t *idx, uint64_t n,
                         double *score, int32_t *feasible, double *pred, double *agg, int32_t nthreads) {
  const uint64_t size = orc_space_size(p);
  const int32_t N = p->n_models;
  if (nthreads < 1) nthreads = 1;
#ifdef _OPENMP
#pragma omp parallel for num_threads(nthreads) schedule(static)
#endif
  for (int64_t t = 0; t < (int64_t)n; ++t) {
    int32_t o[64];
    int32_t f = 0;
    double J = -INFINITY;
    if (idx[t] < size) {
      orc_decode(p, idx[t], o);
      J = orc_util_score_digits(p, fc, o, &f, pred ? pred + 2 * N * t : NULL, agg ? agg + 4 * t : NULL);
    } else if (pred) {
      for (int32_t j = 0; j < 2 * N; ++j) pred[2 * N * t + j] = NAN;
    }
    score[t] = J;
    if (feasible) feasible[t] = f;
  }
}

void orc_util_exhaustive(const orc_problem *p, const orc_fc *fc, uint64_t lo, uint64_t hi, int32_t k,
                         uint64_t *topk_idx, double *topk_score, uint64_t *count, int32_t nthreads) {
  for (int32_t j = 0; j < k; ++j) { topk_idx[j] = UINT64_MAX; topk_score[j] = -INFINITY; }
  uint64_t total_count = 0;
  const uint64_t size = orc_space_size(p);
  if (hi > size) hi = size;
  if (nthreads < 1) nthreads = 1;
#ifdef _OPENMP
#pragma omp parallel num_threads(nthreads)
#endif
  {
    uint64_t *li = (uint64_t *)malloc(sizeof(uint64_t) * (size_t)k);
    double *ls = (double *)malloc(sizeof(double) * (size_t)k);
    for (int32_t j = 0; j < k; ++j) { li[j] = UINT64_MAX; ls[j] = -INFINITY; }
    uint64_t c = 0;
    int32_t o[64];
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 4096)
#endif
    for (int64_t t = (int64_t)lo; t < (int64_t)hi; ++t) {
      int32_t f = 0;
      orc_decode(p, (uint64_t)t, o);
      const double J = orc_util_score_digits(p, fc, o, &f, NULL, NULL);
      if (f) {
        ++c;
        topk_insert(k, li, ls, J, (uint64_t)t);
      }
    }
#ifdef _OPENMP
#pragma omp critical
#endif
    {
      total_count += c;
      for (int32_t j = 0; j < k; ++j)
        if (li[j] != UINT64_MAX) topk_insert(k, topk_idx, topk_score, ls[j], li[j]);
    }
    free(li);
    free(ls);
  }
  *count = total_count;
}

/* ---------------------------------------------------------------------------
 * The paper's GA (Sec. IV-C) on the fixed-context landscape (Sec. III-B holds s_t
 * fixed during the GA search).
 * ------------------------------------------------------------------------- */
enum { GA_CROSS_DO = 6, GA_REPAIR = 7 };

/* J of a genome from the per-option terms (the sum over models of Eq. 3's terms,
 * -inf when a floor fails or the VRAM bound of Eq. 4 is exceeded). */
static double fc_fitness(const orc_problem *p, const double *u, const int32_t *ok, const int32_t *o) {
  double J = 0.0, vram = 0.0;
  int32_t good = 1;
  for (int32_t i = 0; i < p->n_models; ++i) {
    const int64_t r = option_offset(p, i) + o[i];
    J += u[r];
    good = good && ok[r];
    vram += (double)p->demand[3 * r + 1];
  }
  return (good && vram <= (double)p->vram_cap && !isnan(J)) ? J : -INFINITY;
}

/* Repair: replace an infeasible genome by a uniformly drawn feasible one (rejection,
 * at most floor(256 / N) attempts, draws (gen, slot, GA_REPAIR, a * N + i)). */
static double fc_repair(const orc_problem *p, const double *u, const int32_t *ok, uint64_t seed, uint32_t gen,
                        uint32_t slot, int32_t *o, double J) {
  const int32_t n = p->n_models;
  const int32_t attempts = 256 / n;
  int32_t cand[64];
  for (int32_t a = 0; a < attempts && J == -INFINITY; ++a) {
    for (int32_t i = 0; i < n; ++i)
      cand[i] = unif_int(orc_rng(seed, gen, slot, GA_REPAIR, (uint32_t)(a * n + i)), (uint32_t)p->n_options[i]);
    const double Jc = fc_fitness(p, u, ok, cand);
    if (Jc != -INFINITY) {
      memcpy(o, cand, sizeof(int32_t) * (size_t)n);
      J = Jc;
    }
  }
  return J;
}

double orc_fc_ga_run(const orc_problem *p, const orc_fc *fc, const orc_fc_ga_params *g, uint64_t seed,
                     int32_t *best_genome) {
  const int32_t n = p->n_models;
  int64_t rows = 0;
  for (int32_t i = 0; i < n; ++i) rows += p->n_options[i];
  double *fhat = (double *)malloc(sizeof(double) * (size_t)rows);
  double *f = (double *)malloc(sizeof(double) * (size_t)rows);
  double *u = (double *)malloc(sizeof(double) * (size_t)rows);
  int32_t *ok = (int32_t *)malloc(sizeof(int32_t) * (size_t)rows);
  orc_fc_local(p, fc, fhat, f, ok, u);
  int32_t *pop = (int32_t *)malloc(sizeof(int32_t) * (size_t)g->pop * n);
  int32_t *next = (int32_t *)malloc(sizeof(int32_t) * (size_t)g->pop * n);
  double *fit = (double *)malloc(sizeof(double) * (size_t)g->pop);
  double *nfit = (double *)malloc(sizeof(double) * (size_t)g->pop);
  const uint32_t mut_thr = (uint32_t)floor(g->mutation_p * 16777216.0 + 0.5);
  const uint32_t cross_thr = (uint32_t)floor(g->crossover_p * 16777216.0 + 0.5);
  /* initial population: uniform over Lambda, repaired */
  for (int32_t c = 0; c < g->pop; ++c) {
    int32_t *o = pop + (int64_t)c * n;
    for (int32_t i = 0; i < n; ++i)
      o[i] = unif_int(orc_rng(seed, 0, (uint32_t)c, GA_INIT, (uint32_t)i), (uint32_t)p->n_options[i]);
    fit[c] = fc_fitness(p, u, ok, o);
    if (g->repair) fit[c] = fc_repair(p, u, ok, seed, 0, (uint32_t)c, o, fit[c]);
  }
  for (int32_t gen = 0; gen + 1 < g->gens; ++gen) {
    const uint32_t G = (uint32_t)gen + 1u;
    int32_t first = 0;
    if (g->elitism) {
      int32_t e = 0;
      for (int32_t c = 1; c < g->pop; ++c)
        if (fit[c] > fit[e]) e = c;
      memcpy(next, pop + (int64_t)e * n, sizeof(int32_t) * (size_t)n);
      nfit[0] = fit[e];
      first = 1;
    }
    for (int32_t c = first; c < g->pop; ++c) {
      const orc_ga_params tg = {g->pop, g->gens, g->tournament, g->mutation_p, g->elitism};
      const int32_t a = tournament(&tg, fit, seed, G, (uint32_t)c, GA_TOUR_A);
      const int32_t b = tournament(&tg, fit, seed, G, (uint32_t)c, GA_TOUR_B);
      /* crossover with probability crossover_p, else a copy of the first parent */
      const int32_t cross = (uint32_t)(orc_rng(seed, G, (uint32_t)c, GA_CROSS_DO, 0) >> 40) < cross_thr;
      int32_t *o = next + (int64_t)c * n;
      for (int32_t i = 0; i < n; ++i) {
        const uint64_t rc = orc_rng(seed, G, (uint32_t)c, GA_CROSS, (uint32_t)i);
        int32_t gene = (cross && (rc >> 63)) ? pop[(int64_t)b * n + i] : pop[(int64_t)a * n + i];
        const uint64_t rm = orc_rng(seed, G, (uint32_t)c, GA_MUT, (uint32_t)i);
        if ((uint32_t)(rm >> 40) < mut_thr)
          gene = unif_int(orc_rng(seed, G, (uint32_t)c, GA_MUTVAL, (uint32_t)i), (uint32_t)p->n_options[i]);
        o[i] = gene;
      }
      nfit[c] = fc_fitness(p, u, ok, o);
      if (g->repair) nfit[c] = fc_repair(p, u, ok, seed, G, (uint32_t)c, o, nfit[c]);
    }
    memcpy(pop, next, sizeof(int32_t) * (size_t)g->pop * n);
    memcpy(fit, nfit, sizeof(double) * (size_t)g->pop);
  }
  int32_t e = 0;
  for (int32_t c = 1; c < g->pop; ++c)
    if (fit[c] > fit[e]) e = c;
  memcpy(best_genome, pop + (int64_t)e * n, sizeof(int32_t) * (size_t)n);
  const double J = fit[e];
  free(fhat); free(f); free(u); free(ok); free(pop); free(next); free(fit); free(nfit);
  return J;
}
