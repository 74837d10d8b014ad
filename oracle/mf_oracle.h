/*
 * CPU oracle of the MeanField joint-configuration scorer -- TEST INFRASTRUCTURE.
 *
 * Only the tests, the smoke check and the CPU-baseline leg of the benchmark
 * use this library.  It shares no code, header or table with the CUDA path.
 * Arithmetic is fp64 on the float32 inputs; every step is written the way the
 * paper states it, without blocking, fusion or reordering.
 *
 * Parity status per function (pins live in tests/test_oracle_*.py):
 *   orc_space_size, orc_decode        pinned (Eq. 1 sizes, numpy.unravel_index)
 *   orc_pred_scale_list               pinned (equals |output| in the linear case)
 *   orc_score_digits                  pinned (hand example, linear case,
 *                                     aggregate invariant, separable closed form,
 *                                     sigmoid closed form, soft-penalty hand value)
 *   orc_exhaustive                    pinned (brute force, VRAM-only two-pointer
 *                                     count, separable argmax/count, tie order)
 *   orc_rng                           pinned (published SplitMix64 outputs)
 *   orc_ga_init / orc_ga_step         pinned by operator properties (elitism,
 *                                     parent provenance, mutation rate, ranges)
 *   orc_ga_run                        parity unpinned beyond the operator level
 *   orc_fc_local, orc_fc_score_digits,
 *   orc_fc_exhaustive                 pinned (hand example, separable closed form,
 *                                     reload term = alpha c, quadratic margin term,
 *                                     linear case as one matrix product)
 *   orc_vram_feasible                 pinned (two-pointer count, brute-force list)
 *   orc_fc_ga_run                     pinned by properties (near-optimal decisions on the
 *                                     paper-scale space, repair reaches feasibility,
 *                                     seeding); the trajectory itself is parity unpinned
 *   orc_util_*                        pinned (hand example, equal to the fixed-context
 *                                     utility when the aggregate is unused, reduces to
 *                                     the weighted-throughput objective)
 */
#ifndef MF_ORACLE_H
#define MF_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
  int32_t n_models;          /* N */
  const int32_t *n_options;  /* [N] K_i */
  int32_t d_local;           /* d_L */
  int32_t hidden1, hidden2;  /* hidden2 == 0: one hidden layer */
  const float *local_feats;  /* [sum K_i][d_L], model-major */
  const float *demand;       /* [sum K_i][3]: SM share, VRAM GB, BW GB/s */
  const float *weights;      /* per model: W1[h1][d_in], b1, (W2[h2][h1], b2), W3[2][h], b3 */
  const float *agg_scale;    /* [4] or NULL for the default (1/(0.6N), 1/(20N), 1/(1500N), 1/8) */
  const float *sla;          /* [N] latency ceilings */
  const float *obj_w;        /* [N] objective weights */
  float vram_cap;
  float soft_penalty;
  int32_t out_act;           /* 0 identity, 1 sigmoid */
  int32_t objective;         /* 0 weighted throughput + hard SLA, 1 soft latency penalty */
} orc_problem;

/* Number of joint configurations prod K_i (Eq. 1); 0 if it overflows 64 bits. */
uint64_t orc_space_size(const orc_problem *p);

/* Mixed-radix decode of idx into digits o[N], last model fastest (C order). */
void orc_decode(const orc_problem *p, uint64_t idx, int32_t *o);

/* Score one joint configuration given its digits.  Returns J (-inf when
 * infeasible).  Optional outputs: *feasible, pred[N][2] = (thr_i, lat_i),
 * agg[4] = raw aggregate (Sigma SM, Sigma VRAM, Sigma BW, N). */
double orc_score_digits(const orc_problem *p, const int32_t *o, int32_t *feasible,
                        double *pred, double *agg);

/* Score a list of indices (out-of-range indices give -inf, infeasible). */
void orc_score_list(const orc_problem *p, const uint64_t *idx, uint64_t n,
                    double *score, int32_t *feasible, double *pred, double *agg,
                    int32_t nthreads);

/* Per candidate and model, the condition scale of each predictor output:
 * |b3_o| + sum_k |W3[o][k]| |h_k| with the exact last hidden layer h.
 * scale: [n][N][2]. */
void orc_pred_scale_list(const orc_problem *p, const uint64_t *idx, uint64_t n, double *scale,
                         int32_t nthreads);

/* Exhaustive search over [lo, hi): top-k by (J desc, idx asc) and the feasible
 * count.  Unfilled slots are (UINT64_MAX, -inf). */
void orc_exhaustive(const orc_problem *p, uint64_t lo, uint64_t hi, int32_t k,
                    uint64_t *topk_idx, double *topk_score, uint64_t *count,
                    int32_t nthreads);

/* Output number ctr of the SplitMix64 sequence whose state starts at seed. */
uint64_t orc_splitmix64(uint64_t seed, uint64_t ctr);

/* GA random draw for (seed, generation, slot, purpose, j). */
uint64_t orc_rng(uint64_t seed, uint32_t gen, uint32_t slot, uint32_t purpose, uint32_t j);

typedef struct {
  int32_t pop;
  int32_t gens;
  int32_t tournament;
  double mutation_p;
  int32_t elitism;           /* 0 or 1 */
} orc_ga_params;

void orc_ga_init(const orc_problem *p, const orc_ga_params *g, uint64_t seed, int32_t *pop);
void orc_ga_step(const orc_problem *p, const orc_ga_params *g, uint64_t seed, int32_t gen,
                 const int32_t *pop, const double *fitness, int32_t *next);
/* Full GA: returns best fitness; best_genome[N]. */
double orc_ga_run(const orc_problem *p, const orc_ga_params *g, uint64_t seed,
                  int32_t *best_genome, int32_t nthreads);

/* ---------------------------------------------------------------------------
 * Fixed-context mode (Sec. III-B: the observed state s_t = (rho_t, m_t, u_t) is
 * held fixed during the search) with the utility of Eq. 3 and the constraints of
 * Eq. 4: each predictor sees its own option and the observed aggregate state.
 * ------------------------------------------------------------------------- */
typedef struct {
  const float *obs;            /* [4] observed aggregate state, raw units of the
                                  aggregate (Sigma SM, Sigma VRAM, Sigma BW, N) */
  const int32_t *variant;      /* [sum K_i] variant of each option */
  const float *quality;        /* [sum K_i] Q of the option's variant */
  const float *f_min;          /* [sum K_i] throughput extrema of the option's variant */
  const float *f_max;
  const float *omega;          /* [N] priority weights */
  const float *tau;            /* [N] normalised throughput floors */
  const float *reload_cost;    /* [N] c_i^rel */
  const int32_t *prev_variant; /* [N] variant in use (-1: none) */
  float alpha, beta, delta;
} orc_fc;

/* Per option row r (model-major, as local_feats): raw predicted throughput
 * fhat[r], normalised f[r], floor flag ok[r] = (f >= tau_i) and the option's
 * utility term u[r] = omega_i f Q - alpha eta c_i - beta max(0, tau_i + delta - f)^2. */
void orc_fc_local(const orc_problem *p, const orc_fc *fc, double *fhat, double *f, int32_t *ok,
                  double *u);

/* J(lambda) of Eq. 3 in fixed-context mode (-inf, *feasible = 0, when a floor
 * f_i >= tau_i or the VRAM bound of Eq. 4 fails). */
double orc_fc_score_digits(const orc_problem *p, const orc_fc *fc, const int32_t *o, int32_t *feasible);

/* Exhaustive fixed-context search over [lo, hi): top-k by (J desc, idx asc) and
 * the feasible count; unfilled slots are (UINT64_MAX, -inf). */
void orc_fc_exhaustive(const orc_problem *p, const orc_fc *fc, uint64_t lo, uint64_t hi, int32_t k,
                       uint64_t *topk_idx, double *topk_score, uint64_t *count, int32_t nthreads);

/* ---------------------------------------------------------------------------
 * The Eq. 3 utility on the coupled aggregate: each predictor sees the candidate's
 * own summed demands (as orc_score_digits) and its throughput output enters Eq. 3
 * through the per-option terms of orc_fc (obs is not used).  Constraints: Eq. 4
 * floors f_i >= tau_i and the VRAM bound.
 * ------------------------------------------------------------------------- */
double orc_util_score_digits(const orc_problem *p, const orc_fc *fc, const int32_t *o, int32_t *feasible,
                             double *pred, double *agg);
void orc_util_score_list(const orc_problem *p, const orc_fc *fc, const uint64_t *idx, uint64_t n,
                         double *score, int32_t *feasible, double *pred, double *agg, int32_t nthreads);
void orc_util_exhaustive(const orc_problem *p, const orc_fc *fc, uint64_t lo, uint64_t hi, int32_t k,
                         uint64_t *topk_idx, double *topk_score, uint64_t *count, int32_t nthreads);

/* The paper's GA (Sec. IV-C) on the fixed-context landscape: tournament selection,
 * uniform crossover applied with probability crossover_p (else the first parent is
 * copied), per-gene mutation, elitism, and repair of an infeasible individual
 * (J = -inf) by a randomly sampled feasible one.  Reading: the sample is drawn by
 * rejection from the uniform distribution over Lambda, at most floor(256 / N)
 * attempts (the individual stays infeasible if none succeeds); the initial
 * population is uniform over Lambda and repaired the same way. */
typedef struct {
  int32_t pop;
  int32_t gens;
  int32_t tournament;
  double crossover_p;
  double mutation_p;
  int32_t elitism;          /* 0 or 1 */
  int32_t repair;           /* 0 or 1 */
} orc_fc_ga_params;

/* Returns the best fitness of the last population (lowest slot among equals) and
 * its genome in best_genome[N]. */
double orc_fc_ga_run(const orc_problem *p, const orc_fc *fc, const orc_fc_ga_params *g, uint64_t seed,
                     int32_t *best_genome);

/* The VRAM-feasible joint configurations in [lo, hi) (Lambda with the
 * VRAM-infeasible configurations removed), ascending; writes at most cap of
 * them to out and returns how many there are. */
uint64_t orc_vram_feasible(const orc_problem *p, uint64_t lo, uint64_t hi, uint64_t *out, uint64_t cap);

#ifdef __cplusplus
}
#endif
#endif
