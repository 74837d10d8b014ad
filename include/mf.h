/*
 * mf.h -- C ABI of the GB300 MeanField joint-configuration scorer.
 *
 * The library scores joint co-location configurations of N models that share
 * one GPU, following arXiv 2609.02109:
 *   - the joint space Lambda = prod_i Lambda_i of per-model option sets (Sec. II, Eq. 1),
 *     enumerated as a mixed-radix index, last model fastest;
 *   - the aggregate GPU state of a candidate (summed SM share, VRAM and bandwidth
 *     demand of the chosen options, plus N) (Eq. 2, in the coupled reading where the
 *     aggregate is formed from the candidate's own demands);
 *   - one MeanField predictor per model, (thr_i, lat_i) = g_i(local_i, aggregate)
 *     (Sec. III-B, Eq. 6): an MLP Linear-ReLU-[Linear-ReLU]-Linear with an optional
 *     sigmoid on the two outputs;
 *   - the hard constraints sum_i VRAM_i <= R and lat_i <= SLA_i (Eq. 4), infeasible
 *     candidates scoring -inf (Sec. II);
 *   - the objective J = sum_i w_i thr_i (the throughput-weighted term of Eq. 3), or,
 *     with MF_OBJ_SOFT_LAT, J = sum_i w_i thr_i - lambda sum_i max(0, lat_i - SLA_i)
 *     with only the VRAM constraint hard;
 *   - exhaustive argmax / top-k / feasible count over Lambda (Sec. II, Sec. IV-C), and
 *     the GA scheduler's per-generation fitness batch and operators (Sec. IV-C).
 *
 * Conventions for every call:
 *   - Functions return an mf_status and never abort or throw.  mf_last_error()
 *     returns a human-readable detail string for the calling thread's last failure.
 *   - "d_" pointers are device pointers owned by the caller; they must stay valid
 *     until the work on `stream` completes.  `stream` is a cudaStream_t (NULL =
 *     the legacy default stream).  Host pointers are caller-owned too.
 *   - A context is thread-compatible: calls on one context must not run
 *     concurrently from several host threads.  Different contexts are independent.
 *   - Indices are uint64; digits/genes are int32 with 0 <= o_i < K_i.
 *   - The total order of results is (J descending, index ascending).  Infeasible
 *     candidates have J = -INFINITY and never enter a top-k.  Unfilled top-k slots
 *     are (UINT64_MAX, -INFINITY).  No feasible candidate is not an error.
 *   - A candidate whose J is NaN counts as infeasible.
 */
#ifndef MF_H
#define MF_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MF_OK = 0,
  MF_EINVAL = 1,        /* invalid argument (see each call) */
  MF_ENOMEM = 2,        /* device or host allocation failed */
  MF_ECUDA = 3,         /* a CUDA runtime call failed; see mf_last_error() */
  MF_EUNSUPPORTED = 4,  /* valid but unsupported shape/precision combination */
  MF_ETIMEOUT = 5,      /* a bounded device-side wait gave up */
  MF_EDEVICE = 6        /* the device reported an invalid input (e.g. an index >= |Lambda|) */
} mf_status;

/* MF_FP32: fp32 results (scores within 1e-5 of the fp64 definition).  For the
 * d_L 8, 12 -> 64 -> 64 -> 2 predictor shape (up to 8 models) the scoring runs on the
 * tensor cores with every operand split into two tf32 parts (hi.hi + hi.lo + lo.hi,
 * about 22 bits per product, fp32 accumulation); other shapes run on the CUDA cores.
 * MF_FP32_SIMT: the same results on the CUDA cores for every shape.
 * MF_BF16: bf16 tensor-core scoring, search results re-scored in fp32. */
typedef enum { MF_FP32 = 0, MF_BF16 = 1, MF_FP32_SIMT = 2 } mf_precision;
/* MF_OBJ_UTILITY (Eq. 3 utility with floors) is set with mf_set_utility only. */
typedef enum { MF_OBJ_WEIGHTED_THR = 0, MF_OBJ_SOFT_LAT = 1, MF_OBJ_UTILITY = 2 } mf_objective;
typedef enum { MF_ACT_IDENTITY = 0, MF_ACT_SIGMOID = 1 } mf_out_act;

#define MF_MAX_MODELS 16
#define MF_MAX_OPTIONS 255
#define MF_MAX_D_LOCAL 28
#define MF_MAX_HIDDEN 256
#define MF_MAX_TOPK 1024

typedef struct mf_ctx mf_ctx;

/* Problem description (Sec. II and Sec. III-B).  All arrays are host memory and
 * are deep-copied by mf_create; the caller may free them afterwards. */
typedef struct {
  int32_t n_models;            /* N, 1..MF_MAX_MODELS */
  const int32_t *n_options;    /* [N] K_i = |Lambda_i|, each 1..MF_MAX_OPTIONS */
  int32_t d_local;             /* d_L, 1..MF_MAX_D_LOCAL; predictor input d_in = d_L + 4 */
  int32_t hidden1;             /* first hidden width, 1..MF_MAX_HIDDEN */
  int32_t hidden2;             /* second hidden width, 0 (one hidden layer) or 1..MF_MAX_HIDDEN */
  const float *local_feats;    /* [sum K_i][d_L] row-major, model-major option rows */
  const float *demand;         /* [sum K_i][3]: SM share, VRAM GB, bandwidth GB/s */
  const float *weights;        /* per model, PyTorch Linear layout (weight[out][in]):
                                  W1[h1][d_in], b1[h1], (W2[h2][h1], b2[h2]), W3[2][h], b3[2];
                                  output 0 = throughput, output 1 = latency */
  const float *agg_scale;      /* [4] multipliers of (sum SM, sum VRAM, sum BW, N) before the
                                  predictor; NULL = (1/(0.6N), 1/(20N), 1/(1500N), 1/8) */
  const float *sla;            /* [N] latency ceilings SLA_i */
  const float *obj_w;          /* [N] objective weights w_i */
  float vram_cap;              /* R, GB; feasibility needs sum VRAM <= R */
  float soft_penalty;          /* lambda of MF_OBJ_SOFT_LAT (ignored otherwise) */
  int32_t out_act;             /* mf_out_act */
  int32_t objective;           /* mf_objective */
  int32_t precision;           /* mf_precision of the scoring kernels */
  int32_t device;              /* CUDA device ordinal, or -1 for the current device */
} mf_problem;

/* Result of an exhaustive search.  topk_idx/topk_score are caller-owned host
 * arrays of k entries (either may be NULL). */
typedef struct {
  uint64_t best_idx;           /* UINT64_MAX if no feasible candidate */
  float best_score;            /* -INFINITY if no feasible candidate */
  uint64_t feasible_count;
  int32_t k;
  uint64_t *topk_idx;
  float *topk_score;
} mf_result;

/* GA parameters (Sec. IV-C): population, generations, tournament size, per-gene
 * mutation probability, elitism (0 or 1).  Crossover is uniform. */
typedef struct {
  int32_t pop;                 /* 2..65536 */
  int32_t gens;                /* >= 1 fitness evaluations */
  int32_t tournament;          /* 1..256 */
  double mutation_p;           /* [0, 1] */
  int32_t elitism;             /* 0 or 1 */
} mf_ga_params;

/* Instrumentation of the last calls on a context (host-side bookkeeping plus
 * CUDA events recorded on the call's stream; no extra synchronisation). */
typedef struct {
  uint64_t h2d_bytes_create;   /* bytes mf_create copied host -> device */
  uint64_t d2h_bytes_last;     /* bytes the last synchronous call copied device -> host */
  int32_t kernel_launches_last;/* library kernels launched by the last search / GA run */
  int32_t score_launches_last; /* of which scoring launches (one per chunk) */
  float score_ms_last;         /* device time from the first to the end of the last scoring
                                  launch of the last search */
  float total_ms_last;         /* device time of the whole last search (scoring, merge,
                                  re-scoring, result copy) */
  int32_t scoring_path;        /* the context's scoring kernels: 0 fp32 on the CUDA cores,
                                  1 bf16 tensor cores, 2 fp32 tensor cores (3-term tf32) */
} mf_stats;

/* Name of a status code (static string). */
const char *mf_status_string(mf_status s);

/* Detail of the calling thread's last failing call ("" if none). */
const char *mf_last_error(void);

/* Validate `p` (Sec. II problem statement), copy it to the device and prepare
 * the kernels.  MF_EINVAL: N, K_i, d_L or widths out of range, NULL arrays, or
 * prod K_i overflowing uint64.  MF_EUNSUPPORTED: MF_BF16 with a shape the
 * tensor-core kernel does not cover.  On success *out owns device memory until
 * mf_destroy. */
mf_status mf_create(const mf_problem *p, mf_ctx **out);

/* Release the context and its device memory (synchronises the device first).
 * NULL is accepted. */
mf_status mf_destroy(mf_ctx *ctx);

/* |Lambda| = prod_i K_i (Eq. 1). */
mf_status mf_space_size(const mf_ctx *ctx, uint64_t *out);

/* Replace SLA_i and w_i (a new scheduling scenario); NULL keeps the old array.
 * Takes effect for calls issued afterwards. */
mf_status mf_set_objective(mf_ctx *ctx, const float *sla, const float *obj_w);

/* Score n candidates given by index (Eqs. 1-6 and the constraints of Eq. 4).
 *   d_idx      [n] uint64 indices into Lambda
 *   d_score    [n] J (or -INFINITY when infeasible)
 *   d_feasible [n] 1 feasible / 0 not (may be NULL)
 *   d_pred     [n][N][2] (thr_i, lat_i) per model (may be NULL)
 * Asynchronous on `stream`.  An index >= |Lambda| scores -INFINITY, infeasible,
 * and raises the context's device status, read by mf_check_device_status. */
mf_status mf_score_batch(mf_ctx *ctx, const uint64_t *d_idx, uint64_t n, float *d_score,
                         uint8_t *d_feasible, float *d_pred, void *stream);

/* Exhaustive surrogate search over [lo, hi) of Lambda (the argmax of Sec. II,
 * extended to top-k and the feasible count), processed in launches of `chunk`
 * candidates (0 = the library's default) while the running top-k and count are
 * carried across launches.  k in 1..MF_MAX_TOPK.  Synchronous: returns after
 * `out` is filled.  The BF16 precision keeps a shortlist of max(8k, 256)
 * candidates by tensor-core score and re-scores it in fp32, so reported scores
 * and the top-k order are the fp32 ones; its feasible count is taken at bf16
 * precision. */
mf_status mf_search_range(mf_ctx *ctx, uint64_t lo, uint64_t hi, int32_t k, uint64_t chunk,
                          mf_result *out, void *stream);

/* mf_search_range over the whole space [0, |Lambda|). */
mf_status mf_search_exhaustive(mf_ctx *ctx, int32_t k, uint64_t chunk, mf_result *out,
                               void *stream);

/* GA fitness batch (Sec. IV-C): d_pop [P][N] int32 genes -> d_fitness [P] (J or
 * -INFINITY).  Asynchronous.  A gene outside [0, K_i) gives -INFINITY and raises
 * the device status. */
mf_status mf_ga_generation(mf_ctx *ctx, const int32_t *d_pop, int32_t P, float *d_fitness,
                           void *stream);

/* Initial population: gene i of slot c is uniform on [0, K_i) from the
 * counter-based generator (seed, generation 0, c, purpose 0, i).  Asynchronous. */
mf_status mf_ga_init(mf_ctx *ctx, const mf_ga_params *g, uint64_t seed, int32_t *d_pop,
                     void *stream);

/* One GA generation (Sec. IV-C operators): from population `gen` and its
 * fitness to population gen + 1.  Slot 0 keeps the fittest individual (lowest
 * slot among equals) when elitism is on; every other slot draws two parents by
 * tournament (draws with replacement, best fitness, lowest slot among equals),
 * takes each gene from either parent with probability 1/2, and redraws a gene
 * uniformly with probability mutation_p.  All draws are SplitMix64 outputs at
 * counter (gen + 1) << 32 | slot << 12 | purpose << 8 | j of the stream `seed`.
 * Asynchronous.  d_next must not alias d_pop. */
mf_status mf_ga_step(mf_ctx *ctx, const mf_ga_params *g, uint64_t seed, int32_t gen,
                     const int32_t *d_pop, const float *d_fitness, int32_t *d_next,
                     void *stream);

/* A complete GA decision: init, then g->gens fitness batches with a generation
 * step between consecutive ones; returns the fittest individual of the last
 * population (lowest slot among equals) in best_genome[N] (host) and its
 * fitness.  Synchronous.  The operators and random draws are those of
 * mf_ga_init / mf_ga_step.  For fp32 predictors with d_L = 8, h1 = h2 = 64,
 * N <= 8 and pop <= 8 x the SM count, the whole decision runs as one
 * cooperative kernel (mf_stats.kernel_launches_last = 1); otherwise as one CUDA
 * graph of init, fitness and step kernels.  MF_ETIMEOUT if the cooperative
 * kernel's grid barrier gave up waiting (the result is then not valid). */
mf_status mf_ga_run(mf_ctx *ctx, const mf_ga_params *g, uint64_t seed, int32_t *best_genome,
                    float *best_fitness, void *stream);

/* ---------------------------------------------------------------------------
 * Fixed-context mode (Sec. III-B): the observed GPU state s_t is held fixed during
 * the search, so predictor i sees its own option and the observed state only, and
 * the utility of Eq. 3 separates into one term per model:
 *   J = sum_i [omega_i f_i Q_i - alpha eta_i c_i - beta max(0, tau_i + delta - f_i)^2]
 * with f_i = (fhat_i - f_min) / (f_max - f_min) the per-variant min-max normalised
 * predicted throughput (fhat_i: the predictor's throughput output) and eta_i = 1 when
 * option i's variant differs from the variant in use.  Constraints (Eq. 4): the
 * summed VRAM of the chosen options <= vram_cap and f_i >= tau_i for every model;
 * otherwise J = -inf.
 * ------------------------------------------------------------------------- */
typedef struct {
  const float *obs;            /* [4] observed state in the aggregate's raw units
                                  (Sigma SM share, Sigma VRAM GB, Sigma BW GB/s, N);
                                  fed to the predictors scaled by agg_scale */
  const int32_t *variant;      /* [sum K_i] variant of each option (>= 0), model-major */
  const float *quality;        /* [sum K_i] Q of the option's variant */
  const float *f_min;          /* [sum K_i] throughput extrema of the option's variant, */
  const float *f_max;          /*           f_max > f_min */
  const float *omega;          /* [N] priority weights */
  const float *tau;            /* [N] floors on the normalised throughput */
  const float *reload_cost;    /* [N] c_i^rel */
  const int32_t *prev_variant; /* [N] variant in use, -1 for none (eta_i = 0) */
  float alpha, beta, delta;    /* paper: 1/60, 5.0, 0.05 */
} mf_fc_params;

/* Evaluate the sum K_i local predictions under p->obs with the fp32 predictor and
 * build the per-option table (fhat, f, floor flag, utility term) on the device; the
 * context keeps it for mf_fc_search until the next call.  Host arrays, copied.
 * Synchronous on `stream`.  MF_EINVAL: NULL arrays, f_max <= f_min, variant < 0,
 * prev_variant < -1, non-finite constants. */
mf_status mf_fc_set(mf_ctx *ctx, const mf_fc_params *p, void *stream);

/* Copy the table of the last mf_fc_set into caller-owned device arrays of sum K_i
 * entries (model-major; any may be NULL): fhat, f, u (the option's term of J), ok
 * (1: f >= tau_i).  Asynchronous on `stream`.  MF_EINVAL before mf_fc_set. */
mf_status mf_fc_table(mf_ctx *ctx, float *d_fhat, float *d_f, float *d_u, uint8_t *d_ok, void *stream);

/* Fixed-context exhaustive search over [lo, hi): J(lambda) = sum of the options'
 * terms (fp32, model order), the same result contract as mf_search_range (top-k by
 * J desc then index asc, feasible count, empty slots (UINT64_MAX, -inf)).  An
 * ALU-bound table-lookup scan.  MF_EINVAL before mf_fc_set. */
mf_status mf_fc_search(mf_ctx *ctx, uint64_t lo, uint64_t hi, int32_t k, uint64_t chunk, mf_result *out,
                       void *stream);

/* The paper's GA (Sec. IV-C) on the fixed-context landscape of the last mf_fc_set:
 * tournament selection, uniform crossover applied with probability crossover_p (else
 * a copy of the first parent), per-gene mutation, elitism, and repair of an
 * infeasible individual (J = -inf) by a feasible one drawn by rejection from the
 * uniform distribution over Lambda (at most floor(256 / N) attempts; the initial
 * uniform population is repaired the same way).  Fitness is the table sum of
 * mf_fc_search (fp32).  Random draws: the counter-based generator of mf_ga_step
 * plus purposes 6 (crossover coin) and 7 (repair, j = attempt * N + gene).
 * Result (host): the fittest individual of the last population, lowest slot among
 * equals; best_genome has N entries.  Synchronous.  One CTA: pop <= 1024.
 * MF_EINVAL: NULL arguments, called before mf_fc_set, a parameter out of its range. */
typedef struct {
  int32_t pop;                 /* 2..1024 */
  int32_t gens;                /* >= 1 fitness evaluations */
  int32_t tournament;          /* 1..256 */
  double crossover_p;          /* [0, 1]; paper 0.7 */
  double mutation_p;           /* [0, 1]; paper 0.1 */
  int32_t elitism;             /* 0 or 1 */
  int32_t repair;              /* 0 or 1 */
} mf_fc_ga_params;

mf_status mf_fc_ga_run(mf_ctx *ctx, const mf_fc_ga_params *g, uint64_t seed, int32_t *best_genome,
                       float *best_fitness, void *stream);

/* Lambda without its VRAM-infeasible configurations (Eq. 4 applied when Lambda is
 * built): writes the ascending indices of [lo, hi) whose summed VRAM <= vram_cap to
 * d_out (device, capacity cap; indices beyond cap are counted, not written) and
 * their number to *count (host).  Synchronous. */
mf_status mf_vram_feasible(mf_ctx *ctx, uint64_t lo, uint64_t hi, uint64_t *d_out, uint64_t cap,
                           uint64_t *count, void *stream);

/* Score with the Eq. 3 utility on the coupled aggregate: predictor i sees the
 * candidate's own summed demands (as every other call of this library) and its
 * throughput output fhat_i enters J = sum_i [omega_i f_i Q_i - alpha eta_i c_i -
 * beta max(0, tau_i + delta - f_i)^2], f_i = (fhat_i - f_min) / (f_max - f_min) of
 * the option's variant; a candidate is feasible iff its summed VRAM <= vram_cap and
 * f_i >= tau_i for every model (the latency outputs and SLA ceilings are not used).
 * Applies to mf_score_batch, mf_search_range / mf_search_exhaustive (fp32 and bf16),
 * mf_ga_generation and mf_ga_run until mf_set_utility(ctx, NULL) restores the
 * problem's own objective.  p->obs is not used.  MF_EINVAL as mf_fc_set. */
mf_status mf_set_utility(mf_ctx *ctx, const mf_fc_params *p);

/* Read the context's instrumentation (see mf_stats). */
mf_status mf_get_stats(const mf_ctx *ctx, mf_stats *out);

/* Exhaustive search without any device allocation.
 *
 * The paper has no counterpart to this call; it exists for callers that cannot
 * call cudaMalloc -- for example a serving process whose memory pool has already
 * claimed the device's memory, or a per-decision control loop that must not pay
 * cudaMalloc's implicit device synchronisation.  It runs the exact fp32 search of
 * mf_search_exhaustive on the problem `p` (host arrays, as for mf_create;
 * precision must be MF_FP32) and fills `out` (host memory) the same way, without
 * creating a context.  All device memory it uses -- a copy of the problem's
 * tables and weights, the per-CTA running top-k lists, the merge buffers, the
 * feasible counter and the status word -- lives in one fixed array of
 * MF_NOALLOC_SCRATCH_BYTES that the library declares in device memory; every GPU
 * that loads the library holds that array until the process exits.  The call
 * allocates nothing (no cudaMalloc, cudaFree or other allocating routine).
 *
 * Limits (MF_EINVAL with a message beyond them): k <= MF_NOALLOC_MAX_TOPK, packed
 * predictor weights <= MF_NOALLOC_MAX_WEIGHT_BYTES, and the whole layout within
 * MF_NOALLOC_SCRATCH_BYTES.  At most MF_NOALLOC_MAX_CTAS CTAs are launched.
 *
 * The first call on a device looks up the array's device address (once per
 * device, with that device current), and that lookup is what makes the runtime
 * load the library's module and reserve the array on the device: a caller whose
 * memory pool will claim the device's memory makes the first call before the pool
 * does, and before any stream capture.  A cudaDeviceReset releases the array but
 * not the cached address, so after resetting a device do not call this entry point
 * on it again.  A call that fails after it has queued work waits for that work
 * before returning.  Every call on a device shares the one array and overwrites it
 * (what must start at zero is cleared at the start of each call), so calls
 * that overlap on the GPU -- from several host threads or streams -- race and
 * must be serialised by the caller.  Synchronous: returns after `out` is filled. */
#define MF_NOALLOC_SCRATCH_BYTES (4u << 20)
#define MF_NOALLOC_MAX_TOPK 64
#define MF_NOALLOC_MAX_CTAS 256
#define MF_NOALLOC_MAX_WEIGHT_BYTES (1u << 20)
mf_status mf_search_exhaustive_noalloc(const mf_problem *p, int32_t k, uint64_t chunk,
                                       mf_result *out, void *stream);

/* Synchronise `stream`, then return MF_EDEVICE if any asynchronous call since the
 * last check saw an invalid index or gene (and clear that flag), else MF_OK. */
mf_status mf_check_device_status(mf_ctx *ctx, void *stream);

/* For tests of the failure path of the bounded device waits; the paper has no
 * counterpart.  With polls > 0, every later launch on `ctx` of a kernel that waits
 * on the device (the tensor-core scorer behind mf_search_* / mf_score_batch in
 * MF_BF16, and the single-kernel GA of mf_ga_run) first waits on a flag that
 * nothing sets, giving up after `polls` polls (about a millisecond each in the
 * scorer, a few nanoseconds in the GA kernel).  The kernel then flags the context's
 * device status and runs to its end without waiting again, except for its own
 * MMAs and weight copies in flight, which it always drains before it frees its
 * tensor memory; the call returns MF_ETIMEOUT and its results are undefined.  The
 * context stays usable: polls = 0 restores normal operation.  MF_EINVAL: ctx NULL. */
mf_status mf_debug_wait_test(mf_ctx *ctx, uint32_t polls);

#ifdef __cplusplus
}
#endif
#endif /* MF_H */
