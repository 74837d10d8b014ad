// GA operators of the scheduler (arXiv 2609.02109, Sec. IV-C): initial
// population, elitism, tournament selection, uniform crossover and per-gene
// mutation.  Every random draw is a SplitMix64 output at a counter made of
// (generation, slot, purpose, j), so each child is computed independently by
// one thread and the result does not depend on the launch shape.
#include "mf_internal.cuh"

namespace mf {

struct GaArgs {
  int32_t pop, n, tournament, elitism;
  uint32_t mut_thr;              // mutation when (r >> 40) < mut_thr (24-bit fraction)
  int32_t K[MF_MAX_MODELS];
};

__global__ void k_ga_init(GaArgs g, const uint64_t* __restrict__ seed_ptr, uint64_t seed,
                          int32_t* __restrict__ pop) {
  const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= (int64_t)g.pop * g.n) return;
  const uint64_t sd = seed_ptr ? *seed_ptr : seed;
  const int c = (int)(e / g.n), i = (int)(e % g.n);
  pop[e] = ga_unif(ga_rng(sd, 0, (uint32_t)c, kGaInit, (uint32_t)i), (uint32_t)g.K[i]);
}

__device__ __forceinline__ int tournament(const GaArgs& g, const float* __restrict__ fit, uint64_t seed,
                                          uint32_t gen, uint32_t child, uint32_t purpose) {
  int best = -1;
  float bf = 0.f;
  for (int t = 0; t < g.tournament; ++t) {
    const int s = ga_unif(ga_rng(seed, gen, child, purpose, (uint32_t)t), (uint32_t)g.pop);
    const float f = fit[s];
    if (best < 0 || f > bf || (f == bf && s < best)) { best = s; bf = f; }
  }
  return best;
}

// Population `gen` -> `gen + 1`.  One thread per child slot.
__global__ void __launch_bounds__(256)
k_ga_step(GaArgs g, const uint64_t* __restrict__ seed_ptr, uint64_t seed, int32_t gen,
          const int32_t* __restrict__ pop, const float* __restrict__ fit, int32_t* __restrict__ next) {
  __shared__ float sval[32];
  __shared__ int sidx[32];
  const uint64_t sd = seed_ptr ? *seed_ptr : seed;
  const uint32_t G = (uint32_t)gen + 1u;
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (g.elitism && blockIdx.x == 0) {
    const int e = block_argmax(fit, g.pop, sval, sidx);
    if (threadIdx.x < g.n) next[threadIdx.x] = pop[(size_t)e * g.n + threadIdx.x];
  }
  if (c >= g.pop || (g.elitism && c == 0)) return;
  const int a = tournament(g, fit, sd, G, (uint32_t)c, kGaTourA);
  const int b = tournament(g, fit, sd, G, (uint32_t)c, kGaTourB);
  for (int i = 0; i < g.n; ++i) {
    const uint64_t rc = ga_rng(sd, G, (uint32_t)c, kGaCross, (uint32_t)i);
    int gene = (rc >> 63) ? pop[(size_t)b * g.n + i] : pop[(size_t)a * g.n + i];
    const uint64_t rm = ga_rng(sd, G, (uint32_t)c, kGaMut, (uint32_t)i);
    if ((uint32_t)(rm >> 40) < g.mut_thr)
      gene = ga_unif(ga_rng(sd, G, (uint32_t)c, kGaMutVal, (uint32_t)i), (uint32_t)g.K[i]);
    next[(size_t)c * g.n + i] = gene;
  }
}

// Fittest individual of a population -> out_genome[N], out_fit[0].
__global__ void __launch_bounds__(1024)
k_ga_best(int P, int n, const int32_t* __restrict__ pop, const float* __restrict__ fit,
          int32_t* __restrict__ out_genome, float* __restrict__ out_fit) {
  __shared__ float sval[32];
  __shared__ int sidx[32];
  const int e = block_argmax(fit, P, sval, sidx);
  if (threadIdx.x < n) out_genome[threadIdx.x] = pop[(size_t)e * n + threadIdx.x];
  if (threadIdx.x == 0) *out_fit = fit[e];
}

static GaArgs make_args(const mf_ctx* c, const mf_ga_params* g) {
  GaArgs a{};
  a.pop = g->pop;
  a.n = c->P.n_models;
  a.tournament = g->tournament;
  a.elitism = g->elitism;
  a.mut_thr = (uint32_t)floor(g->mutation_p * 16777216.0 + 0.5);
  for (int i = 0; i < a.n; ++i) a.K[i] = c->P.K[i];
  return a;
}

mf_status ga_init(mf_ctx* c, const mf_ga_params* g, uint64_t seed, int32_t* pop, cudaStream_t s) {
  const GaArgs a = make_args(c, g);
  const int64_t n = (int64_t)a.pop * a.n;
  k_ga_init<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(a, nullptr, seed, pop);
  MF_CUDA(cudaGetLastError());
  return MF_OK;
}

mf_status ga_step(mf_ctx* c, const mf_ga_params* g, uint64_t seed, int32_t gen,
                  const int32_t* pop, const float* fit, int32_t* next, cudaStream_t s) {
  const GaArgs a = make_args(c, g);
  k_ga_step<<<(unsigned)((a.pop + 255) / 256), 256, 0, s>>>(a, nullptr, seed, gen, pop, fit, next);
  MF_CUDA(cudaGetLastError());
  return MF_OK;
}

mf_status ga_best(mf_ctx* c, const int32_t* pop, const float* fit, int P, int32_t* out_genome,
                  float* out_fit, cudaStream_t s) {
  k_ga_best<<<1, 1024, 0, s>>>(P, c->P.n_models, pop, fit, out_genome, out_fit);
  MF_CUDA(cudaGetLastError());
  return MF_OK;
}

}  // namespace mf

namespace mf {

// Whole GA decision (init, gens fitness batches, gens - 1 steps, best) captured
// once into a CUDA graph per (GA parameters, objective version); the seed is read
// from device memory so one graph serves every seed.
mf_status ga_run_graph(mf_ctx* c, const mf_ga_params* g, uint64_t seed, cudaStream_t s) {
  const int N = c->P.n_models;
  const int P = g->pop;
  if (P > c->ga_cap) {
    MF_CUDA(cudaStreamSynchronize(s));
    cudaFree(c->d_pop[0]); cudaFree(c->d_pop[1]); cudaFree(c->d_fit); cudaFree(c->d_pred);
    c->d_pop[0] = c->d_pop[1] = nullptr; c->d_fit = c->d_pred = nullptr;
    c->ga_cap = 0;
    MF_CUDA(cudaMalloc(&c->d_pop[0], sizeof(int32_t) * (size_t)P * N));
    MF_CUDA(cudaMalloc(&c->d_pop[1], sizeof(int32_t) * (size_t)P * N));
    MF_CUDA(cudaMalloc(&c->d_fit, sizeof(float) * (size_t)P));
    MF_CUDA(cudaMalloc(&c->d_pred, sizeof(float) * 2 * (size_t)P * N));
    c->ga_cap = P;
    if (c->ga_exec) { cudaGraphExecDestroy(c->ga_exec); c->ga_exec = nullptr; }
  }
  if (!c->d_ga_out) MF_CUDA(cudaMalloc(&c->d_ga_out, 128));
  mf_status st = ensure_host_stage(c, 256);
  if (st != MF_OK) return st;
  if (!c->cap_stream) MF_CUDA(cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking));

  const bool same = c->ga_exec && c->ga_version == c->params_version && c->ga_key.pop == g->pop &&
                    c->ga_key.gens == g->gens && c->ga_key.tournament == g->tournament &&
                    c->ga_key.mutation_p == g->mutation_p && c->ga_key.elitism == g->elitism;
  int32_t* out_genome = (int32_t*)c->d_ga_out;
  float* out_fit = (float*)(out_genome + N);
  uint64_t* d_seed = (uint64_t*)((char*)c->d_ga_out + 64);
  if (!same) {
    if (c->ga_exec) { cudaGraphExecDestroy(c->ga_exec); c->ga_exec = nullptr; }
    const GaArgs a = make_args(c, g);
    cudaStream_t cs = c->cap_stream;
    MF_CUDA(cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal));
    const int64_t ne = (int64_t)P * N;
    k_ga_init<<<(unsigned)((ne + 255) / 256), 256, 0, cs>>>(a, d_seed, 0, c->d_pop[0]);
    int cur = 0;
    mf_status cap = MF_OK;
    for (int gen = 0; gen < g->gens && cap == MF_OK; ++gen) {
      cap = f32_score_list(c, nullptr, c->d_pop[cur], (uint64_t)P, c->d_fit, nullptr, c->d_pred, cs);
      if (cap != MF_OK) break;
      if (gen + 1 < g->gens) {
        k_ga_step<<<(unsigned)((P + 255) / 256), 256, 0, cs>>>(a, d_seed, 0, gen, c->d_pop[cur], c->d_fit,
                                                               c->d_pop[cur ^ 1]);
        cur ^= 1;
      }
    }
    if (cap == MF_OK) k_ga_best<<<1, 1024, 0, cs>>>(P, N, c->d_pop[cur], c->d_fit, out_genome, out_fit);
    cudaGraph_t graph = nullptr;
    cudaError_t e = cudaStreamEndCapture(cs, &graph);
    if (cap != MF_OK) { if (graph) cudaGraphDestroy(graph); return cap; }
    if (e != cudaSuccess) { if (graph) cudaGraphDestroy(graph); return cuda_fail(e, "cudaStreamEndCapture"); }
    e = cudaGraphInstantiate(&c->ga_exec, graph, 0);
    cudaGraphDestroy(graph);
    if (e != cudaSuccess) { c->ga_exec = nullptr; return cuda_fail(e, "cudaGraphInstantiate"); }
    c->ga_key = *g;
    c->ga_version = c->params_version;
  }
  uint64_t* h_seed = (uint64_t*)((char*)c->h_stage + 128);
  *h_seed = seed;
  MF_CUDA(cudaMemcpyAsync(d_seed, h_seed, sizeof(uint64_t), cudaMemcpyHostToDevice, s));
  MF_CUDA(cudaGraphLaunch(c->ga_exec, s));
  return MF_OK;
}

}  // namespace mf

// ---------------------------------------------------------------------------
// Whole GA decision in one cooperative kernel (fp32 predictors d_L 8, 64-64).
//
// CTA b owns the slice [8b, 8b + 8) of the population.  Thread (model m, hidden
// unit j) keeps rows j of W1 and W2 in registers for the whole run, so a weight is
// read from memory once per run.  One generation:
//   layer 1    thread (m, j) for the slice's candidates
//   layer 2-3  thread (m, j) for all 8 candidates (each shared-memory load of four
//              layer-1 activations is one broadcast to the warp); layer 3 sums over
//              the warp in butterfly shuffles where each step halves the values a
//              lane carries
//   objective  warp c for candidate c, lane i for model i (Eq. 7-9)
//   step       warp c breeds child 8b + c: lane t holds tournament entry t and
//              fetches its fitness and genome; the winners' genomes come by
//              shuffle; lane i mutates gene i and adds its demand to the child's
//              aggregate state.  The elite (slot 0) is the best of the CTAs' bests.
// There is no grid-wide barrier.  Every value another CTA reads -- an individual's
// fitness, the two halves of its genome (gene i in byte i mod 4), a CTA's best --
// is a 64-bit word whose high half is the tag g + 1 of its generation g, written
// and read as single 64-bit accesses.  A reader spins on exactly the words it
// needs until their tags match, so each generation waits only for the CTAs whose
// individuals its tournaments drew (and CTA 0, for the elite, for every CTA's
// best).  The words live in a ring of R = min(gens + 1, kGaRingMax) generations;
// before a CTA writes generation g + 1 over g + 1 - R it checks that every CTA has
// finished reading that generation (per-CTA progress counters, read ahead of use).
// Every operator and draw is that of k_ga_step, so the run equals init + (fitness,
// step) x gens up to the fp32 rounding of the fitness.  Every spin gives up after
// kGaSpinLimit polls, sets the timeout bit of the status word and ends the CTA.
// ---------------------------------------------------------------------------
namespace mf {

constexpr int kGaMaxSlice = 8;
constexpr int kGaRingMax = 128;                // generations held in the ring (at most)
constexpr uint32_t kGaSpinLimit = 1u << 22;    // polls of about a microsecond: a few seconds

struct __align__(32) GaRec {   // one individual of one generation
  unsigned long long fw;       // tag | fitness bits
  unsigned long long glo;      // tag | genes 0-3
  unsigned long long ghi;      // tag | genes 4-7
  unsigned long long pad;
};

struct __align__(32) GaBest {  // fittest individual of one CTA's slice
  unsigned long long fw;       // tag | fitness bits
  unsigned long long sw;       // tag | slot
  unsigned long long glo, ghi;
};

struct GaPersist {
  GaRec* rec;            // [ring][pop]
  GaBest* best;          // [ring][ctas]
  unsigned int* prog;    // [ctas] generations whose records the CTA has finished reading
  int32_t* out_genome;
  float* out_fit;
  const uint64_t* seed;
  int gens;
  int ring;
};

__device__ __forceinline__ unsigned long long ld_word(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_word(unsigned long long* p, unsigned long long v) {
  asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ unsigned int ld_u32(const unsigned int* p) {
  unsigned int v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_u32(unsigned int* p, unsigned int v) {
  asm volatile("st.relaxed.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ unsigned long long tagged(uint32_t tag, uint32_t payload) {
  return ((unsigned long long)tag << 32) | payload;
}

__device__ __forceinline__ bool has_tag(unsigned long long w, uint32_t tag) {
  return (uint32_t)(w >> 32) == tag;
}

// (fitness, slot) maximum over the warp: higher fitness, then lower slot; slot < 0 is empty.
__device__ __forceinline__ void warp_best(float& f, int& s) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float of = __shfl_xor_sync(0xffffffffu, f, o);
    const int os = __shfl_xor_sync(0xffffffffu, s, o);
    if (os >= 0 && (s < 0 || of > f || (of == f && os < s))) { f = of; s = os; }
  }
}

// One butterfly step that halves the values a lane carries: the two lanes that
// differ in `bit` each keep one half, so afterwards v[i] (i < n) is the pair's sum
// of value i + n * (that lane bit).
template <int n>
__device__ __forceinline__ void fold(float* v, int bit) {
  const bool b = (threadIdx.x >> bit) & 1;
#pragma unroll
  for (int i = 0; i < n; ++i) {
    const float send = b ? v[i] : v[i + n];
    const float keep = b ? v[i + n] : v[i];
    v[i] = keep + __shfl_xor_sync(0xffffffffu, send, 1 << bit);
  }
}

// Spin until the three words of record r carry `tag` (or the poll limit); false on timeout.
__device__ __forceinline__ bool fetch_rec(const GaRec* r, uint32_t tag, float& f, uint32_t& lo, uint32_t& hi) {
  for (uint32_t n = 0; n < kGaSpinLimit; ++n) {
    const unsigned long long a = ld_word(&r->fw), b = ld_word(&r->glo), c = ld_word(&r->ghi);
    if (has_tag(a, tag) && has_tag(b, tag) && has_tag(c, tag)) {
      f = __uint_as_float((uint32_t)a);
      lo = (uint32_t)b;
      hi = (uint32_t)c;
      return true;
    }
  }
  return false;
}

// Fittest of the CTAs' bests of one generation, on every lane of the warp; false on timeout.
__device__ bool best_of_ctas(const GaBest* bst, int n, uint32_t tag, float& f, int& s, uint32_t& lo,
                             uint32_t& hi) {
  const int lane = threadIdx.x & 31;
  f = -INFINITY;
  s = -1;
  lo = hi = 0;
  bool ok = true;
  for (int b = lane; b < n && ok; b += 32) {
    ok = false;
    for (uint32_t it = 0; it < kGaSpinLimit; ++it) {
      const GaBest* r = bst + b;
      const unsigned long long a = ld_word(&r->fw), w = ld_word(&r->sw), x = ld_word(&r->glo),
                               y = ld_word(&r->ghi);
      if (has_tag(a, tag) && has_tag(w, tag) && has_tag(x, tag) && has_tag(y, tag)) {
        const float rf = __uint_as_float((uint32_t)a);
        const int rs = (int)(uint32_t)w;
        if (s < 0 || rf > f || (rf == f && rs < s)) { f = rf; s = rs; lo = (uint32_t)x; hi = (uint32_t)y; }
        ok = true;
        break;
      }
    }
  }
  ok = __all_sync(0xffffffffu, ok);
  const int mine = s;
  warp_best(f, s);
  const unsigned int src = __ffs(__ballot_sync(0xffffffffu, mine == s)) - 1;
  lo = __shfl_sync(0xffffffffu, lo, src);
  hi = __shfl_sync(0xffffffffu, hi, src);
  return ok;
}

// Random numbers of one child that do not depend on fitness (lane = tournament
// entry t for t < 32, lane = gene i for i < N).
struct ChildDraws {
  int ta, tb;      // tournament A / B entry `lane` (-1: none)
  int take_b;      // gene `lane` comes from parent B
  int mutate;      // gene `lane` mutates
  int mval;        // ... to this option
};

__device__ __forceinline__ ChildDraws child_draws(const GaArgs& g, uint64_t sd, uint32_t G, uint32_t c,
                                                  int lane, int N, int myK) {
  ChildDraws d;
  d.ta = d.tb = -1;
  d.take_b = d.mutate = d.mval = 0;
  if (lane < g.tournament) {
    d.ta = ga_unif(ga_rng(sd, G, c, kGaTourA, (uint32_t)lane), (uint32_t)g.pop);
    d.tb = ga_unif(ga_rng(sd, G, c, kGaTourB, (uint32_t)lane), (uint32_t)g.pop);
  }
  if (lane < N) {
    d.take_b = (int)(ga_rng(sd, G, c, kGaCross, (uint32_t)lane) >> 63);
    d.mutate = (uint32_t)(ga_rng(sd, G, c, kGaMut, (uint32_t)lane) >> 40) < g.mut_thr;
    if (d.mutate) d.mval = ga_unif(ga_rng(sd, G, c, kGaMutVal, (uint32_t)lane), (uint32_t)myK);
  }
  return d;
}

// Winner of one tournament and its genome halves.  Lane t < 32 holds entry t (slot s,
// -1 for none) with its fitness and genome; entries 32.. are fetched here.
__device__ __forceinline__ bool tournament_winner(const GaArgs& g, uint64_t sd, uint32_t G, uint32_t c,
                                                  uint32_t purpose, const GaRec* rec, uint32_t tag, int s,
                                                  float f, uint32_t& lo, uint32_t& hi) {
  const int lane = threadIdx.x & 31;
  bool ok = true;
  for (int t = lane + 32; t < g.tournament && ok; t += 32) {  // tournaments larger than a warp
    const int x = ga_unif(ga_rng(sd, G, c, purpose, (uint32_t)t), (uint32_t)g.pop);
    float v;
    uint32_t xl, xh;
    ok = fetch_rec(rec + x, tag, v, xl, xh);
    if (ok && (s < 0 || v > f || (v == f && x < s))) { f = v; s = x; lo = xl; hi = xh; }
  }
  ok = __all_sync(0xffffffffu, ok);
  const int mine = s;
  warp_best(f, s);
  const unsigned int src = __ffs(__ballot_sync(0xffffffffu, mine == s)) - 1;
  lo = __shfl_sync(0xffffffffu, lo, src);
  hi = __shfl_sync(0xffffffffu, hi, src);
  return ok;
}

template <int MAXT>
__global__ void __launch_bounds__(MAXT, 1)
k_ga_persist(const Params P, const GaArgs g, const GaPersist G) {
  constexpr int H = 64, DL = 8, DIN = DL + 4, SM = kGaMaxSlice;
  constexpr int WPM = H / 32;         // warps per model
  extern __shared__ __align__(16) float sm[];
  __shared__ int s_abort;
  __shared__ float s_fit[SM];
  __shared__ uint32_t s_glo[SM], s_ghi[SM];
  const int N = P.n_models;
  const int sumK = pick(P.off, N - 1) + pick(P.K, N - 1);
  const int pop = g.pop;
  // shared memory; every float region is a multiple of 4 floats so the float4 rows align
  float* sh1 = sm;                                           // [N][SM][H] layer-1 activations
  float* spart = sh1 + (size_t)N * SM * H;                   // [WPM][SM][N][2] layer-3 warp sums
  float* sagg = spart + (size_t)WPM * SM * N * 2;            // [SM][4] scaled aggregate, raw VRAM
  float* sx = sagg + 4 * SM;                                 // [sumK][DL] local features
  float4* sdem = reinterpret_cast<float4*>(sx + (size_t)sumK * DL);  // [sumK]
  int32_t* sgenes = reinterpret_cast<int32_t*>(sdem + sumK); // [SM][N] the slice's genomes

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool unit = tid < N * H;
  const int m = unit ? tid / H : 0;
  const int j = tid % H;
  const int wq = j >> 5;              // warp of the model
  // this thread's weights: rows j of W1 and W2, the layer-3 weights of unit j
  float w1[DIN], w2[H];
  float b1 = 0.f, b2 = 0.f, w3t = 0.f, w3l = 0.f;
  int unit_off = 0;
  if (unit) {
    const float* w = P.w32 + (size_t)m * P.per_model;
#pragma unroll
    for (int k = 0; k < DIN; ++k) w1[k] = __ldg(w + j * DIN + k);
    b1 = __ldg(w + H * DIN + j);
    const float* W2 = w + H * DIN + H;
#pragma unroll
    for (int k = 0; k < H; ++k) w2[k] = __ldg(W2 + j * H + k);
    b2 = __ldg(W2 + H * H + j);
    const float* W3 = W2 + H * H + H;
    w3t = __ldg(W3 + j);
    w3l = __ldg(W3 + H + j);
    unit_off = pick(P.off, m);
  }
  // per-lane constants of model `lane`
  float my_w = 0.f, my_sla = 0.f, my_b3t = 0.f, my_b3l = 0.f;
  float my_uomega = 0.f, my_utau = 0.f, my_ucost = 0.f;
  int my_off = 0, my_K = 1, my_uprev = -1;
  if (lane < N) {
    const float* b3 = P.w32 + (size_t)lane * P.per_model + H * DIN + H + H * H + H + 2 * H;
    my_b3t = __ldg(b3);
    my_b3l = __ldg(b3 + 1);
    my_w = pick(P.w, lane);
    my_sla = pick(P.sla, lane);
    my_off = pick(P.off, lane);
    my_K = pick(P.K, lane);
    my_uomega = pick(P.u_omega, lane);
    my_utau = pick(P.u_tau, lane);
    my_ucost = pick(P.u_cost, lane);
    my_uprev = pick(P.u_prev, lane);
  }
  for (int e = tid; e < N * SM * H; e += blockDim.x) sh1[e] = 0.f;
  for (int e = tid; e < sumK * DL; e += blockDim.x) sx[e] = P.x[e];
  for (int e = tid; e < sumK; e += blockDim.x) sdem[e] = P.dem[e];
  if (tid == 0) s_abort = 0;
  __syncthreads();

  if (P.wait_test) {  // the timeout test: a record word that nothing writes, a few polls
    if (tid == 0) {
      bool got = false;
      for (uint32_t n = 0; n < P.wait_test && !got; ++n)
        got = has_tag(ld_word(&G.best[0].fw), 0xFFFFFFFFu);
      if (!got) {
        atomicOr(P.status, kStatusTimeout);
        s_abort = 1;
      }
    }
    __syncthreads();
    if (s_abort) return;
  }
  const uint64_t sd = *G.seed;
  const int c0 = blockIdx.x * SM;
  const int ns = min(SM, pop - c0);
  const float nz = (float)N * P.agg_scale[3];
  const bool child_warp = warp < ns;
  const int last_warp = (int)(blockDim.x >> 5) - 1;  // never a child warp (blockDim > 32 * SM)
  const uint32_t cg = (uint32_t)(c0 + warp);  // the child slot of a child warp
  auto fail = [&]() {
    atomicOr(P.status, kStatusTimeout);
    s_abort = 1;
  };

  // a child's genes are in place (lane i holds gene i): record it (shared memory and
  // the ring slot of its generation, tag `tag`) and its aggregate state
  auto place = [&](int gene, GaRec* ring_slot, uint32_t tag) {
    float a0 = 0.f, a1 = 0.f, a2 = 0.f;
    if (lane < N) {
      sgenes[warp * N + lane] = gene;
      const float4 d = sdem[my_off + gene];
      a0 = d.x; a1 = d.y; a2 = d.z;
    }
    const uint32_t byte = lane < N ? (uint32_t)gene : 0u;
    const uint32_t lo = __reduce_or_sync(0xffffffffu, lane < 4 ? byte << (8 * lane) : 0u);
    const uint32_t hi = __reduce_or_sync(0xffffffffu, lane >= 4 && lane < 8 ? byte << (8 * (lane - 4)) : 0u);
    if (lane == 0) { s_glo[warp] = lo; st_word(&ring_slot[cg].glo, tagged(tag, lo)); }
    if (lane == 1) { s_ghi[warp] = hi; st_word(&ring_slot[cg].ghi, tagged(tag, hi)); }
#pragma unroll
    for (int o = 4; o > 0; o >>= 1) {  // lanes 0-7 hold the models
      a0 += __shfl_xor_sync(0xffffffffu, a0, o);
      a1 += __shfl_xor_sync(0xffffffffu, a1, o);
      a2 += __shfl_xor_sync(0xffffffffu, a2, o);
    }
    if (lane == 0) {
      sagg[4 * warp + 0] = a0 * P.agg_scale[0];
      sagg[4 * warp + 1] = a1 * P.agg_scale[1];
      sagg[4 * warp + 2] = a2 * P.agg_scale[2];
      sagg[4 * warp + 3] = a1;  // raw VRAM sum for the constraint
    }
  };
  if (child_warp) {  // initial population (generation 0, tag 1)
    const int gene = lane < N ? ga_unif(ga_rng(sd, 0, cg, kGaInit, (uint32_t)lane), (uint32_t)my_K) : 0;
    place(gene, G.rec, 1u);
  }
  __syncthreads();

  for (int gen = 0; gen < G.gens; ++gen) {
    const uint32_t tag = (uint32_t)gen + 1u;
    const int slot = gen % G.ring;
    GaRec* rec_cur = G.rec + (size_t)slot * pop;
    GaRec* rec_nxt = G.rec + (size_t)((gen + 1) % G.ring) * pop;
    GaBest* best_cur = G.best + (size_t)slot * gridDim.x;
    const bool last = gen + 1 == G.gens;
    // ---- the step below overwrites generation gen + 1 - ring: read every CTA's
    // progress now, check it after the objective ----
    const int need = gen + 2 - G.ring;
    unsigned int pv[8] = {~0u, ~0u, ~0u, ~0u, ~0u, ~0u, ~0u, ~0u};
    const bool lag_check = warp == last_warp && need > 0 && !last;
    if (lag_check) {
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (lane + 32 * u < (int)gridDim.x) pv[u] = ld_u32(G.prog + lane + 32 * u);
    }
    // ---- layer 1 ----
    if (unit) {
#pragma unroll
      for (int c = 0; c < SM; ++c) {
        if (c < ns) {
          const float4* xr = reinterpret_cast<const float4*>(sx + (size_t)(unit_off + sgenes[c * N + m]) * DL);
          const float4 v0 = xr[0], v1 = xr[1];
          const float4 a = *reinterpret_cast<const float4*>(sagg + 4 * c);
          float u0 = b1, u1 = 0.f;
          u0 = fmaf(w1[0], v0.x, u0); u1 = fmaf(w1[1], v0.y, u1);
          u0 = fmaf(w1[2], v0.z, u0); u1 = fmaf(w1[3], v0.w, u1);
          u0 = fmaf(w1[4], v1.x, u0); u1 = fmaf(w1[5], v1.y, u1);
          u0 = fmaf(w1[6], v1.z, u0); u1 = fmaf(w1[7], v1.w, u1);
          u0 = fmaf(w1[8], a.x, u0); u1 = fmaf(w1[9], a.y, u1);
          u0 = fmaf(w1[10], a.z, u0); u1 = fmaf(w1[11], nz, u1);
          sh1[((size_t)m * SM + c) * H + j] = relu(u0 + u1);
        }
      }
    }
    __syncthreads();
    if (s_abort) return;
    // ---- layers 2 and 3 (rows past the slice's end hold zeros) ----
    if (unit) {
      const float* h1 = sh1 + (size_t)m * SM * H;
      // even and odd k accumulate apart, two fused multiply-adds per instruction
      float2 acc2[SM];
#pragma unroll
      for (int c = 0; c < SM; ++c) acc2[c] = make_float2(b2, 0.f);
#pragma unroll
      for (int p = 0; p < H / 4; ++p) {
        const float2 wa = make_float2(w2[4 * p + 0], w2[4 * p + 1]);
        const float2 wb = make_float2(w2[4 * p + 2], w2[4 * p + 3]);
#pragma unroll
        for (int c = 0; c < SM; ++c) {
          const float4 hk = *reinterpret_cast<const float4*>(h1 + c * H + 4 * p);
          acc2[c] = fma2(wa, make_float2(hk.x, hk.y), acc2[c]);
          acc2[c] = fma2(wb, make_float2(hk.z, hk.w), acc2[c]);
        }
      }
      float v[2 * SM];
#pragma unroll
      for (int c = 0; c < SM; ++c) {
        const float h2 = relu(acc2[c].x + acc2[c].y);
        v[c] = w3t * h2;
        v[SM + c] = w3l * h2;
      }
      fold<8>(v, 0);
      fold<4>(v, 1);
      fold<2>(v, 2);
      fold<1>(v, 3);
      const float out = v[0] + __shfl_xor_sync(0xffffffffu, v[0], 16);
      // value index 8 * bit0 + 4 * bit1 + 2 * bit2 + bit3: bit0 thr / lat, the rest the candidate
      const int kind = lane & 1;
      const int c = 4 * ((lane >> 1) & 1) + 2 * ((lane >> 2) & 1) + ((lane >> 3) & 1);
      if (lane < 16) spart[((wq * SM + c) * N + m) * 2 + kind] = out;
    }
    __syncthreads();
    // ---- objective and constraints: warp c, lane i = model i ----
    if (child_warp) {
      float J = 0.f, pen = 0.f;
      bool ok = true;
      if (lane < N) {
        float t = my_b3t, l = my_b3l;
#pragma unroll
        for (int w = 0; w < WPM; ++w) {
          t += spart[((w * SM + warp) * N + lane) * 2 + 0];
          l += spart[((w * SM + warp) * N + lane) * 2 + 1];
        }
        t = out_act(P, t);
        l = out_act(P, l);
        if (P.objective == MF_OBJ_UTILITY) {  // Eq. 3 utility, floor f >= tau
          float f;
          J = util_term_of(P, P.util[my_off + sgenes[warp * N + lane]], my_uomega, my_utau, my_ucost, my_uprev, t,
                           &f);
          ok = f >= my_utau;
        } else {
          J = my_w * t;
          ok = l <= my_sla;
          const float over = l - my_sla;
          pen = over > 0.f ? over : 0.f;
        }
      }
#pragma unroll
      for (int o = 4; o > 0; o >>= 1) {  // lanes 0-7 hold the models
        J += __shfl_xor_sync(0xffffffffu, J, o);
        pen += __shfl_xor_sync(0xffffffffu, pen, o);
      }
      ok = __all_sync(0xffffffffu, ok);
      if (lane == 0) {
        bool feas = sagg[4 * warp + 3] <= P.vram_cap;
        if (P.objective == MF_OBJ_SOFT_LAT) J = fmaf(-P.soft_penalty, pen, J);
        else feas = feas && ok;
        if (J != J) feas = false;
        const float f = feas ? J : -INFINITY;
        st_word(&rec_cur[cg].fw, tagged(tag, __float_as_uint(f)));
        s_fit[warp] = f;
      }
    }
    if (lag_check) {
      bool ok = false;
      for (uint32_t n = 0; n < kGaSpinLimit; ++n) {
        bool mine = true;
#pragma unroll
        for (int u = 0; u < 8; ++u) mine = mine && pv[u] >= (unsigned int)need;
        if (__all_sync(0xffffffffu, mine)) { ok = true; break; }
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (lane + 32 * u < (int)gridDim.x) pv[u] = ld_u32(G.prog + lane + 32 * u);
      }
      if (!ok && lane == 0) fail();
    }
    __syncthreads();
    if (s_abort) return;
    // ---- the last warp publishes the slice's fittest individual ----
    if (warp == last_warp) {
      float f = lane < ns ? s_fit[lane] : -INFINITY;
      int s = lane < ns ? c0 + lane : -1;
      warp_best(f, s);
      if (lane == 0) {
        GaBest* b = best_cur + blockIdx.x;
        st_word(&b->glo, tagged(tag, s_glo[s - c0]));
        st_word(&b->ghi, tagged(tag, s_ghi[s - c0]));
        st_word(&b->sw, tagged(tag, (uint32_t)s));
        st_word(&b->fw, tagged(tag, __float_as_uint(f)));
      }
    }
    if (last) {  // CTA 0: the fittest individual of the last generation
      if (blockIdx.x == 0 && warp == 0) {
        float f;
        int s;
        uint32_t lo, hi;
        const bool ok = best_of_ctas(best_cur, gridDim.x, tag, f, s, lo, hi);
        if (!ok) {
          if (lane == 0) atomicOr(P.status, kStatusTimeout);
        } else {
          const uint64_t g8 = (uint64_t)lo | ((uint64_t)hi << 32);
          if (lane < N) G.out_genome[lane] = (int)((g8 >> (8 * lane)) & 0xFF);
          if (lane == 0) *G.out_fit = f;
        }
      }
      return;
    }
    // ---- next generation: warp c breeds child c0 + c ----
    if (child_warp) {
      const uint32_t GEN = (uint32_t)gen + 1u;
      const ChildDraws d = child_draws(g, sd, GEN, cg, lane, N, my_K);
      uint32_t lo = 0, hi = 0;
      bool ok = true;
      const bool elite = g.elitism && cg == 0;
      if (elite) {  // slot 0 keeps the fittest (lowest slot among equals), unmutated
        float f;
        int s;
        ok = best_of_ctas(best_cur, gridDim.x, tag, f, s, lo, hi);
      } else {
        float fa = -INFINITY, fb = -INFINITY;
        uint32_t la = 0, ha = 0, lb = 0, hb = 0;
        if (d.ta >= 0) ok = fetch_rec(rec_cur + d.ta, tag, fa, la, ha);
        if (ok && d.tb >= 0) ok = fetch_rec(rec_cur + d.tb, tag, fb, lb, hb);
        ok = __all_sync(0xffffffffu, ok);
        if (ok) ok = tournament_winner(g, sd, GEN, cg, kGaTourA, rec_cur, tag, d.ta, fa, la, ha);
        if (ok) ok = tournament_winner(g, sd, GEN, cg, kGaTourB, rec_cur, tag, d.tb, fb, lb, hb);
        lo = d.take_b ? lb : la;
        hi = d.take_b ? hb : ha;
      }
      if (!ok) {
        if (lane == 0) fail();
      } else {
        int gene = (int)(((lane < 4 ? lo : hi) >> (8 * (lane & 3))) & 0xFF);
        if (!elite && d.mutate) gene = d.mval;
        place(gene, rec_nxt, tag + 1u);
      }
    }
    __syncthreads();
    if (s_abort) return;
    if (tid == 0) st_u32(G.prog + blockIdx.x, (unsigned int)gen + 1u);  // generation gen fully read
  }
}

mf_status ga_run_persistent(mf_ctx* c, const mf_ga_params* g, uint64_t seed, cudaStream_t s) {
  const Params& P = c->P;
  const int N = P.n_models;
  if (!(P.d_local == 8 && P.h1 == 64 && P.h2 == 64 && N <= 8)) return MF_EUNSUPPORTED;
  const int pop = g->pop;
  const int ctas = (pop + kGaMaxSlice - 1) / kGaMaxSlice;
  if (ctas > 256) return MF_EUNSUPPORTED;  // progress counters: eight per lane of one warp
  // one thread per (model, hidden unit), at least one warp past the 8 child warps;
  // register budgets of 384 (up to six models) and 512 threads
  const int threads = std::max(N * 64, 32 * (kGaMaxSlice + 1));
  const void* fn = threads <= 384 ? (const void*)k_ga_persist<384> : (const void*)k_ga_persist<512>;
  const int sumK = P.off[N - 1] + P.K[N - 1];
  const size_t smem = sizeof(float) * ((size_t)N * kGaMaxSlice * 64 + (size_t)4 * kGaMaxSlice * N +
                                       4 * kGaMaxSlice + (size_t)sumK * 8) +
                      sizeof(float4) * (size_t)sumK + sizeof(int32_t) * (size_t)kGaMaxSlice * N;
  if (smem > 200 * 1024) return MF_EUNSUPPORTED;
  MF_CUDA(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024));
  int per_sm = 0;
  MF_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, threads, smem));
  if (per_sm * c->num_sms < ctas) return MF_EUNSUPPORTED;
  // scratch: records [ring][pop], CTA bests [ring][ctas], progress [ctas]
  const int ring = std::min(g->gens + 1, kGaRingMax);
  const size_t recb = sizeof(GaRec) * ring * (size_t)pop, bestb = sizeof(GaBest) * ring * (size_t)ctas;
  const size_t need = recb + bestb + sizeof(unsigned int) * (size_t)ctas;
  if (need > c->gap_bytes) {
    MF_CUDA(cudaStreamSynchronize(s));
    cudaFree(c->d_gap);
    c->d_gap = nullptr;
    c->gap_bytes = 0;
    MF_CUDA(cudaMalloc(&c->d_gap, need));
    c->gap_bytes = need;
  }
  if (!c->d_ga_out) MF_CUDA(cudaMalloc(&c->d_ga_out, 128));
  mf_status st = ensure_host_stage(c, 256);
  if (st != MF_OK) return st;
  char* base = (char*)c->d_gap;
  GaPersist G{};
  G.rec = (GaRec*)base;
  G.best = (GaBest*)(base + recb);
  G.prog = (unsigned int*)(base + recb + bestb);
  G.out_genome = (int32_t*)c->d_ga_out;
  G.out_fit = (float*)(G.out_genome + N);
  uint64_t* d_seed = (uint64_t*)((char*)c->d_ga_out + 64);
  G.seed = d_seed;
  G.gens = g->gens;
  G.ring = ring;
  uint64_t* h_seed = (uint64_t*)((char*)c->h_stage + 128);
  *h_seed = seed;
  MF_CUDA(cudaMemcpyAsync(d_seed, h_seed, sizeof(uint64_t), cudaMemcpyHostToDevice, s));
  // tags of a previous run must not match: clear the records, bests and counters
  MF_CUDA(cudaMemsetAsync(c->d_gap, 0, need, s));
  GaArgs a = make_args(c, g);
  Params Pc = P;
  void* args[] = {(void*)&Pc, (void*)&a, (void*)&G};
  MF_CUDA(cudaLaunchCooperativeKernel(fn, dim3(ctas), dim3(threads), args, smem, s));
  return MF_OK;
}

}  // namespace mf
