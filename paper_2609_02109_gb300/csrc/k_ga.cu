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

// Index of the fittest individual, lowest slot among equals (block-wide).
__device__ int block_argmax(const float* __restrict__ fit, int P, float* sval, int* sidx) {
  float best = -INFINITY;
  int bi = 0x7fffffff;
  for (int c = threadIdx.x; c < P; c += blockDim.x) {
    const float f = fit[c];
    if (bi == 0x7fffffff || f > best || (f == best && c < bi)) { best = f; bi = c; }
  }
  for (int o = 16; o > 0; o >>= 1) {
    const float ob = __shfl_xor_sync(0xffffffffu, best, o);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (oi != 0x7fffffff && (bi == 0x7fffffff || ob > best || (ob == best && oi < bi))) { best = ob; bi = oi; }
  }
  const int w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  if ((threadIdx.x & 31) == 0) { sval[w] = best; sidx[w] = bi; }
  __syncthreads();
  if (threadIdx.x == 0) {
    float b = sval[0];
    int x = sidx[0];
    for (int j = 1; j < nw; ++j)
      if (sidx[j] != 0x7fffffff && (x == 0x7fffffff || sval[j] > b || (sval[j] == b && sidx[j] < x))) {
        b = sval[j]; x = sidx[j];
      }
    sval[0] = b;
    sidx[0] = x;
  }
  __syncthreads();
  const int r = sidx[0];
  __syncthreads();
  return r;
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
