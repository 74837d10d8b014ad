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

// ---------------------------------------------------------------------------
// Whole GA decision in one cooperative kernel (fp32 predictors d_L 8, 64-64).
//
// Each CTA owns a slice of at most kGaMaxSlice individuals.  One thread per
// (model m, hidden unit j) keeps row j of W1 and W2 of model m in registers for
// the whole run and evaluates that unit for every individual of the slice, so a
// weight is read once per run, not once per individual.  Per generation:
//   aggregate -> layer 1 -> layers 2 and 3 -> objective and constraints of the
//   slice -> grid barrier -> the generation's population and fitness copied
//   from L2 into shared memory in one pass -> the slice's children (elite,
//   tournaments, crossover, mutation: the operators and draws of k_ga_step)
// Population and fitness are double-buffered in global memory.  A buffer written
// in generation g + 2 was last read (copied to shared memory) in generation g,
// before its reader arrived at the barrier that ends generation g + 1, which the
// writer has passed.
// ---------------------------------------------------------------------------
namespace mf {

constexpr int kGaMaxSlice = 8;
constexpr uint32_t kGridPollLimit = 1u << 22;  // polls of about a microsecond: a few seconds

struct GaPersist {
  int32_t* pop0;
  int32_t* pop1;
  float* fit0;           // fitness of even generations
  float* fit1;           // fitness of odd generations
  unsigned int* flags;   // [ctas] last epoch each CTA reached
  int32_t* out_genome;
  float* out_fit;
  const uint64_t* seed;
  int gens;
  int slice;
};

__device__ __forceinline__ unsigned int ld_acquire_gpu(const unsigned int* p) {
  unsigned int v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_gpu(unsigned int* p, unsigned int v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Grid barrier: every CTA publishes `epoch` in its own flag, then polls all flags
// (one per thread).  Gives up after kGridPollLimit polls, flags the status word and
// lets the kernel run to its end.
__device__ void grid_barrier(unsigned int* flags, unsigned int nblocks, unsigned int epoch, uint32_t* status) {
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    st_release_gpu(flags + blockIdx.x, epoch);
  }
  uint32_t n = 0;
  while (true) {
    bool mine = true;
    for (unsigned int q = threadIdx.x; q < nblocks; q += blockDim.x)
      mine = mine && (ld_acquire_gpu(flags + q) >= epoch);
    if (__syncthreads_and(mine)) break;
    if (++n > kGridPollLimit) {
      if (threadIdx.x == 0) atomicOr(status, kStatusTimeout);
      break;
    }
  }
}

template <int DL, int MAXT>
__global__ void __launch_bounds__(MAXT, 1)
k_ga_persist(const Params P, const GaArgs g, const GaPersist G) {
  constexpr int H = 64, DIN = DL + 4, SM = kGaMaxSlice;
  extern __shared__ __align__(16) float sm[];
  const int N = P.n_models;
  const int sumK = P.off[N - 1] + P.K[N - 1];
  const int pop = g.pop;
  const int pop4 = (pop + 3) & ~3;
  // shared memory; every float region is a multiple of 4 floats so the float4 rows align
  float* sh1 = sm;                                           // [N][SM][H] layer-1 activations
  float* spart = sh1 + (size_t)N * SM * H;                   // [2][SM][N][2] layer-3 halves
  float* sagg = spart + 4 * SM * N;                          // [SM][4] scaled aggregate, raw VRAM
  float* sb3 = sagg + 4 * SM;                                // [MF_MAX_MODELS][2]
  float* sfit = sb3 + 2 * MF_MAX_MODELS;                     // [pop] fitness of the generation
  float* sx = sfit + pop4;                                   // [sumK][DL] local features
  float4* sdem = reinterpret_cast<float4*>(sx + (size_t)sumK * DL);  // [sumK]
  int32_t* spop = reinterpret_cast<int32_t*>(sdem + sumK);   // [pop][N] the generation's genomes
  int32_t* sgenes = spop + (((size_t)pop * N + 3) & ~(size_t)3);  // [SM][N] this slice's genomes
  __shared__ float sval[32];
  __shared__ int sidx[32];

  const int tid = threadIdx.x, lane = tid & 31;
  const bool unit = tid < N * H;
  const int m = unit ? tid / H : 0, j = unit ? tid % H : 0;
  // this thread's weights: rows j of W1 and W2 of model m, and its layer-3 column
  float w1[DIN], w2[H];
  float b1 = 0.f, b2 = 0.f, w3t = 0.f, w3l = 0.f;
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
  }
  for (int e = tid; e < N; e += blockDim.x) {
    const float* b3 = P.w32 + (size_t)e * P.per_model + H * DIN + H + H * H + H + 2 * H;
    sb3[2 * e] = b3[0];
    sb3[2 * e + 1] = b3[1];
  }
  for (int e = tid; e < sumK * DL; e += blockDim.x) sx[e] = P.x[e];
  for (int e = tid; e < sumK; e += blockDim.x) sdem[e] = P.dem[e];
  const uint64_t sd = *G.seed;
  const int c0 = blockIdx.x * G.slice;
  const int c1 = min(pop, c0 + G.slice);
  const int ns = c1 - c0;
  for (int e = tid; e < ns * N; e += blockDim.x) {  // initial population of this slice
    const int c = c0 + e / N, i = e % N;
    const int gene = ga_unif(ga_rng(sd, 0, (uint32_t)c, kGaInit, (uint32_t)i), (uint32_t)g.K[i]);
    G.pop0[(size_t)c * N + i] = gene;
    sgenes[e] = gene;
  }
  __syncthreads();
  const float nz = (float)N * P.agg_scale[3];

  for (int gen = 0; gen < G.gens; ++gen) {
    int32_t* cur = (gen & 1) ? G.pop1 : G.pop0;
    int32_t* nxt = (gen & 1) ? G.pop0 : G.pop1;
    float* fit = (gen & 1) ? G.fit1 : G.fit0;
    // ---- aggregate state of every individual of the slice ----
    if (tid < ns) {
      float A0 = 0.f, A1 = 0.f, A2 = 0.f;
      for (int i = 0; i < N; ++i) {
        const float4 d = sdem[P.off[i] + sgenes[tid * N + i]];
        A0 += d.x; A1 += d.y; A2 += d.z;
      }
      sagg[4 * tid + 0] = A0 * P.agg_scale[0];
      sagg[4 * tid + 1] = A1 * P.agg_scale[1];
      sagg[4 * tid + 2] = A2 * P.agg_scale[2];
      sagg[4 * tid + 3] = A1;  // raw VRAM sum for the constraint
    }
    __syncthreads();
    // ---- layer 1: unit j of model m for every individual ----
    if (unit) {
#pragma unroll
      for (int c = 0; c < SM; ++c) {
        if (c < ns) {
          const float4* xr = reinterpret_cast<const float4*>(sx + (size_t)(P.off[m] + sgenes[c * N + m]) * DL);
          float u0 = b1, u1 = 0.f;
#pragma unroll
          for (int q = 0; q < DL / 4; ++q) {
            const float4 v = xr[q];
            u0 = fmaf(w1[4 * q + 0], v.x, u0);
            u1 = fmaf(w1[4 * q + 1], v.y, u1);
            u0 = fmaf(w1[4 * q + 2], v.z, u0);
            u1 = fmaf(w1[4 * q + 3], v.w, u1);
          }
          const float4 a = *reinterpret_cast<const float4*>(sagg + 4 * c);
          u0 = fmaf(w1[DL + 0], a.x, u0);
          u1 = fmaf(w1[DL + 1], a.y, u1);
          u0 = fmaf(w1[DL + 2], a.z, u0);
          u1 = fmaf(w1[DL + 3], nz, u1);
          sh1[((size_t)m * SM + c) * H + j] = relu(u0 + u1);
        }
      }
    }
    __syncthreads();
    // ---- layers 2 and 3: unit j of model m for every individual ----
    if (unit) {
      const float* h1 = sh1 + (size_t)m * SM * H;
      float acc[SM];
#pragma unroll
      for (int c = 0; c < SM; ++c) acc[c] = b2;
#pragma unroll
      for (int k = 0; k < H; k += 4) {
#pragma unroll
        for (int c = 0; c < SM; ++c) {
          if (c < ns) {
            const float4 hk = *reinterpret_cast<const float4*>(h1 + c * H + k);
            acc[c] = fmaf(w2[k + 0], hk.x, acc[c]);
            acc[c] = fmaf(w2[k + 1], hk.y, acc[c]);
            acc[c] = fmaf(w2[k + 2], hk.z, acc[c]);
            acc[c] = fmaf(w2[k + 3], hk.w, acc[c]);
          }
        }
      }
      const int hh = j >> 5;  // which warp of the model's 64 units
#pragma unroll
      for (int c = 0; c < SM; ++c) {
        if (c < ns) {
          const float h2 = relu(acc[c]);
          float tt = w3t * h2, ll = w3l * h2;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) {
            tt += __shfl_xor_sync(0xffffffffu, tt, o);
            ll += __shfl_xor_sync(0xffffffffu, ll, o);
          }
          if (lane == 0) {
            spart[((hh * SM + c) * N + m) * 2 + 0] = tt;
            spart[((hh * SM + c) * N + m) * 2 + 1] = ll;
          }
        }
      }
    }
    __syncthreads();
    // ---- objective and constraints of the slice ----
    if (tid < ns) {
      Acc acc;
      acc.init();
      for (int i = 0; i < N; ++i) {
        const float t = spart[((0 * SM + tid) * N + i) * 2] + spart[((1 * SM + tid) * N + i) * 2] + sb3[2 * i];
        const float l =
            spart[((0 * SM + tid) * N + i) * 2 + 1] + spart[((1 * SM + tid) * N + i) * 2 + 1] + sb3[2 * i + 1];
        acc.add(P, i, out_act(P, t), out_act(P, l));
      }
      acc.finish(P, sagg[4 * tid + 3]);
      fit[c0 + tid] = acc.J;
    }
    grid_barrier(G.flags, gridDim.x, (unsigned int)gen + 1u, P.status);
    // ---- the generation's genomes and fitness into shared memory, through L2 ----
    {
      const int n4 = (pop * N) >> 2;
      const int4* src = reinterpret_cast<const int4*>(cur);
      int4* dst = reinterpret_cast<int4*>(spop);
      for (int e = tid; e < n4; e += blockDim.x) dst[e] = __ldcg(src + e);
      for (int e = 4 * n4 + tid; e < pop * N; e += blockDim.x) spop[e] = __ldcg(cur + e);
      for (int e = tid; e < pop; e += blockDim.x) sfit[e] = __ldcg(fit + e);
    }
    __syncthreads();
    if (gen + 1 == G.gens) break;
    // ---- next generation for the slice ----
    const uint32_t GEN = (uint32_t)gen + 1u;
    if (g.elitism && c0 == 0) {  // slot 0 keeps the fittest (lowest slot among equals)
      const int e = block_argmax(sfit, pop, sval, sidx);
      if (tid < N) sgenes[tid] = spop[(size_t)e * N + tid];
    }
    if (tid < ns && !(g.elitism && c0 + tid == 0)) {
      const int c = c0 + tid;
      const int a = tournament(g, sfit, sd, GEN, (uint32_t)c, kGaTourA);
      const int b = tournament(g, sfit, sd, GEN, (uint32_t)c, kGaTourB);
      for (int i = 0; i < N; ++i) {
        const uint64_t rc = ga_rng(sd, GEN, (uint32_t)c, kGaCross, (uint32_t)i);
        int gene = spop[(size_t)((rc >> 63) ? b : a) * N + i];
        const uint64_t rm = ga_rng(sd, GEN, (uint32_t)c, kGaMut, (uint32_t)i);
        if ((uint32_t)(rm >> 40) < g.mut_thr)
          gene = ga_unif(ga_rng(sd, GEN, (uint32_t)c, kGaMutVal, (uint32_t)i), (uint32_t)g.K[i]);
        sgenes[tid * N + i] = gene;
      }
    }
    __syncthreads();
    for (int e = tid; e < ns * N; e += blockDim.x) nxt[(size_t)c0 * N + e] = sgenes[e];
    __syncthreads();
  }
  // fittest individual of the last population
  if (blockIdx.x == 0) {
    const int e = block_argmax(sfit, pop, sval, sidx);
    if (tid < N) G.out_genome[tid] = spop[(size_t)e * N + tid];
    if (tid == 0) *G.out_fit = sfit[e];
  }
}

size_t ga_persist_smem(int N, int sumK, int pop) {
  const size_t floats = (size_t)N * kGaMaxSlice * 64 + 4 * kGaMaxSlice * (size_t)N + 4 * kGaMaxSlice +
                        2 * MF_MAX_MODELS + (size_t)((pop + 3) & ~3) + (size_t)sumK * 8;
  return floats * sizeof(float) + sizeof(float4) * (size_t)sumK +
         sizeof(int32_t) * ((((size_t)pop * N + 3) & ~(size_t)3) + (size_t)kGaMaxSlice * N);
}

mf_status ga_run_persistent(mf_ctx* c, const mf_ga_params* g, uint64_t seed, cudaStream_t s) {
  const Params& P = c->P;
  const int N = P.n_models;
  if (!(P.d_local == 8 && P.h1 == 64 && P.h2 == 64 && N * 64 <= 512)) return MF_EUNSUPPORTED;
  const int pop = g->pop;
  int slice = (pop + c->num_sms - 1) / c->num_sms;
  if (slice < 1) slice = 1;
  if (slice > kGaMaxSlice) return MF_EUNSUPPORTED;
  const int ctas = (pop + slice - 1) / slice;
  const int threads = ((N * 64 > 256 ? N * 64 : 256) + 31) / 32 * 32;
  const int sumK = P.off[N - 1] + P.K[N - 1];
  const size_t smem = ga_persist_smem(N, sumK, pop);
  if (smem > 200 * 1024) return MF_EUNSUPPORTED;
  // two register budgets: up to 384 threads (N <= 6) and up to 512 (N <= 8)
  const void* fn = threads <= 384 ? (const void*)k_ga_persist<8, 384> : (const void*)k_ga_persist<8, 512>;
  MF_CUDA(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024));
  int per_sm = 0;
  MF_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, threads, smem));
  if (per_sm * c->num_sms < ctas) return MF_EUNSUPPORTED;
  if (pop > c->ga_cap) {
    MF_CUDA(cudaStreamSynchronize(s));
    cudaFree(c->d_pop[0]); cudaFree(c->d_pop[1]); cudaFree(c->d_fit); cudaFree(c->d_pred);
    c->d_pop[0] = c->d_pop[1] = nullptr; c->d_fit = c->d_pred = nullptr;
    c->ga_cap = 0;
    MF_CUDA(cudaMalloc(&c->d_pop[0], sizeof(int32_t) * (size_t)pop * N));
    MF_CUDA(cudaMalloc(&c->d_pop[1], sizeof(int32_t) * (size_t)pop * N));
    MF_CUDA(cudaMalloc(&c->d_fit, sizeof(float) * (size_t)pop));
    MF_CUDA(cudaMalloc(&c->d_pred, sizeof(float) * 2 * (size_t)pop * N));
    c->ga_cap = pop;
    if (c->ga_exec) { cudaGraphExecDestroy(c->ga_exec); c->ga_exec = nullptr; }
  }
  if (!c->d_ga_out) MF_CUDA(cudaMalloc(&c->d_ga_out, 128));
  mf_status st = ensure_host_stage(c, 256);
  if (st != MF_OK) return st;
  int32_t* out_genome = (int32_t*)c->d_ga_out;
  float* out_fit = (float*)(out_genome + N);
  uint64_t* d_seed = (uint64_t*)((char*)c->d_ga_out + 64);
  // the odd generations' fitness and the per-CTA barrier flags live in the per-model
  // output buffer (2 * pop * N words >= pop + ctas)
  float* fit1 = c->d_pred;
  unsigned int* flags = reinterpret_cast<unsigned int*>(c->d_pred + pop);
  uint64_t* h_seed = (uint64_t*)((char*)c->h_stage + 128);
  *h_seed = seed;
  MF_CUDA(cudaMemcpyAsync(d_seed, h_seed, sizeof(uint64_t), cudaMemcpyHostToDevice, s));
  MF_CUDA(cudaMemsetAsync(flags, 0, sizeof(unsigned int) * (size_t)ctas, s));
  GaArgs a = make_args(c, g);
  GaPersist G{c->d_pop[0], c->d_pop[1], c->d_fit, fit1, flags, out_genome, out_fit, d_seed, g->gens, slice};
  Params Pc = P;
  void* args[] = {(void*)&Pc, (void*)&a, (void*)&G};
  MF_CUDA(cudaLaunchCooperativeKernel(fn, dim3(ctas), dim3(threads), args, smem, s));
  return MF_OK;
}

}  // namespace mf
