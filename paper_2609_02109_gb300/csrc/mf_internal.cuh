// Internal declarations of the CUDA path (not part of the public ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "../../include/mf.h"

namespace mf {

constexpr uint64_t kEmptyIdx = ~0ull;
constexpr int kScoreThreads = 512;   // CTA size of the CUDA-core scorer
constexpr int kWideWarps = 8;        // warps per CTA of the warp-per-(candidate, model) scorer

// Everything a kernel needs about a problem, passed by value (a few hundred bytes).
struct Params {
  int32_t n_models, d_local, h1, h2, d_in;
  int32_t objective, out_act;
  float vram_cap, soft_penalty;
  float agg_scale[4];
  int32_t K[MF_MAX_MODELS];           // options per model
  int32_t off[MF_MAX_MODELS];         // first option row of each model
  uint64_t stride[MF_MAX_MODELS];     // prod_{j>i} K_j (mixed-radix place values)
  float sla[MF_MAX_MODELS];
  float w[MF_MAX_MODELS];
  uint64_t total;                     // |Lambda|
  int64_t per_model;                  // floats per packed predictor
  const float* x;                     // [sumK][d_local]
  const float4* dem;                  // [sumK] (sm, vram, bw, 0)
  const float* w32;                   // predictors, packed as given
  const float* wT;                    // predictors with W1, W2 transposed ([in][out])
  uint32_t* status;                   // device status word (bit 0: bad index/gene)
  // Eq. 3 utility (objective MF_OBJ_UTILITY)
  const float4* util;                 // [sumK] (f_min, f_max - f_min, Q, variant as int bits)
  float u_omega[MF_MAX_MODELS], u_tau[MF_MAX_MODELS], u_cost[MF_MAX_MODELS];
  int32_t u_prev[MF_MAX_MODELS];
  float u_alpha, u_beta, u_delta;
  // Test of the timeout path (mf_debug_wait_test): when non-zero, the kernels with
  // bounded device waits first wait on a flag that nothing sets, giving up after this
  // many polls, and then run to their end as after any wait that gave up.
  uint32_t wait_test;
};

// Tensor-core path: operand images and the per-CTA layout (filled by tc_prepare).
struct TcArgs {
  const void* img;                    // B operands (bf16, or tf32 hi/lo), UMMA K-major no-swizzle layout
  uint32_t img_bytes;
  const uint32_t* xw;                 // [sumK][kw] local features: bf16 pairs, or tf32 hi then lo words
  int32_t k1, kw, h1, h2, hl, n3, dle;
  uint32_t off_b1[MF_MAX_MODELS], off_b2[MF_MAX_MODELS], off_b3[MF_MAX_MODELS];  // bytes in img
  int32_t pipes, col_d, col_h, col_ones, col_a, col_d3, pipe_stride;  // TMEM columns
  // the exact fp32 variant (3-term tf32 split): operands as tf32 hi and lo parts; col_hlo
  // holds the hidden layer's lo parts, img_lo1..3 are the byte offsets of each B image's
  // lo part after its hi part
  int32_t tf, col_hlo;
  uint32_t img_lo1, img_lo2, img_lo3;
  uint32_t sm_xw, sm_dem, sm_rows, sm_topk, sm_bar, sm_total;  // shared-memory byte offsets
  uint32_t img_model;                 // bytes of one model's B1 + B2 + B3 images
  int32_t kcap;                       // per-pipeline list length the layout was sized for
  int32_t qcap;                       // per-pipeline candidate queue (128 or 512, a power of two)
  uint32_t step[MF_MAX_MODELS];       // mixed-radix digits of the per-tile index stride (range mode)
  // the same stride for digits packed one per byte (model N - 1 in the lowest byte):
  // byte of model i = step[i] + 256 - K_i, and the bias bytes 256 - K_i
  uint64_t dstep, dbias;
  // models whose weights do not fit shared memory together run in passes of consecutive
  // models [pass_m[p], pass_m[p + 1]); each pass's image is staged on its own
  int32_t npasses;
  int32_t pass_m[MF_MAX_MODELS + 1];
  // per launch: this pass's models and image bytes, and the per-candidate partial record
  int32_t m0, m1, pass_first, pass_last;
  uint32_t img_lo, img_copy, img_total;
  float4* partial;                    // [candidates of the launch] (J, penalty, flags, -)
};

// Device status bits.
constexpr uint32_t kStatusBadInput = 1u;
constexpr uint32_t kStatusTimeout = 2u;

// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------

// (J, idx) total order: J descending, then index ascending.
__device__ __forceinline__ bool precedes(float ja, uint64_t ia, float jb, uint64_t ib) {
  return ja > jb || (ja == jb && ia < ib);
}

// ReLU that keeps NaN (so a NaN weight reaches the outputs and marks the
// candidate infeasible).
__device__ __forceinline__ float relu(float v) { return v < 0.f ? 0.f : v; }

// Digit of model i of index idx (C order: last model fastest).
__device__ __forceinline__ int digit_of(const Params& P, uint64_t idx, int i) {
  if (P.total <= 0x100000000ull) {
    uint32_t q = (uint32_t)idx / (uint32_t)P.stride[i];
    return (int)(q % (uint32_t)P.K[i]);
  }
  return (int)((idx / P.stride[i]) % (uint64_t)P.K[i]);
}

// Output unit of the predictor: identity or sigmoid (the paper's output layer).
__device__ __forceinline__ float out_act(const Params& P, float v) {
  return P.out_act == MF_ACT_SIGMOID ? 1.f / (1.f + expf(-v)) : v;
}

// Objective and constraints of one candidate from per-model outputs.
// Model i's term of the Eq. 3 utility from its predicted throughput fhat (after the
// output activation) for option row `row`: per-variant normalisation, quality,
// reload cost when the variant changes, quadratic margin below tau_i + delta.
// *f: the normalised throughput (its floor is tau_i).
__device__ __forceinline__ float util_term_of(const Params& P, float4 q, float omega, float tau, float cost,
                                             int prev, float fhat, float* f) {
  const float fn = (fhat - q.x) / q.y;
  const int v = __float_as_int(q.w);
  const float eta = (prev >= 0 && v != prev) ? 1.f : 0.f;
  const float margin = tau + P.u_delta - fn;
  *f = fn;
  return omega * fn * q.z - P.u_alpha * eta * cost - P.u_beta * (margin > 0.f ? margin * margin : 0.f);
}

__device__ __forceinline__ float util_term(const Params& P, int i, int row, float fhat, float* f) {
  return util_term_of(P, P.util[row], P.u_omega[i], P.u_tau[i], P.u_cost[i], P.u_prev[i], fhat, f);
}

struct Acc {
  float J, pen;
  bool sla_ok;    // latency ceilings (weighted throughput) or floors (utility)
  __device__ __forceinline__ void init() { J = 0.f; pen = 0.f; sla_ok = true; }
  // thr, lat: predictor outputs after the output activation; row: the option row.
  __device__ __forceinline__ void add(const Params& P, int i, float thr, float lat, int row) {
    if (P.objective == MF_OBJ_UTILITY) {
      float f;
      J += util_term(P, i, row, thr, &f);
      sla_ok = sla_ok && (f >= P.u_tau[i]);
      return;
    }
    J = fmaf(P.w[i], thr, J);
    sla_ok = sla_ok && (lat <= P.sla[i]);
    float over = lat - P.sla[i];
    pen += over > 0.f ? over : 0.f;
  }
  // Returns feasibility; J becomes the final score (-inf when infeasible).
  __device__ __forceinline__ bool finish(const Params& P, float vram_sum) {
    bool feas = vram_sum <= P.vram_cap;
    if (P.objective == MF_OBJ_SOFT_LAT) J = fmaf(-P.soft_penalty, pen, J);
    else feas = feas && sla_ok;
    if (J != J) feas = false;
    if (!feas) J = -INFINITY;
    return feas;
  }
};

// fma.rn.f32x2: two fp32 fused multiply-adds (each rounded as fmaf) in one instruction.
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
  unsigned long long r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;"
      : "=l"(r)
      : "l"(*reinterpret_cast<unsigned long long*>(&a)), "l"(*reinterpret_cast<unsigned long long*>(&b)),
        "l"(*reinterpret_cast<unsigned long long*>(&c)));
  return *reinterpret_cast<float2*>(&r);
}

// a[i] for a per-model array of the kernel parameters, read with constant indices
// (a runtime index into a parameter array would copy it to local memory)
template <typename T>
__device__ __forceinline__ T pick(const T (&a)[MF_MAX_MODELS], int i) {
  T v = a[0];
#pragma unroll
  for (int k = 1; k < MF_MAX_MODELS; ++k) v = k == i ? a[k] : v;
  return v;
}

// Index of the fittest individual of fit[0, n), lowest slot among equals (block-wide;
// every thread of the block calls it; sval/sidx: 32 entries of shared memory).
__device__ __forceinline__ int block_argmax(const float* __restrict__ fit, int n, float* sval, int* sidx) {
  float best = -INFINITY;
  int bi = 0x7fffffff;
  for (int c = threadIdx.x; c < n; c += blockDim.x) {
    const float f = fit[c];
    if (bi == 0x7fffffff || f > best || (f == best && c < bi)) { best = f; bi = c; }
  }
  for (int o = 16; o > 0; o >>= 1) {
    const float ob = __shfl_xor_sync(0xffffffffu, best, o);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (oi != 0x7fffffff && (bi == 0x7fffffff || ob > best || (ob == best && oi < bi))) { best = ob; bi = oi; }
  }
  const int w = threadIdx.x >> 5;
  const int nwb = (blockDim.x + 31) >> 5, nwn = (n + 31) >> 5;
  const int nw = nwn < nwb ? nwn : nwb;  // warps holding entries (the rest found none)
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

// SplitMix64 output number ctr of the sequence whose state starts at seed
// (Steele, Lea and Flood, OOPSLA 2014).
__device__ __forceinline__ uint64_t splitmix64(uint64_t seed, uint64_t ctr) {
  uint64_t z = seed + (ctr + 1ull) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t ga_rng(uint64_t seed, uint32_t gen, uint32_t slot,
                                           uint32_t purpose, uint32_t j) {
  uint64_t ctr = ((uint64_t)gen << 32) | ((uint64_t)(slot & 0xFFFFFu) << 12) |
                 ((uint64_t)(purpose & 0xFu) << 8) | (uint64_t)(j & 0xFFu);
  return splitmix64(seed, ctr);
}

__device__ __forceinline__ int ga_unif(uint64_t r, uint32_t k) {
  return (int)(((r >> 32) * (uint64_t)k) >> 32);
}

enum { kGaInit = 0, kGaTourA = 1, kGaTourB = 2, kGaCross = 3, kGaMut = 4, kGaMutVal = 5, kGaCrossDo = 6,
       kGaRepair = 7 };

// ---------------------------------------------------------------------------
// Per-CTA running top-k in shared memory (sorted by the total order), fed by
// a queue of candidates that beat the current k-th entry.
// ---------------------------------------------------------------------------
struct CtaTopK {
  float* ls; uint64_t* li;   // current list [k]
  float* ns; uint64_t* ni;   // merge output [k]
  float* qs; uint64_t* qi;   // queue [qcap]
  int* qn;
  int k;
};

// Merge the queue into the list.  Called by `nthr` threads (ids 0..nthr-1) after a
// barrier that made the queue visible; `sync()` is a barrier over those threads.
template <class Sync>
__device__ void topk_merge(const CtaTopK& t, int tid, int nthr, Sync sync) {
  const int k = t.k;
  const int q = *t.qn;
  for (int e = tid; e < k; e += nthr) { t.ns[e] = -INFINITY; t.ni[e] = kEmptyIdx; }
  sync();
  for (int e = tid; e < k + q; e += nthr) {
    float s; uint64_t id; int rank;
    if (e < k) {
      s = t.ls[e]; id = t.li[e];
      if (id == kEmptyIdx) continue;
      rank = e;
    } else {
      s = t.qs[e - k]; id = t.qi[e - k];
      int lo = 0, hi = k;
      while (lo < hi) {
        int mid = (lo + hi) >> 1;
        if (precedes(t.ls[mid], t.li[mid], s, id)) lo = mid + 1; else hi = mid;
      }
      rank = lo;
    }
    for (int j = 0; j < q && rank < k; ++j) rank += precedes(t.qs[j], t.qi[j], s, id) ? 1 : 0;
    if (rank < k) { t.ns[rank] = s; t.ni[rank] = id; }
  }
  sync();
  for (int e = tid; e < k; e += nthr) { t.ls[e] = t.ns[e]; t.li[e] = t.ni[e]; }
  if (tid == 0) *t.qn = 0;
  sync();
}

// The same merge for a long queue (up to qcap entries, qcap a power of two): the queue
// is first sorted best-first by a bitonic network over the next power of two (padding
// entries are (-inf, empty), last in the order), so an entry's rank is its position in
// the sorted queue plus the number of list entries ahead of it, found by binary search
// (and a list entry's rank likewise).  O(q log^2 q) work instead of O(q k).
template <class Sync>
__device__ void topk_merge_sorted(const CtaTopK& t, int tid, int nthr, Sync sync) {
  const int k = t.k;
  const int q = *t.qn;
  int n2 = 1;
  while (n2 < q) n2 <<= 1;
  for (int e = q + tid; e < n2; e += nthr) { t.qs[e] = -INFINITY; t.qi[e] = kEmptyIdx; }
  for (int e = tid; e < k; e += nthr) { t.ns[e] = -INFINITY; t.ni[e] = kEmptyIdx; }
  sync();
  for (int size = 2; size <= n2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = tid; i < (n2 >> 1); i += nthr) {
        const int a = 2 * stride * (i / stride) + (i % stride), b = a + stride;
        const float sa = t.qs[a], sb = t.qs[b];
        const uint64_t ia = t.qi[a], ib = t.qi[b];
        const bool best_first = (a & size) == 0;
        if (best_first ? precedes(sb, ib, sa, ia) : precedes(sa, ia, sb, ib)) {
          t.qs[a] = sb; t.qi[a] = ib;
          t.qs[b] = sa; t.qi[b] = ia;
        }
      }
      sync();
    }
  }
  // queue entries: only the first k positions can rank below k
  for (int p = tid; p < k && p < q; p += nthr) {
    const float s = t.qs[p];
    const uint64_t id = t.qi[p];
    int lo = 0, hi = k;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (precedes(t.ls[mid], t.li[mid], s, id)) lo = mid + 1; else hi = mid;
    }
    if (p + lo < k) { t.ns[p + lo] = s; t.ni[p + lo] = id; }
  }
  // list entries
  for (int e = tid; e < k; e += nthr) {
    const float s = t.ls[e];
    const uint64_t id = t.li[e];
    if (id == kEmptyIdx) continue;
    int lo = 0, hi = q;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (precedes(t.qs[mid], t.qi[mid], s, id)) lo = mid + 1; else hi = mid;
    }
    if (e + lo < k) { t.ns[e + lo] = s; t.ni[e + lo] = id; }
  }
  sync();
  for (int e = tid; e < k; e += nthr) { t.ls[e] = t.ns[e]; t.li[e] = t.ni[e]; }
  if (tid == 0) *t.qn = 0;
  sync();
}

}  // namespace mf

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
struct mf_ctx {
  int device = 0;
  int num_sms = 0;
  mf::Params P{};                 // device pointers filled in
  int32_t precision = MF_FP32;
  std::vector<int32_t> K;
  int sumK = 0;
  // device buffers owned by the context
  float* d_x = nullptr;
  float4* d_dem = nullptr;
  float* d_w32 = nullptr;
  float* d_wT = nullptr;
  uint32_t* d_status = nullptr;
  void* d_tc = nullptr;           // packed bf16 operand images (tensor-core path)
  void* d_partial = nullptr;      // per-candidate partial objective between tensor-core passes
  size_t partial_bytes = 0;
  // fixed-context mode: the per-option table of the last mf_fc_set
  void* d_fc = nullptr;           // see mf::FcLayout
  int fc_ready = 0;
  float4* d_util = nullptr;       // [sumK] utility table of mf_set_utility
  int32_t base_objective = 0;     // the problem's own objective
  size_t tc_bytes = 0;
  mf::TcArgs tc{};
  // growable scratch (search lists, merge buffers, shortlist)
  void* d_scratch = nullptr;
  size_t scratch_bytes = 0;
  // pinned host staging for results
  void* h_stage = nullptr;
  size_t h_stage_bytes = 0;
  // GA: populations, fitness, per-model outputs, result, and the captured graph
  int32_t* d_pop[2] = {nullptr, nullptr};
  float* d_fit = nullptr;
  float* d_pred = nullptr;
  void* d_ga_out = nullptr;       // best genome [N] int32, then its fitness (float), then the seed (u64)
  void* d_gap = nullptr;          // cooperative GA kernel: byte genomes, fitness, barrier flags, CTA bests
  size_t gap_bytes = 0;
  int ga_cap = 0;
  cudaStream_t cap_stream = nullptr;
  cudaGraphExec_t ga_exec = nullptr;
  uint64_t params_version = 0;
  uint64_t ga_version = ~0ull;
  mf_ga_params ga_key{};
  // instrumentation
  mf_stats stats{};
  cudaEvent_t ev[3] = {nullptr, nullptr, nullptr};
};

namespace mf {

// Thread-local detail string of the last failure.
void set_error(const std::string& msg);

// Makes the context's device current for the scope of an API call.
struct DeviceGuard {
  int prev = -1;
  bool changed = false;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) changed = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DeviceGuard() {
    if (changed) cudaSetDevice(prev);
  }
};
mf_status cuda_fail(cudaError_t e, const char* what);

#define MF_CUDA(call)                                         \
  do {                                                        \
    cudaError_t _e = (call);                                  \
    if (_e != cudaSuccess) return ::mf::cuda_fail(_e, #call); \
  } while (0)

// Scratch management.
mf_status ensure_scratch(mf_ctx* c, size_t bytes);
mf_status ensure_host_stage(mf_ctx* c, size_t bytes);

// CUDA-core scorer (exact fp32 path).
struct RangeArgs {
  uint64_t base, len;
  int k;
  int first;            // 1: initialise the per-CTA lists
  float* lists_s;       // [grid][k]
  uint64_t* lists_i;    // [grid][k]
  unsigned long long* count;
};
bool f32_supported(const Params& P);
size_t f32_smem_bytes(const Params& P, int k, bool& resident);
int f32_grid(const mf_ctx* c);
mf_status f32_prepare(mf_ctx* c);
mf_status f32_search_chunk(mf_ctx* c, const RangeArgs& a, cudaStream_t s);
// Fixed-context mode: one range launch of the table-lookup scan over the per-option
// table of mf_fc_set.
int fc_grid(const mf_ctx* c);
mf_status fc_search_chunk(mf_ctx* c, const RangeArgs& a, cudaStream_t s);
mf_status f32_search_chunk_params(const Params& P, int grid, const RangeArgs& a, cudaStream_t s);
mf_status f32_score_list(mf_ctx* c, const uint64_t* idx, const int32_t* genes, uint64_t n,
                         float* score, uint8_t* feas, float* pred, cudaStream_t s);
// Exact re-scoring of a shortlist that may contain empty slots (index UINT64_MAX),
// which score -inf without raising the device status.  pred: scratch [n][N][2].
mf_status f32_score_list_ex(mf_ctx* c, const uint64_t* idx, uint64_t n, float* score, float* pred,
                            cudaStream_t s);

// Merge of per-CTA sorted lists into one sorted top-k.
mf_status merge_lists(mf_ctx* c, const float* ls, const uint64_t* li, int nlists, int k,
                      float* tmp_s, uint64_t* tmp_i, float* out_s, uint64_t* out_i,
                      cudaStream_t s);
// Sort n (score, idx) pairs by the total order and keep the first k (n <= 8192).
mf_status select_topk(mf_ctx* c, const float* in_s, const uint64_t* in_i, int n, int k,
                      float* out_s, uint64_t* out_i, cudaStream_t s);

// Tensor-core scorer (bf16 path).
bool tc_supported(const Params& P, std::string* why);
bool tc_exact_supported(const Params& P);  // the exact fp32 (3-term tf32) variant's shapes
bool tc_fits(const mf_ctx* c, int kcap);    // the context's tensor-core layout with lists of kcap
mf_status tc_prepare(mf_ctx* c, bool exact = false);
int tc_grid(const mf_ctx* c);
mf_status tc_search_chunk(mf_ctx* c, const RangeArgs& a, cudaStream_t s, int* nlaunch);
mf_status tc_score_list(mf_ctx* c, const uint64_t* idx, uint64_t n, float* score,
                        uint8_t* feas, float* pred, cudaStream_t s);

// GA kernels.
mf_status ga_init(mf_ctx* c, const mf_ga_params* g, uint64_t seed, int32_t* pop, cudaStream_t s);
mf_status ga_step(mf_ctx* c, const mf_ga_params* g, uint64_t seed, int32_t gen,
                  const int32_t* pop, const float* fit, int32_t* next, cudaStream_t s);
mf_status ga_best(mf_ctx* c, const int32_t* pop, const float* fit, int P, int32_t* out_genome,
                  float* out_fit, cudaStream_t s);
// Whole GA decision as one CUDA graph launch on `s`; the result lands in c->d_ga_out
// and the pinned staging buffer is sized for it.
mf_status ga_run_graph(mf_ctx* c, const mf_ga_params* g, uint64_t seed, cudaStream_t s);
// Whole GA decision in one cooperative kernel; MF_EUNSUPPORTED (nothing launched) when
// the shape or the device does not allow it.
mf_status ga_run_persistent(mf_ctx* c, const mf_ga_params* g, uint64_t seed, cudaStream_t s);

}  // namespace mf
