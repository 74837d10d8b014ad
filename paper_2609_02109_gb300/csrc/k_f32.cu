// Exact fp32 scorer on the CUDA cores.
//
// Per candidate (arXiv 2609.02109): decode the mixed-radix index (Eq. 1), gather
// each model's option row, form the aggregate state (summed SM share, VRAM and
// bandwidth of the chosen options plus N), run each model's MLP predictor
// (Eq. 6), apply the VRAM and SLA constraints (Eq. 4) and the objective (Eq. 3,
// throughput-weighted term, or the soft latency penalty).
//
// Two layouts of the work:
//   k_score_f32  one thread per candidate; predictor weights staged once per CTA
//                in shared memory (all threads read the same weight: a
//                broadcast), a persistent grid of one 512-thread CTA per SM.
//                Used for exhaustive ranges (with a per-CTA running top-k) and
//                for large index lists.
//   k_wide_f32   one warp per (candidate, model): the hidden units are spread
//                over the lanes, weights read transposed from L1/L2.  Used for
//                small batches (a GA population, a re-scoring shortlist), where
//                one thread per candidate would leave most SMs idle.
#include <cstdio>

#include "mf_internal.cuh"

namespace mf {

enum { kModeRange = 0, kModeList = 1, kModeGenes = 2 };

struct ListArgs {
  const uint64_t* idx;     // kModeList
  const int32_t* genes;    // kModeGenes [n][N]
  uint64_t n;
  float* score;
  uint8_t* feas;
  float* pred;             // [n][N][2] or null
};

__host__ __device__ constexpr int round4(int v) { return (v + 3) & ~3; }

// ---------------------------------------------------------------------------
// One model's predictor on one candidate, compile-time shape.
// w: the model's packed weights (16-byte aligned), z: the d_in inputs.
// ---------------------------------------------------------------------------
template <int DL, int H1, int H2>
__device__ __forceinline__ void predict_fixed(const float* __restrict__ w, const float* z,
                                              float& thr, float& lat) {
  constexpr int DIN = DL + 4;
  static_assert(DIN % 4 == 0 && H1 % 4 == 0 && H2 % 4 == 0, "vector loads need multiples of 4");
  const float4* W1 = reinterpret_cast<const float4*>(w);
  const float* b1 = w + H1 * DIN;
  float h1[H1];
#pragma unroll
  for (int j = 0; j < H1; ++j) {
    float s = b1[j];
#pragma unroll
    for (int k4 = 0; k4 < DIN / 4; ++k4) {
      const float4 v = W1[j * (DIN / 4) + k4];
      s = fmaf(v.x, z[4 * k4 + 0], s);
      s = fmaf(v.y, z[4 * k4 + 1], s);
      s = fmaf(v.z, z[4 * k4 + 2], s);
      s = fmaf(v.w, z[4 * k4 + 3], s);
    }
    h1[j] = relu(s);
  }
  const float* p = b1 + H1;
  float t, l;
  if constexpr (H2 > 0) {
    const float4* W2 = reinterpret_cast<const float4*>(p);
    const float* b2 = p + H2 * H1;
    const float* W3 = b2 + H2;
    const float* b3 = W3 + 2 * H2;
    t = b3[0];
    l = b3[1];
#pragma unroll 1
    for (int j = 0; j < H2; j += 4) {
      float a0 = b2[j], a1 = b2[j + 1], a2 = b2[j + 2], a3 = b2[j + 3];
#pragma unroll
      for (int k4 = 0; k4 < H1 / 4; ++k4) {
        const float4 w0 = W2[(j + 0) * (H1 / 4) + k4];
        const float4 w1 = W2[(j + 1) * (H1 / 4) + k4];
        const float4 w2 = W2[(j + 2) * (H1 / 4) + k4];
        const float4 w3 = W2[(j + 3) * (H1 / 4) + k4];
        const float x0 = h1[4 * k4], x1 = h1[4 * k4 + 1], x2 = h1[4 * k4 + 2], x3 = h1[4 * k4 + 3];
        a0 = fmaf(w0.x, x0, a0); a0 = fmaf(w0.y, x1, a0); a0 = fmaf(w0.z, x2, a0); a0 = fmaf(w0.w, x3, a0);
        a1 = fmaf(w1.x, x0, a1); a1 = fmaf(w1.y, x1, a1); a1 = fmaf(w1.z, x2, a1); a1 = fmaf(w1.w, x3, a1);
        a2 = fmaf(w2.x, x0, a2); a2 = fmaf(w2.y, x1, a2); a2 = fmaf(w2.z, x2, a2); a2 = fmaf(w2.w, x3, a2);
        a3 = fmaf(w3.x, x0, a3); a3 = fmaf(w3.y, x1, a3); a3 = fmaf(w3.z, x2, a3); a3 = fmaf(w3.w, x3, a3);
      }
      a0 = relu(a0); a1 = relu(a1); a2 = relu(a2); a3 = relu(a3);
      t = fmaf(W3[j], a0, t); t = fmaf(W3[j + 1], a1, t); t = fmaf(W3[j + 2], a2, t); t = fmaf(W3[j + 3], a3, t);
      l = fmaf(W3[H2 + j], a0, l); l = fmaf(W3[H2 + j + 1], a1, l);
      l = fmaf(W3[H2 + j + 2], a2, l); l = fmaf(W3[H2 + j + 3], a3, l);
    }
  } else {
    const float* W3 = p;
    const float* b3 = W3 + 2 * H1;
    t = b3[0];
    l = b3[1];
#pragma unroll
    for (int j = 0; j < H1; ++j) {
      t = fmaf(W3[j], h1[j], t);
      l = fmaf(W3[H1 + j], h1[j], l);
    }
  }
  thr = t;
  lat = l;
}

// Any shape (runtime sizes; hidden activations in local memory).
__device__ __noinline__ void predict_generic(const Params& P, const float* __restrict__ w,
                                             const float* z, float& thr, float& lat) {
  const int din = P.d_in, h1 = P.h1, h2 = P.h2;
  const float* W1 = w;
  const float* b1 = W1 + h1 * din;
  float a1[MF_MAX_HIDDEN];
  for (int j = 0; j < h1; ++j) {
    float s = b1[j];
    for (int k = 0; k < din; ++k) s = fmaf(W1[j * din + k], z[k], s);
    a1[j] = relu(s);
  }
  const float* p = b1 + h1;
  if (h2 > 0) {
    const float* W2 = p;
    const float* b2 = W2 + h2 * h1;
    const float* W3 = b2 + h2;
    const float* b3 = W3 + 2 * h2;
    float t = b3[0], l = b3[1];
    for (int j = 0; j < h2; ++j) {
      float s = b2[j];
      for (int k = 0; k < h1; ++k) s = fmaf(W2[j * h1 + k], a1[k], s);
      s = relu(s);
      t = fmaf(W3[j], s, t);
      l = fmaf(W3[h2 + j], s, l);
    }
    thr = t;
    lat = l;
  } else {
    const float* W3 = p;
    const float* b3 = W3 + 2 * h1;
    float t = b3[0], l = b3[1];
    for (int j = 0; j < h1; ++j) {
      t = fmaf(W3[j], a1[j], t);
      l = fmaf(W3[h1 + j], a1[j], l);
    }
    thr = t;
    lat = l;
  }
}

// ---------------------------------------------------------------------------
// Thread-per-candidate scorer.
// DL < 0 selects the generic predictor (weights read from global memory).
// ---------------------------------------------------------------------------
template <int DL, int H1, int H2, int MODE, bool RESIDENT>
__global__ void __launch_bounds__(kScoreThreads, 1)
k_score_f32(const Params P, const RangeArgs R, const ListArgs L) {
  extern __shared__ __align__(16) unsigned char smem[];
  constexpr bool kFixed = DL > 0;
  constexpr int kZ = kFixed ? DL + 4 : MF_MAX_D_LOCAL + 4;
  const int tid = threadIdx.x;
  const int N = P.n_models;
  const int stride = (int)P.per_model;  // floats between models (multiple of 4)

  // ---- stage the predictors in shared memory (one copy per CTA) ----
  float* sw = reinterpret_cast<float*>(smem);
  size_t wfloats = RESIDENT ? (size_t)N * stride : 0;
  if (RESIDENT) {
    const float4* src = reinterpret_cast<const float4*>(P.w32);
    float4* dst = reinterpret_cast<float4*>(sw);
    for (size_t e = tid; e < wfloats / 4; e += blockDim.x) dst[e] = src[e];
  }
  // ---- top-k state (range mode) ----
  CtaTopK tk{};
  unsigned int my_count = 0;
  float thr_s = -INFINITY;
  uint64_t thr_i = kEmptyIdx;
  if (MODE == kModeRange) {
    unsigned char* q = smem + wfloats * sizeof(float);
    const int k = R.k;
    tk.li = reinterpret_cast<uint64_t*>(q); q += sizeof(uint64_t) * k;
    tk.ni = reinterpret_cast<uint64_t*>(q); q += sizeof(uint64_t) * k;
    tk.qi = reinterpret_cast<uint64_t*>(q); q += sizeof(uint64_t) * kScoreThreads;
    tk.ls = reinterpret_cast<float*>(q); q += sizeof(float) * k;
    tk.ns = reinterpret_cast<float*>(q); q += sizeof(float) * k;
    tk.qs = reinterpret_cast<float*>(q); q += sizeof(float) * kScoreThreads;
    tk.qn = reinterpret_cast<int*>(q);
    tk.k = k;
    const size_t base = (size_t)blockIdx.x * k;
    for (int e = tid; e < k; e += blockDim.x) {
      tk.ls[e] = R.first ? -INFINITY : R.lists_s[base + e];
      tk.li[e] = R.first ? kEmptyIdx : R.lists_i[base + e];
    }
    if (tid == 0) *tk.qn = 0;
  }
  __syncthreads();
  if (MODE == kModeRange) {
    thr_s = tk.ls[R.k - 1];
    thr_i = tk.li[R.k - 1];
  }

  const uint64_t n = MODE == kModeRange ? R.len : L.n;
  for (uint64_t tile = blockIdx.x; tile * kScoreThreads < n; tile += gridDim.x) {
    const uint64_t t = tile * kScoreThreads + tid;
    bool valid = t < n;
    uint64_t idx = 0;
    if (valid) {
      if (MODE == kModeRange) idx = R.base + t;
      else if (MODE == kModeList) idx = L.idx[t];
      else idx = t;
    }
    if (MODE == kModeList && valid && idx >= P.total) {
      atomicOr(P.status, kStatusBadInput);
      valid = false;
    }
    // digits of every model
    auto digit = [&](int i) -> int {
      if (MODE == kModeGenes) return L.genes[t * N + i];
      return digit_of(P, idx, i);
    };
    // aggregate state: summed demand of the chosen options (model order) and N
    float A0 = 0.f, A1 = 0.f, A2 = 0.f;
    if (valid) {
      for (int i = 0; i < N; ++i) {
        int o = digit(i);
        if (MODE == kModeGenes && (o < 0 || o >= P.K[i])) {
          atomicOr(P.status, kStatusBadInput);
          valid = false;
          break;
        }
        const float4 d = __ldg(&P.dem[P.off[i] + o]);
        A0 += d.x; A1 += d.y; A2 += d.z;
      }
    }
    Acc acc;
    acc.init();
    bool feas = false;
    if (valid) {
      float z[kZ];
      const int dl = kFixed ? DL : P.d_local;
      z[dl + 0] = A0 * P.agg_scale[0];
      z[dl + 1] = A1 * P.agg_scale[1];
      z[dl + 2] = A2 * P.agg_scale[2];
      z[dl + 3] = (float)N * P.agg_scale[3];
      for (int i = 0; i < N; ++i) {
        const int row = P.off[i] + digit(i);
        if constexpr (kFixed) {
          const float4* xr = reinterpret_cast<const float4*>(P.x + (size_t)row * DL);
#pragma unroll
          for (int k4 = 0; k4 < DL / 4; ++k4) {
            const float4 v = __ldg(xr + k4);
            z[4 * k4] = v.x; z[4 * k4 + 1] = v.y; z[4 * k4 + 2] = v.z; z[4 * k4 + 3] = v.w;
          }
        } else {
          for (int k = 0; k < dl; ++k) z[k] = __ldg(P.x + (size_t)row * dl + k);
        }
        const float* wm = RESIDENT ? sw + (size_t)i * stride : P.w32 + (size_t)i * stride;
        float thr, lat;
        if constexpr (kFixed) predict_fixed<(kFixed ? DL : 4), (kFixed ? H1 : 4), (kFixed ? H2 : 0)>(wm, z, thr, lat);
        else predict_generic(P, wm, z, thr, lat);
        thr = out_act(P, thr);
        lat = out_act(P, lat);
        if (MODE != kModeRange && L.pred) {
          L.pred[(t * N + i) * 2 + 0] = thr;
          L.pred[(t * N + i) * 2 + 1] = lat;
        }
        acc.add(P, i, thr, lat, row);
      }
      feas = acc.finish(P, A1);
    } else {
      acc.J = -INFINITY;
      if (MODE != kModeRange && L.pred && t < n)
        for (int i = 0; i < N; ++i) {
          L.pred[(t * N + i) * 2 + 0] = __int_as_float(0x7fc00000);
          L.pred[(t * N + i) * 2 + 1] = __int_as_float(0x7fc00000);
        }
    }

    if (MODE == kModeRange) {
      my_count += feas ? 1u : 0u;
      const bool push = feas && precedes(acc.J, idx, thr_s, thr_i);
      if (push) {
        const int pos = atomicAdd(tk.qn, 1);
        tk.qs[pos] = acc.J;
        tk.qi[pos] = idx;
      }
      // the barrier's OR is block-uniform, so every thread takes the same branch
      if (__syncthreads_or(push)) {  // a long queue (early in a search) is sorted first
        if (*tk.qn > 256) topk_merge_sorted(tk, tid, blockDim.x, [] __device__() { __syncthreads(); });
        else topk_merge(tk, tid, blockDim.x, [] __device__() { __syncthreads(); });
        thr_s = tk.ls[R.k - 1];
        thr_i = tk.li[R.k - 1];
      }
    } else if (t < n) {
      L.score[t] = acc.J;
      if (L.feas) L.feas[t] = feas ? 1 : 0;
    }
  }

  if (MODE == kModeRange) {
    const size_t base = (size_t)blockIdx.x * R.k;
    for (int e = tid; e < R.k; e += blockDim.x) {
      R.lists_s[base + e] = tk.ls[e];
      R.lists_i[base + e] = tk.li[e];
    }
    unsigned int c = my_count;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
    if ((tid & 31) == 0 && c) atomicAdd(R.count, (unsigned long long)c);
  }
}

// ---------------------------------------------------------------------------
// Warp-per-(candidate, model) predictor for small batches.
// U1 = ceil(h1 / 32) units per lane in layer 1, U2 = ceil(h2 / 32) (0: no layer 2).
// Weights come from the transposed copy: W1T[d_in][h1], b1, W2T[h1][h2], b2, W3[2][h], b3.
// ---------------------------------------------------------------------------
template <int U1, int U2>
__global__ void __launch_bounds__(kWideWarps * 32)
k_wide_f32(const Params P, const uint64_t* __restrict__ idx, const int32_t* __restrict__ genes,
           uint64_t n, float* __restrict__ pred, int allow_empty) {
  const int lane = threadIdx.x & 31;
  const uint64_t warp = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t nwarps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  const int N = P.n_models, dl = P.d_local, din = P.d_in, h1 = P.h1, h2 = P.h2;
  const uint64_t tasks = n * (uint64_t)N;
  for (uint64_t task = warp; task < tasks; task += nwarps) {
    const uint64_t cand = task / N;
    const int m = (int)(task % N);
    // lane j < N resolves model j's option and demand
    int o = 0;
    bool ok = true;
    float4 d = make_float4(0.f, 0.f, 0.f, 0.f);
    if (lane < N) {
      if (genes) {
        o = genes[cand * N + lane];
        ok = o >= 0 && o < P.K[lane];
      } else {
        const uint64_t id = idx[cand];
        ok = id < P.total;
        if (ok) o = digit_of(P, id, lane);
      }
      if (ok) d = __ldg(&P.dem[P.off[lane] + o]);
    }
    const bool all_ok = __all_sync(0xffffffffu, ok);
    if (!all_ok) {
      if (lane == 0) {
        const bool empty = allow_empty && !genes && idx[cand] == kEmptyIdx;
        if (m == 0 && !empty) atomicOr(P.status, kStatusBadInput);
        pred[(cand * N + m) * 2 + 0] = __int_as_float(0x7fc00000);
        pred[(cand * N + m) * 2 + 1] = __int_as_float(0x7fc00000);
      }
      continue;
    }
    // aggregate: sum over models in model order (lane 0 accumulates by shuffles)
    float A0 = 0.f, A1 = 0.f, A2 = 0.f;
    for (int j = 0; j < N; ++j) {
      A0 += __shfl_sync(0xffffffffu, d.x, j);
      A1 += __shfl_sync(0xffffffffu, d.y, j);
      A2 += __shfl_sync(0xffffffffu, d.z, j);
    }
    const int om = __shfl_sync(0xffffffffu, o, m);
    const int row = P.off[m] + om;
    float zown = 0.f;
    if (lane < dl) zown = __ldg(P.x + (size_t)row * dl + lane);
    else if (lane == dl) zown = A0 * P.agg_scale[0];
    else if (lane == dl + 1) zown = A1 * P.agg_scale[1];
    else if (lane == dl + 2) zown = A2 * P.agg_scale[2];
    else if (lane == dl + 3) zown = (float)N * P.agg_scale[3];

    const float* w = P.wT + (size_t)m * P.per_model;
    const float* W1T = w;
    const float* b1 = W1T + (size_t)din * h1;
    float hv1[U1];
#pragma unroll
    for (int u = 0; u < U1; ++u) {
      const int j = lane + 32 * u;
      float s = j < h1 ? __ldg(b1 + j) : 0.f;
      for (int k = 0; k < din; ++k) {
        const float zk = __shfl_sync(0xffffffffu, zown, k);
        if (j < h1) s = fmaf(__ldg(W1T + (size_t)k * h1 + j), zk, s);
      }
      hv1[u] = j < h1 ? relu(s) : 0.f;
    }
    const float* p = b1 + h1;
    float t = 0.f, l = 0.f;
    if constexpr (U2 > 0) {
      const float* W2T = p;
      const float* b2 = W2T + (size_t)h1 * h2;
      const float* W3 = b2 + h2;
      float acc2[U2];
#pragma unroll
      for (int u2 = 0; u2 < U2; ++u2) {
        const int j = lane + 32 * u2;
        acc2[u2] = j < h2 ? __ldg(b2 + j) : 0.f;
      }
#pragma unroll
      for (int u = 0; u < U1; ++u) {
#pragma unroll
        for (int kk = 0; kk < 32; ++kk) {
          const int k = 32 * u + kk;
          if (k < h1) {
            const float hk = __shfl_sync(0xffffffffu, hv1[u], kk);
#pragma unroll
            for (int u2 = 0; u2 < U2; ++u2) {
              const int j = lane + 32 * u2;
              if (j < h2) acc2[u2] = fmaf(__ldg(W2T + (size_t)k * h2 + j), hk, acc2[u2]);
            }
          }
        }
      }
#pragma unroll
      for (int u2 = 0; u2 < U2; ++u2) {
        const int j = lane + 32 * u2;
        if (j < h2) {
          const float a = relu(acc2[u2]);
          t = fmaf(__ldg(W3 + j), a, t);
          l = fmaf(__ldg(W3 + h2 + j), a, l);
        }
      }
    } else {
      const float* W3 = p;
#pragma unroll
      for (int u = 0; u < U1; ++u) {
        const int j = lane + 32 * u;
        if (j < h1) {
          t = fmaf(__ldg(W3 + j), hv1[u], t);
          l = fmaf(__ldg(W3 + h1 + j), hv1[u], l);
        }
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      t += __shfl_xor_sync(0xffffffffu, t, off);
      l += __shfl_xor_sync(0xffffffffu, l, off);
    }
    if (lane == 0) {
      const int hl = h2 > 0 ? h2 : h1;
      const float* b3 = w + (size_t)din * h1 + h1 + (h2 > 0 ? (size_t)h1 * h2 + h2 : 0) + 2 * hl;
      pred[(cand * N + m) * 2 + 0] = out_act(P, t + __ldg(b3));
      pred[(cand * N + m) * 2 + 1] = out_act(P, l + __ldg(b3 + 1));
    }
  }
}

// Objective and constraints from per-model outputs (thread per candidate).
__global__ void k_combine(const Params P, const uint64_t* __restrict__ idx,
                          const int32_t* __restrict__ genes, uint64_t n,
                          const float* __restrict__ pred, float* __restrict__ score,
                          uint8_t* __restrict__ feas, int allow_empty) {
  const uint64_t t = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n) return;
  const int N = P.n_models;
  bool ok = true;
  float A1 = 0.f;
  uint64_t id = genes ? 0 : idx[t];
  if (!genes && id >= P.total) ok = false;
  for (int i = 0; i < N && ok; ++i) {
    const int o = genes ? genes[t * N + i] : digit_of(P, id, i);
    if (o < 0 || o >= P.K[i]) { ok = false; break; }
    A1 += __ldg(&P.dem[P.off[i] + o]).y;
  }
  bool f = false;
  float J = -INFINITY;
  if (ok) {
    Acc acc;
    acc.init();
    for (int i = 0; i < N; ++i) {
      const int o = genes ? genes[t * N + i] : digit_of(P, id, i);
      acc.add(P, i, pred[(t * N + i) * 2], pred[(t * N + i) * 2 + 1], P.off[i] + o);
    }
    f = acc.finish(P, A1);
    J = acc.J;
  }
  score[t] = J;
  if (feas) feas[t] = f ? 1 : 0;
}

// ---------------------------------------------------------------------------
// Host-side dispatch
// ---------------------------------------------------------------------------
namespace {

struct ShapeKey { int dl, h1, h2; };
constexpr ShapeKey kFixedShapes[] = {{8, 32, 0}, {8, 64, 64}, {8, 64, 32}, {16, 128, 128}, {8, 32, 32}};

int fixed_shape_id(const Params& P) {
  for (int s = 0; s < (int)(sizeof(kFixedShapes) / sizeof(kFixedShapes[0])); ++s)
    if (kFixedShapes[s].dl == P.d_local && kFixedShapes[s].h1 == P.h1 && kFixedShapes[s].h2 == P.h2)
      return s;
  return -1;
}

using ScoreFn = void (*)(const Params, const RangeArgs, const ListArgs);

template <int MODE, bool RES>
ScoreFn pick(int shape) {
  switch (shape) {
    case 0: return k_score_f32<8, 32, 0, MODE, RES>;
    case 1: return k_score_f32<8, 64, 64, MODE, RES>;
    case 2: return k_score_f32<8, 64, 32, MODE, RES>;
    case 3: return k_score_f32<16, 128, 128, MODE, RES>;
    case 4: return k_score_f32<8, 32, 32, MODE, RES>;
    default: return k_score_f32<-1, 0, 0, MODE, false>;
  }
}

ScoreFn pick_fn(int mode, int shape, bool res) {
  if (shape < 0) res = false;
  if (mode == kModeRange) return res ? pick<kModeRange, true>(shape) : pick<kModeRange, false>(shape);
  if (mode == kModeList) return res ? pick<kModeList, true>(shape) : pick<kModeList, false>(shape);
  return res ? pick<kModeGenes, true>(shape) : pick<kModeGenes, false>(shape);
}

constexpr size_t kSmemBudget = 200 * 1024;

size_t topk_bytes(int k) {
  return (sizeof(uint64_t) + sizeof(float)) * (2 * (size_t)k + kScoreThreads) + 16;
}

}  // namespace

bool f32_supported(const Params& P) { return P.d_local <= MF_MAX_D_LOCAL; }

size_t f32_smem_bytes(const Params& P, int k, bool& resident) {
  const size_t wbytes = (size_t)P.n_models * P.per_model * sizeof(float);
  const size_t tk = k > 0 ? topk_bytes(k) : 0;
  resident = fixed_shape_id(P) >= 0 && wbytes + tk <= kSmemBudget;
  return (resident ? wbytes : 0) + tk;
}

int f32_grid(const mf_ctx* c) { return c->num_sms; }

mf_status f32_prepare(mf_ctx* c) {
  const int shape = fixed_shape_id(c->P);
  for (int mode = 0; mode < 3; ++mode)
    for (int res = 0; res < 2; ++res) {
      ScoreFn fn = pick_fn(mode, shape, res != 0);
      MF_CUDA(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024));
    }
  return MF_OK;
}

mf_status f32_search_chunk(mf_ctx* c, const RangeArgs& a, cudaStream_t s) {
  bool res;
  const size_t smem = f32_smem_bytes(c->P, a.k, res);
  ScoreFn fn = pick_fn(kModeRange, fixed_shape_id(c->P), res);
  ListArgs L{};
  fn<<<f32_grid(c), kScoreThreads, smem, s>>>(c->P, a, L);
  MF_CUDA(cudaGetLastError());
  return MF_OK;
}

template <int U1, int U2>
static void launch_wide(const Params& P, const uint64_t* idx, const int32_t* genes, uint64_t n,
                        float* pred, int grid, cudaStream_t s, int allow_empty) {
  k_wide_f32<U1, U2><<<grid, kWideWarps * 32, 0, s>>>(P, idx, genes, n, pred, allow_empty);
}

static mf_status score_wide(mf_ctx* c, const uint64_t* idx, const int32_t* genes, uint64_t n,
                            float* score, uint8_t* feas, float* pred, cudaStream_t s, int allow_empty) {
  const Params& P = c->P;
  const uint64_t tasks = n * (uint64_t)P.n_models;
  {  // grid: up to four 8-warp CTAs per SM, warps loop over the tasks
    const int u1 = (P.h1 + 31) / 32, u2 = (P.h2 + 31) / 32;
    const uint64_t blocks = (tasks + kWideWarps - 1) / kWideWarps;
    const int grid = (int)(blocks < 4ull * c->num_sms ? blocks : 4ull * c->num_sms);
    if (u2 == 0) {
      if (u1 <= 1) launch_wide<1, 0>(P, idx, genes, n, pred, grid, s, allow_empty);
      else if (u1 <= 2) launch_wide<2, 0>(P, idx, genes, n, pred, grid, s, allow_empty);
      else if (u1 <= 4) launch_wide<4, 0>(P, idx, genes, n, pred, grid, s, allow_empty);
      else launch_wide<8, 0>(P, idx, genes, n, pred, grid, s, allow_empty);
    } else {
      const int u = u1 > u2 ? u1 : u2;
      if (u <= 1) launch_wide<1, 1>(P, idx, genes, n, pred, grid, s, allow_empty);
      else if (u <= 2) launch_wide<2, 2>(P, idx, genes, n, pred, grid, s, allow_empty);
      else if (u <= 4) launch_wide<4, 4>(P, idx, genes, n, pred, grid, s, allow_empty);
      else launch_wide<8, 8>(P, idx, genes, n, pred, grid, s, allow_empty);
    }
    MF_CUDA(cudaGetLastError());
    k_combine<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(P, idx, genes, n, pred, score, feas,
                                                           allow_empty);
    MF_CUDA(cudaGetLastError());
    return MF_OK;
  }
}

mf_status f32_score_list_ex(mf_ctx* c, const uint64_t* idx, uint64_t n, float* score, float* pred,
                            cudaStream_t s) {
  if (n == 0) return MF_OK;
  return score_wide(c, idx, nullptr, n, score, nullptr, pred, s, 1);
}

mf_status f32_score_list(mf_ctx* c, const uint64_t* idx, const int32_t* genes, uint64_t n,
                         float* score, uint8_t* feas, float* pred, cudaStream_t s) {
  if (n == 0) return MF_OK;
  const Params& P = c->P;
  const uint64_t tasks = n * (uint64_t)P.n_models;
  // Small batches: warp per (candidate, model), then a combine pass.
  if (tasks <= 64ull * 1024 && pred != nullptr) return score_wide(c, idx, genes, n, score, feas, pred, s, 0);
  bool res;
  const size_t smem = f32_smem_bytes(P, 0, res);
  ScoreFn fn = pick_fn(genes ? kModeGenes : kModeList, fixed_shape_id(P), res);
  RangeArgs R{};
  ListArgs L{idx, genes, n, score, feas, pred};
  const uint64_t tiles = (n + kScoreThreads - 1) / kScoreThreads;
  const int grid = (int)(tiles < (uint64_t)c->num_sms ? tiles : (uint64_t)c->num_sms);
  fn<<<grid, kScoreThreads, smem, s>>>(P, R, L);
  MF_CUDA(cudaGetLastError());
  return MF_OK;
}

}  // namespace mf

namespace mf {

// Range-mode launch from a bare parameter block (no context): sets the kernel's
// shared-memory limit and launches one chunk on `grid` CTAs.
mf_status f32_search_chunk_params(const Params& P, int grid, const RangeArgs& a, cudaStream_t s) {
  bool res;
  const size_t smem = f32_smem_bytes(P, a.k, res);
  ScoreFn fn = pick_fn(kModeRange, fixed_shape_id(P), res);
  MF_CUDA(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024));
  ListArgs L{};
  fn<<<grid, kScoreThreads, smem, s>>>(P, a, L);
  MF_CUDA(cudaGetLastError());
  return MF_OK;
}

}  // namespace mf
