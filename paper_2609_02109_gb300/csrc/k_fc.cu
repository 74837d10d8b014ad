// Fixed-context mode (arXiv 2609.02109, Sec. III-B): the observed GPU state s_t is
// held fixed during the search, so predictor g_i(lambda_i, s_t) depends on model i's
// option only.  The sum K_i local predictions are evaluated once (k_fc_local) into a
// per-option table of the utility term of Eq. 3,
//   u = omega_i f Q - alpha eta c_i - beta max(0, tau_i + delta - f)^2,
//   f = (fhat - f_min) / (f_max - f_min)   (per-variant normalisation),
// and a joint configuration's J is the sum of its options' terms (Eq. 3), -inf when a
// floor f_i >= tau_i or the VRAM bound of Eq. 4 fails.  The exhaustive search is then
// a table-lookup scan (k_fc_scan, ALU-bound); k_vram_count / k_vram_write build the
// VRAM-feasible space (Lambda without its VRAM-infeasible configurations) as an
// ascending index list.
#include <cmath>
#include <cstring>
#include <string>
#include <vector>

#include "mf_internal.cuh"

namespace mf {

// Device layout of mf_ctx::d_fc.
struct FcLayout {
  float2* tab;       // [sumK] (u, or -inf below the floor; VRAM of the option)
  float* fhat;       // [sumK]
  float* f;          // [sumK]
  float* u;          // [sumK]
  uint8_t* ok;       // [sumK]
  // inputs, copied
  float* obs;        // [4]
  int32_t* variant;  // [sumK]
  float* quality;    // [sumK]
  float* f_min;      // [sumK]
  float* f_max;      // [sumK]
  float* omega;      // [N]
  float* tau;        // [N]
  float* cost;       // [N]
  int32_t* prev;     // [N]
};

static size_t fc_bytes(int sumK, int N, FcLayout* L, char* base) {
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o = (o + bytes + 255) / 256 * 256;
    return base ? base + at : nullptr;
  };
  char* p;
  p = take(sizeof(float2) * sumK); if (L) L->tab = (float2*)p;
  p = take(sizeof(float) * sumK); if (L) L->fhat = (float*)p;
  p = take(sizeof(float) * sumK); if (L) L->f = (float*)p;
  p = take(sizeof(float) * sumK); if (L) L->u = (float*)p;
  p = take(sumK); if (L) L->ok = (uint8_t*)p;
  p = take(sizeof(float) * 4); if (L) L->obs = (float*)p;
  p = take(sizeof(int32_t) * sumK); if (L) L->variant = (int32_t*)p;
  p = take(sizeof(float) * sumK); if (L) L->quality = (float*)p;
  p = take(sizeof(float) * sumK); if (L) L->f_min = (float*)p;
  p = take(sizeof(float) * sumK); if (L) L->f_max = (float*)p;
  p = take(sizeof(float) * N); if (L) L->omega = (float*)p;
  p = take(sizeof(float) * N); if (L) L->tau = (float*)p;
  p = take(sizeof(float) * N); if (L) L->cost = (float*)p;
  p = take(sizeof(int32_t) * N); if (L) L->prev = (int32_t*)p;
  return o;
}

struct FcConst {
  float alpha, beta, delta;
};

// ---------------------------------------------------------------------------
// Local predictions: one CTA per option row.  z = [x_i(o) | obs * s_A]; the hidden
// layers spread their units over the threads; the throughput head reduces over
// warp 0.  Thread 0 forms f, the floor flag and u.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
k_fc_local(const Params P, const FcLayout L, const FcConst C) {
  __shared__ float z[MF_MAX_D_LOCAL + 4];
  __shared__ float h1[MF_MAX_HIDDEN], h2[MF_MAX_HIDDEN];
  __shared__ int s_model;
  const int r = blockIdx.x, tid = threadIdx.x;
  const int N = P.n_models;
  if (tid == 0) {
    int m = 0;
    for (int i = 0; i < N; ++i)
      if (r >= pick(P.off, i)) m = i;
    s_model = m;
  }
  const int dl = P.d_local, din = P.d_in, H1 = P.h1, H2 = P.h2;
  for (int k = tid; k < dl; k += blockDim.x) z[k] = P.x[(size_t)r * dl + k];
  if (tid < 4) z[dl + tid] = L.obs[tid] * P.agg_scale[tid];
  __syncthreads();
  const int m = s_model;
  const float* w = P.w32 + (size_t)m * P.per_model;
  const float* W1 = w;
  const float* b1 = W1 + (size_t)H1 * din;
  for (int j = tid; j < H1; j += blockDim.x) {
    float s = b1[j];
    for (int k = 0; k < din; ++k) s = fmaf(W1[(size_t)j * din + k], z[k], s);
    h1[j] = relu(s);
  }
  __syncthreads();
  const float* next = b1 + H1;
  const float* h = h1;
  int hl = H1;
  if (H2 > 0) {
    const float* W2 = next;
    const float* b2 = W2 + (size_t)H2 * H1;
    for (int j = tid; j < H2; j += blockDim.x) {
      float s = b2[j];
      for (int k = 0; k < H1; ++k) s = fmaf(W2[(size_t)j * H1 + k], h1[k], s);
      h2[j] = relu(s);
    }
    __syncthreads();
    next = b2 + H2;
    h = h2;
    hl = H2;
  }
  if (tid < 32) {
    const float* W3 = next;  // row 0: the throughput head
    float s = 0.f;
    for (int k = tid; k < hl; k += 32) s = fmaf(W3[k], h[k], s);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (tid == 0) {
      const float fhat = out_act(P, s + W3[2 * hl]);
      const float f = (fhat - L.f_min[r]) / (L.f_max[r] - L.f_min[r]);
      const float tau = L.tau[m];
      const bool ok = f >= tau;
      const float eta = (L.prev[m] >= 0 && L.variant[r] != L.prev[m]) ? 1.f : 0.f;
      const float margin = tau + C.delta - f;
      const float u = L.omega[m] * f * L.quality[r] - C.alpha * eta * L.cost[m] -
                      C.beta * (margin > 0.f ? margin * margin : 0.f);
      L.fhat[r] = fhat;
      L.f[r] = f;
      L.u[r] = u;
      L.ok[r] = ok ? 1 : 0;
      L.tab[r] = make_float2(ok ? u : -INFINITY, P.dem[r].y);
    }
  }
}

// ---------------------------------------------------------------------------
// Table-lookup scan.  Each thread walks its own contiguous slice of the range, so from
// one candidate to the next only the last model's option advances: the partial sum over
// the other models is reused until a carry, and a carry that stops at model N - 2 (all
// but one in K_{N-2}) costs one lookup.  J is summed in model order either way.
// Running top-k: a thread queues a candidate only if it beats the list's k-th entry
// (held in registers), at most kFcBudget between two merge checks (a thread that runs
// out stops until the merge); a merge check follows every cycle of the last model's
// options, at least kFcMinRun candidates (kFcMinRunLong in slices long enough that the
// list settles early).  WL (k <= kFcWarpK): each warp keeps its own list and queue and
// merges with warp barriers only, the CTA's list taking the warps' lists at the end;
// otherwise one list per CTA, the merge check a CTA barrier.
// ---------------------------------------------------------------------------
constexpr int kFcThreads = 512;
constexpr int kFcBudget = 8;   // the queue: kFcThreads x kFcBudget entries
constexpr int kFcMinRun = 16, kFcMinRunLong = 64;
constexpr int kFcWarpK = 64, kFcWarps = kFcThreads / 32;
constexpr int kFcWarpQ = 32 * kFcBudget;              // a warp's queue
constexpr int kFcEndQ = kFcWarps * kFcWarpK;          // the warps' lists, merged at the end (a power of two)
constexpr uint64_t kFcLongSlice = 8192;

struct FcScan {
  const float2* tab;
};

// Shared-memory bytes of k_fc_scan<.., WL> after the table.
__host__ __device__ inline size_t fc_scan_list_bytes(int k, bool wl) {
  const size_t e = sizeof(uint64_t) + sizeof(float);
  if (!wl) return e * (2 * (size_t)k + kFcThreads * kFcBudget) + 16;
  return e * (2 * (size_t)k + kFcEndQ) + 16 + kFcWarps * (e * (2 * (size_t)k + kFcWarpQ) + 16);
}

template <int NMAX, bool WL>
__global__ void __launch_bounds__(kFcThreads, 1)
k_fc_scan(const Params P, const FcScan S, const RangeArgs R) {
  // NMAX: a bound on N for the unrolled per-model loops
  extern __shared__ __align__(16) unsigned char sm[];
  const int N = P.n_models;
  const int sumK = pick(P.off, N - 1) + pick(P.K, N - 1);
  constexpr int QCAP = WL ? kFcEndQ : kFcThreads * kFcBudget;
  float2* tab = reinterpret_cast<float2*>(sm);
  unsigned char* q = sm + (((size_t)sumK * sizeof(float2) + 15) & ~(size_t)15);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // one list + queue block: li, ni [k], qi [qcap], ls, ns [k], qs [qcap], qn
  auto carve = [&](CtaTopK& t, int qcap) {
    t.li = reinterpret_cast<uint64_t*>(q); q += sizeof(uint64_t) * R.k;
    t.ni = reinterpret_cast<uint64_t*>(q); q += sizeof(uint64_t) * R.k;
    t.qi = reinterpret_cast<uint64_t*>(q); q += sizeof(uint64_t) * qcap;
    t.ls = reinterpret_cast<float*>(q); q += sizeof(float) * R.k;
    t.ns = reinterpret_cast<float*>(q); q += sizeof(float) * R.k;
    t.qs = reinterpret_cast<float*>(q); q += sizeof(float) * qcap;
    t.qn = reinterpret_cast<int*>(q); q += 16;
    t.k = R.k;
  };
  CtaTopK tk, wt;  // the CTA's list; this warp's (WL), else the CTA's again
  carve(tk, QCAP);
  if (WL) {  // the warps' blocks follow the CTA's, in warp order
    q += (size_t)warp * ((sizeof(uint64_t) + sizeof(float)) * (2 * (size_t)R.k + kFcWarpQ) + 16);
    carve(wt, kFcWarpQ);
    for (int e = lane; e < R.k; e += 32) { wt.ls[e] = -INFINITY; wt.li[e] = kEmptyIdx; }
    if (lane == 0) *wt.qn = 0;
  } else {
    wt = tk;
  }
  // an option below its floor (utility -inf, or NaN) carries VRAM +inf here, so one
  // compare against the cap decides feasibility
  for (int e = tid; e < sumK; e += blockDim.x) {
    float2 v = S.tab[e];
    if (!(v.x > -INFINITY)) v.y = INFINITY;
    tab[e] = v;
  }
  const size_t gl = (size_t)blockIdx.x * R.k;
  for (int e = tid; e < R.k; e += blockDim.x) {
    tk.ls[e] = R.first ? -INFINITY : R.lists_s[gl + e];
    tk.li[e] = R.first ? kEmptyIdx : R.lists_i[gl + e];
  }
  if (tid == 0) *tk.qn = 0;
  // Thread g of the grid scans the contiguous slice [g S, (g + 1) S) of the range.
  // S = ceil(len / threads); in long scans rounded up to a multiple of the last model's
  // option count, so all lanes of a warp run the same cycles of the last model's options
  // (the same table entries, no divergence), while short scans keep slices short (a small
  // first merge, spread over more CTAs).
  const uint64_t nthreads = (uint64_t)gridDim.x * blockDim.x;
  const int last = N - 1;
  const int off_last = pick(P.off, last);
  const int klast = pick(P.K, last);
  const uint64_t slice0 = (R.len + nthreads - 1) / nthreads;
  const uint64_t slice = slice0 >= 4 * (uint64_t)klast ? (slice0 + klast - 1) / klast * klast : slice0;
  const uint64_t s0 = ((uint64_t)blockIdx.x * blockDim.x + tid) * slice;
  const uint64_t s1 = s0 + slice < R.len ? s0 + slice : R.len;
  int row[NMAX];  // option rows of models 0 .. N - 2
  int o;          // the last model's option
  {
    const uint64_t idx0 = R.base + (s0 < R.len ? s0 : 0);
#pragma unroll
    for (int i = 0; i < NMAX; ++i)
      if (i < last) row[i] = P.off[i] + (int)((idx0 / P.stride[i]) % (uint64_t)P.K[i]);
    o = (int)((idx0 / pick(P.stride, last)) % (uint64_t)klast);
  }
  __syncthreads();
  float thr_s = tk.ls[R.k - 1];
  uint64_t thr_i = tk.li[R.k - 1];
  const float cap = P.vram_cap;
  // prefix sums in model order: p2 over models 0 .. N - 3, p over 0 .. N - 2; rp is
  // model N - 2's option row (the one a carry usually stops at), endp its end
  float pJ2 = 0.f, pV2 = 0.f, pJ = 0.f, pV = 0.f;
  int rp = 0, endp = 0;
  auto prefix = [&]() {
    pJ2 = 0.f;
    pV2 = 0.f;
#pragma unroll
    for (int i = 0; i < NMAX; ++i)
      if (i < last - 1) { const float2 e = tab[row[i]]; pJ2 += e.x; pV2 += e.y; }
    pJ = pJ2;
    pV = pV2;
    if (last >= 1) {
#pragma unroll
      for (int i = 0; i < NMAX; ++i)
        if (i == last - 1) rp = row[i];
      const float2 e = tab[rp];
      pJ += e.x;
      pV += e.y;
    }
  };
  if (last >= 1) endp = pick(P.off, last - 1) + pick(P.K, last - 1);
  prefix();
  const float thr0_s = thr_s;  // (WL: the bar until the warp's own list is full)
  const uint64_t thr0_i = thr_i;
  // the last model's option wrapped: the next option of the models before it
  auto carry = [&]() {
    if (++rp < endp) {
      const float2 e = tab[rp];
      pJ = pJ2 + e.x;
      pV = pV2 + e.y;
      return;
    }
    bool c = true;  // model N - 2 wrapped as well
#pragma unroll
    for (int i = NMAX - 1; i >= 0; --i)
      if (i < last && c) {
        const int off = P.off[i];
        int d = (i == last - 1 ? rp : row[i] + 1) - off;
        c = d == P.K[i];
        if (c) d = 0;
        row[i] = off + d;
      }
    prefix();
  };
  const float2* tl = tab + off_last;
  const int minrun = slice >= kFcLongSlice ? kFcMinRunLong : kFcMinRun;
  uint64_t t = s0;  // this thread's next candidate (offset in the range)
  bool done = t >= s1;
  unsigned int my_count = 0;
  for (;;) {
    int pushed = 0, ran = 0;
    while (!done && ran < minrun) {
      const int n_here = s1 - t < (uint64_t)(klast - o) ? (int)(s1 - t) : klast - o;
      const float2* e0 = tl + o;
      // fast pass: the count, and whether any candidate might enter the list
      bool hit = false;
      const float2 pjv = make_float2(pJ, pV);
#pragma unroll 8
      for (int u = 0; u < n_here; ++u) {
        const float2 jv = __fadd2_rn(pjv, e0[u]);  // (J, V) = (pJ + x, pV + y), one paired add
        const bool feas = jv.y <= cap;  // NaN compares false
        my_count += feas ? 1u : 0u;
        hit |= feas & (jv.x >= thr_s);
      }
      int u = n_here;
      if (hit) {  // rare once the list is full: queue what beats its k-th entry
        for (u = 0; u < n_here; ++u) {
          const float2 e = e0[u];
          const float J = pJ + e.x, V = pV + e.y;
          if (V <= cap && J >= thr_s) {
            const uint64_t idx = R.base + t + u;
            if (precedes(J, idx, thr_s, thr_i)) {
              if (pushed == kFcBudget) break;  // this candidate and the rest wait for the merge
              const int pos = atomicAdd(wt.qn, 1);
              wt.qs[pos] = J;
              wt.qi[pos] = idx;
              ++pushed;
            }
          }
        }
        for (int w = u; w < n_here; ++w) my_count -= (pV + e0[w].y <= cap) ? 1u : 0u;  // counted again later
      }
      t += u;
      o += u;
      ran += u;
      if (t >= s1) done = true;
      else if (o == klast) { o = 0; carry(); }
      if (u < n_here) break;
    }
    if (WL) {
      const bool more = __any_sync(0xffffffffu, !done);
      if (__any_sync(0xffffffffu, pushed > 0)) {
        __syncwarp();
        if (*(volatile int*)wt.qn > 32) topk_merge_sorted(wt, lane, 32, [] __device__() { __syncwarp(); });
        else topk_merge(wt, lane, 32, [] __device__() { __syncwarp(); });
        const bool full = wt.li[R.k - 1] != kEmptyIdx;  // (its entries all beat the CTA's bar)
        thr_s = full ? wt.ls[R.k - 1] : thr0_s;
        thr_i = full ? wt.li[R.k - 1] : thr0_i;
      }
      if (!more) break;
    } else {
      const bool more = __syncthreads_or(!done);
      if (*(volatile int*)tk.qn > 0) {  // (read by every thread after the barrier: uniform)
        // a long queue (the first merges of a search) is sorted first
        if (*(volatile int*)tk.qn > 256) topk_merge_sorted(tk, tid, blockDim.x, [] __device__() { __syncthreads(); });
        else topk_merge(tk, tid, blockDim.x, [] __device__() { __syncthreads(); });
        thr_s = tk.ls[R.k - 1];
        thr_i = tk.li[R.k - 1];
      }
      if (!more) break;
    }
  }
  if (WL) {  // the warps' lists join the CTA's
    __syncthreads();
    for (int e = lane; e < R.k; e += 32)
      if (wt.li[e] != kEmptyIdx) {
        const int pos = atomicAdd(tk.qn, 1);
        tk.qs[pos] = wt.ls[e];
        tk.qi[pos] = wt.li[e];
      }
    __syncthreads();
    if (*(volatile int*)tk.qn > 0) {
      if (*(volatile int*)tk.qn > 256) topk_merge_sorted(tk, tid, blockDim.x, [] __device__() { __syncthreads(); });
      else topk_merge(tk, tid, blockDim.x, [] __device__() { __syncthreads(); });
    }
  }
  for (int e = tid; e < R.k; e += blockDim.x) {
    R.lists_s[gl + e] = tk.ls[e];
    R.lists_i[gl + e] = tk.li[e];
  }
  unsigned int c = my_count;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if ((tid & 31) == 0 && c) atomicAdd(R.count, (unsigned long long)c);
}

// ---------------------------------------------------------------------------
// VRAM-feasible space: CTA b scans the contiguous segment [b*seg, (b+1)*seg) of the
// range, in steps of 512 consecutive candidates.  k_vram_count counts; after an
// exclusive scan of the counts, k_vram_write writes each CTA's indices in order.
// ---------------------------------------------------------------------------
constexpr int kVramThreads = 512;

struct VramArgs {
  uint64_t lo, len, seg;
  uint32_t step[MF_MAX_MODELS];   // mixed-radix digits of 512
  unsigned long long* counts;     // [grid]
  uint64_t* out;
  uint64_t cap;
};

template <bool WRITE>
__global__ void __launch_bounds__(kVramThreads)
k_vram(const Params P, const VramArgs A) {
  extern __shared__ __align__(16) float vr[];  // [sumK] VRAM of each option
  __shared__ unsigned int s_warp[kVramThreads / 32];
  __shared__ unsigned long long s_base;
  const int N = P.n_models;
  const int sumK = pick(P.off, N - 1) + pick(P.K, N - 1);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int e = tid; e < sumK; e += blockDim.x) vr[e] = P.dem[e].y;
  const uint64_t s0 = (uint64_t)blockIdx.x * A.seg;
  const uint64_t s1 = s0 + A.seg < A.len ? s0 + A.seg : A.len;
  int row[MF_MAX_MODELS];
  {
    const uint64_t idx0 = A.lo + (s0 + tid < A.len ? s0 + tid : 0);
#pragma unroll
    for (int i = 0; i < MF_MAX_MODELS; ++i)
      if (i < N) row[i] = P.off[i] + (int)((idx0 / P.stride[i]) % (uint64_t)P.K[i]);
  }
  if (tid == 0) s_base = WRITE ? A.counts[blockIdx.x] : 0ull;
  __syncthreads();
  unsigned long long mine = 0;
  for (uint64_t b = s0; b < s1; b += kVramThreads) {
    const uint64_t t = b + tid;
    float V = 0.f;
#pragma unroll
    for (int i = 0; i < MF_MAX_MODELS; ++i)
      if (i < N) V += vr[row[i]];
    const bool ok = t < s1 && V <= P.vram_cap;
    if (WRITE) {
      // ascending positions: this warp's earlier lanes, then the earlier warps
      const unsigned int bal = __ballot_sync(0xffffffffu, ok);
      if (lane == 0) s_warp[warp] = __popc(bal);
      __syncthreads();
      unsigned int before = __popc(bal & ((1u << lane) - 1u));
      unsigned int total = 0;
      for (int w = 0; w < kVramThreads / 32; ++w) {
        if (w < warp) before += s_warp[w];
        total += s_warp[w];
      }
      const unsigned long long pos = s_base + before;
      if (ok && pos < A.cap) A.out[pos] = A.lo + t;
      __syncthreads();
      if (tid == 0) s_base += total;
    } else {
      mine += ok ? 1ull : 0ull;
    }
    uint32_t carry = 0;
#pragma unroll
    for (int i = MF_MAX_MODELS - 1; i >= 0; --i)
      if (i < N) {
        const int off = P.off[i];
        const uint32_t K = (uint32_t)P.K[i];
        uint32_t d = (uint32_t)(row[i] - off) + A.step[i] + carry;
        carry = d >= K;
        if (carry) d -= K;
        row[i] = off + (int)d;
      }
  }
  if (!WRITE) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mine += __shfl_xor_sync(0xffffffffu, mine, o);
    if (lane == 0) atomicAdd(&A.counts[blockIdx.x], mine);
  }
}

// Exclusive scan of n counts in place (one CTA; n <= 4096); total to *total.
__global__ void __launch_bounds__(1024)
k_scan_counts(unsigned long long* c, int n, unsigned long long* total) {
  __shared__ unsigned long long s[4096];
  for (int e = threadIdx.x; e < n; e += blockDim.x) s[e] = c[e];
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long run = 0;
    for (int e = 0; e < n; ++e) {
      const unsigned long long v = s[e];
      s[e] = run;
      run += v;
    }
    *total = run;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < n; e += blockDim.x) c[e] = s[e];
}

static void radix_digits(const Params& P, uint64_t v, uint32_t* step) {
  v %= P.total;
  for (int i = P.n_models - 1; i >= 0; --i) {
    step[i] = (uint32_t)(v % (uint64_t)P.K[i]);
    v /= (uint64_t)P.K[i];
  }
}

// ---------------------------------------------------------------------------
// The paper's GA (Sec. IV-C) on the fixed-context landscape, one CTA: thread c breeds
// individual c; fitness is the table sum of fc mode.  Operators and draws follow the
// GA of k_ga.cu with two more: crossover applied with probability crossover_p (draw
// kGaCrossDo, else the first parent is copied) and repair of an infeasible individual
// by rejection sampling from the uniform distribution over Lambda (draws kGaRepair,
// j = a * N + i, at most 256 / N attempts, the first feasible one kept).  The block has
// 1024 threads whatever the population, and a generation's repairs share all of them
// (see repair).
// ---------------------------------------------------------------------------
struct FcGaArgs {
  const float2* tab;
  int pop, gens, tournament, elitism, repair;
  uint32_t mut_thr, cross_thr;     // 24-bit thresholds
  uint64_t seed;
  int32_t* out_genome;
  float* out_fit;
};

__device__ __forceinline__ float fc_fit(const Params& P, const float2* tab, const uint8_t* g) {
  float J = 0.f, V = 0.f;
  for (int i = 0; i < P.n_models; ++i) {
    const float2 e = tab[pick(P.off, i) + g[i]];
    J += e.x;
    V += e.y;
  }
  return (V <= P.vram_cap && J > -INFINITY) ? J : -INFINITY;
}

__global__ void __launch_bounds__(1024)
k_fc_ga(const Params P, const FcGaArgs A) {
  extern __shared__ __align__(16) unsigned char sm[];
  __shared__ float sval[32];
  __shared__ int sidx[32];
  __shared__ int s_wcnt[32];
  __shared__ int s_pend[1024];
  const int N = P.n_models, pop = A.pop;
  const int sumK = pick(P.off, N - 1) + pick(P.K, N - 1);
  float2* tab = reinterpret_cast<float2*>(sm);
  float* fit0 = reinterpret_cast<float*>(tab + sumK);
  float* fit1 = fit0 + pop;
  uint8_t* g0 = reinterpret_cast<uint8_t*>(fit1 + pop);
  uint8_t* g1 = g0 + (size_t)pop * N;
  const int c = threadIdx.x;
  for (int e = c; e < sumK; e += blockDim.x) tab[e] = A.tab[e];
  __syncthreads();
  // Does any configuration meet the floors and the VRAM bound?  Exactly when every model
  // has an option with a finite term and the smallest such VRAM demands, summed in model
  // order as the fitness sums them, fit the cap (fp32 rounding is monotone, so no other
  // configuration sums to less).  If none does, every repair would draw all its attempts
  // in vain; its draws come from their own stream, so skipping it changes nothing else.
  __shared__ int s_any_feasible;
  if (c < 32) {
    float V = 0.f;
    bool every = true;
    for (int i = 0; i < N; ++i) {
      const int off = pick(P.off, i), K = pick(P.K, i);
      float m = INFINITY;
      for (int o = c; o < K; o += 32) {
        const float2 e = tab[off + o];
        if (e.x > -INFINITY && e.y < m) m = e.y;
      }
#pragma unroll
      for (int w = 16; w > 0; w >>= 1) m = fminf(m, __shfl_xor_sync(0xffffffffu, m, w));
      every = every && m < INFINITY;
      V += m;
    }
    if (c == 0) s_any_feasible = every && V <= P.vram_cap ? 1 : 0;
  }
  __syncthreads();
  const bool repairable = A.repair && s_any_feasible;
  const uint64_t sd = A.seed;
  const int attempts = 256 / N;
  // Repair of the generation's infeasible children (need): the cnt of them, in ascending
  // order, each get a group of gs lanes of one warp (gs a power of two, as many lanes as
  // the block has for cnt rounded up to a power of two, at most 32), which tries the
  // child's attempts gs at a time; the lowest feasible attempt of a group's first
  // successful round is the sequential search's result.  The winning lane writes the
  // child's genes and fitness over the unrepaired ones already in shared memory.
  const int lane = c & 31, warp = c >> 5, nwarps = (int)(blockDim.x >> 5);
  auto repair = [&](uint32_t G, bool need, uint8_t* genes, float* fit) {
    const unsigned bal = __ballot_sync(0xffffffffu, need);
    if (lane == 0) s_wcnt[warp] = __popc(bal);
    __syncthreads();
    int before = 0, cnt = 0;
    for (int w = 0; w < (pop + 31) / 32; ++w) {  // (only the population's warps breed)
      const int v = s_wcnt[w];
      before += w < warp ? v : 0;
      cnt += v;
    }
    if (need) s_pend[before + __popc(bal & ((1u << lane) - 1u))] = c;
    __syncthreads();
    if (cnt == 0) return;  // (uniform)
    int m = 1;
    while (m < cnt) m <<= 1;
    int gs = nwarps * 32 / m;
    gs = gs > 32 ? 32 : (gs < 1 ? 1 : gs);
    const int grp = lane / gs, lig = lane % gs;
    const int gid = warp * (32 / gs) + grp;
    const int child = gid < cnt ? s_pend[gid] : -1;
    const unsigned gmask = gs == 32 ? 0xffffffffu : ((1u << gs) - 1u) << (grp * gs);
    bool done = child < 0;
    for (int a0 = 0; a0 < attempts; a0 += gs) {
      if (!__any_sync(0xffffffffu, !done)) break;
      const int a = a0 + lig;
      float Jc = -INFINITY;
      uint8_t cand[MF_MAX_MODELS];
      if (!done && a < attempts) {  // fc_fit's sums, with the draws kept in registers
        float Js = 0.f, Vs = 0.f;
#pragma unroll
        for (int i = 0; i < MF_MAX_MODELS; ++i) {
          if (i < N) {
            cand[i] = (uint8_t)ga_unif(ga_rng(sd, G, (uint32_t)child, kGaRepair, (uint32_t)(a * N + i)),
                                       (uint32_t)pick(P.K, i));
            const float2 e = tab[pick(P.off, i) + cand[i]];
            Js += e.x;
            Vs += e.y;
          }
        }
        Jc = (Vs <= P.vram_cap && Js > -INFINITY) ? Js : -INFINITY;
      }
      const unsigned ok = __ballot_sync(0xffffffffu, Jc != -INFINITY) & gmask;
      if (!done && ok) {
        if (lane == __ffs(ok) - 1) {
#pragma unroll
          for (int i = 0; i < MF_MAX_MODELS; ++i)
            if (i < N) genes[(size_t)child * N + i] = cand[i];
          fit[child] = Jc;
        }
        done = true;
      }
    }
  };
  bool need = false;
  if (c < pop) {  // initial population: uniform over Lambda, repaired
    uint8_t* g = g0 + (size_t)c * N;
    for (int i = 0; i < N; ++i) g[i] = (uint8_t)ga_unif(ga_rng(sd, 0, (uint32_t)c, kGaInit, (uint32_t)i), (uint32_t)pick(P.K, i));
    const float J = fc_fit(P, tab, g);
    fit0[c] = J;
    need = repairable && J == -INFINITY;
  }
  repair(0u, need, g0, fit0);
  __syncthreads();
  uint8_t* gc = g0;
  uint8_t* gn = g1;
  float* fc_ = fit0;
  float* fn = fit1;
  for (int gen = 0; gen + 1 < A.gens; ++gen) {
    const uint32_t G = (uint32_t)gen + 1u;
    int first = 0;
    if (A.elitism) {  // slot 0 keeps the fittest (lowest slot among equals)
      const int e = block_argmax(fc_, pop, sval, sidx);
      if (c < N) gn[c] = gc[(size_t)e * N + c];
      if (c == 0) fn[0] = fc_[e];
      first = 1;
    }
    need = false;
    if (c >= first && c < pop) {
      int win[2];
      for (int w = 0; w < 2; ++w) {
        int best = -1;
        float bf = 0.f;
        for (int t = 0; t < A.tournament; ++t) {
          const int s2 = ga_unif(ga_rng(sd, G, (uint32_t)c, w ? kGaTourB : kGaTourA, (uint32_t)t), (uint32_t)pop);
          const float f = fc_[s2];
          if (best < 0 || f > bf || (f == bf && s2 < best)) { best = s2; bf = f; }
        }
        win[w] = best;
      }
      const bool cross = (uint32_t)(ga_rng(sd, G, (uint32_t)c, kGaCrossDo, 0u) >> 40) < A.cross_thr;
      uint8_t* g = gn + (size_t)c * N;
      for (int i = 0; i < N; ++i) {
        const uint64_t rc = ga_rng(sd, G, (uint32_t)c, kGaCross, (uint32_t)i);
        uint8_t gene = (cross && (rc >> 63)) ? gc[(size_t)win[1] * N + i] : gc[(size_t)win[0] * N + i];
        const uint64_t rm = ga_rng(sd, G, (uint32_t)c, kGaMut, (uint32_t)i);
        if ((uint32_t)(rm >> 40) < A.mut_thr)
          gene = (uint8_t)ga_unif(ga_rng(sd, G, (uint32_t)c, kGaMutVal, (uint32_t)i), (uint32_t)pick(P.K, i));
        g[i] = gene;
      }
      const float J = fc_fit(P, tab, g);
      fn[c] = J;
      need = repairable && J == -INFINITY;
    }
    repair(G, need, gn, fn);
    __syncthreads();
    uint8_t* tg = gc; gc = gn; gn = tg;
    float* tf = fc_; fc_ = fn; fn = tf;
  }
  const int e = block_argmax(fc_, pop, sval, sidx);
  if (c < N) A.out_genome[c] = gc[(size_t)e * N + c];
  if (c == 0) *A.out_fit = fc_[e];
}

int fc_grid(const mf_ctx* c) { return c->num_sms; }

mf_status fc_search_chunk(mf_ctx* c, const RangeArgs& a, cudaStream_t s) {
  FcLayout L;
  fc_bytes(c->sumK, c->P.n_models, &L, (char*)c->d_fc);
  FcScan S{};
  S.tab = L.tab;
  const bool wl = a.k <= kFcWarpK;  // per-warp lists
  const size_t smem = (((size_t)c->sumK * sizeof(float2) + 15) & ~(size_t)15) + fc_scan_list_bytes(a.k, wl);
  if (smem > 227 * 1024) {
    set_error("fixed-context search: top-k lists do not fit shared memory; use a smaller k");
    return MF_EUNSUPPORTED;
  }
  using ScanFn = void (*)(const Params, const FcScan, const RangeArgs);
  const bool n8 = c->P.n_models <= 8;
  const ScanFn fn = wl ? (n8 ? k_fc_scan<8, true> : k_fc_scan<MF_MAX_MODELS, true>)
                       : (n8 ? k_fc_scan<8, false> : k_fc_scan<MF_MAX_MODELS, false>);
  MF_CUDA(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  fn<<<fc_grid(c), kFcThreads, smem, s>>>(c->P, S, a);
  MF_CUDA(cudaGetLastError());
  return MF_OK;
}

}  // namespace mf

using namespace mf;

static mf_status fc_einval(const std::string& m) {
  set_error(m);
  return MF_EINVAL;
}

mf_status mf_fc_set(mf_ctx* ctx, const mf_fc_params* p, void* stream) {
  set_error("");
  if (!ctx || !p) return fc_einval("NULL argument");
  if (!p->obs || !p->variant || !p->quality || !p->f_min || !p->f_max || !p->omega || !p->tau ||
      !p->reload_cost || !p->prev_variant)
    return fc_einval("mf_fc_params: every array is required");
  const int N = ctx->P.n_models, sumK = ctx->sumK;
  for (int r = 0; r < sumK; ++r) {
    if (!(p->f_max[r] > p->f_min[r])) return fc_einval("mf_fc_params: f_max must exceed f_min for every option");
    if (p->variant[r] < 0) return fc_einval("mf_fc_params: variants must be >= 0");
  }
  for (int i = 0; i < N; ++i)
    if (p->prev_variant[i] < -1) return fc_einval("mf_fc_params: prev_variant must be >= -1");
  if (!std::isfinite(p->alpha) || !std::isfinite(p->beta) || !std::isfinite(p->delta))
    return fc_einval("mf_fc_params: alpha, beta and delta must be finite");
  DeviceGuard guard(ctx->device);
  cudaStream_t s = (cudaStream_t)stream;
  const size_t bytes = fc_bytes(sumK, N, nullptr, nullptr);
  if (!ctx->d_fc) MF_CUDA(cudaMalloc(&ctx->d_fc, bytes));
  FcLayout L;
  fc_bytes(sumK, N, &L, (char*)ctx->d_fc);
  // inputs to the device (pinned staging, one copy each, then a synchronisation)
  std::vector<unsigned char> host(bytes);
  auto put = [&](void* dev, const void* src, size_t n) {
    std::memcpy(host.data() + ((char*)dev - (char*)ctx->d_fc), src, n);
  };
  put(L.obs, p->obs, sizeof(float) * 4);
  put(L.variant, p->variant, sizeof(int32_t) * sumK);
  put(L.quality, p->quality, sizeof(float) * sumK);
  put(L.f_min, p->f_min, sizeof(float) * sumK);
  put(L.f_max, p->f_max, sizeof(float) * sumK);
  put(L.omega, p->omega, sizeof(float) * N);
  put(L.tau, p->tau, sizeof(float) * N);
  put(L.cost, p->reload_cost, sizeof(float) * N);
  put(L.prev, p->prev_variant, sizeof(int32_t) * N);
  const size_t in_lo = (char*)L.obs - (char*)ctx->d_fc;
  MF_CUDA(cudaMemcpyAsync((char*)ctx->d_fc + in_lo, host.data() + in_lo, bytes - in_lo, cudaMemcpyHostToDevice, s));
  const FcConst C{p->alpha, p->beta, p->delta};
  k_fc_local<<<sumK, 256, 0, s>>>(ctx->P, L, C);
  MF_CUDA(cudaGetLastError());
  MF_CUDA(cudaStreamSynchronize(s));
  ctx->fc_ready = 1;
  return MF_OK;
}

mf_status mf_fc_table(mf_ctx* ctx, float* d_fhat, float* d_f, float* d_u, uint8_t* d_ok, void* stream) {
  set_error("");
  if (!ctx) return fc_einval("NULL argument");
  if (!ctx->fc_ready) return fc_einval("mf_fc_set has not been called on this context");
  DeviceGuard guard(ctx->device);
  cudaStream_t s = (cudaStream_t)stream;
  FcLayout L;
  fc_bytes(ctx->sumK, ctx->P.n_models, &L, (char*)ctx->d_fc);
  const size_t n = (size_t)ctx->sumK;
  if (d_fhat) MF_CUDA(cudaMemcpyAsync(d_fhat, L.fhat, sizeof(float) * n, cudaMemcpyDeviceToDevice, s));
  if (d_f) MF_CUDA(cudaMemcpyAsync(d_f, L.f, sizeof(float) * n, cudaMemcpyDeviceToDevice, s));
  if (d_u) MF_CUDA(cudaMemcpyAsync(d_u, L.u, sizeof(float) * n, cudaMemcpyDeviceToDevice, s));
  if (d_ok) MF_CUDA(cudaMemcpyAsync(d_ok, L.ok, n, cudaMemcpyDeviceToDevice, s));
  return MF_OK;
}

mf_status mf_vram_feasible(mf_ctx* ctx, uint64_t lo, uint64_t hi, uint64_t* d_out, uint64_t cap,
                           uint64_t* count, void* stream) {
  set_error("");
  if (!ctx || !count) return fc_einval("NULL argument");
  if (lo > hi || hi > ctx->P.total) return fc_einval("need lo <= hi <= |Lambda|");
  if (cap > 0 && !d_out) return fc_einval("d_out is NULL");
  DeviceGuard guard(ctx->device);
  cudaStream_t s = (cudaStream_t)stream;
  const uint64_t len = hi - lo;
  // segments of whole steps, at most 4096 CTAs
  const uint64_t steps = (len + kVramThreads - 1) / kVramThreads;
  uint64_t grid = 4ull * ctx->num_sms;
  if (grid > steps) grid = steps > 0 ? steps : 1;
  const uint64_t seg = ((steps + grid - 1) / grid) * kVramThreads;
  grid = len > 0 ? (len + seg - 1) / seg : 1;
  mf_status st = ensure_scratch(ctx, sizeof(unsigned long long) * (grid + 1));
  if (st != MF_OK) return st;
  unsigned long long* counts = (unsigned long long*)ctx->d_scratch;
  VramArgs A{};
  A.lo = lo;
  A.len = len;
  A.seg = seg;
  radix_digits(ctx->P, kVramThreads, A.step);
  A.counts = counts;
  A.out = d_out;
  A.cap = cap;
  const size_t smem = sizeof(float) * (size_t)ctx->sumK;
  MF_CUDA(cudaMemsetAsync(counts, 0, sizeof(unsigned long long) * (grid + 1), s));
  k_vram<false><<<(unsigned)grid, kVramThreads, smem, s>>>(ctx->P, A);
  MF_CUDA(cudaGetLastError());
  k_scan_counts<<<1, 1024, 0, s>>>(counts, (int)grid, counts + grid);
  MF_CUDA(cudaGetLastError());
  if (cap > 0) {
    k_vram<true><<<(unsigned)grid, kVramThreads, smem, s>>>(ctx->P, A);
    MF_CUDA(cudaGetLastError());
  }
  st = ensure_host_stage(ctx, sizeof(unsigned long long));
  if (st != MF_OK) return st;
  unsigned long long* h = (unsigned long long*)ctx->h_stage;
  MF_CUDA(cudaMemcpyAsync(h, counts + grid, sizeof(unsigned long long), cudaMemcpyDeviceToHost, s));
  MF_CUDA(cudaStreamSynchronize(s));
  *count = *h;
  return MF_OK;
}

mf_status mf_fc_ga_run(mf_ctx* ctx, const mf_fc_ga_params* g, uint64_t seed, int32_t* best_genome,
                       float* best_fitness, void* stream) {
  set_error("");
  if (!ctx || !g || !best_genome || !best_fitness) return fc_einval("NULL argument");
  if (!ctx->fc_ready) return fc_einval("mf_fc_set has not been called on this context");
  if (g->pop < 2 || g->pop > 1024) return fc_einval("pop must be in 2..1024");
  if (g->gens < 1) return fc_einval("gens must be >= 1");
  if (g->tournament < 1 || g->tournament > 256) return fc_einval("tournament must be in 1..256");
  if (!(g->crossover_p >= 0.0 && g->crossover_p <= 1.0) || !(g->mutation_p >= 0.0 && g->mutation_p <= 1.0))
    return fc_einval("crossover_p and mutation_p must be in [0, 1]");
  if ((g->elitism != 0 && g->elitism != 1) || (g->repair != 0 && g->repair != 1))
    return fc_einval("elitism and repair must be 0 or 1");
  DeviceGuard guard(ctx->device);
  cudaStream_t s = (cudaStream_t)stream;
  const int N = ctx->P.n_models;
  FcLayout L;
  fc_bytes(ctx->sumK, N, &L, (char*)ctx->d_fc);
  // result: genome (16 ints) then the fitness
  mf_status st = ensure_scratch(ctx, sizeof(int32_t) * 17);
  if (st != MF_OK) return st;
  st = ensure_host_stage(ctx, sizeof(int32_t) * 17);
  if (st != MF_OK) return st;
  FcGaArgs A{};
  A.tab = L.tab;
  A.pop = g->pop;
  A.gens = g->gens;
  A.tournament = g->tournament;
  A.elitism = g->elitism;
  A.repair = g->repair;
  A.mut_thr = (uint32_t)std::floor(g->mutation_p * 16777216.0 + 0.5);
  A.cross_thr = (uint32_t)std::floor(g->crossover_p * 16777216.0 + 0.5);
  A.seed = seed;
  A.out_genome = (int32_t*)ctx->d_scratch;
  A.out_fit = (float*)((int32_t*)ctx->d_scratch + 16);
  const size_t smem = sizeof(float2) * ctx->sumK + sizeof(float) * 2 * g->pop + (size_t)2 * g->pop * N;
  const int threads = 1024;  // (the repairs use every warp)
  MF_CUDA(cudaFuncSetAttribute(k_fc_ga, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  k_fc_ga<<<1, threads, smem, s>>>(ctx->P, A);
  MF_CUDA(cudaGetLastError());
  int32_t* h = (int32_t*)ctx->h_stage;
  MF_CUDA(cudaMemcpyAsync(h, ctx->d_scratch, sizeof(int32_t) * 17, cudaMemcpyDeviceToHost, s));
  MF_CUDA(cudaStreamSynchronize(s));
  std::memcpy(best_genome, h, sizeof(int32_t) * N);
  std::memcpy(best_fitness, h + 16, sizeof(float));
  return MF_OK;
}
