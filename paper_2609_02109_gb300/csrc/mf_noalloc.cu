// Exhaustive search for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc: a serving process whose memory pool has
// already claimed the device's memory, or a control loop that must not pay
// cudaMalloc's implicit device synchronisation on every scheduling decision.
// mf_search_exhaustive_noalloc runs the exact fp32 exhaustive search with all
// of its device memory (the problem's tables and weights, the per-CTA running
// top-k lists, the merge buffers, the feasible counter and the status word) in
// one file-scope __device__ array of fixed size.  The runtime loads the module that
// holds the array lazily, so the array is reserved on a device by the first call
// there (its cudaGetSymbolAddress loads the module): a caller whose pool will claim
// the device's memory makes that first call before the pool does, and before any
// stream capture.  From then on the device holds the array until the process exits,
// and the entry point calls no cudaMalloc, cudaFree or other allocating routine.  A
// cudaDeviceReset releases the array while the address looked up at the first call
// stays cached, so a process that resets a device must not call this entry point on
// that device again.
#include <mutex>

#include "mf_internal.cuh"

static_assert(MF_NOALLOC_SCRATCH_BYTES % 256 == 0, "scratch size must keep 256-byte alignment");

// The whole device memory of mf_search_exhaustive_noalloc, one copy per GPU.
static __device__ __align__(256) unsigned char g_noalloc_scratch[MF_NOALLOC_SCRATCH_BYTES];

namespace mf {
namespace {

constexpr int kMaxDevices = 64;
std::mutex g_setup_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the array for the current device.  The array's name in host
// code is only a host-side stand-in, so the address comes from the runtime, once
// per device, with that device current.
mf_status scratch_address(int dev, unsigned char** out) {
  if (dev < 0 || dev >= kMaxDevices) {
    set_error("device ordinal out of range for the no-allocation path");
    return MF_EINVAL;
  }
  std::lock_guard<std::mutex> lock(g_setup_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(g_noalloc_scratch)");
    g_scratch_addr[dev] = p;
  }
  *out = static_cast<unsigned char*>(g_scratch_addr[dev]);
  return MF_OK;
}

// Internal layouts from the caller's arrays (already copied into the scratch):
// demand rows padded to float4, predictors padded to a multiple of 4 floats.
__global__ void k_noalloc_layout(const float* __restrict__ dem3, int sumK, float4* __restrict__ dem4,
                                 const float* __restrict__ w, int n_models, int64_t per,
                                 int64_t per_pad, float* __restrict__ wpad) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t nth = (int64_t)gridDim.x * blockDim.x;
  for (int64_t r = tid; r < sumK; r += nth)
    dem4[r] = make_float4(dem3[3 * r], dem3[3 * r + 1], dem3[3 * r + 2], 0.f);
  for (int64_t e = tid; e < (int64_t)n_models * per_pad; e += nth) {
    const int64_t m = e / per_pad, j = e - m * per_pad;
    wpad[e] = j < per ? w[m * per + j] : 0.f;
  }
}

size_t up256(size_t v) { return (v + 255) & ~size_t(255); }

mf_status einval(const char* msg) {
  set_error(msg);
  return MF_EINVAL;
}

}  // namespace
}  // namespace mf

using namespace mf;

extern "C" mf_status mf_search_exhaustive_noalloc(const mf_problem* p, int32_t k, uint64_t chunk,
                                                  mf_result* out, void* stream) {
  set_error("");
  if (!p || !out) return einval("NULL argument");
  const int N = p->n_models;
  if (N < 1 || N > MF_MAX_MODELS) return einval("n_models must be in 1..16");
  if (!p->n_options || !p->local_feats || !p->demand || !p->weights || !p->sla || !p->obj_w)
    return einval("a required array is NULL");
  if (p->d_local < 1 || p->d_local > MF_MAX_D_LOCAL) return einval("d_local must be in 1..28");
  if (p->hidden1 < 1 || p->hidden1 > MF_MAX_HIDDEN) return einval("hidden1 must be in 1..256");
  if (p->hidden2 < 0 || p->hidden2 > MF_MAX_HIDDEN) return einval("hidden2 must be in 0..256");
  if (p->objective != MF_OBJ_WEIGHTED_THR && p->objective != MF_OBJ_SOFT_LAT) return einval("unknown objective");
  if (p->out_act != MF_ACT_IDENTITY && p->out_act != MF_ACT_SIGMOID) return einval("unknown out_act");
  if (p->precision != MF_FP32 && p->precision != MF_FP32_SIMT)
    return einval("the no-allocation search runs the fp32 path only");
  if (p->vram_cap != p->vram_cap) return einval("vram_cap is NaN");
  if (k < 1 || k > MF_NOALLOC_MAX_TOPK) return einval("k must be in 1..64 for the no-allocation search");

  Params P;
  memset(&P, 0, sizeof(P));
  uint64_t total = 1;
  int sumK = 0;
  for (int i = 0; i < N; ++i) {
    const int kk = p->n_options[i];
    if (kk < 1 || kk > MF_MAX_OPTIONS) return einval("n_options[i] must be in 1..255");
    if (total > UINT64_MAX / (uint64_t)kk) return einval("prod n_options overflows uint64");
    P.K[i] = kk;
    P.off[i] = sumK;
    P.sla[i] = p->sla[i];
    P.w[i] = p->obj_w[i];
    total *= (uint64_t)kk;
    sumK += kk;
  }
  uint64_t st = 1;
  for (int i = N - 1; i >= 0; --i) { P.stride[i] = st; st *= (uint64_t)P.K[i]; }
  P.total = total;
  P.n_models = N;
  P.d_local = p->d_local;
  P.h1 = p->hidden1;
  P.h2 = p->hidden2;
  P.d_in = p->d_local + 4;
  P.objective = p->objective;
  P.out_act = p->out_act;
  P.vram_cap = p->vram_cap;
  P.soft_penalty = p->soft_penalty;
  if (p->agg_scale) {
    for (int j = 0; j < 4; ++j) P.agg_scale[j] = p->agg_scale[j];
  } else {
    P.agg_scale[0] = (float)(1.0 / (0.6 * N));
    P.agg_scale[1] = (float)(1.0 / (20.0 * N));
    P.agg_scale[2] = (float)(1.0 / (1500.0 * N));
    P.agg_scale[3] = (float)(1.0 / 8.0);
  }
  const int64_t din = P.d_in, h1 = P.h1, h2 = P.h2;
  int64_t per = h1 * din + h1;
  int64_t last = h1;
  if (h2 > 0) { per += h2 * h1 + h2; last = h2; }
  per += 2 * last + 2;
  const int64_t per_pad = (per + 3) & ~int64_t(3);
  P.per_model = per_pad;

  int dev = p->device;
  if (dev < 0 && cudaGetDevice(&dev) != cudaSuccess) return einval("no current CUDA device");
  int prev = -1;
  MF_CUDA(cudaGetDevice(&prev));
  if (prev != dev) MF_CUDA(cudaSetDevice(dev));
  struct Restore {
    int d, prev;
    ~Restore() { if (d != prev) cudaSetDevice(prev); }
  } restore{dev, prev};

  int grid = 0;
  MF_CUDA(cudaDeviceGetAttribute(&grid, cudaDevAttrMultiProcessorCount, dev));
  if (grid > MF_NOALLOC_MAX_CTAS) grid = MF_NOALLOC_MAX_CTAS;

  // carve the scratch array
  const size_t b_x = sizeof(float) * (size_t)sumK * p->d_local;
  const size_t b_d3 = sizeof(float) * 3 * (size_t)sumK;
  const size_t b_d4 = sizeof(float4) * (size_t)sumK;
  const size_t b_w = sizeof(float) * (size_t)N * per;
  const size_t b_wp = sizeof(float) * (size_t)N * per_pad;
  if (b_w > MF_NOALLOC_MAX_WEIGHT_BYTES)
    return einval("predictor weights exceed the no-allocation limit (MF_NOALLOC_MAX_WEIGHT_BYTES)");
  const size_t entries = (size_t)grid * k;
  const size_t half = (size_t)((grid + 1) / 2) * k;
  size_t o = 0;
  const size_t o_x = o; o = up256(o + b_x);
  const size_t o_d3 = o; o = up256(o + b_d3);
  const size_t o_d4 = o; o = up256(o + b_d4);
  const size_t o_w = o; o = up256(o + b_w);
  const size_t o_wp = o; o = up256(o + b_wp);
  const size_t o_status = o; o = up256(o + sizeof(uint32_t));
  const size_t o_cnt = o; o = up256(o + sizeof(unsigned long long));
  const size_t o_ls = o; o = up256(o + sizeof(float) * entries);
  const size_t o_li = o; o = up256(o + sizeof(uint64_t) * entries);
  const size_t o_ts = o; o = up256(o + sizeof(float) * 2 * half);
  const size_t o_ti = o; o = up256(o + sizeof(uint64_t) * 2 * half);
  const size_t o_fs = o; o = up256(o + sizeof(float) * k);
  const size_t o_fi = o; o = up256(o + sizeof(uint64_t) * k);
  if (o > MF_NOALLOC_SCRATCH_BYTES)
    return einval("problem does not fit the no-allocation scratch (MF_NOALLOC_SCRATCH_BYTES)");

  unsigned char* base = nullptr;
  mf_status s0 = scratch_address(dev, &base);
  if (s0 != MF_OK) return s0;
  cudaStream_t s = (cudaStream_t)stream;
  // From the first enqueue on, a failing return first waits for the work already on the
  // stream, so no copy or kernel of this call is still using the shared array when the
  // caller's next call starts.
  struct Drain {
    cudaStream_t s;
    bool armed = true;
    ~Drain() {
      if (armed) cudaStreamSynchronize(s);
    }
  } drain{s};

  // inputs: the caller's host arrays into the scratch, then the internal layouts
  MF_CUDA(cudaMemcpyAsync(base + o_x, p->local_feats, b_x, cudaMemcpyHostToDevice, s));
  MF_CUDA(cudaMemcpyAsync(base + o_d3, p->demand, b_d3, cudaMemcpyHostToDevice, s));
  MF_CUDA(cudaMemcpyAsync(base + o_w, p->weights, b_w, cudaMemcpyHostToDevice, s));
  k_noalloc_layout<<<64, 256, 0, s>>>((const float*)(base + o_d3), sumK, (float4*)(base + o_d4),
                                      (const float*)(base + o_w), N, per, per_pad, (float*)(base + o_wp));
  MF_CUDA(cudaGetLastError());
  // the array keeps the previous call's contents: clear what must start at zero
  MF_CUDA(cudaMemsetAsync(base + o_status, 0, sizeof(uint32_t), s));
  MF_CUDA(cudaMemsetAsync(base + o_cnt, 0, sizeof(unsigned long long), s));
  P.x = (const float*)(base + o_x);
  P.dem = (const float4*)(base + o_d4);
  P.w32 = (const float*)(base + o_wp);
  P.wT = nullptr;
  P.status = (uint32_t*)(base + o_status);

  if (chunk == 0) chunk = 1ull << 24;
  if (chunk > (1ull << 31)) chunk = 1ull << 31;
  RangeArgs a{};
  a.k = k;
  a.lists_s = (float*)(base + o_ls);
  a.lists_i = (uint64_t*)(base + o_li);
  a.count = (unsigned long long*)(base + o_cnt);
  a.first = 1;
  for (uint64_t b = 0; b < total; b += chunk) {
    a.base = b;
    a.len = (total - b) < chunk ? (total - b) : chunk;
    mf_status r = f32_search_chunk_params(P, grid, a, s);
    if (r != MF_OK) return r;
    a.first = 0;
  }
  mf_status r = merge_lists(nullptr, a.lists_s, a.lists_i, grid, k, (float*)(base + o_ts),
                            (uint64_t*)(base + o_ti), (float*)(base + o_fs), (uint64_t*)(base + o_fi), s);
  if (r != MF_OK) return r;

  // outputs straight into the caller's host memory
  uint64_t best_i = 0;
  float best_s = 0.f;
  unsigned long long cnt = 0;
  uint32_t status = 0;
  MF_CUDA(cudaMemcpyAsync(&best_i, base + o_fi, sizeof(uint64_t), cudaMemcpyDeviceToHost, s));
  MF_CUDA(cudaMemcpyAsync(&best_s, base + o_fs, sizeof(float), cudaMemcpyDeviceToHost, s));
  MF_CUDA(cudaMemcpyAsync(&cnt, base + o_cnt, sizeof(cnt), cudaMemcpyDeviceToHost, s));
  MF_CUDA(cudaMemcpyAsync(&status, base + o_status, sizeof(status), cudaMemcpyDeviceToHost, s));
  if (out->topk_idx)
    MF_CUDA(cudaMemcpyAsync(out->topk_idx, base + o_fi, sizeof(uint64_t) * k, cudaMemcpyDeviceToHost, s));
  if (out->topk_score)
    MF_CUDA(cudaMemcpyAsync(out->topk_score, base + o_fs, sizeof(float) * k, cudaMemcpyDeviceToHost, s));
  MF_CUDA(cudaStreamSynchronize(s));
  drain.armed = false;
  if (status & kStatusTimeout) {
    set_error("a bounded device wait gave up");
    return MF_ETIMEOUT;
  }
  out->best_idx = best_i;
  out->best_score = best_s;
  out->feasible_count = cnt;
  out->k = k;
  return MF_OK;
}
