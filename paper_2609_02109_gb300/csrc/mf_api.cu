// C ABI of the scorer: argument validation, context set-up, launch sequencing.
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>

#include "mf_internal.cuh"

namespace mf {

static thread_local std::string g_last_error;

void set_error(const std::string& msg) { g_last_error = msg; }

mf_status cuda_fail(cudaError_t e, const char* what) {
  g_last_error = std::string(what) + ": " + cudaGetErrorName(e) + " (" + cudaGetErrorString(e) + ")";
  return e == cudaErrorMemoryAllocation ? MF_ENOMEM : MF_ECUDA;
}

static mf_status einval(const std::string& msg) {
  g_last_error = msg;
  return MF_EINVAL;
}

static size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

mf_status ensure_scratch(mf_ctx* c, size_t bytes) {
  if (bytes <= c->scratch_bytes) return MF_OK;
  if (c->d_scratch) {
    MF_CUDA(cudaDeviceSynchronize());
    cudaFree(c->d_scratch);
    c->d_scratch = nullptr;
    c->scratch_bytes = 0;
  }
  MF_CUDA(cudaMalloc(&c->d_scratch, bytes));
  c->scratch_bytes = bytes;
  return MF_OK;
}

mf_status ensure_host_stage(mf_ctx* c, size_t bytes) {
  if (bytes <= c->h_stage_bytes) return MF_OK;
  if (c->h_stage) {
    MF_CUDA(cudaDeviceSynchronize());
    cudaFreeHost(c->h_stage);
    c->h_stage = nullptr;
    c->h_stage_bytes = 0;
  }
  MF_CUDA(cudaMallocHost(&c->h_stage, bytes));
  c->h_stage_bytes = bytes;
  return MF_OK;
}

static void free_ctx(mf_ctx* c) {
  if (!c) return;
  cudaFree(c->d_x);
  cudaFree(c->d_dem);
  cudaFree(c->d_w32);
  cudaFree(c->d_wT);
  cudaFree(c->d_status);
  cudaFree(c->d_tc);
  cudaFree(c->d_partial);
  cudaFree(c->d_fc);
  cudaFree(c->d_util);
  cudaFree(c->d_scratch);
  cudaFree(c->d_pop[0]);
  cudaFree(c->d_pop[1]);
  cudaFree(c->d_fit);
  cudaFree(c->d_pred);
  cudaFree(c->d_ga_out);
  cudaFree(c->d_gap);
  if (c->ga_exec) cudaGraphExecDestroy(c->ga_exec);
  if (c->cap_stream) cudaStreamDestroy(c->cap_stream);
  for (int j = 0; j < 3; ++j)
    if (c->ev[j]) cudaEventDestroy(c->ev[j]);
  if (c->h_stage) cudaFreeHost(c->h_stage);
  delete c;
}

// Floats of one packed predictor (W1, b1, [W2, b2], W3, b3).
static int64_t params_per_model(int d_local, int h1, int h2) {
  const int64_t din = d_local + 4;
  int64_t n = h1 * din + h1;
  int64_t last = h1;
  if (h2 > 0) { n += (int64_t)h2 * h1 + h2; last = h2; }
  return n + 2 * last + 2;
}

}  // namespace mf

using namespace mf;

extern "C" {

const char* mf_status_string(mf_status s) {
  switch (s) {
    case MF_OK: return "MF_OK";
    case MF_EINVAL: return "MF_EINVAL";
    case MF_ENOMEM: return "MF_ENOMEM";
    case MF_ECUDA: return "MF_ECUDA";
    case MF_EUNSUPPORTED: return "MF_EUNSUPPORTED";
    case MF_ETIMEOUT: return "MF_ETIMEOUT";
    case MF_EDEVICE: return "MF_EDEVICE";
  }
  return "MF_UNKNOWN";
}

const char* mf_last_error(void) { return g_last_error.c_str(); }

mf_status mf_create(const mf_problem* p, mf_ctx** out) {
  g_last_error.clear();
  if (!out) return einval("out is NULL");
  *out = nullptr;
  if (!p) return einval("problem is NULL");
  const int N = p->n_models;
  if (N < 1 || N > MF_MAX_MODELS) return einval("n_models must be in 1..16");
  if (!p->n_options || !p->local_feats || !p->demand || !p->weights || !p->sla || !p->obj_w)
    return einval("a required array is NULL");
  if (p->d_local < 1 || p->d_local > MF_MAX_D_LOCAL) return einval("d_local must be in 1..28");
  if (p->hidden1 < 1 || p->hidden1 > MF_MAX_HIDDEN) return einval("hidden1 must be in 1..256");
  if (p->hidden2 < 0 || p->hidden2 > MF_MAX_HIDDEN) return einval("hidden2 must be in 0..256");
  if (p->objective != MF_OBJ_WEIGHTED_THR && p->objective != MF_OBJ_SOFT_LAT)
    return einval("unknown objective");
  if (p->out_act != MF_ACT_IDENTITY && p->out_act != MF_ACT_SIGMOID) return einval("unknown out_act");
  if (p->precision != MF_FP32 && p->precision != MF_BF16 && p->precision != MF_FP32_SIMT)
    return einval("unknown precision");
  if (std::isnan(p->vram_cap)) return einval("vram_cap is NaN");
  uint64_t total = 1;
  int sumK = 0;
  for (int i = 0; i < N; ++i) {
    const int k = p->n_options[i];
    if (k < 1 || k > MF_MAX_OPTIONS) return einval("n_options[i] must be in 1..255");
    if (total > UINT64_MAX / (uint64_t)k) return einval("prod n_options overflows uint64");
    total *= (uint64_t)k;
    sumK += k;
  }

  int dev = p->device;
  if (dev < 0) MF_CUDA(cudaGetDevice(&dev));
  DeviceGuard guard(dev);
  int cur = -1;
  MF_CUDA(cudaGetDevice(&cur));
  if (cur != dev) return einval("cannot select the requested device");

  mf_ctx* c = new mf_ctx();
  c->device = dev;
  c->precision = p->precision;
  c->K.assign(p->n_options, p->n_options + N);
  c->sumK = sumK;
  cudaDeviceProp prop;
  cudaError_t e = cudaGetDeviceProperties(&prop, dev);
  if (e != cudaSuccess) { free_ctx(c); return cuda_fail(e, "cudaGetDeviceProperties"); }
  c->num_sms = prop.multiProcessorCount;

  Params& P = c->P;
  std::memset(&P, 0, sizeof(P));
  P.n_models = N;
  P.d_local = p->d_local;
  P.h1 = p->hidden1;
  P.h2 = p->hidden2;
  P.d_in = p->d_local + 4;
  P.objective = p->objective;
  c->base_objective = p->objective;
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
  int off = 0;
  for (int i = 0; i < N; ++i) {
    P.K[i] = p->n_options[i];
    P.off[i] = off;
    off += p->n_options[i];
    P.sla[i] = p->sla[i];
    P.w[i] = p->obj_w[i];
  }
  uint64_t st = 1;
  for (int i = N - 1; i >= 0; --i) { P.stride[i] = st; st *= (uint64_t)P.K[i]; }
  P.total = total;
  const int64_t per = params_per_model(p->d_local, p->hidden1, p->hidden2);
  const int64_t per_pad = (per + 3) & ~int64_t(3);
  P.per_model = per_pad;

  // host-side images
  std::vector<float> dem4((size_t)sumK * 4, 0.f);
  for (int r = 0; r < sumK; ++r)
    for (int j = 0; j < 3; ++j) dem4[(size_t)r * 4 + j] = p->demand[(size_t)r * 3 + j];
  std::vector<float> w32((size_t)N * per_pad, 0.f), wT((size_t)N * per_pad, 0.f);
  const int din = P.d_in, h1 = P.h1, h2 = P.h2, hl = h2 > 0 ? h2 : h1;
  for (int i = 0; i < N; ++i) {
    const float* src = p->weights + (size_t)i * per;
    float* d32 = w32.data() + (size_t)i * per_pad;
    float* dT = wT.data() + (size_t)i * per_pad;
    std::memcpy(d32, src, sizeof(float) * per);
    size_t o = 0;
    for (int j = 0; j < h1; ++j)
      for (int k = 0; k < din; ++k) dT[(size_t)k * h1 + j] = src[o + (size_t)j * din + k];
    o += (size_t)h1 * din;
    for (int j = 0; j < h1; ++j) dT[o + j] = src[o + j];
    o += h1;
    if (h2 > 0) {
      for (int j = 0; j < h2; ++j)
        for (int k = 0; k < h1; ++k) dT[o + (size_t)k * h2 + j] = src[o + (size_t)j * h1 + k];
      o += (size_t)h2 * h1;
      for (int j = 0; j < h2; ++j) dT[o + j] = src[o + j];
      o += h2;
    }
    for (size_t j = 0; j < (size_t)2 * hl + 2; ++j) dT[o + j] = src[o + j];
  }

  auto upload = [&](void** dst, const void* src, size_t bytes) -> cudaError_t {
    cudaError_t err = cudaMalloc(dst, bytes);
    if (err != cudaSuccess) return err;
    return cudaMemcpy(*dst, src, bytes, cudaMemcpyHostToDevice);
  };
  if ((e = upload((void**)&c->d_x, p->local_feats, sizeof(float) * (size_t)sumK * p->d_local)) != cudaSuccess ||
      (e = upload((void**)&c->d_dem, dem4.data(), sizeof(float) * dem4.size())) != cudaSuccess ||
      (e = upload((void**)&c->d_w32, w32.data(), sizeof(float) * w32.size())) != cudaSuccess ||
      (e = upload((void**)&c->d_wT, wT.data(), sizeof(float) * wT.size())) != cudaSuccess ||
      (e = cudaMalloc((void**)&c->d_status, sizeof(uint32_t))) != cudaSuccess ||
      (e = cudaMemset(c->d_status, 0, sizeof(uint32_t))) != cudaSuccess ||
      (e = cudaEventCreate(&c->ev[0])) != cudaSuccess || (e = cudaEventCreate(&c->ev[1])) != cudaSuccess ||
      (e = cudaEventCreate(&c->ev[2])) != cudaSuccess) {
    mf_status st2 = cuda_fail(e, "mf_create upload");
    free_ctx(c);
    return st2;
  }
  c->stats.h2d_bytes_create = sizeof(float) * ((size_t)sumK * p->d_local + dem4.size() + w32.size() + wT.size());
  P.x = c->d_x;
  P.dem = c->d_dem;
  P.w32 = c->d_w32;
  P.wT = c->d_wT;
  P.status = c->d_status;

  mf_status st3 = f32_prepare(c);
  if (st3 == MF_OK && c->precision == MF_BF16) {
    std::string why;
    if (!tc_supported(P, &why)) {
      g_last_error = "bf16 tensor-core path: " + why;
      st3 = MF_EUNSUPPORTED;
    } else {
      st3 = tc_prepare(c);
    }
  } else if (st3 == MF_OK && c->precision == MF_FP32 && tc_exact_supported(P)) {
    // the exact tensor-core variant where its operands fit; else the CUDA-core path
    if (tc_prepare(c, true) != MF_OK) {
      cudaFree(c->d_tc);
      c->d_tc = nullptr;
      std::memset(&c->tc, 0, sizeof(c->tc));
      g_last_error.clear();
    }
  }
  if (st3 != MF_OK) {
    free_ctx(c);
    return st3;
  }
  *out = c;
  return MF_OK;
}

mf_status mf_destroy(mf_ctx* ctx) {
  if (!ctx) return MF_OK;
  DeviceGuard guard(ctx->device);
  cudaDeviceSynchronize();
  free_ctx(ctx);
  return MF_OK;
}

mf_status mf_space_size(const mf_ctx* ctx, uint64_t* out) {
  if (!ctx || !out) return einval("NULL argument");
  *out = ctx->P.total;
  return MF_OK;
}

mf_status mf_set_utility(mf_ctx* ctx, const mf_fc_params* p) {
  g_last_error.clear();
  if (!ctx) return einval("ctx is NULL");
  DeviceGuard guard(ctx->device);
  Params& P = ctx->P;
  if (!p) {  // back to the problem's own objective
    P.objective = ctx->base_objective;
    ctx->params_version++;
    return MF_OK;
  }
  if (!p->variant || !p->quality || !p->f_min || !p->f_max || !p->omega || !p->tau || !p->reload_cost ||
      !p->prev_variant)
    return einval("mf_fc_params: every array but obs is required");
  const int N = P.n_models, sumK = ctx->sumK;
  std::vector<float4> tab(sumK);
  for (int r = 0; r < sumK; ++r) {
    if (!(p->f_max[r] > p->f_min[r])) return einval("mf_fc_params: f_max must exceed f_min for every option");
    if (p->variant[r] < 0) return einval("mf_fc_params: variants must be >= 0");
    float v;
    std::memcpy(&v, &p->variant[r], sizeof(float));
    tab[r] = make_float4(p->f_min[r], p->f_max[r] - p->f_min[r], p->quality[r], v);
  }
  for (int i = 0; i < N; ++i)
    if (p->prev_variant[i] < -1) return einval("mf_fc_params: prev_variant must be >= -1");
  if (!std::isfinite(p->alpha) || !std::isfinite(p->beta) || !std::isfinite(p->delta))
    return einval("mf_fc_params: alpha, beta and delta must be finite");
  if (!ctx->d_util) MF_CUDA(cudaMalloc(&ctx->d_util, sizeof(float4) * (size_t)sumK));
  MF_CUDA(cudaMemcpy(ctx->d_util, tab.data(), sizeof(float4) * (size_t)sumK, cudaMemcpyHostToDevice));
  P.util = ctx->d_util;
  for (int i = 0; i < N; ++i) {
    P.u_omega[i] = p->omega[i];
    P.u_tau[i] = p->tau[i];
    P.u_cost[i] = p->reload_cost[i];
    P.u_prev[i] = p->prev_variant[i];
  }
  P.u_alpha = p->alpha;
  P.u_beta = p->beta;
  P.u_delta = p->delta;
  P.objective = MF_OBJ_UTILITY;
  ctx->params_version++;
  return MF_OK;
}

mf_status mf_set_objective(mf_ctx* ctx, const float* sla, const float* obj_w) {
  if (!ctx) return einval("ctx is NULL");
  for (int i = 0; i < ctx->P.n_models; ++i) {
    if (sla) ctx->P.sla[i] = sla[i];
    if (obj_w) ctx->P.w[i] = obj_w[i];
  }
  ctx->params_version++;
  return MF_OK;
}

mf_status mf_score_batch(mf_ctx* ctx, const uint64_t* d_idx, uint64_t n, float* d_score,
                         uint8_t* d_feasible, float* d_pred, void* stream) {
  g_last_error.clear();
  if (!ctx) return einval("ctx is NULL");
  if (n == 0) return MF_OK;
  if (!d_idx || !d_score) return einval("d_idx and d_score are required");
  DeviceGuard guard(ctx->device);
  cudaStream_t s = (cudaStream_t)stream;
  if (ctx->precision == MF_BF16 || ctx->tc.tf) return tc_score_list(ctx, d_idx, n, d_score, d_feasible, d_pred, s);
  float* pred = d_pred;
  const uint64_t tasks = n * (uint64_t)ctx->P.n_models;
  if (!pred && tasks <= 64ull * 1024) {
    // the small-batch kernel passes per-model outputs through memory
    mf_status st = ensure_scratch(ctx, sizeof(float) * 2 * tasks);
    if (st != MF_OK) return st;
    pred = (float*)ctx->d_scratch;
  }
  return f32_score_list(ctx, d_idx, nullptr, n, d_score, d_feasible, pred, s);
}

static mf_status read_status(mf_ctx* ctx, cudaStream_t s, uint32_t* word, bool clear) {
  MF_CUDA(cudaMemcpyAsync(word, ctx->d_status, sizeof(uint32_t), cudaMemcpyDeviceToHost, s));
  MF_CUDA(cudaStreamSynchronize(s));
  if (clear && *word) MF_CUDA(cudaMemsetAsync(ctx->d_status, 0, sizeof(uint32_t), s));
  return MF_OK;
}

// The exhaustive-search driver: per-CTA running lists over chunks of [lo, hi), their
// merge, the fp32 re-scoring of a bf16 shortlist, the result.  fc: the fixed-context
// table-lookup scan instead of the predictors.
static mf_status search_impl(mf_ctx* ctx, uint64_t lo, uint64_t hi, int32_t k, uint64_t chunk,
                             mf_result* out, void* stream, bool fc);

mf_status mf_search_range(mf_ctx* ctx, uint64_t lo, uint64_t hi, int32_t k, uint64_t chunk,
                          mf_result* out, void* stream) {
  g_last_error.clear();
  return search_impl(ctx, lo, hi, k, chunk, out, stream, false);
}

mf_status mf_fc_search(mf_ctx* ctx, uint64_t lo, uint64_t hi, int32_t k, uint64_t chunk, mf_result* out,
                       void* stream) {
  g_last_error.clear();
  if (ctx && !ctx->fc_ready) return einval("mf_fc_set has not been called on this context");
  return search_impl(ctx, lo, hi, k, chunk, out, stream, true);
}

static mf_status search_impl(mf_ctx* ctx, uint64_t lo, uint64_t hi, int32_t k, uint64_t chunk,
                             mf_result* out, void* stream, bool fc) {
  if (!ctx || !out) return einval("NULL argument");
  if (k < 1 || k > MF_MAX_TOPK) return einval("k must be in 1..1024");
  if (lo > hi || hi > ctx->P.total) return einval("need lo <= hi <= |Lambda|");
  if (chunk == 0) chunk = 1ull << 24;
  if (chunk > (1ull << 31)) chunk = 1ull << 31;
  DeviceGuard guard(ctx->device);
  cudaStream_t s = (cudaStream_t)stream;
  const bool tc = !fc && ctx->precision == MF_BF16;
  // the exact (3-term tf32) tensor-core variant, where its lists fit next to the weights
  const bool tx = !fc && !tc && ctx->tc.tf && tc_fits(ctx, k);
  const int kcap = tc ? (k * 8 > 256 ? k * 8 : 256) : k;
  const int grid = fc ? fc_grid(ctx) : (tc || tx) ? tc_grid(ctx) : f32_grid(ctx);

  // scratch: per-CTA lists, two merge buffers, merged list, rescored shortlist, count
  const size_t entries = (size_t)grid * kcap;
  const size_t half = (size_t)((grid + 1) / 2) * kcap;
  size_t o = 0;
  const size_t o_ls = o; o = align_up(o + sizeof(float) * entries, 256);
  const size_t o_li = o; o = align_up(o + sizeof(uint64_t) * entries, 256);
  const size_t o_ts = o; o = align_up(o + sizeof(float) * 2 * half, 256);
  const size_t o_ti = o; o = align_up(o + sizeof(uint64_t) * 2 * half, 256);
  const size_t o_ms = o; o = align_up(o + sizeof(float) * kcap, 256);
  const size_t o_mi = o; o = align_up(o + sizeof(uint64_t) * kcap, 256);
  const size_t o_rs = o; o = align_up(o + sizeof(float) * kcap, 256);
  const size_t o_rp = o; o = align_up(o + sizeof(float) * 2 * kcap * ctx->P.n_models, 256);
  const size_t o_fs = o; o = align_up(o + sizeof(float) * k, 256);
  const size_t o_fi = o; o = align_up(o + sizeof(uint64_t) * k, 256);
  const size_t o_cnt = o; o = align_up(o + sizeof(unsigned long long), 256);
  mf_status st = ensure_scratch(ctx, o);
  if (st != MF_OK) return st;
  char* base = (char*)ctx->d_scratch;
  float* ls = (float*)(base + o_ls);
  uint64_t* li = (uint64_t*)(base + o_li);
  float* ts = (float*)(base + o_ts);
  uint64_t* ti = (uint64_t*)(base + o_ti);
  float* ms = (float*)(base + o_ms);
  uint64_t* mi = (uint64_t*)(base + o_mi);
  float* rs = (float*)(base + o_rs);
  float* rp = (float*)(base + o_rp);
  float* fs = (float*)(base + o_fs);
  uint64_t* fi = (uint64_t*)(base + o_fi);
  unsigned long long* cnt = (unsigned long long*)(base + o_cnt);
  MF_CUDA(cudaMemsetAsync(cnt, 0, sizeof(unsigned long long), s));

  int launches = 0, score_launches = 0;
  MF_CUDA(cudaEventRecord(ctx->ev[0], s));
  RangeArgs a{};
  a.k = kcap;
  a.lists_s = ls;
  a.lists_i = li;
  a.count = cnt;
  a.first = 1;
  if (hi == lo) {
    // empty range: initialise the lists through a zero-length launch of the scorer
    a.base = lo;
    a.len = 0;
    int nl = 1;
    st = fc ? fc_search_chunk(ctx, a, s) : (tc || tx) ? tc_search_chunk(ctx, a, s, &nl) : f32_search_chunk(ctx, a, s);
    if (st != MF_OK) return st;
    launches += nl;
    score_launches += nl;
  }
  for (uint64_t b = lo; b < hi; b += chunk) {
    a.base = b;
    a.len = (hi - b) < chunk ? (hi - b) : chunk;
    int nl = 1;
    st = fc ? fc_search_chunk(ctx, a, s) : (tc || tx) ? tc_search_chunk(ctx, a, s, &nl) : f32_search_chunk(ctx, a, s);
    if (st != MF_OK) return st;
    a.first = 0;
    launches += nl;
    score_launches += nl;
  }
  MF_CUDA(cudaEventRecord(ctx->ev[1], s));
  st = merge_lists(ctx, ls, li, grid, kcap, ts, ti, ms, mi, s);
  ++launches;
  if (st != MF_OK) return st;
  if (tc) {
    // exact fp32 re-scoring of the tensor-core shortlist, then the final top-k
    st = f32_score_list_ex(ctx, mi, kcap, rs, rp, s);
    if (st != MF_OK) return st;
    st = select_topk(ctx, rs, mi, kcap, k, fs, fi, s);
    launches += 3;
  } else {
    MF_CUDA(cudaMemcpyAsync(fs, ms, sizeof(float) * k, cudaMemcpyDeviceToDevice, s));
    MF_CUDA(cudaMemcpyAsync(fi, mi, sizeof(uint64_t) * k, cudaMemcpyDeviceToDevice, s));
  }
  if (st != MF_OK) return st;

  const size_t hbytes = sizeof(uint64_t) * k + sizeof(float) * k + sizeof(unsigned long long) + 16;
  st = ensure_host_stage(ctx, hbytes);
  if (st != MF_OK) return st;
  char* h = (char*)ctx->h_stage;
  uint64_t* h_i = (uint64_t*)h;
  float* h_s = (float*)(h + sizeof(uint64_t) * k);
  unsigned long long* h_c = (unsigned long long*)(h + sizeof(uint64_t) * k + sizeof(float) * k);
  uint32_t* h_status = (uint32_t*)(h_c + 1);
  MF_CUDA(cudaMemcpyAsync(h_i, fi, sizeof(uint64_t) * k, cudaMemcpyDeviceToHost, s));
  MF_CUDA(cudaMemcpyAsync(h_s, fs, sizeof(float) * k, cudaMemcpyDeviceToHost, s));
  MF_CUDA(cudaMemcpyAsync(h_c, cnt, sizeof(unsigned long long), cudaMemcpyDeviceToHost, s));
  MF_CUDA(cudaEventRecord(ctx->ev[2], s));
  st = read_status(ctx, s, h_status, true);
  if (st != MF_OK) return st;
  ctx->stats.kernel_launches_last = launches;
  ctx->stats.score_launches_last = score_launches;
  ctx->stats.d2h_bytes_last = (sizeof(uint64_t) + sizeof(float)) * k + sizeof(unsigned long long) + sizeof(uint32_t);
  MF_CUDA(cudaEventElapsedTime(&ctx->stats.score_ms_last, ctx->ev[0], ctx->ev[1]));
  MF_CUDA(cudaEventElapsedTime(&ctx->stats.total_ms_last, ctx->ev[0], ctx->ev[2]));
  if (*h_status & kStatusTimeout) {
    g_last_error = "a bounded device wait gave up";
    return MF_ETIMEOUT;
  }
  out->feasible_count = *h_c;
  out->best_idx = h_i[0];
  out->best_score = h_s[0];
  out->k = k;
  if (out->topk_idx) std::memcpy(out->topk_idx, h_i, sizeof(uint64_t) * k);
  if (out->topk_score) std::memcpy(out->topk_score, h_s, sizeof(float) * k);
  return MF_OK;
}

mf_status mf_search_exhaustive(mf_ctx* ctx, int32_t k, uint64_t chunk, mf_result* out, void* stream) {
  if (!ctx) return einval("ctx is NULL");
  return mf_search_range(ctx, 0, ctx->P.total, k, chunk, out, stream);
}

mf_status mf_ga_generation(mf_ctx* ctx, const int32_t* d_pop, int32_t P, float* d_fitness, void* stream) {
  g_last_error.clear();
  if (!ctx) return einval("ctx is NULL");
  if (P < 0) return einval("P < 0");
  if (P == 0) return MF_OK;
  if (!d_pop || !d_fitness) return einval("NULL device pointer");
  DeviceGuard guard(ctx->device);
  const size_t need = sizeof(float) * 2 * (size_t)P * ctx->P.n_models;
  mf_status st = ensure_scratch(ctx, need);
  if (st != MF_OK) return st;
  return f32_score_list(ctx, nullptr, d_pop, (uint64_t)P, d_fitness, nullptr, (float*)ctx->d_scratch,
                        (cudaStream_t)stream);
}

static mf_status check_ga(const mf_ctx* ctx, const mf_ga_params* g) {
  if (!ctx || !g) return einval("NULL argument");
  if (g->pop < 2 || g->pop > 65536) return einval("pop must be in 2..65536");
  if (g->gens < 1) return einval("gens must be >= 1");
  if (g->tournament < 1 || g->tournament > 256) return einval("tournament must be in 1..256");
  if (!(g->mutation_p >= 0.0 && g->mutation_p <= 1.0)) return einval("mutation_p must be in [0, 1]");
  if (g->elitism != 0 && g->elitism != 1) return einval("elitism must be 0 or 1");
  return MF_OK;
}

mf_status mf_ga_init(mf_ctx* ctx, const mf_ga_params* g, uint64_t seed, int32_t* d_pop, void* stream) {
  g_last_error.clear();
  mf_status st = check_ga(ctx, g);
  if (st != MF_OK) return st;
  if (!d_pop) return einval("d_pop is NULL");
  DeviceGuard guard(ctx->device);
  return ga_init(ctx, g, seed, d_pop, (cudaStream_t)stream);
}

mf_status mf_ga_step(mf_ctx* ctx, const mf_ga_params* g, uint64_t seed, int32_t gen, const int32_t* d_pop,
                     const float* d_fitness, int32_t* d_next, void* stream) {
  g_last_error.clear();
  mf_status st = check_ga(ctx, g);
  if (st != MF_OK) return st;
  if (!d_pop || !d_fitness || !d_next) return einval("NULL device pointer");
  if (d_next == d_pop) return einval("d_next must not alias d_pop");
  if (gen < 0) return einval("gen must be >= 0");
  DeviceGuard guard(ctx->device);
  return ga_step(ctx, g, seed, gen, d_pop, d_fitness, d_next, (cudaStream_t)stream);
}

mf_status mf_ga_run(mf_ctx* ctx, const mf_ga_params* g, uint64_t seed, int32_t* best_genome,
                    float* best_fitness, void* stream) {
  g_last_error.clear();
  mf_status st = check_ga(ctx, g);
  if (st != MF_OK) return st;
  if (!best_genome || !best_fitness) return einval("NULL output");
  DeviceGuard guard(ctx->device);
  cudaStream_t s = (cudaStream_t)stream;
  int launches = 1;  // one cooperative kernel
  st = ga_run_persistent(ctx, g, seed, s);
  if (st == MF_EUNSUPPORTED) {
    st = ga_run_graph(ctx, g, seed, s);
    launches = 2 + g->gens * 2 + (g->gens - 1);  // init, (wide + combine) x gens, steps, best
  }
  if (st != MF_OK) return st;
  const int N = ctx->P.n_models;
  int32_t* h_g = (int32_t*)ctx->h_stage;
  float* h_f = (float*)(h_g + N);
  uint32_t* h_status = (uint32_t*)(h_f + 1);
  MF_CUDA(cudaMemcpyAsync(h_g, ctx->d_ga_out, sizeof(int32_t) * N + sizeof(float), cudaMemcpyDeviceToHost, s));
  st = read_status(ctx, s, h_status, true);
  if (st != MF_OK) return st;
  if (*h_status & kStatusTimeout) {
    g_last_error = "the GA kernel's grid barrier gave up waiting";
    return MF_ETIMEOUT;
  }
  std::memcpy(best_genome, h_g, sizeof(int32_t) * N);
  *best_fitness = *h_f;
  ctx->stats.d2h_bytes_last = sizeof(int32_t) * N + sizeof(float) + sizeof(uint32_t);
  ctx->stats.kernel_launches_last = launches;
  return MF_OK;
}

mf_status mf_get_stats(const mf_ctx* ctx, mf_stats* out) {
  if (!ctx || !out) return einval("NULL argument");
  *out = ctx->stats;
  out->scoring_path = ctx->precision == MF_BF16 ? 1 : ctx->tc.tf ? 2 : 0;
  return MF_OK;
}

mf_status mf_debug_wait_test(mf_ctx* ctx, uint32_t polls) {
  if (!ctx) return einval("ctx is NULL");
  ctx->P.wait_test = polls;
  return MF_OK;
}

mf_status mf_check_device_status(mf_ctx* ctx, void* stream) {
  if (!ctx) return einval("ctx is NULL");
  DeviceGuard guard(ctx->device);
  mf_status st = ensure_host_stage(ctx, 64);
  if (st != MF_OK) return st;
  uint32_t* w = (uint32_t*)ctx->h_stage;
  st = read_status(ctx, (cudaStream_t)stream, w, true);
  if (st != MF_OK) return st;
  if (*w & kStatusTimeout) { g_last_error = "a bounded device wait gave up"; return MF_ETIMEOUT; }
  if (*w & kStatusBadInput) { g_last_error = "an index or gene was out of range"; return MF_EDEVICE; }
  return MF_OK;
}

}  // extern "C"
