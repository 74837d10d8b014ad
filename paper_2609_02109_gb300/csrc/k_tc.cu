// Tensor-core (tcgen05: bf16 x bf16 -> fp32, or 3-term tf32 -> fp32) scorer for sm_103a.
//
// Same computation as the exact fp32 path (arXiv 2609.02109: Eq. 1 decode, the
// aggregate GPU state, the per-model MeanField MLP of Eq. 6, the constraints of
// Eq. 4 and the objective of Eq. 3), with the MLP layers run as UMMA tiles:
//
//   layer 1   D1[128 x h1]  = A1[128 x k1] . B1^T    A1 = [x_i | agg hi | 1 | agg lo]
//   layer 2   D2[128 x h2]  = H1[128 x h1] . W2^T    (+ b2, ReLU in the epilogue)
//   layer 3   D3[128 x n3] += H2[128 x h2] . B3_i^T  B3_i puts W3_i's two rows in
//                                                    columns i (thr) and n3/2 + i (lat),
//                                                    so D3 accumulates all N models
//                                                    (b3 is added in the final epilogue).
//
// One persistent CTA per SM runs up to four independent 128-row pipelines.  Each has
// four epilogue warps (warp q of a pipeline owns TMEM lanes 32q..32q+31) and one warp
// that only issues the pipeline's MMAs: every MMA group starts on a named-barrier
// rendezvous with the epilogue warps once its operands are stored, and is committed to
// an mbarrier the epilogue warps wait on (bounded; a wait that gives up raises the
// status word and the kernel runs to completion without further waits).  Every A
// operand stays in tensor memory (layer inputs written with tcgen05.st, hidden
// activations converted from the fp32 accumulators with cvt.rn.relu.bf16x2), so the
// tensor core reads only the weights (B) from shared memory, staged once per CTA (per
// pass of models) with TMA bulk copies.
//
// b1 rides in A1's constant-1 column and b2 in a constant block of ones that sits
// in tensor memory right after H1 (one extra K = 16 step whose B rows hold the bias
// as a bf16 hi/lo pair), so the hidden epilogues are only load -> ReLU + round ->
// store.  b3 is added in fp32 in the final epilogue: a bias step of layer 3 would
// cost a whole MMA issue for two numbers.  The aggregate enters layer 1 as a bf16
// hi/lo pair as well (two columns per component with the same weight), so its
// rounding error is ~2^-16, not 2^-9.
//
// Each thread keeps its candidate's digits (option index per model) and steps them
// from tile to tile by adding the digits of the tile stride with carries, so no
// division runs in the hot loop: packed in registers in the six-model instantiation,
// else in shared memory.
//
// The exact fp32 variant (TF) runs the same kernel on tf32 operands: every operand is
// a tf32 hi part plus a tf32 lo part (the rest), and each K = 8 step issues
// hi.hi + hi.lo + lo.hi MMAs of kind::tf32 into the fp32 accumulator (lo.lo, about
// 2^-22 of a product, is dropped), which keeps the scores within the fp32 path's
// 1e-5.  Its tensor-memory layout (256 columns per pipeline) leaves room for two
// pipelines.
#include <cuda_bf16.h>

#include <cstring>
#include <type_traits>
#include <vector>

#include "mf_internal.cuh"

namespace mf {

// ---------------------------------------------------------------------------
// PTX wrappers (tcgen05 / mbarrier / bulk copy), written from the PTX ISA.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

// Suspends the thread until the phase completes or about 1 ms passes.
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(1000000u)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// wait for this thread's tensor-memory loads; the two registers loaded last are tied to
// the wait, so no use of them is scheduled before it
__device__ __forceinline__ void tmem_wait_ld_2(uint32_t& a, uint32_t& b) {
  asm volatile("tcgen05.wait::ld.sync.aligned;" : "+r"(a), "+r"(b)::"memory");
}

__device__ __forceinline__ void named_bar(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// OR of `pred` over the threads of a named barrier (also a barrier).
__device__ __forceinline__ bool named_bar_or(int id, int nthreads, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred pi, po;\n setp.ne.u32 pi, %1, 0;\n bar.red.or.pred po, %2, %3, pi;\n"
      " selp.u32 %0, 1, 0, po;\n}"
      : "=r"(r)
      : "r"((uint32_t)pred), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}

// UMMA shared-memory descriptor: K-major, no swizzle.  lbo = byte distance of
// core matrices adjacent in K, sbo = byte distance of adjacent 8-row groups.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | (1ull << 46);
}

// Instruction descriptor of kind::f16: bf16 A and B (K-major), fp32 D, M = 128.
__host__ __device__ constexpr uint32_t idesc_bf16(int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
}

// Instruction descriptor of kind::tf32: tf32 A and B (K-major), fp32 D, M = 128.
__host__ __device__ constexpr uint32_t idesc_tf32(int n) {
  return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
}

// D[tmem] (+)= A[tmem] . B[smem]^T, one 128 x n x 16 MMA.
__device__ __forceinline__ void mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}

// ReLU then round to bf16, two values per register: `lo` in the low half.
__device__ __forceinline__ uint32_t relu_bf16x2(uint32_t lo, uint32_t hi) {
  uint32_t d;
  asm("cvt.rn.relu.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(__uint_as_float(hi)), "f"(__uint_as_float(lo)));
  return d;
}

__device__ __forceinline__ uint32_t bf16_bits(float v) {
  return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v));
}

// v rounded to tf32 (nearest, ties away from zero): its fp32 bits, low 13 bits zero.
__device__ __forceinline__ uint32_t tf32_bits(float v) {
  uint32_t d;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(d) : "f"(v));
  return d;
}

__device__ __forceinline__ uint32_t tmem_ld_x1(uint32_t taddr) {
  uint32_t r;
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(r) : "r"(taddr));
  return r;
}

__device__ __forceinline__ void tmem_ld_x16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
               : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld_x32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
               : "r"(taddr));
}

__device__ __forceinline__ void tmem_st_x4(uint32_t taddr, const uint32_t (&v)[4]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1,%2,%3,%4};"
               :: "r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3])
               : "memory");
}

__device__ __forceinline__ void tmem_st_x8(uint32_t taddr, const uint32_t (&v)[8]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};"
               :: "r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7])
               : "memory");
}

__device__ __forceinline__ void tmem_st_x32(uint32_t taddr, const uint32_t (&v)[32]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};"
               :: "r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]),
                  "r"(v[16]), "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
               : "memory");
}

__device__ __forceinline__ void tmem_st_x16(uint32_t taddr, const uint32_t (&v)[16]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};"
               :: "r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
               : "memory");
}


// ---------------------------------------------------------------------------
// The kernel
// ---------------------------------------------------------------------------
enum { kTcRange = 0, kTcList = 1 };
constexpr int kTcMaxPipes = 4;
// Each 128-row pipeline has four epilogue warps (warp w reaches tensor-memory lanes
// 32 (w % 4) ..) and one warp that issues its MMAs: warps [0, 4 pipes) are the epilogue
// warps (pipeline w / 4), warps [4 pipes, 5 pipes) the issuing warps (pipeline w - 4 pipes,
// so the issuers sit on different schedulers).
constexpr int kTcPipeThreads = 160;
constexpr uint32_t kWaitLimit = 4096;  // suspended retries (~1 ms each at most)

struct TcList {
  const uint64_t* idx;
  uint64_t n;
  float* score;
  uint8_t* feas;
  float* pred;
};

struct NamedSync128 {
  int id;
  __device__ void operator()() const { named_bar(id, 128); }
};

// The pipeline's top-k merge, out of line: it runs rarely and its registers stay off
// the hot loop.
__device__ __noinline__ void tc_topk_merge(const CtaTopK& tk, int row, int barid) {
  if (*tk.qn <= 128) topk_merge(tk, row, 128, NamedSync128{barid});
  else topk_merge_sorted(tk, row, 128, NamedSync128{barid});
}

// The rest of a bounded wait, out of line: on giving up it flags the status word and
// every later wait returns at once, so the kernel still runs to its end.
__device__ __noinline__ void mbar_wait_slow(uint64_t* bar, uint32_t parity, volatile int* abort, uint32_t* status) {
  if (*abort) return;
  uint32_t n = 0;
  while (!mbar_try_wait(bar, parity)) {
    if (++n == kWaitLimit) {
      *abort = 1;
      atomicOr(status, kStatusTimeout);
      return;
    }
  }
}

struct PipeWait {
  volatile int* abort;
  uint32_t* status;
  // Bounded wait for `parity` of `bar`: first up to 96 non-blocking polls (an MMA group
  // usually completes within a few hundred cycles of the wait, and a polling warp sees
  // it sooner than a suspended one is woken), then suspended tries.
  __device__ __forceinline__ void operator()(uint64_t* bar, uint32_t parity) const {
    for (int i = 0; i < 96; ++i) {
      uint32_t ok;
      asm volatile(
          "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
          " selp.u32 %0, 1, 0, p;\n}"
          : "=r"(ok)
          : "r"(smem_u32(bar)), "r"(parity)
          : "memory");
      if (ok) return;
    }
    if (!mbar_try_wait(bar, parity)) mbar_wait_slow(bar, parity, abort, status);
  }
};

// A wait that ignores an earlier give-up, for the work this CTA itself has in flight
// (its MMAs, its weight copy) before the tensor memory is freed; bounded all the same.
__device__ __noinline__ void mbar_wait_drain(uint64_t* bar, uint32_t parity, uint32_t* status) {
  for (uint32_t n = 0; n < kWaitLimit; ++n)
    if (mbar_try_wait(bar, parity)) return;
  atomicOr(status, kStatusTimeout);
}

// The planted wait of the timeout test: a barrier that nothing arrives on, `polls`
// suspended tries; giving up flags the status word and sets the CTA's give-up flag.
__device__ __noinline__ void mbar_wait_test(uint64_t* never, uint32_t polls, volatile int* abort,
                                            uint32_t* status) {
  for (uint32_t n = 0; n < polls; ++n)
    if (mbar_try_wait(never, 0)) return;
  *abort = 1;
  atomicOr(status, kStatusTimeout);
}

// The predictor's output unit; the sigmoid out of line keeps the scorer's loop small.
__device__ __noinline__ float tc_sigmoid(float v) { return 1.f / (1.f + expf(-v)); }
__device__ __forceinline__ float tc_out(const Params& P, float v) {
  return P.out_act == MF_ACT_SIGMOID ? tc_sigmoid(v) : v;
}

// MMA issue by a whole warp: every lane executes the instruction stream (so the
// operands stay warp-uniform) and one elected lane issues.  The same lane is elected
// for the MMAs and for the commit that tracks them.
__device__ __forceinline__ void mma_ts_warp(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p, e;\n setp.ne.b32 p, %4, 0;\n elect.sync _|e, 0xffffffff;\n"
      " @e tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit_warp(uint64_t* bar) {
  asm volatile(
      "{\n .reg .pred e;\n elect.sync _|e, 0xffffffff;\n"
      " @e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n}" ::"r"(smem_u32(bar))
      : "memory");
}

// The same for kind::tf32 (one 128 x n x 8 MMA).
__device__ __forceinline__ void mma_ts_warp_tf32(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                                 uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p, e;\n setp.ne.b32 p, %4, 0;\n elect.sync _|e, 0xffffffff;\n"
      " @e tcgen05.mma.cta_group::1.kind::tf32 [%0], [%1], %2, %3, p;\n}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// The three products of the exact fp32 variant, A = a_hi + a_lo and B = b_hi + b_lo in
// tf32 parts: KH K-steps of A_hi B_hi, then KX of A_hi B_lo and of A_lo B_hi (A_lo B_lo,
// about 2^-22 of the product, is left out).  A K-step is 8 columns of A and 256 bytes
// of B.
template <int KH, int KX>
__device__ __forceinline__ void mma_tf3(uint32_t d, uint32_t a_hi, uint32_t a_lo, uint64_t b_hi, uint64_t b_lo,
                                        uint32_t idesc, uint32_t acc0) {
#pragma unroll
  for (int k = 0; k < KH; ++k) mma_ts_warp_tf32(d, a_hi + 8u * k, b_hi + 16u * k, idesc, k > 0 ? 1u : acc0);
#pragma unroll
  for (int k = 0; k < KX; ++k) mma_ts_warp_tf32(d, a_hi + 8u * k, b_lo + 16u * k, idesc, 1u);
#pragma unroll
  for (int k = 0; k < KX; ++k) mma_ts_warp_tf32(d, a_lo + 8u * k, b_hi + 16u * k, idesc, 1u);
}

// `steps` MMAs of K = 16 along one K extent; S > 0 unrolls a compile-time count.
template <int S>
__device__ __forceinline__ void mma_steps(int steps, uint32_t d_tmem, uint32_t a_tmem, uint64_t desc,
                                          uint32_t idesc, uint32_t acc0) {
  if constexpr (S > 0) {
#pragma unroll
    for (int s = 0; s < S; ++s) mma_ts_warp(d_tmem, a_tmem + 8u * s, desc + 16u * s, idesc, s > 0 ? 1u : acc0);
  } else {
    for (int s = 0; s < steps; ++s) mma_ts_warp(d_tmem, a_tmem + 8u * s, desc + 16u * s, idesc, s > 0 ? 1u : acc0);
  }
}

// Hidden epilogue: fp32 accumulators [0, width) at `src` -> ReLU -> bf16 pairs at `dst`.
// 64 columns are loaded before one wait.  `after_load` runs once the last accumulator
// column is in registers (the accumulator columns are then free for the next layer);
// `before_store` runs once, before the first stores (the layer-1 epilogue waits there for the
// previous model's layer 3, which reads the same tensor-memory columns).
template <int W, class FL, class FS>
__device__ __forceinline__ void hidden_epilogue(int width, uint32_t src, uint32_t dst, FL after_load,
                                                FS before_store) {
  if constexpr (W > 0 && W % 64 == 0) {
#pragma unroll 1
    for (int c0 = 0; c0 < W; c0 += 64) {
      uint32_t a[32], b[32];
      tmem_ld_x32(src + c0, a);
      tmem_ld_x32(src + c0 + 32, b);
      tmem_wait_ld();
      if (c0 + 64 == W) after_load();
      uint32_t h[16], g[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) h[j] = relu_bf16x2(a[2 * j], a[2 * j + 1]);
#pragma unroll
      for (int j = 0; j < 16; ++j) g[j] = relu_bf16x2(b[2 * j], b[2 * j + 1]);
      if (c0 == 0) before_store();
      tmem_st_x16(dst + (c0 >> 1), h);
      tmem_st_x16(dst + (c0 >> 1) + 16, g);
    }
  } else {
    for (int c0 = 0; c0 < width; c0 += 32) {
      uint32_t a[32];
      tmem_ld_x32(src + c0, a);
      tmem_wait_ld();
      if (c0 + 32 >= width) after_load();
      uint32_t h[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) h[j] = relu_bf16x2(a[2 * j], a[2 * j + 1]);
      if (c0 == 0) before_store();
      tmem_st_x16(dst + (c0 >> 1), h);
    }
  }
}

// The exact fp32 variant's hidden epilogue: fp32 accumulators [0, W) at `src` -> ReLU
// (NaN kept) -> tf32 hi part at `dst_hi`, the rest (fp32; the tensor core reads its top
// tf32 bits) at `dst_lo`, one column per value.
template <int W, class FL, class FS>
__device__ __forceinline__ void hidden_epilogue_tf(uint32_t src, uint32_t dst_hi, uint32_t dst_lo, FL after_load,
                                                   FS before_store) {
  static_assert(W > 0 && W % 32 == 0, "32-column chunks");
  uint32_t a[W / 32][32];
#pragma unroll
  for (int c = 0; c < W / 32; ++c) tmem_ld_x32(src + 32 * c, a[c]);
  tmem_wait_ld();
  after_load();
  before_store();
#pragma unroll
  for (int c = 0; c < W / 32; ++c) {
    uint32_t h[32], l[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const float v = __uint_as_float(a[c][j]);
      const float r = v < 0.f ? 0.f : v;
      // tf32 rounding, nearest with ties away from zero: half a tf32 ulp (2^12 in the
      // fp32 bits) added to the magnitude, the 13 dropped bits cleared (r >= 0 or NaN)
      h[j] = (__float_as_uint(r) + 0x1000u) & 0xFFFFE000u;
      l[j] = __float_as_uint(r - __uint_as_float(h[j]));
    }
    tmem_st_x32(dst_hi + 32 * c, h);
    tmem_st_x32(dst_lo + 32 * c, l);
  }
}

// The aggregate words of a tile's A1 rows: h (and for the tf32 variant l, the lo parts).
struct AggW {
  uint4 h, l;
};

// KW: 32-bit words of an A1 row (8 or 16); AWO: word where the aggregate starts, or
// -1 to take it from T at run time.  S1, S2, S3: K-steps of the three layers (0 = run time).
// N3: columns of the layer-3 accumulator (16, or 0 = run time).  MP: the models run in
// several passes (T.m0..T.m1 and a partial record per candidate); otherwise all N models
// in one launch.  UT: the Eq. 3 utility objective.  NM: the number of models, when fixed at
// compile time (0: run time); the per-model loop is then unrolled, so every per-model
// offset, descriptor and branch is a constant.
//
// Per 128-row pipeline and model i, the issuing warp runs three MMA groups, each on a
// hand-off (named barrier) from the pipeline's four epilogue warps:
//   H1 stored     -> layer 2 of model i (commit A)
//   D2 read, the next A1 row written -> layer 1 of model i + 1, or of the next tile's
//                    first model (commit A)
//   H2 stored     -> layer 3 of model i (commit B)
// and the epilogue warps, per model: D1 -> H1 (stored once the previous layer 3 has read
// H); while layer 2 runs, the objective terms of the previous model (at the first model:
// the previous tile's last, and that tile's constraints and top-k), a stage of the next
// tile's digits and aggregate, and the next A1 row; then D2 -> H2.  The issuing warp does
// nothing else, so an MMA group starts as soon as its operands are stored.
template <int MODE, int KW, int AWO, int S1, int S2, int S3, int N3, bool MP, bool UT, int NM, bool TF>
__global__ void __launch_bounds__((TF ? 2 : kTcMaxPipes) * kTcPipeThreads, 1)
k_score_tc(const Params P, const TcArgs T, const RangeArgs R, const TcList L) {
  static_assert(AWO < 0 || AWO == 4 || AWO == 8, "partial A1 rows are written for these layouts only");
  static_assert(NM <= 7, "packed digits hold at most seven models");
  static_assert(!TF || (KW == 16 && S1 == 2 && S2 == 9 && S3 == 8 && N3 == 16),
                "the exact variant runs the d_L 8, 64-64 shape");
  constexpr int KS = TF ? 8 : 16;  // K of one MMA
  // With the model count fixed at compile time (range mode), a tile's digits live in
  // registers, packed one per byte (model N - 1 in the lowest byte); otherwise in shared
  // memory, one byte per model and row, two tiles.
  constexpr bool RD = NM > 0 && MODE == kTcRange;
  using DS = typename std::conditional<RD, uint64_t, uint8_t*>::type;
  extern __shared__ __align__(1024) unsigned char smem[];
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort;
  __shared__ float s_b3[MF_MAX_MODELS][2];
  const int tid = threadIdx.x;
  // compile-time K-step counts must be the layout's (else no MMA may run)
  if ((S1 > 0 && S1 != T.k1 / KS) || (S2 > 0 && S2 != T.h1 / KS + 1) || (S3 > 0 && S3 != T.hl / KS) ||
      (N3 > 0 && N3 != T.n3) || (NM > 0 && (NM != P.n_models || MP)) || TF != (T.tf != 0)) {
    if (tid == 0) atomicOr(P.status, kStatusBadInput);
    return;
  }
  // the warp index through a shuffle from lane 0, so the compiler knows it is warp-uniform
  // and keeps everything derived from it (pipeline, tensor-memory addresses, issuer roles)
  // in uniform registers with uniform branches
  const int warp = __shfl_sync(0xffffffffu, tid >> 5, 0), lane = tid & 31;
  const int N = NM > 0 ? NM : P.n_models;
  const int npipes = T.pipes;
  const bool issuer = warp >= 4 * npipes;  // the pipeline's MMA-issuing warp
  const int pipe = issuer ? warp - 4 * npipes : warp >> 2, wq = warp & 3;
  const int row = wq * 32 + lane;

  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + T.sm_bar);
  const uint4* xw_s = reinterpret_cast<const uint4*>(smem + T.sm_xw);
  float4* dem_s = reinterpret_cast<float4*>(smem + T.sm_dem);
  // this thread's digits (option index within the model) of every model, two tiles:
  // digits[b * MF_MAX_MODELS * 128 + i * 128 + row]
  uint8_t* digits = reinterpret_cast<uint8_t*>(smem + T.sm_rows) + (size_t)pipe * 2 * MF_MAX_MODELS * 128;

  if (tid == 0) {
    s_abort = 0;
    for (int j = 0; j < 1 + 2 * npipes; ++j) mbar_init(&bars[j], 1);
    mbar_init(&bars[1 + 2 * npipes], 1);           // the timeout test's barrier: nothing arrives
    mbar_init(&bars[2 + 2 * npipes], npipes);  // drain: one commit per issuing warp
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&s_tmem)),
                 "r"(512)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  __syncthreads();
  const uint32_t smem_base = smem_u32(smem);
  if (tid == 0) {
    // weights: one TMA bulk copy per 32 KB piece, all completing on bars[0]
    mbar_arrive_expect_tx(&bars[0], T.img_copy);
    for (uint32_t o = 0; o < T.img_copy; o += 32768u) {
      const uint32_t b = T.img_copy - o < 32768u ? T.img_copy - o : 32768u;
      bulk_g2s(smem + o, static_cast<const unsigned char*>(T.img) + T.img_lo + o, b, &bars[0]);
    }
  }
  if (tid >= T.m0 && tid < T.m1) {
    const float* b3 = P.w32 + (size_t)tid * P.per_model + (size_t)T.h1 * P.d_in + T.h1 +
                      (T.h2 > 0 ? (size_t)T.h2 * T.h1 + T.h2 : 0) + 2 * (size_t)T.hl;
    s_b3[tid][0] = b3[0];
    s_b3[tid][1] = b3[1];
  }
  // option tables with ordinary loads
  const int sumK = P.off[N - 1] + P.K[N - 1];
  {
    uint32_t* xw32 = reinterpret_cast<uint32_t*>(smem + T.sm_xw);
    for (int e = tid; e < sumK * T.kw; e += blockDim.x) xw32[e] = T.xw[e];
  }
  for (int e = tid; e < sumK; e += blockDim.x) dem_s[e] = P.dem[e];

  // per-pipeline running top-k (range mode), its pointers rebuilt where they are used
  const int kcap = R.k;
  auto topk = [&]() {
    CtaTopK tk;
    unsigned char* q = smem + T.sm_topk +
                       (size_t)pipe * ((sizeof(uint64_t) + sizeof(float)) * (2 * (size_t)kcap + T.qcap) + 16);
    tk.li = reinterpret_cast<uint64_t*>(q); q += sizeof(uint64_t) * kcap;
    tk.ni = reinterpret_cast<uint64_t*>(q); q += sizeof(uint64_t) * kcap;
    tk.qi = reinterpret_cast<uint64_t*>(q); q += sizeof(uint64_t) * T.qcap;
    tk.ls = reinterpret_cast<float*>(q); q += sizeof(float) * kcap;
    tk.ns = reinterpret_cast<float*>(q); q += sizeof(float) * kcap;
    tk.qs = reinterpret_cast<float*>(q); q += sizeof(float) * T.qcap;
    tk.qn = reinterpret_cast<int*>(q);
    tk.k = kcap;
    return tk;
  };
  if (MODE == kTcRange && !issuer) {
    const CtaTopK tk = topk();
    const size_t gl = ((size_t)blockIdx.x * npipes + pipe) * kcap;
    for (int e = row; e < kcap; e += 128) {
      tk.ls[e] = R.first ? -INFINITY : R.lists_s[gl + e];
      tk.li[e] = R.first ? kEmptyIdx : R.lists_i[gl + e];
    }
    if (row == 0) *tk.qn = 0;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = __shfl_sync(0xffffffffu, s_tmem, 0);
  const PipeWait wait_bar{&s_abort, P.status};

  const uint32_t tp = tmem + (uint32_t)(pipe * T.pipe_stride);
  const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
  const uint32_t tD = tp + T.col_d, tA = tp + T.col_a, tD3 = tp + T.col_d3, tOnes = tp + T.col_ones;
  // layer-2 and layer-3 A operands (bf16 pairs, or tf32 hi parts with their lo parts at tHlo)
  const uint32_t tH1 = tOnes - (uint32_t)(TF ? T.h1 : T.h1 / 2);
  const uint32_t tH2 = T.h2 > 0 ? tOnes - (uint32_t)(TF ? T.h2 : T.h2 / 2) : tH1;
  const uint32_t tHlo = tp + T.col_hlo;
  uint64_t* barA = &bars[1 + 2 * pipe];  // layers 1 and 2 completed (alternating)
  uint64_t* barB = &bars[2 + 2 * pipe];  // layer 3 completed
  uint32_t phA = 0, phB = 0;
  // epilogue -> issuer hand-offs alternate between two named barriers per pipeline, each
  // a full rendezvous of the 160 threads: the epilogue warps cannot run ahead of the
  // issuing warp even where their mbarrier waits return early (after a wait gave up),
  // which with arrive-only hand-offs could complete a barrier without the issuing warp
  // and leave it waiting at the next one; the pipeline's top-k uses a third barrier
  // among its epilogue warps
  const int sig0 = 1 + 2 * pipe, barid = 1 + 2 * npipes + pipe;
  const uint32_t id1 = TF ? idesc_tf32(T.h1) : idesc_bf16(T.h1), id2 = TF ? idesc_tf32(T.h2) : idesc_bf16(T.h2),
                 id3 = TF ? idesc_tf32(T.n3) : idesc_bf16(T.n3);
  const int s1 = T.k1 / KS, s2 = T.h1 / KS + 1, s3 = T.hl / KS;
  const int m0 = MP ? T.m0 : 0, m1 = MP ? T.m1 : N;  // this pass's models
  const float vcap = P.vram_cap;
  if (!issuer) {  // constant ones block: (1, 1) feeds the bias hi/lo rows of B2
    if constexpr (TF) {
      uint32_t v[8] = {0x3F800000u, 0x3F800000u, 0u, 0u, 0u, 0u, 0u, 0u};
      tmem_st_x8(tOnes + lane_off, v);
      uint32_t z[32] = {};  // the A1 rows' unused words stay zero
      tmem_st_x32(tA + lane_off, z);
    } else {
      uint32_t v[8] = {0x3F803F80u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
      tmem_st_x8(tOnes + lane_off, v);
    }
  }
  if (P.wait_test) mbar_wait_test(&bars[1 + 2 * npipes], P.wait_test, &s_abort, P.status);

  unsigned int my_count = 0;

  const uint64_t n = MODE == kTcRange ? R.len : L.n;
  const uint64_t gpipe = (uint64_t)blockIdx.x * npipes + pipe;
  const uint64_t gstride = (uint64_t)gridDim.x * npipes;

  // UMMA descriptors: every model's image has the same size, so model i's B operands sit
  // (i - m0) images after model m0's
  const uint32_t sb1 = smem_base;  // the pass's image starts with model m0's B1
  const uint32_t sb2 = smem_base + (T.off_b2[0] - T.off_b1[0]);
  const uint32_t sb3 = smem_base + (T.off_b3[0] - T.off_b1[0]);
  // (tf32: 4 values per 16-byte core-matrix row, and each B image's lo part follows its hi part)
  auto issue_mma1 = [&](int i) {
    const uint64_t b = smem_desc(sb1 + (uint32_t)(i - m0) * T.img_model, 128u, (uint32_t)(T.k1 / (TF ? 4 : 8)) * 128u);
    if constexpr (TF) mma_tf3<S1, S1>(tD, tA, tA + 16u, b, b + (T.img_lo1 >> 4), id1, 0u);
    else mma_steps<S1>(s1, tD, tA, b, id1, 0u);
  };
  auto issue_mma2 = [&](int i) {
    const uint64_t b = smem_desc(sb2 + (uint32_t)(i - m0) * T.img_model, 128u,
                                 (uint32_t)((T.h1 + (TF ? 8 : 16)) / (TF ? 4 : 8)) * 128u);
    if constexpr (TF) mma_tf3<S2, S2 - 1>(tD, tH1, tHlo, b, b + (T.img_lo2 >> 4), id2, 0u);
    else mma_steps<S2>(s2, tD, tH1, b, id2, 0u);
  };
  auto issue_mma3 = [&](int i) {
    const uint64_t b = smem_desc(sb3 + (uint32_t)(i - m0) * T.img_model, 128u, (uint32_t)(T.hl / (TF ? 4 : 8)) * 128u);
    if constexpr (TF) mma_tf3<S3, S3>(tD3, tH2, tHlo, b, b + (T.img_lo3 >> 4), id3, i > m0 ? 1u : 0u);
    else mma_steps<S3>(s3, tD3, tH2, b, id3, i > m0 ? 1u : 0u);
  };
  // The epilogue warps wait on the commits' mbarriers (suspended until the phase completes).
  auto await_a = [&]() {
    wait_bar(barA, phA);
    phA ^= 1u;
    tc_fence_after();
  };
  auto await_b = [&]() {
    wait_bar(barB, phB);
    phB ^= 1u;
    tc_fence_after();
  };
  uint32_t ksig = 0;
  // epilogue warps: this thread's tensor-memory loads and stores so far are complete and
  // ordered before the issuing warp's next MMAs
  auto signal = [&]() {
    tmem_wait_st();
    tc_fence_before();
    named_bar(sig0 + (int)(ksig & 1u), 160);
    ++ksig;
  };
  // issuing warp: the epilogue warps' next hand-off
  auto take = [&]() {
    named_bar(sig0 + (int)(ksig & 1u), 160);
    ++ksig;
    tc_fence_after();
  };

  // ---- A1 rows: [local features | aggregate hi | 1 | aggregate lo] ----
  // The aggregate words are the same for every model of a tile: they are written with the
  // tile's first A1 row, and the later models rewrite only the local-feature words (when
  // the aggregate's position is a compile-time constant).
  const int awo = AWO >= 0 ? AWO : (T.dle >> 1);
  // digit of model i in a digit set
  auto dig = [&](DS ds, int i) -> uint32_t {
    if constexpr (RD) return (uint32_t)(ds >> (8 * (NM - 1 - i))) & 0xFFu;
    else return ds[i * 128 + row];
  };
  auto write_a1 = [&](int i, DS dg, bool with_agg, AggW aw) {
    const uint4* src = xw_s + (size_t)(P.off[i] + dig(dg, i)) * (KW >> 2);
    if constexpr (TF) {  // words 0-7: x hi, 8-11: aggregate hi and 1; 16-23: x lo, 24-27: aggregate lo
      const uint4 a = src[0], b = src[1], c = src[2], d = src[3];
      const uint32_t vh[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
      const uint32_t vl[8] = {c.x, c.y, c.z, c.w, d.x, d.y, d.z, d.w};
      tmem_st_x8(tA + lane_off, vh);
      tmem_st_x8(tA + 16u + lane_off, vl);
      if (with_agg) {
        const uint32_t ah[4] = {aw.h.x, aw.h.y, aw.h.z, aw.h.w};
        const uint32_t al[4] = {aw.l.x, aw.l.y, aw.l.z, aw.l.w};
        tmem_st_x4(tA + 8u + lane_off, ah);
        tmem_st_x4(tA + 24u + lane_off, al);
      }
      return;
    }
    const uint4 aw4 = aw.h;
    if (AWO >= 0 && !with_agg) {
      uint32_t v[AWO > 0 ? AWO : 1];
#pragma unroll
      for (int q = 0; q < AWO / 4; ++q) {
        const uint4 w4 = src[q];
        v[4 * q + 0] = w4.x; v[4 * q + 1] = w4.y; v[4 * q + 2] = w4.z; v[4 * q + 3] = w4.w;
      }
      if constexpr (AWO == 4) tmem_st_x4(tA + lane_off, v);
      else if constexpr (AWO == 8) tmem_st_x8(tA + lane_off, v);
      return;
    }
    uint32_t v[KW];
#pragma unroll
    for (int q = 0; q < KW / 4; ++q) {
      const uint4 w4 = src[q];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int j = 4 * q + e;
        const int a = j - awo;
        const uint32_t x = e == 0 ? w4.x : e == 1 ? w4.y : e == 2 ? w4.z : w4.w;
        v[j] = a == 0 ? aw4.x : a == 1 ? aw4.y : a == 2 ? aw4.z : a == 3 ? aw4.w : x;
      }
    }
    if constexpr (KW == 8) tmem_st_x8(tA + lane_off, v);
    else tmem_st_x16(tA + lane_off, v);
  };
  // Digits of tile `tile` (in shared memory: written to buffer `into`).  Range mode:
  // from the index at the first tile, else `from` (the previous tile's digits) stepped
  // by the tile stride.
  auto tile_digits = [&](uint64_t tile, uint8_t* into, DS from, bool first) -> DS {
    const uint64_t t = tile * 128 + row;
    if constexpr (RD) {
      if (first) {
        const uint64_t idx = R.base + t;
        uint64_t d = 0;
#pragma unroll
        for (int i = 0; i < NM; ++i) d |= (uint64_t)((idx / P.stride[i]) % P.K[i]) << (8 * (NM - 1 - i));
        return d;
      }
      // One add steps every digit: with each byte biased by 256 - K_i, a byte overflows
      // exactly when its digit wraps, and the carry moves on to the next model's byte.
      // Bytes that did not wrap then drop their bias again.
      constexpr uint64_t ones = 0x0101010101010101ull & ((1ull << (8 * NM)) - 1);
      const uint64_t x = from + T.dstep;
      const uint64_t wrapped = ((x ^ from ^ T.dstep) >> 8) & ones;  // carry out of each byte
      return (x - (~(wrapped * 0xFFull) & T.dbias)) & ((1ull << (8 * NM)) - 1);
    } else if (MODE == kTcRange) {
      if (first) {
        const uint64_t idx = R.base + t;
#pragma unroll (NM > 0 ? NM : 1)
        for (int i = 0; i < N; ++i) into[i * 128 + row] = (uint8_t)((idx / P.stride[i]) % P.K[i]);
      } else {  // add the tile stride to the digits, last model first
        uint32_t carry = 0;
#pragma unroll (NM > 0 ? NM : 1)
        for (int i = N - 1; i >= 0; --i) {
          uint32_t d = (uint32_t)from[i * 128 + row] + T.step[i] + carry;
          carry = d >= (uint32_t)P.K[i];
          if (carry) d -= (uint32_t)P.K[i];
          into[i * 128 + row] = (uint8_t)d;
        }
      }
      return into;
    } else {
      uint64_t idx = t < n ? L.idx[t] : 0;
      if (t < n && idx >= P.total) {
        atomicOr(P.status, kStatusBadInput);
        idx = 0;  // compute on candidate 0, discard at the end
      }
      for (int i = 0; i < N; ++i) into[i * 128 + row] = (uint8_t)digit_of(P, idx, i);
      return into;
    }
  };
  // The aggregate state of a tile (fp32, model order) as the A1 words: bf16 hi/lo pairs;
  // its VRAM component (the same sum, unscaled) is the candidate's VRAM demand.
  auto tile_agg = [&](DS dg, float& vram) -> AggW {
    float A0 = 0.f, A1 = 0.f, A2 = 0.f;
#pragma unroll (NM > 0 ? NM : 1)
    for (int i = 0; i < N; ++i) {
      const float4 d = dem_s[P.off[i] + dig(dg, i)];
      A0 += d.x; A1 += d.y; A2 += d.z;
    }
    vram = A1;
    const float v0 = A0 * P.agg_scale[0], v1 = A1 * P.agg_scale[1], v2 = A2 * P.agg_scale[2];
    if constexpr (TF) {  // tf32 hi parts and 1.0; the lo parts
      const uint32_t h0 = tf32_bits(v0), h1 = tf32_bits(v1), h2 = tf32_bits(v2);
      return AggW{make_uint4(h0, h1, h2, 0x3F800000u),
                  make_uint4(__float_as_uint(v0 - __uint_as_float(h0)), __float_as_uint(v1 - __uint_as_float(h1)),
                             __float_as_uint(v2 - __uint_as_float(h2)), 0u)};
    }
    const uint32_t h0 = bf16_bits(v0), h1 = bf16_bits(v1), h2 = bf16_bits(v2);
    const uint32_t l0 = bf16_bits(v0 - __uint_as_float(h0 << 16));
    const uint32_t l1 = bf16_bits(v1 - __uint_as_float(h1 << 16));
    const uint32_t l2 = bf16_bits(v2 - __uint_as_float(h2 << 16));
    return AggW{make_uint4(h0 | (h1 << 16), h2 | (0x3F80u << 16) /* bf16 1.0 */, l0 | (l1 << 16), l2),
                make_uint4(0u, 0u, 0u, 0u)};
  };
  // Digits of a pipeline's first tile and its first A1 row (model m0) with the aggregate words.
  auto load_tile = [&](uint64_t tile, uint8_t* into, float& vram) -> DS {
    const DS d = tile_digits(tile, into, DS{}, true);
    write_a1(m0, d, true, tile_agg(d, vram));
    return d;
  };
  // the model-i A1 row of the current tile (aggregate words already in place when AWO >= 0)
  auto next_a1 = [&](int i, DS dg) {
    if (TF || AWO >= 0) {
      write_a1(i, dg, false, AggW{});
    } else {  // run-time layout: the whole row, aggregate recomputed
      float A0 = 0.f, A1 = 0.f, A2 = 0.f;
      for (int j = 0; j < N; ++j) {
        const float4 d = dem_s[P.off[j] + dig(dg, j)];
        A0 += d.x; A1 += d.y; A2 += d.z;
      }
      const float v0 = A0 * P.agg_scale[0], v1 = A1 * P.agg_scale[1], v2 = A2 * P.agg_scale[2];
      const uint32_t h0 = bf16_bits(v0), h1 = bf16_bits(v1), h2 = bf16_bits(v2);
      const uint32_t l0 = bf16_bits(v0 - __uint_as_float(h0 << 16));
      const uint32_t l1 = bf16_bits(v1 - __uint_as_float(h1 << 16));
      const uint32_t l2 = bf16_bits(v2 - __uint_as_float(h2 << 16));
      write_a1(i, dg, true, AggW{make_uint4(h0 | (h1 << 16), h2 | (0x3F80u << 16), l0 | (l1 << 16), l2), {}});
    }
  };

  // ---- objective and constraints, model by model, from the layer-3 outputs ----
  // Model j's two outputs (columns j and n3/2 + j of D3) are read once its layer 3 has
  // landed, and its terms join this thread's running objective for the tile; later
  // models' layer-3 MMAs add zero to those columns.
  const int half3 = N3 == 16 ? 8 : (T.n3 >> 1);
  constexpr float kBand = TF ? 0.f : 2e-2f;
  float acc_J = 0.f, acc_pen = 0.f;
  bool acc_ok = true, acc_near = true;
  // (the two loads are issued first; other work may run before `add_model` waits for them)
  auto load_model = [&](int j, uint32_t& a, uint32_t& b) {
    a = tmem_ld_x1(tD3 + lane_off + (uint32_t)j);
    b = tmem_ld_x1(tD3 + lane_off + (uint32_t)(half3 + j));
  };
  auto add_model = [&](int j, uint32_t a, uint32_t b, DS dg, uint64_t tile_f) {
    tmem_wait_ld_2(a, b);
    const float thr = tc_out(P, __uint_as_float(a) + s_b3[j][0]);
    const float lat = tc_out(P, __uint_as_float(b) + s_b3[j][1]);
    if (MODE == kTcList && L.pred) {
      const uint64_t t = tile_f * 128 + row;
      if (t < n && L.idx[t] < P.total) {
        L.pred[(t * N + j) * 2 + 0] = thr;
        L.pred[(t * N + j) * 2 + 1] = lat;
      }
    }
    if (UT) {  // Eq. 3 utility, floors f >= tau
      float f;
      acc_J += util_term(P, j, P.off[j] + dig(dg, j), thr, &f);
      const float tau = P.u_tau[j];
      acc_ok = acc_ok && (f >= tau);
      acc_near = acc_near && (f >= tau - kBand * fmaxf(fabsf(tau), fabsf(f)));
      return;
    }
    acc_J = fmaf(P.w[j], thr, acc_J);
    const float sla = P.sla[j];
    acc_ok = acc_ok && (lat <= sla);
    // shortlist test: within the bf16 error band of the ceiling (none for the exact variant)
    acc_near = acc_near && (lat <= sla + kBand * fmaxf(fabsf(sla), fabsf(lat)));
    const float over = lat - sla;
    acc_pen += over > 0.f ? over : 0.f;
  };
  // The end of a tile whose every model has been added: the VRAM bound, the earlier
  // passes' record, feasibility, the count and the top-k queue; then a fresh objective.
  // The list's k-th entry (the bar a candidate must pass to be queued) changes only in a
  // merge; each thread keeps a copy.
  float bar_s = -INFINITY;
  uint64_t bar_i = kEmptyIdx;
  auto reload_bar = [&]() {
    if (MODE == kTcRange) {
      const CtaTopK tk = topk();
      bar_s = tk.ls[kcap - 1];
      bar_i = tk.li[kcap - 1];
    }
  };
  auto finish_tile = [&](uint64_t tile_f, float vram) {
    const uint64_t t = tile_f * 128 + row;
    bool valid = t < n;
    uint64_t idx;
    if (MODE == kTcRange) {
      idx = R.base + t;
    } else {
      idx = valid ? L.idx[t] : 0;
      valid = valid && idx < P.total;
    }
    float J = acc_J, pen = acc_pen;
    bool sla_ok = acc_ok, sla_near = acc_near;
    acc_J = 0.f;
    acc_pen = 0.f;
    acc_ok = true;
    acc_near = true;
    if (MP && !T.pass_first && t < n) {  // the earlier passes' models
      const float4 pr = T.partial[t];
      J += pr.x;
      pen += pr.y;
      const uint32_t fl = __float_as_uint(pr.z);
      sla_ok = sla_ok && (fl & 1u);
      sla_near = sla_near && (fl & 2u);
    }
    if (MP && !T.pass_last) {  // (uniform) hand the partial objective to the next pass
      if (t < n) T.partial[t] = make_float4(J, pen, __uint_as_float((sla_ok ? 1u : 0u) | (sla_near ? 2u : 0u)), 0.f);
      return;
    }
    bool feas = valid && vram <= vcap;
    bool cand = feas;
    if (!UT && P.objective == MF_OBJ_SOFT_LAT) {
      J = fmaf(-P.soft_penalty, pen, J);
    } else {  // latency ceilings, or the utility's floors
      feas = feas && sla_ok;
      cand = cand && sla_near;
    }
    if (J != J) { feas = false; cand = false; }
    if (MODE == kTcList) {
      if (t < n) {
        L.score[t] = feas ? J : -INFINITY;
        if (L.feas) L.feas[t] = feas ? 1 : 0;
      }
    } else {
      my_count += feas ? 1u : 0u;
      const CtaTopK tk = topk();
      const bool push = cand && precedes(J, idx, bar_s, bar_i);
      if (push) {
        const int pos = atomicAdd(tk.qn, 1);
        tk.qs[pos] = J;
        tk.qi[pos] = idx;
      }
      // Candidates wait in the queue (against the list's k-th entry of the last merge)
      // until another tile's 128 might not fit; then one merge takes them all.
      named_bar(barid, 128);
      if (*(volatile int*)tk.qn > T.qcap - 128) {
        tc_topk_merge(tk, row, barid);
        reload_bar();
      }
    }
  };
  if (issuer) {
    // ---- the issuing warp: one MMA group per hand-off of the epilogue warps ----
    wait_bar(&bars[0], 0);  // weights landed
    uint64_t tile = gpipe;
    if (tile * 128 < n) {
      take();  // the first A1 row
      issue_mma1(m0);
      mma_commit_warp(barA);
    }
    for (; tile * 128 < n; tile += gstride) {
      const bool has_next = (tile + gstride) * 128 < n;
#pragma unroll (NM > 0 ? NM : 1)
      for (int i = m0; i < m1; ++i) {
        const bool next_l1 = i + 1 < m1 || has_next;
        if (T.h2 > 0) {
          take();  // H1 of model i stored
          issue_mma2(i);
          mma_commit_warp(barA);
        }
        if (next_l1) {
          take();  // accumulators read, the next A1 row written
          issue_mma1(i + 1 < m1 ? i + 1 : m0);
          mma_commit_warp(barA);
        }
        take();  // the last hidden layer of model i stored
        issue_mma3(i);
        mma_commit_warp(barB);
      }
    }
  } else {
    // ---- the epilogue warps ----
    reload_bar();
    uint64_t tile = gpipe;
    int buf = 0;
    float vram_cur = 0.f, vram_prev = 0.f, vram_nx = 0.f;  // VRAM demand of this thread's rows
    DS dcur{}, dprev{}, dnx{};
    if (tile * 128 < n) {
      dcur = load_tile(tile, digits, vram_cur);
      signal();  // ones block and the first A1 row
    }
    // the previous tile is finished once its last layer 3 (issued at the end of that
    // tile) has landed, during this tile's first model
    bool pending = false;
    // the next tile's digits, aggregate and first A1 row are prepared in stages, each
    // while one model's layer 2 runs
    const int st_dig = m0 + 1 < m1 ? m0 + 1 : m1 - 1;
    const int st_agg = m0 + 2 < m1 ? m0 + 2 : m1 - 1;
    AggW aw_nx{};
    for (; tile * 128 < n; tile += gstride) {
      uint8_t* buf_nx = digits + (buf ^ 1) * (MF_MAX_MODELS * 128);  // (shared-memory digits)
      const bool has_next = (tile + gstride) * 128 < n;
      auto stage = [&](int i) {
        if (has_next && i == st_dig) dnx = tile_digits(tile + gstride, buf_nx, dcur, false);
        if (has_next && i == st_agg) aw_nx = tile_agg(dnx, vram_nx);
      };
      // Work off the critical path, while layer 2 of model i runs (or, with one hidden
      // layer, after its layer-1 epilogue): the objective terms of the model whose layer
      // 3 has landed (at the first model: the previous tile's last, and that tile's end),
      // a stage of the next tile, the next A1 row.  The layer-3 outputs are loaded first
      // and used last.
      auto side_work = [&](int i) {
        uint32_t oa = 0u, ob = 0u;
        if (i > m0) {
          load_model(i - 1, oa, ob);
          stage(i);
          if (i + 1 < m1) next_a1(i + 1, dcur);
          add_model(i - 1, oa, ob, dcur, tile);
        } else {
          if (pending) load_model(m1 - 1, oa, ob);
          if (i + 1 < m1) next_a1(i + 1, dcur);
          if (pending) {  // (before the stage: with one model it overwrites these digits)
            add_model(m1 - 1, oa, ob, dprev, tile - gstride);
            finish_tile(tile - gstride, vram_prev);
          }
          stage(i);
        }
        if (i + 1 >= m1 && has_next) write_a1(m0, dnx, true, aw_nx);
      };
#pragma unroll (NM > 0 ? NM : 1)
      for (int i = m0; i < m1; ++i) {
        const bool l3 = i > m0 || pending;
        const bool next_l1 = i + 1 < m1 || has_next;
        // ---- layer 1 of model i landed: D1 -> H1 ----
        await_a();
        if constexpr (TF) {
          hidden_epilogue_tf<(S2 - 1) * 8>(tD + lane_off, tH1 + lane_off, tHlo + lane_off, []() {}, [&]() {
            if (l3) await_b();  // the previous model's layer 3 has read H
          });
        } else {
          hidden_epilogue<(S2 > 0 ? (S2 - 1) * 16 : 0)>(T.h1, tD + lane_off, tH1 + lane_off, []() {}, [&]() {
            if (l3) await_b();  // the previous model's layer 3 has read H
          });
        }
        if (T.h2 == 0) {  // one hidden layer: the next layer 1, then layer 3 of model i
          side_work(i);
          if (next_l1) signal();
          signal();
          continue;
        }
        signal();  // H1 stored: layer 2 of model i
        side_work(i);
        // ---- layer 2 of model i landed: D2 -> H2 ----
        await_a();
        if constexpr (TF) {
          hidden_epilogue_tf<S3 * 8>(
              tD + lane_off, tH2 + lane_off, tHlo + lane_off,
              [&]() {
                if (next_l1) signal();  // accumulators read, next A1 written: the next layer 1
              },
              []() {});
        } else {
          hidden_epilogue<(S3 > 0 ? S3 * 16 : 0)>(
              T.h2, tD + lane_off, tH2 + lane_off,
              [&]() {
                if (next_l1) signal();  // accumulators read, next A1 written: the next layer 1
              },
              []() {});
        }
        signal();  // H2 stored: layer 3 of model i
      }
      pending = true;
      dprev = dcur;
      dcur = dnx;
      vram_prev = vram_cur;
      vram_cur = vram_nx;
      buf ^= 1;
    }
    if (pending) {  // the last tile's last layer 3
      await_b();
      uint32_t oa, ob;
      load_model(m1 - 1, oa, ob);
      add_model(m1 - 1, oa, ob, dprev, tile - gstride);
      finish_tile(tile - gstride, vram_prev);
    }
  }
  if (MODE == kTcRange && (!MP || T.pass_last) && !issuer) {  // what is still queued joins the list
    const CtaTopK tk = topk();
    named_bar(barid, 128);
    if (*(volatile int*)tk.qn > 0) tc_topk_merge(tk, row, barid);
  }

  if (MODE == kTcRange && (!MP || T.pass_last) && !issuer) {
    const CtaTopK tk = topk();
    const size_t gl = ((size_t)blockIdx.x * npipes + pipe) * kcap;
    for (int e = row; e < kcap; e += 128) {
      R.lists_s[gl + e] = tk.ls[e];
      R.lists_i[gl + e] = tk.li[e];
    }
    unsigned int c = my_count;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
    if (lane == 0 && c) atomicAdd(R.count, (unsigned long long)c);
  }
  // Nothing of this CTA may still run when its tensor memory is freed: each issuing warp
  // commits its MMAs to the drain barrier, and everyone waits for them and for the weight
  // copy (after a wait that gave up, these are the only waits still made).
  if (issuer) mma_commit_warp(&bars[2 + 2 * npipes]);
  mbar_wait_drain(&bars[2 + 2 * npipes], 0, P.status);
  mbar_wait_drain(&bars[0], 0, P.status);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512) : "memory");
  }
}

// ---------------------------------------------------------------------------
// Host side: operand images, layout, launches
// ---------------------------------------------------------------------------
namespace {

uint16_t f2bf(float f) {  // round to nearest even
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7FFFFFFFu) > 0x7F800000u) return 0x7FC0;
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

float bf2f(uint16_t b) {
  const uint32_t u = (uint32_t)b << 16;
  float f;
  std::memcpy(&f, &u, 4);
  return f;
}

// Byte offset of element (r, k) of a K-major no-swizzle UMMA operand with kdim columns:
// 8-row x 16-byte core matrices, K-adjacent cores 128 B apart, 8-row groups kdim*16 B apart.
size_t umma_off(int r, int k, int kdim) {
  return (size_t)(r >> 3) * (size_t)(kdim / 8) * 128u + (size_t)(k >> 3) * 128u + (size_t)(r & 7) * 16u +
         (size_t)(k & 7) * 2u;
}

// The same for 4-byte (tf32) elements: 4 per 16-byte core-matrix row.
size_t umma_off4(int r, int k, int kdim) {
  return (size_t)(r >> 3) * (size_t)(kdim / 4) * 128u + (size_t)(k >> 2) * 128u + (size_t)(r & 7) * 16u +
         (size_t)(k & 3) * 4u;
}

// v rounded to tf32 (nearest, ties away from zero), as an fp32 value.
float tf32_round(double v) {
  const float f = (float)v;
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7F800000u) != 0x7F800000u) u = (u + 0x1000u) & 0xFFFFE000u;  // (inf and NaN as they are)
  float r;
  std::memcpy(&r, &u, 4);
  return r;
}

int round_up(int v, int a) { return (v + a - 1) / a * a; }

size_t topk_bytes_pipe(int kcap, int qcap) {
  return (sizeof(uint64_t) + sizeof(float)) * (2 * (size_t)kcap + qcap) + 16;
}

size_t image_bytes(const Params& P, int k1, int n3) {
  const int hl = P.h2 > 0 ? P.h2 : P.h1;
  const size_t per = (size_t)P.h1 * k1 * 2 + (size_t)P.h2 * (P.h1 + 16) * 2 + (size_t)n3 * hl * 2;
  return per * P.n_models;
}

constexpr uint32_t kSmemLimit = 227 * 1024 - 1024;  // static shared variables take the rest

// Shared-memory layout for a launch with per-pipeline lists of kcap entries.
void layout_smem(const Params& P, TcArgs& T, int kcap) {
  const int sumK = P.off[P.n_models - 1] + P.K[P.n_models - 1];
  uint32_t o = round_up((int)T.img_bytes, 1024);
  T.sm_xw = o; o += round_up(sumK * T.kw * 4, 16);
  T.sm_dem = o; o += sumK * 16;
  T.sm_rows = o; o += T.pipes * 2 * MF_MAX_MODELS * 128;  // byte digits of two tiles per pipeline
  // the candidate queue: 512 entries (a merge every few tiles) where shared memory allows,
  // else one tile's 128 (a merge after every tile that queued a candidate)
  const uint32_t rest = o + 16 + 8 * (3 + 2 * kTcMaxPipes);
  T.qcap = 128;
  if (kcap > 0 && rest + T.pipes * topk_bytes_pipe(kcap, 512) <= kSmemLimit) T.qcap = 512;
  T.sm_topk = o; o += kcap > 0 ? (uint32_t)(T.pipes * topk_bytes_pipe(kcap, T.qcap)) : 0u;
  o = round_up((int)o, 16);
  T.sm_bar = o; o += 8 * (3 + 2 * kTcMaxPipes);
  T.sm_total = o;
  T.kcap = kcap;
}

constexpr size_t kPassImageBudget = 160 * 1024;      // weights staged per pass

using TcFn = void (*)(const Params, const TcArgs, const RangeArgs, const TcList);

// Instantiations: the two benchmark shapes (d_L 8, 64-64 and d_L 16, 128-128, up to 8
// models) with all counts fixed at compile time, and a run-time fallback per A1 row width.
template <int MODE, bool MP, bool UT>
TcFn tc_kernel_mode(const TcArgs& T, int n_models) {
  // the exact fp32 variant (d_L 8, 64-64): S1 = k1 / 8, S2 = h1 / 8 + 1, S3 = hl / 8
  if (T.tf) return k_score_tc<MODE, 16, 8, 2, 9, 8, 16, MP, UT, 0, true>;
  // S1 = k1 / 16, S2 = h1 / 16 + 1 (the b2 step), S3 = hl / 16
  if (T.kw == 8 && T.dle == 8 && T.h1 == 64 && T.h2 == 64 && T.n3 == 16) {
    if constexpr (MODE == kTcRange && !MP && !UT) {
      if (n_models == 6) return k_score_tc<MODE, 8, 4, 1, 5, 4, 16, MP, UT, 6, false>;  // the 24^6 workload's shape
    }
    return k_score_tc<MODE, 8, 4, 1, 5, 4, 16, MP, UT, 0, false>;
  }
  if (T.kw == 16 && T.dle == 16 && T.h1 == 128 && T.h2 == 128 && T.n3 == 16)
    return k_score_tc<MODE, 16, 8, 2, 9, 8, 16, MP, UT, 0, false>;
  if (T.kw == 8) return k_score_tc<MODE, 8, -1, 0, 0, 0, 0, MP, UT, 0, false>;
  return k_score_tc<MODE, 16, -1, 0, 0, 0, 0, MP, UT, 0, false>;
}

template <bool UT>
TcFn tc_kernel_ut(int mode, const TcArgs& T, int n) {
  if (T.npasses > 1)
    return mode == kTcRange ? tc_kernel_mode<kTcRange, true, UT>(T, n) : tc_kernel_mode<kTcList, true, UT>(T, n);
  return mode == kTcRange ? tc_kernel_mode<kTcRange, false, UT>(T, n) : tc_kernel_mode<kTcList, false, UT>(T, n);
}

TcFn tc_kernel(int mode, const TcArgs& T, bool util, int n) {
  return util ? tc_kernel_ut<true>(mode, T, n) : tc_kernel_ut<false>(mode, T, n);
}
constexpr uint32_t kSmemFloor = 120 * 1024;          // keeps one CTA (one TMEM owner) per SM

}  // namespace

namespace {

// Candidates per launch when the models run in several passes (the partial records of
// one launch: 16 B each, 256 MiB).
constexpr uint64_t kPassSpan = 1ull << 24;

// Per-launch fields of pass p.
void set_pass(TcArgs& T, int p, float4* partial) {
  T.m0 = T.pass_m[p];
  T.m1 = T.pass_m[p + 1];
  T.pass_first = p == 0;
  T.pass_last = p + 1 == T.npasses;
  T.img_lo = T.off_b1[T.m0];
  T.img_copy = (p + 1 < T.npasses ? T.off_b1[T.m1] : T.img_total) - T.img_lo;
  T.partial = partial;
}

mf_status ensure_partial(mf_ctx* c, uint64_t n, cudaStream_t s, float4** out) {
  *out = nullptr;
  if (c->tc.npasses == 1) return MF_OK;
  const size_t need = sizeof(float4) * (size_t)(n < kPassSpan ? (n > 0 ? n : 1) : kPassSpan);
  if (need > c->partial_bytes) {
    MF_CUDA(cudaStreamSynchronize(s));
    cudaFree(c->d_partial);
    c->d_partial = nullptr;
    c->partial_bytes = 0;
    MF_CUDA(cudaMalloc(&c->d_partial, need));
    c->partial_bytes = need;
  }
  *out = static_cast<float4*>(c->d_partial);
  return MF_OK;
}

}  // namespace

bool tc_supported(const Params& P, std::string* why) {
  auto no = [&](const char* m) { if (why) *why = m; return false; };
  if (P.h1 % 32 || P.h1 > 256) return no("hidden1 must be a multiple of 32 up to 256");
  if (P.h2 % 32 || P.h2 > 256) return no("hidden2 must be 0 or a multiple of 32 up to 256");
  if (P.d_local > 24) return no("d_local must be <= 24");
  const int hmax = P.h1 > P.h2 ? P.h1 : P.h2;
  const int dle = P.d_local + (P.d_local & 1);
  const int k1 = round_up(dle + 8, 16);
  const int n3 = 2 * P.n_models <= 16 ? 16 : 32;
  const int col_a = hmax + hmax / 2 + 8;
  const int col_d3 = round_up(col_a + k1 / 2, 16);
  if (round_up(col_d3 + n3, 32) > 512) return no("tensor-memory footprint above 512 columns");
  if (image_bytes(P, k1, n3) / P.n_models > kPassImageBudget)
    return no("one model's bf16 weights exceed the shared-memory budget");
  return true;
}

bool tc_exact_supported(const Params& P) {
  return P.d_local == 8 && P.h1 == 64 && P.h2 == 64 && P.n_models <= 8;
}

bool tc_fits(const mf_ctx* c, int kcap) {
  TcArgs T = c->tc;
  layout_smem(c->P, T, kcap);
  return T.sm_total <= kSmemLimit;
}

int tc_grid(const mf_ctx* c) { return c->num_sms * c->tc.pipes; }

namespace {

// The exact fp32 variant's layout and operand images (d_L 8, 12 -> 64 -> 64 -> 2): every
// operand as a tf32 hi part and the rest (a lo part, also tf32), so that hi.hi + hi.lo +
// lo.hi carries about 22 bits of each product.
mf_status tc_prepare_exact(mf_ctx* c) {
  const Params& P = c->P;
  TcArgs& T = c->tc;
  const int N = P.n_models, dl = P.d_local, h1 = P.h1, h2 = P.h2, hl = h2, din = P.d_in;
  T.tf = 1;
  T.dle = dl;
  T.k1 = 16;   // [x (8) | aggregate (3) | 1 | 0 0 0 0]
  T.kw = 16;   // words per option: x hi (8), x lo (8)
  T.h1 = h1;
  T.h2 = h2;
  T.hl = hl;
  T.n3 = 16;
  // TMEM columns of a pipeline: D (64 fp32) | H hi (64) | ones (8) | H lo (64) | A1 hi (16), A1 lo (16) | D3 (16)
  T.col_d = 0;
  T.col_h = h1;
  T.col_ones = 2 * h1;
  T.col_hlo = T.col_ones + 8;
  T.col_a = T.col_hlo + h1;
  T.col_d3 = round_up(T.col_a + 32, 16);
  T.pipe_stride = round_up(T.col_d3 + T.n3, 32);
  T.pipes = 512 / T.pipe_stride;
  if (T.pipes > 2) T.pipes = 2;
  // per model: B1 [h1 x 16], B2 [h2 x (h1 + 8)] (its last K-step holds b2 hi, lo against
  // the ones block), B3 [16 x hl], each as a hi image followed by a lo image
  const int k2 = h1 + 8;
  const size_t b1 = (size_t)h1 * T.k1 * 4, b2 = (size_t)h2 * k2 * 4, b3 = (size_t)T.n3 * hl * 4;
  T.img_lo1 = (uint32_t)b1;
  T.img_lo2 = (uint32_t)b2;
  T.img_lo3 = (uint32_t)b3;
  std::vector<float> w(P.per_model * N);
  cudaError_t e = cudaMemcpy(w.data(), P.w32, sizeof(float) * w.size(), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "tc_prepare: read weights");
  std::vector<unsigned char> img;
  auto put = [&](size_t base, size_t lo_off, int r, int k, int kdim, double v) {
    const float hi = tf32_round(v), lo = tf32_round(v - (double)hi);
    std::memcpy(img.data() + base + umma_off4(r, k, kdim), &hi, 4);
    std::memcpy(img.data() + base + lo_off + umma_off4(r, k, kdim), &lo, 4);
  };
  const double s3 = P.agg_scale[3];
  for (int i = 0; i < N; ++i) {
    const float* W1 = w.data() + (size_t)i * P.per_model;
    const float* bb1 = W1 + (size_t)h1 * din;
    const float* W2 = bb1 + h1;
    const float* bb2 = W2 + (size_t)h2 * h1;
    const float* W3 = bb2 + h2;
    T.off_b1[i] = (uint32_t)img.size();
    img.resize(img.size() + 2 * b1, 0);
    for (int j = 0; j < h1; ++j) {
      for (int k = 0; k < dl + 3; ++k) put(T.off_b1[i], b1, j, k, T.k1, W1[(size_t)j * din + k]);
      // the constant-1 column: b1 plus the weight of the constant feature N * s_3
      put(T.off_b1[i], b1, j, dl + 3, T.k1, (double)bb1[j] + (double)W1[(size_t)j * din + dl + 3] * s3 * N);
    }
    T.off_b2[i] = (uint32_t)img.size();
    img.resize(img.size() + 2 * b2, 0);
    for (int j = 0; j < h2; ++j) {
      for (int k = 0; k < h1; ++k) put(T.off_b2[i], b2, j, k, k2, W2[(size_t)j * h1 + k]);
      // b2 as two tf32 values (hi, then the rest) in the hi image, against the ones (1, 1)
      const float bh = tf32_round(bb2[j]), bl = tf32_round((double)bb2[j] - (double)bh);
      std::memcpy(img.data() + T.off_b2[i] + umma_off4(j, h1, k2), &bh, 4);
      std::memcpy(img.data() + T.off_b2[i] + umma_off4(j, h1 + 1, k2), &bl, 4);
    }
    T.off_b3[i] = (uint32_t)img.size();
    img.resize(img.size() + 2 * b3, 0);
    T.img_model = (uint32_t)(2 * (b1 + b2 + b3));
    for (int k = 0; k < hl; ++k) {
      put(T.off_b3[i], b3, i, k, hl, W3[k]);
      put(T.off_b3[i], b3, T.n3 / 2 + i, k, hl, W3[hl + k]);
    }
  }
  img.resize(round_up((int)img.size(), 16), 0);
  T.img_total = (uint32_t)img.size();
  T.npasses = 0;
  T.pass_m[0] = 0;
  for (int i = 0; i < N;) {
    int j = i + 1;
    while (j < N && (size_t)((j + 1 < N ? T.off_b1[j + 1] : T.img_total) - T.off_b1[i]) <= kPassImageBudget) ++j;
    T.pass_m[++T.npasses] = j;
    i = j;
  }
  T.img_bytes = 0;
  for (int p = 0; p < T.npasses; ++p) {
    const uint32_t lo = T.off_b1[T.pass_m[p]];
    const uint32_t hi = p + 1 < T.npasses ? T.off_b1[T.pass_m[p + 1]] : T.img_total;
    if (hi - lo > T.img_bytes) T.img_bytes = hi - lo;
  }
  set_pass(T, 0, nullptr);
  if (T.npasses == 1) { T.pass_last = 1; }
  // option words: x hi (8), x lo (8)
  const int sumK = c->sumK;
  std::vector<float> x((size_t)sumK * dl);
  e = cudaMemcpy(x.data(), P.x, sizeof(float) * x.size(), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "tc_prepare: read tables");
  std::vector<float> xw((size_t)sumK * T.kw, 0.f);
  for (int r = 0; r < sumK; ++r)
    for (int k = 0; k < dl; ++k) {
      const float v = x[(size_t)r * dl + k], hi = tf32_round(v);
      xw[(size_t)r * T.kw + k] = hi;
      xw[(size_t)r * T.kw + 8 + k] = tf32_round((double)v - (double)hi);
    }
  const size_t o_xw = round_up((int)img.size(), 256);
  const size_t total = o_xw + round_up((int)(xw.size() * 4), 256);
  MF_CUDA(cudaMalloc(&c->d_tc, total));
  c->tc_bytes = total;
  unsigned char* base = static_cast<unsigned char*>(c->d_tc);
  MF_CUDA(cudaMemcpy(base, img.data(), img.size(), cudaMemcpyHostToDevice));
  MF_CUDA(cudaMemcpy(base + o_xw, xw.data(), xw.size() * 4, cudaMemcpyHostToDevice));
  c->stats.h2d_bytes_create += img.size() + xw.size() * 4;
  T.img = base;
  T.xw = reinterpret_cast<const uint32_t*>(base + o_xw);
  for (int u = 0; u < 2; ++u) {
    MF_CUDA(cudaFuncSetAttribute(tc_kernel(kTcRange, T, u, P.n_models), cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit));
    MF_CUDA(cudaFuncSetAttribute(tc_kernel(kTcList, T, u, P.n_models), cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit));
  }
  layout_smem(P, T, 0);
  if (T.sm_total > kSmemLimit) {
    set_error("exact tensor-core path: tables and weights exceed shared memory");
    return MF_EUNSUPPORTED;
  }
  return MF_OK;
}

}  // namespace

mf_status tc_prepare(mf_ctx* c, bool exact) {
  const Params& P = c->P;
  TcArgs& T = c->tc;
  std::memset(&T, 0, sizeof(T));
  if (exact) return tc_prepare_exact(c);
  const int N = P.n_models, dl = P.d_local, h1 = P.h1, h2 = P.h2, hl = h2 > 0 ? h2 : h1;
  const int din = P.d_in;
  T.dle = dl + (dl & 1);
  T.k1 = round_up(T.dle + 8, 16);
  T.kw = T.k1 / 2;
  T.h1 = h1;
  T.h2 = h2;
  T.hl = hl;
  T.n3 = 2 * N <= 16 ? 16 : 32;
  const int hmax = h1 > h2 ? h1 : h2;
  T.col_d = 0;
  T.col_h = hmax;
  T.col_ones = hmax + hmax / 2;
  T.col_a = T.col_ones + 8;
  T.col_d3 = round_up(T.col_a + T.kw, 16);
  T.pipe_stride = round_up(T.col_d3 + T.n3, 32);
  T.pipes = 512 / T.pipe_stride;
  if (T.pipes > kTcMaxPipes) T.pipes = kTcMaxPipes;

  // B operand images (K-major): B1 [h1 x k1], B2 [h2 x (h1 + 16)], B3 [n3 x hl]
  const int k2 = h1 + 16, k3 = hl;
  const size_t b1_bytes = (size_t)h1 * T.k1 * 2, b2_bytes = (size_t)h2 * k2 * 2, b3_bytes = (size_t)T.n3 * k3 * 2;
  std::vector<unsigned char> img;
  const double s3 = P.agg_scale[3];
  std::vector<float> w(P.per_model * N);
  cudaError_t e = cudaMemcpy(w.data(), P.w32, sizeof(float) * w.size(), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "tc_prepare: read weights");
  auto put = [&](uint32_t base, int r, int k, int kdim, double v) {
    const uint16_t b = f2bf((float)v);
    std::memcpy(img.data() + base + umma_off(r, k, kdim), &b, 2);
  };
  // a bias as a bf16 pair (hi, lo) whose sum carries ~16 mantissa bits
  auto put_bias = [&](uint32_t base, int r, int k, int kdim, float v) {
    const uint16_t hi = f2bf(v);
    put(base, r, k, kdim, bf2f(hi));
    put(base, r, k + 1, kdim, (double)v - (double)bf2f(hi));
  };
  for (int i = 0; i < N; ++i) {
    const float* src = w.data() + (size_t)i * P.per_model;
    const float* W1 = src;
    const float* b1 = W1 + (size_t)h1 * din;
    const float* W2 = b1 + h1;
    const float* b2 = W2 + (size_t)h2 * h1;
    const float* W3 = h2 > 0 ? b2 + h2 : W2;
    T.off_b1[i] = (uint32_t)img.size();
    img.resize(img.size() + b1_bytes, 0);
    for (int j = 0; j < h1; ++j) {
      for (int k = 0; k < dl; ++k) put(T.off_b1[i], j, k, T.k1, W1[(size_t)j * din + k]);
      // A1 carries the scaled aggregate (hi and lo parts), so these columns hold W1 as is;
      // the constant-1 column carries b1 plus the weight of the constant feature N * s_3
      for (int q = 0; q < 3; ++q) {
        put(T.off_b1[i], j, T.dle + q, T.k1, W1[(size_t)j * din + dl + q]);
        put(T.off_b1[i], j, T.dle + 4 + q, T.k1, W1[(size_t)j * din + dl + q]);
      }
      put(T.off_b1[i], j, T.dle + 3, T.k1, (double)b1[j] + (double)W1[(size_t)j * din + dl + 3] * s3 * N);
    }
    T.off_b2[i] = (uint32_t)img.size();
    img.resize(img.size() + b2_bytes, 0);
    for (int j = 0; j < h2; ++j) {
      for (int k = 0; k < h1; ++k) put(T.off_b2[i], j, k, k2, W2[(size_t)j * h1 + k]);
      put_bias(T.off_b2[i], j, h1, k2, b2[j]);
    }
    T.off_b3[i] = (uint32_t)img.size();
    img.resize(img.size() + b3_bytes, 0);
    T.img_model = (uint32_t)(b1_bytes + b2_bytes + b3_bytes);  // the kernel steps descriptors by it
    for (int k = 0; k < hl; ++k) {
      put(T.off_b3[i], i, k, k3, W3[k]);
      put(T.off_b3[i], T.n3 / 2 + i, k, k3, W3[hl + k]);
    }
  }
  img.resize(round_up((int)img.size(), 16), 0);
  T.img_total = (uint32_t)img.size();
  // passes: consecutive models whose images fit the budget together
  T.npasses = 0;
  T.pass_m[0] = 0;
  for (int i = 0; i < N;) {
    int j = i + 1;
    while (j < N && (size_t)((j + 1 < N ? T.off_b1[j + 1] : T.img_total) - T.off_b1[i]) <= kPassImageBudget) ++j;
    T.pass_m[++T.npasses] = j;
    i = j;
  }
  T.img_bytes = 0;
  for (int p = 0; p < T.npasses; ++p) {
    const uint32_t lo = T.off_b1[T.pass_m[p]];
    const uint32_t hi = p + 1 < T.npasses ? T.off_b1[T.pass_m[p + 1]] : T.img_total;
    if (hi - lo > T.img_bytes) T.img_bytes = hi - lo;
  }
  set_pass(T, 0, nullptr);  // single-pass defaults (a pass-0 image of all models)
  if (T.npasses == 1) { T.pass_last = 1; }

  // local-feature words
  const int sumK = c->sumK;
  std::vector<float> x((size_t)sumK * dl);
  e = cudaMemcpy(x.data(), P.x, sizeof(float) * x.size(), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "tc_prepare: read tables");
  std::vector<uint32_t> xw((size_t)sumK * T.kw, 0u);
  for (int r = 0; r < sumK; ++r)
    for (int k = 0; k < dl; ++k)
      xw[(size_t)r * T.kw + k / 2] |= (uint32_t)f2bf(x[(size_t)r * dl + k]) << (16 * (k & 1));
  const size_t o_xw = round_up((int)img.size(), 256);
  const size_t total = o_xw + round_up((int)(xw.size() * 4), 256);
  MF_CUDA(cudaMalloc(&c->d_tc, total));
  c->tc_bytes = total;
  unsigned char* base = static_cast<unsigned char*>(c->d_tc);
  MF_CUDA(cudaMemcpy(base, img.data(), img.size(), cudaMemcpyHostToDevice));
  MF_CUDA(cudaMemcpy(base + o_xw, xw.data(), xw.size() * 4, cudaMemcpyHostToDevice));
  c->stats.h2d_bytes_create += img.size() + xw.size() * 4;
  T.img = base;
  T.xw = reinterpret_cast<const uint32_t*>(base + o_xw);
  for (int u = 0; u < 2; ++u) {
    MF_CUDA(cudaFuncSetAttribute(tc_kernel(kTcRange, T, u, P.n_models), cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit));
    MF_CUDA(cudaFuncSetAttribute(tc_kernel(kTcList, T, u, P.n_models), cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit));
  }
  layout_smem(P, T, 0);
  if (T.sm_total > kSmemLimit) {
    set_error("tensor-core path: tables and weights exceed shared memory");
    return MF_EUNSUPPORTED;
  }
  return MF_OK;
}


mf_status tc_search_chunk(mf_ctx* c, const RangeArgs& a, cudaStream_t s, int* nlaunch) {
  TcArgs T = c->tc;
  layout_smem(c->P, T, a.k);
  if (T.sm_total > kSmemLimit) {
    set_error("tensor-core path: top-k lists do not fit shared memory; use a smaller k");
    return MF_EUNSUPPORTED;
  }
  // digits of the per-tile index stride (grid x pipes x 128), modulo |Lambda|
  const uint64_t stride = ((uint64_t)c->num_sms * T.pipes * 128) % c->P.total;
  uint64_t v = stride;
  T.dstep = 0;
  T.dbias = 0;
  for (int i = c->P.n_models - 1; i >= 0; --i) {
    T.step[i] = (uint32_t)(v % (uint64_t)c->P.K[i]);
    v /= (uint64_t)c->P.K[i];
    if (c->P.n_models <= 7) {
      const int sh = 8 * (c->P.n_models - 1 - i);
      T.dstep |= (uint64_t)(T.step[i] + 256u - (uint32_t)c->P.K[i]) << sh;
      T.dbias |= (uint64_t)(256u - (uint32_t)c->P.K[i]) << sh;
    }
  }
  const uint32_t smem = T.sm_total > kSmemFloor ? T.sm_total : kSmemFloor;
  TcList L{};
  float4* partial = nullptr;
  mf_status st = ensure_partial(c, a.len, s, &partial);
  if (st != MF_OK) return st;
  // one launch per pass and span of candidates; the lists and the count belong to the
  // last pass only
  const uint64_t span = T.npasses == 1 ? (a.len > 0 ? a.len : 1) : kPassSpan;
  int launches = 0;
  RangeArgs r = a;
  for (uint64_t b = 0; b == 0 || b < a.len; b += span) {
    r.base = a.base + b;
    r.len = a.len - b < span ? a.len - b : span;
    r.first = a.first && b == 0;
    for (int p = 0; p < T.npasses; ++p) {
      set_pass(T, p, partial);
      tc_kernel(kTcRange, T, c->P.objective == MF_OBJ_UTILITY, c->P.n_models)<<<c->num_sms, T.pipes * kTcPipeThreads, smem, s>>>(c->P, T, r, L);
      MF_CUDA(cudaGetLastError());
      ++launches;
    }
  }
  *nlaunch = launches;
  return MF_OK;
}

mf_status tc_score_list(mf_ctx* c, const uint64_t* idx, uint64_t n, float* score, uint8_t* feas, float* pred,
                        cudaStream_t s) {
  if (n == 0) return MF_OK;
  TcArgs T = c->tc;
  layout_smem(c->P, T, 0);
  const uint32_t smem = T.sm_total > kSmemFloor ? T.sm_total : kSmemFloor;
  float4* partial = nullptr;
  mf_status st = ensure_partial(c, n, s, &partial);
  if (st != MF_OK) return st;
  const uint64_t span = T.npasses == 1 ? n : kPassSpan;
  const int N = c->P.n_models;
  RangeArgs R{};
  for (uint64_t b = 0; b < n; b += span) {
    const uint64_t m = n - b < span ? n - b : span;
    const uint64_t tiles = (m + 127) / 128;
    const uint64_t per_cta = (uint64_t)T.pipes;
    uint64_t grid = (tiles + per_cta - 1) / per_cta;
    if (grid > (uint64_t)c->num_sms) grid = c->num_sms;
    TcList L{idx + b, m, score + b, feas ? feas + b : nullptr, pred ? pred + b * N * 2 : nullptr};
    for (int p = 0; p < T.npasses; ++p) {
      set_pass(T, p, partial);
      tc_kernel(kTcList, T, c->P.objective == MF_OBJ_UTILITY, c->P.n_models)<<<(unsigned)grid, T.pipes * kTcPipeThreads, smem, s>>>(c->P, T, R, L);
      MF_CUDA(cudaGetLastError());
    }
  }
  return MF_OK;
}

}  // namespace mf
