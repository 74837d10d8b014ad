// Reductions of the exhaustive search (the argmax of Sec. II extended to a
// top-k): merging the per-CTA running lists, and selecting the top-k of a
// re-scored shortlist.  Order: J descending, index ascending.
#include "mf_internal.cuh"

namespace mf {

// Pairwise merge tree over `nlists` sorted lists of length k, by one CTA.
// Each element's output position is its position in its own list plus the
// number of elements of the partner list that precede it (binary search);
// elements at positions >= k are dropped.  Indices are distinct, so positions
// never collide.
__global__ void __launch_bounds__(1024)
k_merge_lists(const float* __restrict__ in_s, const uint64_t* __restrict__ in_i, int nlists, int k,
              float* a_s, uint64_t* a_i, float* b_s, uint64_t* b_i,
              float* __restrict__ out_s, uint64_t* __restrict__ out_i) {
  const float* src_s = in_s;
  const uint64_t* src_i = in_i;
  float* dst_s = a_s;
  uint64_t* dst_i = a_i;
  int n = nlists;
  while (n > 1) {
    const int m = (n + 1) / 2;
    for (int e = threadIdx.x; e < m * k; e += blockDim.x) { dst_s[e] = -INFINITY; dst_i[e] = kEmptyIdx; }
    __syncthreads();
    for (int e = threadIdx.x; e < 2 * m * k; e += blockDim.x) {
      const int p = e / (2 * k);
      const int r = e - p * 2 * k;
      const int which = r / k;
      const int pos = r - which * k;
      const int mine = 2 * p + which;
      if (mine >= n) continue;
      const float s = src_s[(size_t)mine * k + pos];
      const uint64_t id = src_i[(size_t)mine * k + pos];
      if (id == kEmptyIdx) continue;
      int cnt = 0;
      const int other = 2 * p + 1 - which;
      if (other < n) {
        const float* os = src_s + (size_t)other * k;
        const uint64_t* oi = src_i + (size_t)other * k;
        int lo = 0, hi = k;
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if (precedes(os[mid], oi[mid], s, id)) lo = mid + 1; else hi = mid;
        }
        cnt = lo;
      }
      const int rank = pos + cnt;
      if (rank < k) { dst_s[(size_t)p * k + rank] = s; dst_i[(size_t)p * k + rank] = id; }
    }
    __syncthreads();
    src_s = dst_s;
    src_i = dst_i;
    dst_s = (dst_s == a_s) ? b_s : a_s;
    dst_i = (dst_i == a_i) ? b_i : a_i;
    n = m;
  }
  for (int e = threadIdx.x; e < k; e += blockDim.x) { out_s[e] = src_s[e]; out_i[e] = src_i[e]; }
}

// Bitonic sort of up to 8192 (score, index) pairs in shared memory by the total
// order; the first k go to the output.
__global__ void __launch_bounds__(1024)
k_select_topk(const float* __restrict__ in_s, const uint64_t* __restrict__ in_i, int n, int n2, int k,
              float* __restrict__ out_s, uint64_t* __restrict__ out_i) {
  extern __shared__ __align__(16) unsigned char smem[];
  uint64_t* si = reinterpret_cast<uint64_t*>(smem);
  float* ss = reinterpret_cast<float*>(si + n2);
  for (int e = threadIdx.x; e < n2; e += blockDim.x) {
    if (e < n) { ss[e] = in_s[e]; si[e] = in_i[e]; }
    else { ss[e] = -INFINITY; si[e] = kEmptyIdx; }
    if (ss[e] == -INFINITY) si[e] = kEmptyIdx;  // infeasible entries sort last
  }
  __syncthreads();
  for (int size = 2; size <= n2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < n2; i += blockDim.x) {
        const int j = i ^ stride;
        if (j > i) {
          const bool up = (i & size) == 0;
          const bool sw = up ? precedes(ss[j], si[j], ss[i], si[i]) : precedes(ss[i], si[i], ss[j], si[j]);
          if (sw) {
            const float ts = ss[i]; ss[i] = ss[j]; ss[j] = ts;
            const uint64_t ti = si[i]; si[i] = si[j]; si[j] = ti;
          }
        }
      }
      __syncthreads();
    }
  }
  for (int e = threadIdx.x; e < k; e += blockDim.x) { out_s[e] = ss[e]; out_i[e] = si[e]; }
}

mf_status merge_lists(mf_ctx* c, const float* ls, const uint64_t* li, int nlists, int k,
                      float* tmp_s, uint64_t* tmp_i, float* out_s, uint64_t* out_i,
                      cudaStream_t s) {
  // tmp holds two buffers of ceil(nlists / 2) * k entries each
  const size_t half = (size_t)((nlists + 1) / 2) * k;
  k_merge_lists<<<1, 1024, 0, s>>>(ls, li, nlists, k, tmp_s, tmp_i, tmp_s + half, tmp_i + half,
                                   out_s, out_i);
  MF_CUDA(cudaGetLastError());
  (void)c;
  return MF_OK;
}

mf_status select_topk(mf_ctx* c, const float* in_s, const uint64_t* in_i, int n, int k,
                      float* out_s, uint64_t* out_i, cudaStream_t s) {
  int n2 = 1;
  while (n2 < n) n2 <<= 1;
  if (n2 < k) n2 = k;
  int p2 = 1;
  while (p2 < n2) p2 <<= 1;
  n2 = p2;
  if (n2 > 8192) {
    set_error("select_topk: more than 8192 entries");
    return MF_EINVAL;
  }
  const size_t smem = (size_t)n2 * (sizeof(float) + sizeof(uint64_t));
  MF_CUDA(cudaFuncSetAttribute(k_select_topk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  k_select_topk<<<1, 1024, smem, s>>>(in_s, in_i, n, n2, k, out_s, out_i);
  MF_CUDA(cudaGetLastError());
  (void)c;
  return MF_OK;
}

}  // namespace mf
