// Tensor-core (tcgen05, bf16) scorer -- placeholder until the kernel lands.
#include "mf_internal.cuh"

namespace mf {

bool tc_supported(const Params& P, std::string* why) {
  (void)P;
  if (why) *why = "not built in this version";
  return false;
}
mf_status tc_prepare(mf_ctx* c) { (void)c; return MF_EUNSUPPORTED; }
int tc_grid(const mf_ctx* c) { return c->num_sms; }
mf_status tc_search_chunk(mf_ctx* c, const RangeArgs& a, cudaStream_t s) {
  (void)c; (void)a; (void)s;
  return MF_EUNSUPPORTED;
}
mf_status tc_score_list(mf_ctx* c, const uint64_t* idx, uint64_t n, float* score, uint8_t* feas,
                        float* pred, cudaStream_t s) {
  (void)c; (void)idx; (void)n; (void)score; (void)feas; (void)pred; (void)s;
  return MF_EUNSUPPORTED;
}

}  // namespace mf
