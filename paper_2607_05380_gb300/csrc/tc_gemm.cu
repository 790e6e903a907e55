// tc_gemm.cu -- tensor-core grouped GEMM plan (placeholder: disabled).
#include "tc_gemm.cuh"

namespace tp {

tp_status tc_build_plan(TcPlan& plan, const tp_config&, const std::vector<int32_t>&, const std::vector<int32_t>&,
                        const std::vector<uint8_t>&, const std::vector<std::array<int64_t, kMaxDepth + 1>>&,
                        const std::vector<std::array<int64_t, kMaxDepth>>&,
                        const std::vector<std::array<int64_t, kMaxDepth>>&, int, int, const __nv_bfloat16*,
                        const void*, const void*, const void*, std::string&) {
  plan.enabled = false;
  return TP_OK;
}
tp_status tc_run_fwd(TcPlan&, cudaStream_t, int, int, int, uint32_t, int, uint64_t, const float*, const MemberDev*,
                     std::string& err) {
  err = "tensor-core plan disabled";
  return TP_ESTATE;
}
tp_status tc_run_bwd(TcPlan&, cudaStream_t, int, int, int, float*, const MemberDev*, std::string& err) {
  err = "tensor-core plan disabled";
  return TP_ESTATE;
}
void tc_free_plan(TcPlan& plan) { plan.enabled = false; }

}  // namespace tp
