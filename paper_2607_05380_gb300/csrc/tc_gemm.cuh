// tc_gemm.cuh -- grouped ragged bf16 GEMMs on the 5th-generation tensor cores
// (tcgen05 + TMEM, operands staged by TMA) for the bf16 mode.
#pragma once

#include <array>
#include <string>
#include <vector>

#include "tabpack.h"
#include "tp_internal.cuh"

namespace tp {

struct TcPlan {
  bool enabled = false;
};

tp_status tc_build_plan(TcPlan& plan, const tp_config& cfg, const std::vector<int32_t>& depth,
                        const std::vector<int32_t>& width, const std::vector<uint8_t>& active,
                        const std::vector<std::array<int64_t, kMaxDepth + 1>>& W_off,
                        const std::vector<std::array<int64_t, kMaxDepth>>& act_off,
                        const std::vector<std::array<int64_t, kMaxDepth>>& dz_off, int d_in_pad, int B_cap,
                        const __nv_bfloat16* wq, const void* xb, const void* act, const void* dz,
                        std::string& err);
tp_status tc_run_fwd(TcPlan& plan, cudaStream_t st, int layer, int B, int B_pad, uint32_t step, int train,
                     uint64_t seed, const float* params, const MemberDev* mem, std::string& err);
tp_status tc_run_bwd(TcPlan& plan, cudaStream_t st, int layer, int B, int B_pad, float* grads,
                     const MemberDev* mem, std::string& err);
void tc_free_plan(TcPlan& plan);

}  // namespace tp
