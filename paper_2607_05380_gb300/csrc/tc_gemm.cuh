// tc_gemm.cuh -- grouped ragged bf16 GEMMs on the 5th-generation tensor cores
// (tcgen05.mma with accumulators in TMEM, operands staged by TMA) used by the
// bf16 mode for the forward, dgrad and wgrad products of every member.
#pragma once

#include <cuda.h>

#include <array>
#include <string>
#include <vector>

#include "tabpack.h"
#include "tp_internal.cuh"

namespace tp {

// One 128 x n_len output tile of one member's product.
//   kFwd   C[b, j]  = sum_k H[b, k] W[j, k]       A = H (K-major), B = W (K-major)
//   kDgrad C[b, k]  = sum_j dZ[b, j] W[j, k]      A = dZ (K-major), B = W (MN-major)
//   kWgrad C[j, k]  = sum_b dZ[b, j] H[b, k]      A = dZ (MN-major), B = H (MN-major)
struct TcTile {
  int32_t kind, member, layer;
  int32_t m0, n0, n_len;   // tile origin; n_len = MMA N (multiple of 16, <= 256)
  int32_t m_real, n_real;  // output bounds (m_real 0: the step's padded batch)
  int32_t k_len;           // reduction length (0: the step's padded batch)
  int32_t map_a, map_b;    // indices into the tensor-map table
  int32_t ldc;
  int64_t c_off;           // output offset: act (kFwd), dz (kDgrad), grads (kWgrad)
  int64_t aux_off;         // kFwd: bias offset in params; kDgrad: H_l offset in act (mask)
};

struct TcPlan {
  bool enabled = false;
  int n_sm = 0;
  CUtensorMap* maps_dev = nullptr;
  int n_maps = 0;
  TcTile* tiles_dev = nullptr;
  int cap_tiles = 0;
  std::vector<std::pair<int, int>> fwd_rng, bwd_rng;  // tile ranges per depth index
  int* err_dev = nullptr;  // device error word (bounded waits that gave up)
  // inputs used at build time
  std::vector<int> map_act, map_dz, map_w;  // per (member * kMaxDepth + layer)
};

tp_status tc_build_plan(TcPlan& plan, const tp_config& cfg, const std::vector<int32_t>& depth,
                        const std::vector<int32_t>& width, const std::vector<uint8_t>& active,
                        const std::vector<std::array<int64_t, kMaxDepth + 1>>& W_off,
                        const std::vector<std::array<int64_t, kMaxDepth + 1>>& b_off,
                        const std::vector<std::array<int64_t, kMaxDepth>>& act_off,
                        const std::vector<std::array<int64_t, kMaxDepth>>& dz_off, int d_in_pad, int B_cap,
                        const __nv_bfloat16* wq, const void* xb, const void* act, const void* dz,
                        std::string& err);
tp_status tc_run_fwd(TcPlan& plan, cudaStream_t st, int layer, int B, int B_pad, uint32_t step, int train,
                     uint64_t seed, const float* params, const MemberDev* mem, void* act, std::string& err);
tp_status tc_run_bwd(TcPlan& plan, cudaStream_t st, int layer, int B, int B_pad, float* grads,
                     const MemberDev* mem, void* act, void* dz, std::string& err);
// Reads and clears the device error word (synchronises the stream).
tp_status tc_check(TcPlan& plan, cudaStream_t st, std::string& err);
void tc_free_plan(TcPlan& plan);

}  // namespace tp
