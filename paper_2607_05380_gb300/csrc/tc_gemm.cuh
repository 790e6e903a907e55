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

// One output tile of one member's product: 128 * (CTAs per tile) rows from
// m0 (a CTA pair holds row blocks m0 and m0 + 128) by n_len columns from n0.
//   kFwd   C[b, j]  = sum_k H[b, k] W[j, k]         A = H (K-major), B = W (K-major)
//   kDgrad C[b, k]  = sum_j dZ[b, j] W[j, k]        A = dZ (K-major), B = W (MN-major)
//   kWgrad C[j, k]  = sum_b dZ[b, j] [H | 1][b, k]  A = dZ (MN-major), B = [H | 1] (MN-major);
//          columns k < in_pad are dW, column in_pad is db -- or, where the
//          input width is a multiple of 256 (bias_from_colsums), B = H and
//          the tiles with n0 = 0 write db_j = sum_b dZ[b, j] from the column
//          sums that the producer of dZ (head kernel or dgrad epilogue)
//          stored beside it, added in batch order
struct TcTile {
  int32_t kind, member, layer;
  int32_t m0, n0, n_len;   // tile origin; n_len = MMA N (multiple of 16, <= 256)
  int32_t m_real, n_real;  // output bounds (m_real 0: the step's padded batch);
                           // kWgrad: n_real = in_pad + 1 (the bias column)
  int32_t k_len;           // reduction length (0: the step's padded batch)
  int32_t map_a, map_b;    // indices into the tensor-map table (weight maps of copy 0)
  int32_t ldc, ld_aux;
  // Dataflow within one launch: before loading A the producer of row block
  // mi of the tile waits until counters d .. d + n - 1 each reach dep_need
  // (dep_n = 1: d = dep + mi, n = 1; dep_n = 0: d = dep, n = the step's
  // B_pad / 128); after storing its output every epilogue warp adds 1 to
  // counter sig + mi.  -1: none.  Newton-Schulz tiles: counters dep and
  // sig themselves, shared by the CTAs of a pair (one per matrix and product).
  int32_t dep, dep_n, dep_need, sig;
  int32_t mask_off;        // kFwd of a member with dropout: word offset of its keep words in the
                           // mask arena ([ceil(n_real / 32), mask rows]); -1: none
  int32_t ns_scale;        // kNsGram / kNsApply of the first iteration: 1 + the Muon matrix whose
                           // 1 / |U|_F scales the product (X0 holds U unnormalised); 0: none
  int32_t db_rows;         // kWgrad: batch rows per column-sum partial of dZ (64: written by the
                           // head kernel, 32: by dgrad epilogues); kDgrad: 32 = store the column
                           // sums of the output, 0 = do not
  int64_t c_off;           // output: act (kFwd), dz (kDgrad), weight offset in the arena (kWgrad)
  int64_t aux_off;         // kFwd: bias offset in params; kDgrad: H_l offset in act (mask);
                           // kWgrad: bias offset in the arena
  int64_t db_off;          // kWgrad: the column-sum partials of its dZ in the partial arena
                           // ([B_pad / db_rows][w], partial after partial); -1: db from the
                           // bias column
};

struct TcPlan {
  bool enabled = false;
  int n_sm = 0;
  CUtensorMap* maps_dev = nullptr;
  int n_maps = 0;
  int w_shift = 0;         // index distance from a weight map of copy 0 to copy 1
  int kmaj_off = 0;        // index distance from a map to its 128-row-box twin
  TcTile* tiles_dev = nullptr;
  int cap_tiles = 0;
  std::pair<int, int> fwd_rng, bwd_rng;  // tile ranges of the forward / backward launch
  // The Newton-Schulz launch: every iteration's kNsGram, kNsPoly and
  // kNsApply tiles, with their own completion counters (3 per Muon matrix),
  // which must be zero before the launch (the Muon momentum kernel that
  // precedes it clears them)
  std::pair<int, int> ns_rng = {};
  int* ns_cnt_dev = nullptr;
  int n_ns_cnt = 0;
  bool ns_maps = false;    // the map table holds the Muon matrices' maps
  // Row-block completion counters: act of (member, layer) then dz of
  // (member, layer), B_cap / 128 each.  They must be zero before a launch
  // (the gather kernel that precedes every forward clears them).
  int* cnt_dev = nullptr;
  int n_cnt = 0;
  int cta = 1;             // CTAs per tile (2: CTA pairs with cta_group::2 MMAs)
  int max_clusters = 0;    // tiles in flight at once (resident CTAs / cta)
  int* err_dev = nullptr;  // device error word (bounded waits that gave up)
  uint64_t wait_ns = 2000000000ull;  // budget of every wait that can give up
  std::vector<int> map_act, map_dz, map_w;  // per (member * kMaxDepth + layer)
  std::vector<int> map_ns;                  // per Muon matrix: X0, X1, A, Bm
};

struct TcLayout {          // what the plan needs to know about the pack's arenas
  const std::vector<int32_t>* depth;
  const std::vector<int32_t>* width;
  const std::vector<uint8_t>* active;
  const std::vector<std::array<int64_t, kMaxDepth + 1>>* W_off;
  const std::vector<std::array<int64_t, kMaxDepth + 1>>* b_off;
  const std::vector<std::array<int64_t, kMaxDepth>>* act_off;
  const std::vector<std::array<int64_t, kMaxDepth>>* dz_off;
  int m, d_in_pad, ldx, B_cap;
  const __nv_bfloat16* wq[2];
  const void* xb;
  const void* act;
  const void* dz;
  bool fwd_only = false;   // forward tiles only (prediction): no dz maps, counters or backward tiles
  bool bias_colsums = false;  // bias gradients from dZ column sums where bias_from_colsums (else the
                              // bias column everywhere)
  // Muon: the matrices whose Newton-Schulz products get tiles (NULL: none)
  // and the bf16 arena holding their X, A and Bm buffers
  const std::vector<MuonMat>* muon = nullptr;
  const void* ns = nullptr;
  int ns_steps = 0;        // Newton-Schulz iterations per Muon step
  int64_t xb_stride = 0;   // > 0: a batch matrix per member (stacked batches), this many elements apart
  // Periodic embeddings: member i's first layer reads the matrix at xb +
  // x0_off[i] ([B_cap, in0_pad[i] + 16]) and, with de_off, its input gradient
  // dE_i [B_cap, in0_pad[i]] is written to dz + de_off[i] (NULL: none)
  const std::vector<int32_t>* in0_pad = nullptr;
  const std::vector<int64_t>* x0_off = nullptr;
  const std::vector<int64_t>* de_off = nullptr;
  // per (member, layer): word offset of the dropout keep words, -1 for none (NULL: no masks)
  const std::vector<std::array<int64_t, kMaxDepth>>* mask_off = nullptr;
};

tp_status tc_build_plan(TcPlan& plan, const TcLayout& lay, std::string& err);
// Forward products of every hidden layer of every active member (one
// launch), reading weight copy `wcur`.  train = 1: dropout with the keep
// words of the step in `masks` (rows = mask_rows per 32-column chunk).
tp_status tc_run_fwd(TcPlan& plan, cudaStream_t st, int B, int B_pad, int wcur, int train, const uint32_t* masks,
                     int mask_rows, const float* params, const MemberDev* mem, void* act, std::string& err);
// Backward products (dgrad + wgrad) of every hidden layer (one launch).
// update = 0: the weight and bias gradients are stored in `grads`;
// update = 1: AdamW is applied in the epilogue (adam.wq_out = the other
// weight copy).  dbp: the column-sum partials of dZ (float, element
// dz_off / 32 + g * w + j for partial g of a [B_cap, w] dZ at dz_off) of
// the layers whose bias gradient comes from them; the head kernel has
// written those of each member's last hidden layer, the dgrad epilogues
// write the others.
tp_status tc_run_bwd(TcPlan& plan, cudaStream_t st, int B, int B_pad, int wcur, const MemberDev* mem, void* act,
                     void* dz, float* grads, float* dbp, int update, const AdamDev& adam, std::string& err);
// Every Newton-Schulz iteration of every Muon matrix in one launch (U in
// buffer 0, scaled by ns_scale[matrix] = 1 / |U|_F inside the first
// iteration's products; the result in buffer ns_steps & 1).
tp_status tc_run_ns(TcPlan& plan, cudaStream_t st, void* ns, const float* ns_scale, const MemberDev* mem,
                    std::string& err);
// Reads and clears the device error word (synchronises the stream).
tp_status tc_check(TcPlan& plan, cudaStream_t st, std::string& err);
// Tests: the first forward tile with a dependency waits for a count the
// launch never reaches (then its CTA gives up after plan.wait_ns).
tp_status tc_debug_poison(TcPlan& plan, cudaStream_t st, std::string& err);
void tc_free_plan(TcPlan& plan);

}  // namespace tp
