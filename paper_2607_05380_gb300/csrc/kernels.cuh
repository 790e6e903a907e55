// kernels.cuh -- kernel argument blocks and launchers of the tabpack library.
#pragma once

#include <algorithm>

#include "tp_internal.cuh"

namespace tp {

template <typename T>
struct GemmArgs {
  const GemmProblem* probs;
  const GemmTile* tiles;
  const T* xb;
  T* act;
  T* dz;
  const T* wq;            // matrix-product copy of the weights (the fp32 params in fp32 mode)
  const float* params;    // fp32 master (biases)
  float* grads;
  const MemberDev* mem;
  int32_t B, B_pad;
  uint32_t step;
  int32_t train;          // 1: dropout on
  uint64_t seed;
  const StepDyn* dyn;     // non-NULL: take the step from here
  int64_t xb_stride;      // stacked batches: elements between members' batch matrices (0: shared)
  T* ns;                  // Muon's Newton-Schulz arena (kNs* problems)
  const T* ex;            // the embedding matrices (kSrcEmb)
};

// Muon steps around the Newton-Schulz products (see MuonMat).
template <typename T>
struct MuonArgs {
  const MuonMat* mats;
  const int32_t* chunk_mat;  // flat chunk -> matrix
  const float* grads;
  float* mom;                // momentum buffers (the AdamW first-moment arena)
  float* params;
  T* ns;
  double* part;              // per flat chunk: sum of squares of U
  __nv_bfloat16* wq_out;     // bf16 copy to refresh (NULL in fp32 mode)
  const MemberDev* mem;
  float mu;
  int32_t x_final;           // the X buffer that holds the result
  int* ns_cnt;               // the Newton-Schulz launch's counters, cleared by the momentum kernel
  int32_t n_ns_cnt;
  // x0_fused = 1 (the tensor-core iteration): the momentum kernel also writes
  // U, unnormalised, as X0 and, from the last chunk of each matrix to finish,
  // ns_scale[matrix] = 1 / max(|U|_F, 1e-7); mat_done counts the chunks done
  // (back to 0 after each step).  k_muon_x0 is then not launched.
  int32_t x0_fused;
  float* ns_scale;
  int* mat_done;
};

template <typename T>
struct HeadArgs {
  const HeadJob* jobs;
  const MemberDev* mem;
  const T* act;
  T* dz;
  const float* params;
  float* head_part;
  float* loss_part;
  float* logits;          // [m, B_cap, d_out]
  const int32_t* idx;
  const void* y;
  int32_t B, B_pad, B_cap, d_out, task, n_blk_cap;
  const StepDyn* dyn;     // non-NULL: take idx and y from here
  int32_t idx_stride;     // member i's rows are idx[i * idx_stride ..] (0: one shared batch)
  int32_t w_max;          // widest member (bf16: shared-memory size of the staged head kernel)
  int32_t stage;          // bf16: 1 = the staged head kernel where it fits in shared memory
  int* err;               // device error word for a bounded wait that runs out (NULL: none)
  float* dbp;             // bf16 tensor-core mode: the column sums of dZ_L as stored (bf16) over
                          // each 64-row block (element dz_off / 32 + blk * w + j) of the jobs
                          // with colsum set, from which the weight-gradient tiles take db
};

// Staged head kernel (bf16): shared memory per block for members up to w_max
// wide and DO classes, and the most a block may take.
constexpr int kHeadStageSmemMax = 232448;
__host__ __device__ constexpr int head_stage_pitch(int w) { return (int)round_up((int64_t)w * 2, 128) + 16; }
__host__ __device__ constexpr int head_stage_split(int w, int DO) {
  int S = 1;
  while (S < 8 && (w / 4) * S * 2 <= 256 && S * 2 * DO <= 32) S *= 2;
  return S;
}
__host__ __device__ constexpr int64_t head_stage_smem(int w_max, int DO) {
  return (int64_t)kHeadRows * head_stage_pitch(w_max) +
         4 * ((int64_t)DO * w_max + (int64_t)8 * kHeadRows * DO + (int64_t)kHeadRows * (DO == 1 ? 1 : (DO + 3) & ~3) +
              kHeadRows) + 16;
}
void head_stage_prepare();

struct HeadReduceArgs {
  const HeadReduceJob* jobs;
  const uint8_t* active;
  const int64_t* part_stride;
  const float* head_part;
  const float* loss_part;
  float* grads;           // store mode: head gradients land here
  float* loss_out;        // caller's [m] or NULL
  float* loss_last;       // pack's own copy [m]
  int32_t B, B_pad, d_out, n_blk_cap;
  int32_t update;         // 1: apply AdamW to the head parameters instead of storing the gradients
  AdamDev adam;
  const StepDyn* dyn;     // non-NULL: take loss_out from here
};

struct AdamArgs {
  const Chunk* chunks;
  const Segment* segs;
  const MemberDev* mem;
  const float2* bias_corr;
  float* params;
  const float* grads;
  float* m;
  float* v;
  __nv_bfloat16* wq;      // NULL in fp32 mode
  float beta1, beta2, eps;
  int32_t wd_on_bias;
  MaskGen mg;             // the next step's dropout masks, filled by the same threads
};

struct InitArgs {
  const Chunk* chunks;
  const Segment* segs;
  float* params;
  float* grads;
  float* m;
  float* v;
  __nv_bfloat16* wq0;
  __nv_bfloat16* wq1;
  uint64_t seed;
};

template <typename T>
struct PredictHeadArgs {
  const HeadJob* jobs;
  const MemberDev* mem;
  const T* act;
  const float* params;
  float* out;
  int64_t N, n0;
  int32_t rows, d_out, task, _pad;
};

// dyn non-NULL: X and idx are taken from it
template <typename T>
void launch_gather(cudaStream_t st, const float* X, const int32_t* idx, const StepDyn* dyn, int B, int B_pad,
                   int d_in, int d_in_pad, int ldx, T* xb, int advance, int32_t* t_dev, float2* bias_corr,
                   const int32_t* active_ids, int n_active, float beta1, float beta2, int* zero = nullptr,
                   int n_zero = 0, int stacked = 0, int64_t xb_stride = 0);
template <typename T>
void launch_gemm_simt(cudaStream_t st, const GemmArgs<T>& g, int tile_base, int n_tiles);
template <typename T>
void launch_head(cudaStream_t st, const HeadArgs<T>& g, int n_jobs);
// grid: m members x ceil(max_elems / 256) chunks (max_elems = max_i d_out (w_i + 1))
void launch_head_reduce(cudaStream_t st, const HeadReduceArgs& g, int m, int max_elems);
void launch_adamw(cudaStream_t st, const AdamArgs& g, int n_chunks);
void launch_init(cudaStream_t st, const InitArgs& g, int n_chunks);
void launch_masks(cudaStream_t st, const MaskGen& mg);

// Periodic embeddings: E of every active member from the rows idx (NULL:
// rows 0..) of X (member i's rows at idx + i * idx_stride), rows >= B zero;
// and the gradients of their parameters from dE.
template <typename T>
struct EmbArgs {
  const EmbMember* em;
  const int32_t* active_ids;
  const float* X;
  const int32_t* idx;
  const StepDyn* dyn;       // non-NULL: X and idx from here
  const float* params;
  float* grads;
  T* ex;                    // embedding arena (forward: written)
  const T* dz;              // dz arena (backward: dE read)
  int32_t idx_stride, B, B_pad, d_in;
};
// cols_max: the largest in0_pad of the members
template <typename T>
void launch_emb_fwd(cudaStream_t st, const EmbArgs<T>& a, int n_active, int cols_max);
template <typename T>
void launch_emb_bwd(cudaStream_t st, const EmbArgs<T>& a, int n_active, int cols_max);
template <typename T>
void launch_muon(cudaStream_t st, const MuonArgs<T>& a, int n_chunks, int phase);  // 0 momentum, 1 X0, 2 apply
void launch_refresh_wq(cudaStream_t st, const float* p, __nv_bfloat16* wq0, __nv_bfloat16* wq1, int64_t n);
template <typename T>
void launch_fill_ones(cudaStream_t st, const OnesJob* jobs, int n_jobs, T* xb, T* act, T* ex);
template <typename T>
void launch_predict_head(cudaStream_t st, const PredictHeadArgs<T>& g, int n_jobs);
void launch_debug_masks(cudaStream_t st, uint8_t* out, int B, int w, uint64_t seed, uint32_t member,
                        uint32_t layer, uint32_t step, uint32_t T);
void launch_debug_philox(cudaStream_t st, const uint32_t* in, uint32_t* out, int n);

// Sets the per-thread message pack_last_error(NULL) returns (tabpack.cu).
void record_thread_error(const char* msg);

// greedy selection (select.cu)
struct SelectScratch {
  double* S;              // running ensemble sum [N, d_out]
  double* partial;        // [P, n_blk]
  int32_t* state;         // [4 + m_ens + P]: n, done, last, pad | selected | used
  double* cur;            // [1]: current score
  uint32_t* keys;         // ROC-AUC score: sort keys, two buffers of N per candidate
  uint8_t* lab;           // and their labels
};
// score: scratch for the ROC-AUC score's sorts only when score == TP_SCORE_AUC
int64_t select_scratch_bytes(int32_t P, int64_t N, int32_t d_out, int32_t m_ens, int32_t score);
SelectScratch select_carve(void* base, int32_t P, int64_t N, int32_t d_out, int32_t m_ens, int32_t score);
// excl: device uint8 [P] or NULL; candidates with excl[c] != 0 take no part.
// solo: device double [P] or NULL; receives every candidate's score on its
// own (the first iteration's values; NaN for excluded candidates).
int select_enqueue(cudaStream_t st, const SelectScratch& s, const float* preds, int32_t P, int64_t N,
                   int32_t d_out, const void* y, int32_t task, int32_t score, int32_t m_ens,
                   const uint8_t* excl, double* solo, int64_t* launches);

}  // namespace tp
