// tp_internal.cuh -- shared internals of the tabpack CUDA library (sm_103a).
//
// Device data layout (one pack):
//   params / grads / adam_m / adam_v : fp32 arenas of n_params elements.  Member i
//       owns one contiguous run: for l = 0..L_i (L_i = head) the weight block
//       [out, in_pad] row-major then the bias [out]; every block starts on a
//       32-element boundary.  Layer 0 has in_pad = round_up(d_in, 8) columns
//       (the pad columns stay exactly zero); other layers in_pad = in.
//   wq[2]  : bf16 copies of the whole param arena (same offsets).  A step reads
//       wq[cur] in its matrix products and its fused AdamW writes wq[cur ^ 1],
//       so the step's dgrad can still read the weights its wgrad is updating.
//   xb     : the gathered batch [B_cap, ldx] (T), ldx = d_in_pad + 16.
//   act    : H_{l+1} = output of hidden layer l of member i, [B_cap, ldh_i] (T),
//            ldh_i = w_i + 16.
//   dz     : dL/dZ_l of hidden layer l of member i, [B_cap, w_i] (T).
// Column in_pad of xb and column w of every act matrix hold 1 (the next 15
// columns 0): the weight-gradient product dZ^T [H | 1] then yields the bias
// gradient dZ^T 1 as its extra output column (except where the tensor-core
// products take it from column sums of dZ, bias_from_colsums below).
// T = __nv_bfloat16 in bf16 mode, float in fp32 mode.  Batches are padded to
// B_pad = round_up(B, 128) rows; padded rows carry zero loss gradient, so they
// add nothing to weight or bias gradients.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace tp {

constexpr int kMaxDepth = 14;   // hidden blocks per member (4-bit layer field of the Philox counter)
constexpr int kMaxDout = 32;
constexpr int kRowTile = 128;   // batch rows per tile; B_pad is a multiple of this
constexpr int kHeadRows = 64;   // batch rows per head-kernel block
constexpr int kSegAlign = 32;   // elements
constexpr int kOnesCols = 16;   // the ones column plus zero padding to 16 columns

enum GemmKind : int32_t { kFwd = 0, kDgrad = 1, kWgrad = 2, kNsGram = 3, kNsPoly = 4, kNsApply = 5 };
enum Src : int32_t { kSrcXb = 0, kSrcAct = 1, kSrcDz = 2, kSrcWq = 3, kSrcNs = 4, kSrcEmb = 5 };

// Muon (Sec. 3.4; Jordan et al. 2024) on the hidden-layer weight matrices:
// the products of one Newton-Schulz iteration over the normalised momentum
// X [r, c] (r <= c; the transposed gradient when W has more rows than
// columns), all members and layers at once:
//   kNsGram  A  = X X^T            (A, B operands: X, K-major)
//   kNsPoly  Bm = b A + c A A      (A, B operands: A, K-major; A symmetric)
//   kNsApply X' = a X + Bm X       (A: Bm K-major, B: X MN-major)
// Coefficients (a, b, c) = (3.4445, -4.7750, 2.0315).
constexpr float kNsA = 3.4445f, kNsB = -4.7750f, kNsC = 2.0315f;

struct MuonMat {          // one Muon matrix: W_l of a member, [rows, cols] in the arena
  int64_t w_off;          // weight block offset in the parameter arena (pitch cols)
  int64_t x_off[2];       // X ping-pong buffers [r, c] in the Newton-Schulz arena
  int64_t a_off, bm_off;  // A and Bm [r, r]
  int32_t member, layer;
  int32_t rows, cols;     // w and in_pad
  int32_t r, c, tr;       // tr = 1: X = U^T (rows > cols)
  float scale, lr;        // max(1, rows / real columns)^(1/2); the member's Muon lr
  int32_t chunk0, n_chunks;  // its element chunks (of kMuonChunk) in the flat list
};
constexpr int kMuonChunk = 4096;

// One matrix product of one member and layer (CUDA-core path).
// Output C[r, c] = sum_k A(r, k) B(c, k).
//   kFwd   : A = H_l [B, in] (act or xb), B = W_l [w, in];  C = H_{l+1} [B, w]
//   kDgrad : A = dZ_l [B, w], B(c, k) = W_l[k, c];          C = dZ_{l-1} [B, in]
//   kWgrad : A(r, k) = dZ_l[k, r], B(c, k) = [H_l | 1][k, c]; C = dW_l [w, in_pad],
//            column in_pad = db_l
struct GemmProblem {
  int32_t kind, member, layer, ld_aux;
  int32_t M, N, K;        // M == 0 / K == 0: the step's B_pad rows
  int32_t a_src, b_src;
  int32_t lda, ldb, ldc;  // row pitches in elements
  int64_t a_off, b_off, c_off;
  int64_t aux_off;        // kFwd: bias offset in params; kDgrad: offset of H_l (mask) in act;
                          // kWgrad: bias offset in grads
  int64_t _pad1;
};

struct GemmTile {
  int32_t prob, m0, n0, n_len;  // output tile origin; n_len = columns of this tile
};

struct MemberDev {
  int32_t L, w;
  float p, scale;         // dropout rate, 1 / (1 - p)
  float lr, wd;
  uint32_t drop_T;        // drop iff Philox word < drop_T
  int32_t _pad;
};

// Contiguous run of parameters of one layer (weights or bias) of one member.
struct Segment {
  int64_t off;            // element offset in the param arena
  int32_t member, layer;
  int32_t rows, cols, cols_pad;  // weights: [rows, cols_pad], cols real; bias: rows x 1
  int32_t is_bias, fan_in;
  int32_t w_elems;        // unpadded weight count of the layer (bias init index base)
};

struct Chunk {            // element-wise work unit (init, AdamW): never crosses a segment
  int64_t off;
  int32_t len, seg;
};

struct HeadJob {          // head forward / loss / backward of one member on one 64-row block
  int32_t member, blk;
  int32_t h_ld;           // pitch of H_L
  int32_t split;          // row sets of the gradient pass (head_split)
  int32_t colsum, _pad;   // 1: store the column sums of dZ (bf16 tensor-core mode, bias_from_colsums)
  int64_t h_off;          // H_L in act
  int64_t dz_off;         // dZ_{L-1} in dz (pitch w)
  int64_t w_off, b_off;   // head weight / bias offsets in params
  int64_t part_off;       // partial dW_h of this block: [d_out, w] then [d_out] db
};

struct HeadReduceJob {
  int32_t member, n_blk;
  int64_t part_off;       // first block's partial; blocks follow at part_stride[member]
  int64_t gw_off, gb_off; // head weight / bias offsets (params, grads, m, v share them)
  int32_t w, _pad;
};

struct OnesJob {          // column `col` of rows 0..rows-1 of a matrix with pitch `ld` := 1
  int64_t off;
  int32_t ld, col, rows;
  int32_t arena;          // 0: xb, 1: act, 2: the embedding matrices
};

// The per-call arguments of a training step, read from device memory by the
// kernels of a replayed CUDA graph (the graph itself stays unchanged).
struct StepDyn {
  const float* X;
  const int32_t* idx;
  const void* y;
  float* loss_out;
  uint32_t step;
  uint32_t _pad;
};

// What a fused AdamW update needs besides the element itself.
struct AdamDev {
  float* params;
  float* m;
  float* v;
  __nv_bfloat16* wq_out;  // bf16 copy to write (NULL: none)
  const float2* bias_corr;  // per member (1 - beta1^t, 1 - beta2^t) of the step
  const MemberDev* mem;
  float beta1, beta2, eps;
  int32_t wd_on_bias;
};

// AdamW on one element (PyTorch semantics): decoupled decay, moments, bias-
// corrected step.  ib1 = 1 / (1 - beta1^t), ib2 = 1 / (1 - beta2^t).
__device__ __forceinline__ void adamw_elem(float& p, float& m, float& v, float g, float lr, float wd, float b1,
                                           float b2, float eps, float ib1, float ib2) {
  p = p - lr * wd * p;
  m = b1 * m + (1.f - b1) * g;
  v = b2 * v + (1.f - b2) * g * g;
  p = p - lr * (m * ib1) / (sqrtf(v * ib2) + eps);
}

// ---------------------------------------------------------------- Philox4x32-10
// Salmon, Moraes, Dror, Shaw (SC'11): ten rounds of
//   (c0, c1, c2, c3) -> (hi(Mb c2) ^ c1 ^ k0, lo(Mb c2), hi(Ma c0) ^ c3 ^ k1, lo(Ma c0)),
// keys bumped by the Weyl increments between rounds.
struct U4 { uint32_t x, y, z, w; };

__device__ __forceinline__ U4 philox10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                       uint32_t k0, uint32_t k1) {
  const uint32_t Ma = 0xD2511F53u, Mb = 0xCD9E8D57u;
  const uint32_t Wa = 0x9E3779B9u, Wb = 0xBB67AE85u;
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    uint32_t lo_a = Ma * c0, hi_a = __umulhi(Ma, c0);
    uint32_t lo_b = Mb * c2, hi_b = __umulhi(Mb, c2);
    uint32_t n0 = hi_b ^ c1 ^ k0, n2 = hi_a ^ c3 ^ k1;
    c0 = n0; c1 = lo_b; c2 = n2; c3 = lo_a;
    k0 += Wa; k1 += Wb;
  }
  return U4{c0, c1, c2, c3};
}

// Keep bits of columns (col4 * 4 .. col4 * 4 + 3) of row `row`: bit q = keep(col4 * 4 + q).
__device__ __forceinline__ uint32_t keep_bits4(uint64_t seed, uint32_t member, uint32_t layer,
                                               uint32_t step, uint32_t row, uint32_t col4,
                                               uint32_t T) {
  if (T == 0u) return 0xFu;
  U4 r = philox10(row, col4, step, (member << 4) | layer, (uint32_t)seed, (uint32_t)(seed >> 32));
  return (uint32_t)(r.x >= T) | ((uint32_t)(r.y >= T) << 1) | ((uint32_t)(r.z >= T) << 2) |
         ((uint32_t)(r.w >= T) << 3);
}

// Periodic feature embeddings of one member (App. "Feature Embeddings"):
// E[b, j d + k] = alpha_jk f_k + beta_jk with f_0 = x_bj and f_k =
// cos(w_j,k-1 x_bj + b_j,k-1); the parameters [w, b, alpha, beta] at p_off
// in the parameter (and gradient) arena.
struct EmbMember {
  int32_t d, in0, in0_pad, _pad;
  int64_t e_off;          // E in the embedding arena, pitch in0_pad + 16
  int64_t de_off;         // dE in the dz arena, pitch in0_pad
  int64_t p_off;
};

// Dropout keep bits of 32 consecutive columns of one row, word bit j =
// keep(32 * chunk + j): the eight Philox draws of the chunk, one after the
// other (few registers: the kernels that fill the mask arena stream memory
// beside it).
__device__ __forceinline__ uint32_t keep_word(uint64_t seed, uint32_t member, uint32_t layer, uint32_t step,
                                              uint32_t row, uint32_t chunk, uint32_t T) {
  uint32_t keep = 0;
#pragma unroll 1
  for (int g4 = 0; g4 < 8; ++g4) keep |= keep_bits4(seed, member, layer, step, row, 8 * chunk + g4, T) << (4 * g4);
  return keep;
}

// Precomputed dropout masks (bf16 mode).  Each (member, layer) with p > 0
// owns [ceil(w / 32), B_cap] keep words of one step in the mask arena; the
// forward epilogue reads its row's word of each 32-column chunk instead of
// evaluating Philox.  The chunks of all such (member, layer) pairs are
// numbered in one flat list for the kernels that fill the arena.
struct MaskSeg {
  int64_t off;            // word offset in the mask arena
  int32_t member, layer;
  uint32_t drop_T;
  int32_t chunk0;         // its first chunk in the flat list
};

struct MaskGen {          // what a kernel needs to fill the mask arena for one step
  uint32_t* masks;
  const MaskSeg* segs;
  const int32_t* chunk_seg;  // flat chunk -> segment
  int32_t n_chunks;          // 0: nothing to fill
  int32_t rows;              // B_cap
  uint64_t seed;
  uint32_t step;             // the step (dyn == NULL)
  uint32_t step_add;         // dyn != NULL: the step is dyn->step + step_add
  const StepDyn* dyn;
};

// Fill the mask arena (threads tid of nthreads; consecutive threads take
// consecutive rows of a chunk, so the stores coalesce).
__device__ __forceinline__ void fill_masks(const MaskGen& mg, int64_t tid, int64_t nthreads) {
  if (mg.n_chunks == 0) return;
  const uint32_t step = mg.dyn ? mg.dyn->step + mg.step_add : mg.step;
  const int64_t total = (int64_t)mg.n_chunks * mg.rows;
  for (int64_t e = tid; e < total; e += nthreads) {
    const int gc = (int)(e / mg.rows), row = (int)(e - (int64_t)gc * mg.rows);
    const MaskSeg s = mg.segs[mg.chunk_seg[gc]];
    const int chunk = gc - s.chunk0;
    mg.masks[s.off + (int64_t)chunk * mg.rows + row] =
        keep_word(mg.seed, (uint32_t)s.member, (uint32_t)s.layer, step, (uint32_t)row, (uint32_t)chunk, s.drop_T);
  }
}

// ---------------------------------------------------------------- element types
template <typename T> struct Elem;
template <> struct Elem<float> {
  static __device__ __forceinline__ float to_f(float v) { return v; }
  static __device__ __forceinline__ float from_f(float v) { return v; }
};
template <> struct Elem<__nv_bfloat16> {
  static __device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }
  static __device__ __forceinline__ __nv_bfloat16 from_f(float v) { return __float2bfloat16_rn(v); }
};

// ---------------------------------------------------- dependent launches
// Every kernel of the step is launched with programmatic stream
// serialisation: it lets the next kernel of the stream begin launching at
// once (pdl_trigger) -- whose CTAs then do their set-up on SMs this kernel has
// left -- and waits for the previous kernel to complete and its writes to be
// visible (pdl_wait) before it touches any data.  Without the launch
// attribute both instructions are no-ops.
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline void launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);  // errors surface via cudaGetLastError
}

__host__ __device__ constexpr int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

// Head kernels: class-count bucket (the loops over classes are unrolled to
// it) and columns per thread of the gradient pass for a bucket.
__host__ __device__ constexpr int head_bucket(int d_out) {
  return d_out <= 1 ? 1 : d_out <= 2 ? 2 : d_out <= 4 ? 4 : d_out <= 8 ? 8 : d_out <= 10 ? 10 : d_out <= 16 ? 16 : kMaxDout;
}
__host__ __device__ constexpr int head_cols(int DO) { return DO <= 2 ? 8 : DO <= 10 ? 4 : DO <= 16 ? 2 : 1; }
// Row sets of a head block's gradient pass: the block's 256 threads take
// w / head_cols column groups; narrow heads split the block's rows into up
// to 8 sets so that more threads work.
__host__ __device__ constexpr int head_split(int w, int d_out) {
  const int n_cg = w / head_cols(head_bucket(d_out));
  int S = 1;
  while (S < 8 && n_cg * S * 2 <= 256) S *= 2;
  return S;
}
__host__ __device__ constexpr int64_t ceil_div(int64_t x, int64_t a) { return (x + a - 1) / a; }

// Tensor-core weight-gradient products of a layer whose input width is a
// multiple of 256 (the widest column tile) take the bias gradient from
// column sums of dZ that its producer (head kernel or dgrad epilogue)
// stores beside it: a bias column of ones in the B operand would cost a
// whole extra column tile there.  Other widths keep the ones column, which
// fits in the last tile's spare columns.  Both sum dZ as stored (bf16).
__host__ __device__ constexpr bool bias_from_colsums(int in_pad) { return in_pad % 256 == 0; }

// The element chunks of a Muon matrix: kMuonChunk consecutive elements of W,
// or for a transposed one (tr) a kMuonTileR x kMuonTileC tile of W, so that
// the element kernels can move its X rows (W's columns) as whole segments.
constexpr int kMuonTileR = 32, kMuonTileC = 128;
static_assert(kMuonTileR * kMuonTileC == kMuonChunk, "a tile is one chunk");
__host__ __device__ constexpr int64_t muon_chunks(const MuonMat& mt) {
  return mt.tr ? ceil_div(mt.rows, kMuonTileR) * ceil_div(mt.cols, kMuonTileC)
               : ceil_div((int64_t)mt.rows * mt.cols, kMuonChunk);
}

}  // namespace tp
