// kernels.cu -- element-wise, reduction and CUDA-core matrix kernels of the
// packed training step (gather, CUDA-core grouped GEMM, head + loss + head
// AdamW, AdamW, init, predict head, mask dump).
#include <algorithm>
#include <cmath>
#include <type_traits>

#include "kernels.cuh"

namespace tp {

// ------------------------------------------------------------------ gather
// Four values at once: 8-byte bf16 / 16-byte fp32 stores.
__device__ __forceinline__ void store4(__nv_bfloat16* p, float4 v) {
  uint2 u;
  __nv_bfloat162* b = reinterpret_cast<__nv_bfloat162*>(&u);
  b[0] = __floats2bfloat162_rn(v.x, v.y);
  b[1] = __floats2bfloat162_rn(v.z, v.w);
  *reinterpret_cast<uint2*>(p) = u;
}
__device__ __forceinline__ void store4(float* p, float4 v) { *reinterpret_cast<float4*>(p) = v; }

// xb[b, k] = X[idx[b], k] for b < B, k < d_in; zero for the rest of the first
// d_in_pad columns of rows < B_pad (column d_in_pad holds the constant 1).
// Grid: ceil(B_pad / 8) blocks of 8 warps, a row per warp.
// Block 0 also advances the step count of every active member and stores the
// AdamW bias corrections 1 - beta^t of the new step (when `advance`); the
// grid clears `zero[0 .. n_zero)` (the GEMMs' row-block completion counters).
// stacked != 0 (a batch per member, Sec. 3.6): blockIdx.y is an active
// member's index, whose rows are idx[member * B ..] and whose batch matrix
// starts xb_stride elements after the previous member's.
template <typename T>
__global__ void k_gather(const float* __restrict__ X, const int32_t* __restrict__ idx, const StepDyn* dyn,
                         int32_t B, int32_t B_pad, int32_t d_in, int32_t d_in_pad, int32_t ldx, T* __restrict__ xb,
                         int32_t advance, int32_t* __restrict__ t_dev, float2* __restrict__ bias_corr,
                         const int32_t* __restrict__ active_ids, int32_t n_active, float ln_beta1,
                         float ln_beta2, int32_t* __restrict__ zero, int32_t n_zero, int32_t stacked,
                         int64_t xb_stride) {
  pdl_trigger();
  pdl_wait();
  if (dyn) {
    X = dyn->X;
    idx = dyn->idx;
  }
  if (stacked) {
    const int member = active_ids[blockIdx.y];
    if (idx) idx += (int64_t)member * B;
    xb += (int64_t)member * xb_stride;
  }
  if (blockIdx.y == 0)
    for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < n_zero; e += gridDim.x * blockDim.x) zero[e] = 0;
  if (advance && blockIdx.x == 0 && blockIdx.y == 0) {
    for (int a = threadIdx.x; a < n_active; a += blockDim.x) {
      int i = active_ids[a];
      int t = t_dev[i] + 1;
      t_dev[i] = t;
      // Adam's bias corrections 1 - beta^t = -expm1(t ln beta), in fp32 to
      // about 1e-7 relative (fp64 runs at a small fraction of the fp32 rate)
      bias_corr[i] = make_float2(-expm1f((float)t * ln_beta1), -expm1f((float)t * ln_beta2));
    }
  }
  // one warp per batch row: float4 reads of the source row when it is
  // 16-byte aligned, four converted values written at once
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * (blockDim.x >> 5) + warp;
  if (b >= B_pad) return;
  T* dst = xb + (int64_t)b * ldx;
  const bool live = b < B;
  const int64_t row = live ? (idx ? (int64_t)idx[b] : (int64_t)b) : 0;
  const float* src = X + row * d_in;
  int k0 = 0;
  if (live && (d_in & 3) == 0 && ((uintptr_t)src & 15) == 0) {
    const float4* s4 = reinterpret_cast<const float4*>(src);
    for (int c = lane; c < (d_in >> 2); c += 32) {
      store4(dst + 4 * c, __ldg(s4 + c));
    }
    k0 = d_in;
  }
  for (int k = k0 + lane; k < d_in_pad; k += 32) dst[k] = Elem<T>::from_f(live && k < d_in ? src[k] : 0.f);
}

// Column `col` of the first `rows` rows := 1 (xb and every act matrix, once).
template <typename T>
__global__ void k_fill_ones(const OnesJob* __restrict__ jobs, T* __restrict__ xb, T* __restrict__ act,
                            T* __restrict__ ex) {
  const OnesJob jb = jobs[blockIdx.x];
  T* base = (jb.arena == 0 ? xb : jb.arena == 1 ? act : ex) + jb.off;
  for (int r = threadIdx.x; r < jb.rows; r += blockDim.x) base[(int64_t)r * jb.ld + jb.col] = Elem<T>::from_f(1.f);
}

// ------------------------------------------------------- CUDA-core GEMM
// One 64 x 64 output tile per block, 256 threads, 4 x 4 outputs per thread,
// k-slabs of 16 staged in shared memory.  Each output accumulates its k terms
// in increasing k order with fused multiply-adds (fp32).
template <typename T>
__global__ void __launch_bounds__(256) k_gemm_simt(GemmArgs<T> g, int32_t tile_base) {
  pdl_trigger();
  pdl_wait();
  const GemmTile t = g.tiles[tile_base + blockIdx.x];
  const GemmProblem P = g.probs[t.prob];
  const int M = P.M ? P.M : g.B_pad;
  const int N = P.N;
  const int K = P.K ? P.K : g.B_pad;
  if (t.m0 >= M) return;
  const uint32_t step = g.dyn ? g.dyn->step : g.step;
  const T* bases[6] = {g.xb, g.act, g.dz, g.wq, g.ns, g.ex};
  // stacked batches: the member's own batch matrix
  const int64_t xs = (int64_t)P.member * g.xb_stride;
  const T* A = bases[P.a_src] + P.a_off + (P.a_src == kSrcXb ? xs : 0);
  const T* Bm = bases[P.b_src] + P.b_off + (P.b_src == kSrcXb ? xs : 0);
  int64_t a_rs, a_ks, b_rs, b_ks;
  if (P.kind == kFwd || P.kind == kNsGram || P.kind == kNsPoly) {
    a_rs = P.lda; a_ks = 1; b_rs = P.ldb; b_ks = 1;
  } else if (P.kind == kDgrad || P.kind == kNsApply) {
    a_rs = P.lda; a_ks = 1; b_rs = 1; b_ks = P.ldb;
  } else {
    a_rs = 1; a_ks = P.lda; b_rs = 1; b_ks = P.ldb;
  }
  __shared__ float As[16][68];
  __shared__ float Bs[16][68];
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  for (int k0 = 0; k0 < K; k0 += 16) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      int e = threadIdx.x + q * 256;
      int r, kk;
      if (a_ks == 1) { kk = e & 15; r = e >> 4; } else { r = e & 63; kk = e >> 6; }
      int gr = t.m0 + r, gk = k0 + kk;
      float v = 0.f;
      if (gr < M && gk < K) v = Elem<T>::to_f(A[gr * a_rs + gk * a_ks]);
      As[kk][r] = v;
      int c, kb;
      if (b_ks == 1) { kb = e & 15; c = e >> 4; } else { c = e & 63; kb = e >> 6; }
      int gc = t.n0 + c, gkb = k0 + kb;
      float u = 0.f;
      if (gc < N && gkb < K) u = Elem<T>::to_f(Bm[gc * b_rs + gkb * b_ks]);
      Bs[kb][c] = u;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  const int c0 = t.n0 + tx * 4;
  if (c0 >= N) return;
  const MemberDev md = g.mem[P.member];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = t.m0 + ty + 16 * i;
    if (r >= M) continue;
    if (P.kind >= kNsGram) {  // Newton-Schulz: alpha acc + beta aux (N a multiple of 8)
      const float al = P.kind == kNsPoly ? kNsC : 1.f;
      const float be = P.kind == kNsPoly ? kNsB : (P.kind == kNsApply ? kNsA : 0.f);
      T* C = g.ns + P.c_off;
      const T* Aux = g.ns + P.aux_off;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        float v = al * acc[i][j];
        if (P.kind != kNsGram) v += be * Elem<T>::to_f(Aux[(int64_t)r * P.ld_aux + c0 + j]);
        C[(int64_t)r * P.ldc + c0 + j] = Elem<T>::from_f(v);
      }
    } else if (P.kind == kFwd) {  // N = w, a multiple of 16
      uint32_t keep = g.train ? keep_bits4(g.seed, (uint32_t)P.member, (uint32_t)P.layer, step,
                                           (uint32_t)r, (uint32_t)(c0 >> 2), md.drop_T)
                              : 0xFu;
      const float sc = g.train ? md.scale : 1.f;
      T* C = g.act + P.c_off;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        float z = acc[i][j] + g.params[P.aux_off + c0 + j];
        float a = z > 0.f ? z : 0.f;
        float h = ((keep >> j) & 1u) ? a * sc : 0.f;
        C[(int64_t)r * P.ldc + c0 + j] = Elem<T>::from_f(h);
      }
    } else if (P.kind == kDgrad) {  // N = w (the first layer's input gradient: no mask, aux_off < 0)
      T* C = g.dz + P.c_off;
      if (P.aux_off < 0) {
#pragma unroll
        for (int j = 0; j < 4; ++j) C[(int64_t)r * P.ldc + c0 + j] = Elem<T>::from_f(acc[i][j]);
      } else {
        const T* Hm = g.act + P.aux_off;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          float h = Elem<T>::to_f(Hm[(int64_t)r * P.ld_aux + c0 + j]);
          C[(int64_t)r * P.ldc + c0 + j] = Elem<T>::from_f(h > 0.f ? acc[i][j] * md.scale : 0.f);
        }
      }
    } else {  // N = in_pad + 1: the last column is the bias gradient
      float* C = g.grads + P.c_off;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int c = c0 + j;
        if (c < N - 1) C[(int64_t)r * P.ldc + c] = acc[i][j];
        else if (c == N - 1) g.grads[P.aux_off + r] = acc[i][j];
      }
    }
  }
}

// ---------------------------------------------------------- vector helpers
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// 8 consecutive values as floats (16-byte bf16 / 2 x 16-byte fp32 loads).
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float (&h)[8]) {
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat16* b = reinterpret_cast<const __nv_bfloat16*>(&u);
#pragma unroll
  for (int k = 0; k < 8; ++k) h[k] = __bfloat162float(b[k]);
}
__device__ __forceinline__ void load8(const float* p, float (&h)[8]) {
  const float4 a = *reinterpret_cast<const float4*>(p), b = *reinterpret_cast<const float4*>(p + 4);
  h[0] = a.x; h[1] = a.y; h[2] = a.z; h[3] = a.w; h[4] = b.x; h[5] = b.y; h[6] = b.z; h[7] = b.w;
}
__device__ __forceinline__ void store8(__nv_bfloat16* p, const float (&v)[8]) {
  uint4 u;
  __nv_bfloat162* b = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
  for (int k = 0; k < 4; ++k) b[k] = __floats2bfloat162_rn(v[2 * k], v[2 * k + 1]);
  *reinterpret_cast<uint4*>(p) = u;
}
__device__ __forceinline__ void store8(float* p, const float (&v)[8]) {
  *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  *reinterpret_cast<float4*>(p + 4) = make_float4(v[4], v[5], v[6], v[7]);
}

// Per-row loss and d(mean loss)/d(logits) of one row (fp32).
template <int DO>
__device__ __forceinline__ float row_loss(int task, int d_out, const float (&z)[DO], const void* y, int64_t row,
                                          float invB, float (&dl)[DO]) {
  float loss;
  if (task == 1) {  // multiclass: softmax cross-entropy
    const int yv = ((const int32_t*)y)[row];
    float mx = z[0];
#pragma unroll
    for (int c = 1; c < DO; ++c) if (c < d_out) mx = fmaxf(mx, z[c]);
    float s = 0.f;
#pragma unroll
    for (int c = 0; c < DO; ++c) if (c < d_out) s += expf(z[c] - mx);
    const float lse = mx + logf(s);
    float zy = 0.f;
#pragma unroll
    for (int c = 0; c < DO; ++c) {
      if (c == yv) zy = z[c];
      dl[c] = c < d_out ? (expf(z[c] - lse) - (c == yv ? 1.f : 0.f)) * invB : 0.f;
    }
    loss = lse - zy;
  } else if (task == 0) {  // binary: logistic loss on one logit
    const float yv = (float)((const int32_t*)y)[row];
    const float x = z[0];
    loss = fmaxf(x, 0.f) - x * yv + log1pf(expf(-fabsf(x)));
#pragma unroll
    for (int c = 0; c < DO; ++c) dl[c] = 0.f;
    dl[0] = (1.f / (1.f + expf(-x)) - yv) * invB;
  } else {  // regression: squared error
    const float d = z[0] - ((const float*)y)[row];
    loss = d * d;
#pragma unroll
    for (int c = 0; c < DO; ++c) dl[c] = 0.f;
    dl[0] = 2.f * d * invB;
  }
  return loss;
}

// ------------------------------------------------------------- head + loss
// Values of G consecutive columns as floats, and back.
template <int G>
__device__ __forceinline__ void loadG(const __nv_bfloat16* p, float (&h)[G]) {
  if constexpr (G == 8) {
    load8(p, h);
  } else if constexpr (G == 4) {
    const uint2 u = *reinterpret_cast<const uint2*>(p);
    const __nv_bfloat16* b = reinterpret_cast<const __nv_bfloat16*>(&u);
#pragma unroll
    for (int k = 0; k < 4; ++k) h[k] = __bfloat162float(b[k]);
  } else if constexpr (G == 2) {
    const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(p));
    h[0] = f.x;
    h[1] = f.y;
  } else {
    h[0] = __bfloat162float(*p);
  }
}
template <int G>
__device__ __forceinline__ void loadG(const float* p, float (&h)[G]) {
  if constexpr (G == 8) {
    load8(p, h);
  } else if constexpr (G == 4) {
    const float4 a = *reinterpret_cast<const float4*>(p);
    h[0] = a.x; h[1] = a.y; h[2] = a.z; h[3] = a.w;
  } else if constexpr (G == 2) {
    const float2 a = *reinterpret_cast<const float2*>(p);
    h[0] = a.x; h[1] = a.y;
  } else {
    h[0] = *p;
  }
}
template <int G>
__device__ __forceinline__ void storeG(__nv_bfloat16* p, const float (&v)[G]) {
  if constexpr (G == 8) {
    store8(p, v);
  } else if constexpr (G == 4) {
    uint2 u;
    __nv_bfloat162* b = reinterpret_cast<__nv_bfloat162*>(&u);
    b[0] = __floats2bfloat162_rn(v[0], v[1]);
    b[1] = __floats2bfloat162_rn(v[2], v[3]);
    *reinterpret_cast<uint2*>(p) = u;
  } else if constexpr (G == 2) {
    *reinterpret_cast<__nv_bfloat162*>(p) = __floats2bfloat162_rn(v[0], v[1]);
  } else {
    *p = __float2bfloat16_rn(v[0]);
  }
}
template <int G>
__device__ __forceinline__ void storeG(float* p, const float (&v)[G]) {
  if constexpr (G == 8) {
    store8(p, v);
  } else if constexpr (G == 4) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  } else if constexpr (G == 2) {
    *reinterpret_cast<float2*>(p) = make_float2(v[0], v[1]);
  } else {
    *p = v[0];
  }
}

// G consecutive elements of T loaded with one vector load and converted to
// float when used, so that several rows' loads can be in flight at once.
template <typename T, int G>
struct RawG;
template <int G>
struct RawG<__nv_bfloat16, G> {
  using V = std::conditional_t<G == 8, uint4, std::conditional_t<G == 4, uint2,
                               std::conditional_t<G == 2, uint32_t, unsigned short>>>;
  V v;
  __device__ __forceinline__ void load(const __nv_bfloat16* p) { v = *reinterpret_cast<const V*>(p); }
  __device__ __forceinline__ void to_float(float (&h)[G]) const {
    const __nv_bfloat16* b = reinterpret_cast<const __nv_bfloat16*>(&v);
#pragma unroll
    for (int k = 0; k < G; ++k) h[k] = __bfloat162float(b[k]);
  }
};
template <int G>
struct RawG<float, G> {
  float v[G];
  __device__ __forceinline__ void load(const float* p) { loadG<G>(p, v); }
  __device__ __forceinline__ void to_float(float (&h)[G]) const {
#pragma unroll
    for (int k = 0; k < G; ++k) h[k] = v[k];
  }
};

// The logit pass of a head block (128 rows of one member, 8 warps of 16
// rows).  LPR lanes share a row (the smallest power of two >= the row's
// 8-column groups, at most 32; lanes walk the groups with 16-byte loads) and
// a warp's 32 / LPR lane groups take different rows, R rows per group at a
// time, so that every head-weight load serves R rows.  After the call the
// group's lane 0 holds the R rows' logits (bias added); `rl0` is the block-
// local index of the group's first row and `live` whether the group has
// rows in this pass.  Returns the number of passes.
template <typename T, int DO, int R>
struct HeadLogits {
  static constexpr int kRowsPerWarp = kHeadRows / 8;
  int lpr, groups, grp, gl;
  __device__ __forceinline__ HeadLogits(int w, int lane) {
    const int ng = w >> 3;
    lpr = 1;
    while (lpr < ng && lpr < 32) lpr <<= 1;
    groups = min(32 / lpr, kRowsPerWarp / R);
    grp = lane / lpr;
    gl = lane % lpr;
  }
  __device__ __forceinline__ int step() const { return groups * R; }
  // rows rl0 .. rl0 + R - 1 (block-local) of H (block origin), head weights Wh [d_out, w]
  __device__ __forceinline__ void run(const T* __restrict__ H, int ldh, const float* __restrict__ Wh,
                                      const float* __restrict__ bh, int w, int d_out,
                                      int rl0, bool live, float (&acc)[R][DO]) const {
#pragma unroll
    for (int q = 0; q < R; ++q)
#pragma unroll
      for (int c = 0; c < DO; ++c) acc[q][c] = 0.f;
    if (live) {
      // two-deep register pipeline over the column groups: the next group's
      // rows are in flight while this group's products run
      const int ng = w >> 3;
      RawG<T, 8> cur[R], nxt[R];
      if (gl < ng)
#pragma unroll
        for (int q = 0; q < R; ++q) cur[q].load(H + (int64_t)(rl0 + q) * ldh + 8 * gl);
      for (int gi = gl; gi < ng; gi += lpr) {
        if (gi + lpr < ng)
#pragma unroll
          for (int q = 0; q < R; ++q) nxt[q].load(H + (int64_t)(rl0 + q) * ldh + 8 * (gi + lpr));
        float h[R][8];
#pragma unroll
        for (int q = 0; q < R; ++q) cur[q].to_float(h[q]);
#pragma unroll
        for (int c = 0; c < DO; ++c) {
          if (c < d_out) {
            float w8[8];
            load8(Wh + (int64_t)c * w + 8 * gi, w8);
#pragma unroll
            for (int q = 0; q < R; ++q)
#pragma unroll
              for (int k = 0; k < 8; ++k) acc[q][c] = fmaf(h[q][k], w8[k], acc[q][c]);
          }
        }
#pragma unroll
        for (int q = 0; q < R; ++q) cur[q] = nxt[q];
      }
    }
    // sum over the group's lanes (every lane of the warp takes part)
    for (int o = lpr >> 1; o > 0; o >>= 1)
#pragma unroll
      for (int q = 0; q < R; ++q)
#pragma unroll
        for (int c = 0; c < DO; ++c)
          if (c < d_out) acc[q][c] += __shfl_xor_sync(0xffffffffu, acc[q][c], o);
#pragma unroll
    for (int q = 0; q < R; ++q)
#pragma unroll
      for (int c = 0; c < DO; ++c)
        if (c < d_out) acc[q][c] += bh[c];
  }
};

// One block per (member, 128-row block), 256 threads.
//   1. logits, per-row loss and dlogits (HeadLogits; the group's lane 0 takes
//      the loss of its rows) into shared memory;
//   2. the gradient pass: a thread owns G = head_cols(DO) columns and keeps
//      their head weights and partial weight gradients in registers while it
//      walks its rows in order: dZ of the last hidden layer
//      = (dlogits W_h) * [H > 0] / (1 - p), and dW_h += dlogits^T H.  Narrow
//      heads split the rows into jb.split sets, added in order in shared
//      memory, so that every block writes one partial.
// One output: three blocks per SM (80 registers a thread, no spills; the
// kernel waits on memory, 64 to 68 us per wide step for three against two).
template <typename T, int DO>
__global__ void __launch_bounds__(256, DO == 1 ? 3 : 2) k_head(HeadArgs<T> g) {
  constexpr int R = DO <= 4 ? 4 : 2;
  constexpr int G = head_cols(DO);
  constexpr int DOP = DO == 1 ? 1 : (DO + 3) & ~3;  // padded row of dlogits in shared memory
  pdl_trigger();
  pdl_wait();
  const HeadJob jb = g.jobs[blockIdx.x];
  const int r0 = jb.blk * kHeadRows;
  if (r0 >= g.B_pad) return;
  const MemberDev md = g.mem[jb.member];
  const int w = md.w, d_out = g.d_out, ldh = jb.h_ld;
  const T* __restrict__ H = g.act + jb.h_off + (int64_t)r0 * ldh;
  const float* __restrict__ Wh = g.params + jb.w_off;
  const float* __restrict__ bh = g.params + jb.b_off;
  __shared__ __align__(16) float dlog[kHeadRows][DOP];
  __shared__ float lrow[kHeadRows];
  __shared__ __align__(16) float red[256 * G * DO];  // row-set partials when the rows are split
  constexpr bool kColSums = std::is_same_v<T, __nv_bfloat16>;  // dZ column sums (tensor-core mode only)
  __shared__ __align__(16) float redz[kColSums ? 256 * G : 4];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float invB = 1.f / (float)g.B;

  const HeadLogits<T, DO, R> hl(w, lane);
  for (int p0 = 0; p0 < HeadLogits<T, DO, R>::kRowsPerWarp; p0 += hl.step()) {
    const int rl0 = warp * HeadLogits<T, DO, R>::kRowsPerWarp + p0 + hl.grp * R;
    const bool live = hl.grp < hl.groups;
    float acc[R][DO];
    hl.run(H, ldh, Wh, bh, w, d_out, rl0, live, acc);
    // the group's lanes take its R rows in turn (every lane holds the sums)
    for (int q = hl.gl; live && q < R; q += hl.lpr) {
      float z[DO];
#pragma unroll
      for (int c = 0; c < DO; ++c) z[c] = acc[0][c];
#pragma unroll
      for (int qq = 1; qq < R; ++qq)
        if (q == qq)
#pragma unroll
          for (int c = 0; c < DO; ++c) z[c] = acc[qq][c];
      const int32_t* idx = g.dyn ? g.dyn->idx : g.idx;
      const void* yv = g.dyn ? g.dyn->y : g.y;
      const int r = r0 + rl0 + q;
      float dl[DO];
      float loss = 0.f;
#pragma unroll
      for (int c = 0; c < DO; ++c) dl[c] = 0.f;
      if (r < g.B) {
        const int64_t row = idx ? (int64_t)idx[(int64_t)jb.member * g.idx_stride + r] : (int64_t)r;
        loss = row_loss<DO>(g.task, d_out, z, yv, row, invB, dl);
        float* lg = g.logits + ((int64_t)jb.member * g.B_cap + r) * d_out;
#pragma unroll
        for (int c = 0; c < DO; ++c)
          if (c < d_out) lg[c] = z[c];
      }
#pragma unroll
      for (int c = 0; c < DOP; ++c) dlog[rl0 + q][c] = c < DO ? dl[c < DO ? c : 0] : 0.f;
      lrow[rl0 + q] = loss;
    }
  }
  __syncthreads();

  const int n_cg = w / G;
  const int S = jb.split;
  const int rows_per_set = kHeadRows / S;
  T* __restrict__ dZ = g.dz + jb.dz_off + (int64_t)r0 * w;
  float* part = g.head_part + jb.part_off;
  float* dbp = kColSums && g.dbp && jb.colsum ? g.dbp + jb.dz_off / 32 + (int64_t)jb.blk * w : nullptr;
  for (int u = threadIdx.x; u < n_cg * S; u += blockDim.x) {
    const int cg = u % n_cg, set = u / n_cg;
    const int col = G * cg;
    float Wr[DO][G], a[DO][G], cz[G];
#pragma unroll
    for (int k = 0; k < G; ++k) cz[k] = 0.f;
#pragma unroll
    for (int c = 0; c < DO; ++c) {
      if (c < d_out) loadG<G>(Wh + (int64_t)c * w + col, Wr[c]);
      else {
#pragma unroll
        for (int k = 0; k < G; ++k) Wr[c][k] = 0.f;
      }
#pragma unroll
      for (int k = 0; k < G; ++k) a[c][k] = 0.f;
    }
    const int rb = set * rows_per_set;
    // rows in batches of U (rows_per_set is a multiple of 8): the batch's
    // loads are all issued before its products
    constexpr int U = G * DO >= 32 ? 4 : 8;
    for (int rb0 = rb; rb0 < rb + rows_per_set; rb0 += U) {
      RawG<T, G> raw[U];
#pragma unroll
      for (int u2 = 0; u2 < U; ++u2) raw[u2].load(H + (int64_t)(rb0 + u2) * ldh + col);
#pragma unroll
      for (int u2 = 0; u2 < U; ++u2) {
      const int rr = rb0 + u2;
      float h[G], s[G];
      raw[u2].to_float(h);
      float dl[DOP];
      if constexpr (DOP % 4 == 0) {
#pragma unroll
        for (int c = 0; c < DOP; c += 4) {
          const float4 v = *reinterpret_cast<const float4*>(&dlog[rr][c]);
          dl[c] = v.x; dl[c + 1] = v.y; dl[c + 2] = v.z; dl[c + 3] = v.w;
        }
      } else {
#pragma unroll
        for (int c = 0; c < DOP; ++c) dl[c] = dlog[rr][c];
      }
#pragma unroll
      for (int k = 0; k < G; ++k) s[k] = 0.f;
#pragma unroll
      for (int c = 0; c < DO; ++c)
#pragma unroll
        for (int k = 0; k < G; ++k) {
          s[k] = fmaf(dl[c], Wr[c][k], s[k]);
          a[c][k] = fmaf(dl[c], h[k], a[c][k]);
        }
#pragma unroll
      for (int k = 0; k < G; ++k) {
        s[k] = h[k] > 0.f ? s[k] * md.scale : 0.f;
        if constexpr (kColSums)
          if (dbp) cz[k] += __bfloat162float(__float2bfloat16_rn(s[k]));  // dZ as stored
      }
      storeG<G>(dZ + (int64_t)rr * w + col, s);
      }
    }
    if (S == 1) {
#pragma unroll
      for (int c = 0; c < DO; ++c)
        if (c < d_out) storeG<G>(part + (int64_t)c * w + col, a[c]);
      if (dbp) storeG<G>(dbp + col, cz);
    } else {  // n_cg * S <= 256: one (column group, row set) per thread
#pragma unroll
      for (int c = 0; c < DO; ++c)
        if (c < d_out) storeG<G>(&red[((set * DO + c) * n_cg + cg) * G], a[c]);
      if constexpr (kColSums) storeG<G>(&redz[(set * n_cg + cg) * G], cz);
    }
  }
  if (S > 1) {  // the block's partial: row sets added in order
    __syncthreads();
    for (int e = threadIdx.x; e < d_out * w; e += blockDim.x) {
      const int c = e / w, k = e - c * w;
      const int cg = k / G, kk = k - cg * G;
      float v = 0.f;
      for (int set = 0; set < S; ++set) v += red[((set * DO + c) * n_cg + cg) * G + kk];
      part[e] = v;
    }
    if (dbp)
      for (int e = threadIdx.x; e < w; e += blockDim.x) {
        const int cg = e / G, kk = e - cg * G;
        float v = 0.f;
        for (int set = 0; set < S; ++set) v += redz[(set * n_cg + cg) * G + kk];
        dbp[e] = v;
      }
  }
  // bias partial and loss partial of the block (rows in order)
  if (threadIdx.x < d_out) {
    float v = 0.f;
    for (int rr = 0; rr < kHeadRows; ++rr) v += dlog[rr][threadIdx.x];
    part[(int64_t)d_out * w + threadIdx.x] = v;
  }
  if (threadIdx.x == 0) {
    float s = 0.f;
    for (int rr = 0; rr < kHeadRows; ++rr) s += lrow[rr];
    g.loss_part[(int64_t)jb.member * g.n_blk_cap + jb.blk] = s;
  }
}

constexpr int kStageWarps = 8;

__device__ __forceinline__ uint32_t smem_addr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

// ----------------------------------------------- head + loss, staged (bf16)
// The same work as k_head for one member on one 64-row block in bf16 mode,
// with the block's H_L rows (one bulk copy per row) and the head weights (one
// bulk copy) staged in shared memory, so that H is read from HBM once and
// both passes run from shared memory:
//   1. logits: warp v takes the 8-column groups v, v + 8, ... and lane l rows
//      l and l + 32 (16-byte loads; the row pitch is 16 bytes past a
//      multiple of 128, so the eight rows of a quarter-warp fall in distinct
//      banks), with the head weights read warp-uniformly (broadcast); the
//      eight warps' partial logits are added in warp order through shared
//      memory, and one thread per row takes its loss and dlogits;
//   2. gradients: a thread owns 4 consecutive columns of a row set and walks
//      its rows: dZ = (dlogits W_h) [H > 0] / (1 - p) stored in bf16, dW_h
//      partials in registers; row sets (narrow members) are added in order
//      through shared memory.
// Shared memory: H [64][pitch] | W_h [DO][w] | partial logits [8][DO][64] |
// dlogits [64][DOP] | row losses [64] | mbarrier.
template <int DO>
__global__ void __launch_bounds__(256) k_head_stage(HeadArgs<__nv_bfloat16> g) {
  constexpr int DOP = DO == 1 ? 1 : (DO + 3) & ~3;
  // no early trigger: the next kernels' CTAs (the backward GEMM's hold most
  // of an SM's shared memory) must not park beside these blocks
  pdl_wait();
  const HeadJob jb = g.jobs[blockIdx.x];
  const int r0 = jb.blk * kHeadRows;
  if (r0 >= g.B_pad) return;
  const MemberDev md = g.mem[jb.member];
  const int w = md.w, d_out = g.d_out, ldh = jb.h_ld;
  const int pitch = head_stage_pitch(w);
  extern __shared__ __align__(128) unsigned char smem[];
  unsigned char* Hs = smem;
  float* Ws = reinterpret_cast<float*>(smem + (int64_t)kHeadRows * pitch);      // [d_out][w]
  float* zpart = Ws + (int64_t)DO * w;                                          // [8][DO][64]
  float* dlog = zpart + kStageWarps * kHeadRows * DO;                          // [64][DOP]
  float* lrow = dlog + kHeadRows * DOP;                                         // [64]
  uint64_t* bar = reinterpret_cast<uint64_t*>(lrow + kHeadRows + 2);            // 8-byte aligned
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const __nv_bfloat16* __restrict__ H = g.act + jb.h_off + (int64_t)r0 * ldh;
  const float* __restrict__ Wg = g.params + jb.w_off;
  const float* __restrict__ bh = g.params + jb.b_off;
  const uint32_t row_bytes = (uint32_t)w * 2u;
  const uint32_t w_bytes = (uint32_t)(d_out * w) * 4u;

  // stage the 64 rows and the head weights (warp 0 issues the bulk copies)
  if (threadIdx.x == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_addr(bar)) : "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  __syncthreads();
  if (warp == 0) {
    if (lane == 0) {
      asm volatile("fence.proxy.async.global;" ::: "memory");
      asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                   "r"(row_bytes * (uint32_t)kHeadRows + w_bytes)
                   : "memory");
      asm volatile(
          "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
              smem_addr(Ws)),
          "l"(Wg), "r"(w_bytes), "r"(smem_addr(bar))
          : "memory");
    }
    __syncwarp();
    for (int r = lane; r < kHeadRows; r += 32)
      asm volatile(
          "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
              smem_addr(Hs + (int64_t)r * pitch)),
          "l"(H + (int64_t)r * ldh), "r"(row_bytes), "r"(smem_addr(bar))
          : "memory");
  }
  {  // bounded wait for the copies (2 s); on expiry record site 20 and leave
    uint32_t ok = 0;
    uint64_t t0 = 0;
    for (int it = 0;; ++it) {
      asm volatile(
          "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\n selp.u32 %0, 1, 0, p;\n}\n"
          : "=r"(ok)
          : "r"(smem_addr(bar))
          : "memory");
      if (ok) break;
      uint64_t t;
      asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
      if (it == 0) {
        t0 = t;
      } else if (t - t0 > 2000000000ull) {
        if (g.err) atomicCAS(g.err, 0, 20);
        return;
      }
    }
  }

  // 1. logits
  {
    float acc[2][DO];
#pragma unroll
    for (int q = 0; q < 2; ++q)
#pragma unroll
      for (int c = 0; c < DO; ++c) acc[q][c] = 0.f;
    const int ng = w >> 3;
#pragma unroll 2
    for (int gi = warp; gi < ng; gi += kStageWarps) {
      float h[2][8];
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const uint4 v = *reinterpret_cast<const uint4*>(Hs + (int64_t)(lane + 32 * q) * pitch + 16 * gi);
        const __nv_bfloat16* b = reinterpret_cast<const __nv_bfloat16*>(&v);
#pragma unroll
        for (int k = 0; k < 8; ++k) h[q][k] = __bfloat162float(b[k]);
      }
#pragma unroll
      for (int c = 0; c < DO; ++c) {
        if (c < d_out) {
          const float4 wa = *reinterpret_cast<const float4*>(Ws + c * w + 8 * gi);
          const float4 wb = *reinterpret_cast<const float4*>(Ws + c * w + 8 * gi + 4);
          const float w8[8] = {wa.x, wa.y, wa.z, wa.w, wb.x, wb.y, wb.z, wb.w};
#pragma unroll
          for (int q = 0; q < 2; ++q)
#pragma unroll
            for (int k = 0; k < 8; ++k) acc[q][c] = fmaf(h[q][k], w8[k], acc[q][c]);
        }
      }
    }
#pragma unroll
    for (int q = 0; q < 2; ++q)
#pragma unroll
      for (int c = 0; c < DO; ++c) zpart[(warp * DO + c) * kHeadRows + lane + 32 * q] = acc[q][c];
  }
  __syncthreads();
  if (threadIdx.x < kHeadRows) {
    const int rl = threadIdx.x, r = r0 + rl;
    float z[DO];
#pragma unroll
    for (int c = 0; c < DO; ++c) {
      float v = 0.f;
      for (int v8 = 0; v8 < kStageWarps; ++v8) v += zpart[(v8 * DO + c) * kHeadRows + rl];
      z[c] = c < d_out ? v + bh[c] : 0.f;
    }
    float dl[DO];
    float loss = 0.f;
#pragma unroll
    for (int c = 0; c < DO; ++c) dl[c] = 0.f;
    if (r < g.B) {
      const int32_t* idx = g.dyn ? g.dyn->idx : g.idx;
      const void* yv = g.dyn ? g.dyn->y : g.y;
      const int64_t row = idx ? (int64_t)idx[(int64_t)jb.member * g.idx_stride + r] : (int64_t)r;
      loss = row_loss<DO>(g.task, d_out, z, yv, row, 1.f / (float)g.B, dl);
      float* lg = g.logits + ((int64_t)jb.member * g.B_cap + r) * d_out;
#pragma unroll
      for (int c = 0; c < DO; ++c)
        if (c < d_out) lg[c] = z[c];
    }
#pragma unroll
    for (int c = 0; c < DOP; ++c) dlog[rl * DOP + c] = c < DO ? dl[c < DO ? c : 0] : 0.f;
    lrow[rl] = loss;
  }
  __syncthreads();

  // 2. dZ of the last hidden layer and the head-weight gradient partial
  const int n_cg = w >> 2;
  const int S = head_stage_split(w, DO);
  const int rows_per_set = kHeadRows / S;
  __nv_bfloat16* __restrict__ dZ = g.dz + jb.dz_off + (int64_t)r0 * w;
  float* part = g.head_part + jb.part_off;
  float* dbp = g.dbp && jb.colsum ? g.dbp + jb.dz_off / 32 + (int64_t)jb.blk * w : nullptr;
  float a[DO][4], cz[4] = {0.f, 0.f, 0.f, 0.f};
  int cg = 0, set = 0;
  for (int u = threadIdx.x; u < n_cg * S; u += blockDim.x) {
    cg = u % n_cg;
    set = u / n_cg;
    const int col = 4 * cg;
#pragma unroll
    for (int k = 0; k < 4; ++k) cz[k] = 0.f;
    float Wr[DO][4];
#pragma unroll
    for (int c = 0; c < DO; ++c) {
      if (c < d_out) {
        const float4 v = *reinterpret_cast<const float4*>(Ws + c * w + col);
        Wr[c][0] = v.x;
        Wr[c][1] = v.y;
        Wr[c][2] = v.z;
        Wr[c][3] = v.w;
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) Wr[c][k] = 0.f;
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) a[c][k] = 0.f;
    }
    const int rb = set * rows_per_set;
#pragma unroll 4
    for (int rr = rb; rr < rb + rows_per_set; ++rr) {
      const uint2 hv = *reinterpret_cast<const uint2*>(Hs + (int64_t)rr * pitch + 2 * col);
      const __nv_bfloat16* hb = reinterpret_cast<const __nv_bfloat16*>(&hv);
      float h[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) h[k] = __bfloat162float(hb[k]);
      float dl[DOP];
      if constexpr (DOP % 4 == 0) {
#pragma unroll
        for (int c = 0; c < DOP; c += 4) {
          const float4 v = *reinterpret_cast<const float4*>(&dlog[rr * DOP + c]);
          dl[c] = v.x;
          dl[c + 1] = v.y;
          dl[c + 2] = v.z;
          dl[c + 3] = v.w;
        }
      } else {
#pragma unroll
        for (int c = 0; c < DOP; ++c) dl[c] = dlog[rr * DOP + c];
      }
      float sacc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int c = 0; c < DO; ++c)
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          sacc[k] = fmaf(dl[c], Wr[c][k], sacc[k]);
          a[c][k] = fmaf(dl[c], h[k], a[c][k]);
        }
      __align__(8) __nv_bfloat16 o[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        o[k] = __float2bfloat16_rn(h[k] > 0.f ? sacc[k] * md.scale : 0.f);
        if (dbp) cz[k] += __bfloat162float(o[k]);  // dZ as stored
      }
      *reinterpret_cast<uint2*>(dZ + (int64_t)rr * w + col) = *reinterpret_cast<const uint2*>(o);
    }
    if (S == 1) {
#pragma unroll
      for (int c = 0; c < DO; ++c)
        if (c < d_out)
          *reinterpret_cast<float4*>(part + (int64_t)c * w + col) = make_float4(a[c][0], a[c][1], a[c][2], a[c][3]);
      if (dbp) *reinterpret_cast<float4*>(dbp + col) = make_float4(cz[0], cz[1], cz[2], cz[3]);
    }
  }
  if (S > 1) {  // one (column group, row set) per thread; sets added in order (the H area is free now)
    __syncthreads();
    float* red = reinterpret_cast<float*>(Hs);   // [S][DO][w], then [S][w] of dZ column sums
    float* redz = red + (int64_t)S * DO * w;     // S (DO + 1) w <= 24 w floats fit in 64 rows of H
    if (threadIdx.x < n_cg * S) {
#pragma unroll
      for (int c = 0; c < DO; ++c)
        if (c < d_out)
          *reinterpret_cast<float4*>(red + ((int64_t)set * DO + c) * w + 4 * cg) =
              make_float4(a[c][0], a[c][1], a[c][2], a[c][3]);
      *reinterpret_cast<float4*>(redz + (int64_t)set * w + 4 * cg) = make_float4(cz[0], cz[1], cz[2], cz[3]);
    }
    __syncthreads();
    for (int e = threadIdx.x; e < d_out * w; e += blockDim.x) {
      const int c = e / w, k = e - c * w;
      float v = 0.f;
      for (int st = 0; st < S; ++st) v += red[((int64_t)st * DO + c) * w + k];
      part[e] = v;
    }
    if (dbp)
      for (int e = threadIdx.x; e < w; e += blockDim.x) {
        float v = 0.f;
        for (int st = 0; st < S; ++st) v += redz[(int64_t)st * w + e];
        dbp[e] = v;
      }
  }
  pdl_trigger();
  // bias partial and loss partial of the block (rows in order)
  if (threadIdx.x < d_out) {
    float v = 0.f;
    for (int rr = 0; rr < kHeadRows; ++rr) v += dlog[rr * DOP + threadIdx.x];
    part[(int64_t)d_out * w + threadIdx.x] = v;
  }
  if (threadIdx.x == 0) {
    float sl = 0.f;
    for (int rr = 0; rr < kHeadRows; ++rr) sl += lrow[rr];
    g.loss_part[(int64_t)jb.member * g.n_blk_cap + jb.blk] = sl;
  }
}

// ------------------------------------------ one-output head, one pass (bf16)
// The head of a one-output task (binary or regression) for one member on one
// 64-row block, with H_L read once.  The block's 256 threads form S = 256 / T
// row sets of T threads (T = w / 8 rounded up to a power of two, at least
// 32); thread t of a set owns the 8-column group t, keeps its head weights
// and its partial weight gradient in registers, and walks the set's rows
// kOneRows at a time with the next rows' 16-byte loads in flight:
//   1. partial logits of the rows, summed over the warp by shuffles and over
//      the set's warps in warp order through shared memory, bias added; one
//      thread per row takes its loss and dlogit;
//   2. dZ of the last hidden layer = dlogit W_h [H > 0] / (1 - p) stored in
//      bf16, and dW_h += dlogit H.
// The sets' partials are added in set order, so each block writes one
// partial of dW_h, db_h and the loss (rows in order), the layout k_head
// writes for k_head_reduce, and (dbp) the column sums of its dZ rows.
// Widths up to 2048.
constexpr int kOneRows = 8;

__global__ void __launch_bounds__(256, 2) k_head_one(HeadArgs<__nv_bfloat16> g) {
  pdl_trigger();
  pdl_wait();
  const HeadJob jb = g.jobs[blockIdx.x];
  const int r0 = jb.blk * kHeadRows;
  if (r0 >= g.B_pad) return;
  const MemberDev md = g.mem[jb.member];
  const int w = md.w, ldh = jb.h_ld, ng = w >> 3;
  int T = 32;
  while (T < ng) T <<= 1;
  const int S = 256 / T, set = threadIdx.x / T, t = threadIdx.x % T;
  const int rows_set = kHeadRows / S, n_steps = rows_set / kOneRows, wpset = T >> 5;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool has = t < ng;
  const int col = 8 * t;
  __shared__ float zp[8][kOneRows];
  __shared__ float dls[8][kOneRows];
  __shared__ float dlrow[kHeadRows], lrow[kHeadRows];
  __shared__ __align__(16) float red[8 * 256];  // [S][w]: S * w <= 8 * T * S = 2048
  __shared__ __align__(16) float redz[8 * 256]; // the same for the column sums of dZ
  const __nv_bfloat16* __restrict__ H = g.act + jb.h_off + (int64_t)(r0 + set * rows_set) * ldh + col;
  __nv_bfloat16* __restrict__ dZ = g.dz + jb.dz_off + (int64_t)(r0 + set * rows_set) * w + col;
  const float bias = g.params[jb.b_off];
  const float invB = 1.f / (float)g.B;
  const int32_t* idx = g.dyn ? g.dyn->idx : g.idx;
  const void* yv = g.dyn ? g.dyn->y : g.y;
  float Wr[8], a[8], cz[8];
  if (has) load8(g.params + jb.w_off + col, Wr);
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    if (!has) Wr[k] = 0.f;
    a[k] = 0.f;
    cz[k] = 0.f;
  }
  uint4 cur[kOneRows], nxt[kOneRows];
#pragma unroll
  for (int u = 0; u < kOneRows; ++u) {
    cur[u] = has ? *reinterpret_cast<const uint4*>(H + (int64_t)u * ldh) : make_uint4(0u, 0u, 0u, 0u);
    nxt[u] = make_uint4(0u, 0u, 0u, 0u);
  }
  for (int st = 0; st < n_steps; ++st) {
    if (has && st + 1 < n_steps)
#pragma unroll
      for (int u = 0; u < kOneRows; ++u)
        nxt[u] = *reinterpret_cast<const uint4*>(H + (int64_t)((st + 1) * kOneRows + u) * ldh);
    // 1. logits of the set's kOneRows rows
    float p[kOneRows];
#pragma unroll
    for (int u = 0; u < kOneRows; ++u) {
      const __nv_bfloat16* b = reinterpret_cast<const __nv_bfloat16*>(&cur[u]);
      float s = 0.f;
#pragma unroll
      for (int k = 0; k < 8; ++k) s = fmaf(__bfloat162float(b[k]), Wr[k], s);
      p[u] = s;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
#pragma unroll
      for (int u = 0; u < kOneRows; ++u) p[u] += __shfl_xor_sync(0xffffffffu, p[u], o);
    if (lane == 0)
#pragma unroll
      for (int u = 0; u < kOneRows; ++u) zp[warp][u] = p[u];
    __syncthreads();
    if (threadIdx.x < S * kOneRows) {
      const int s2 = threadIdx.x / kOneRows, u = threadIdx.x % kOneRows;
      float zz[1] = {0.f};
      for (int v = 0; v < wpset; ++v) zz[0] += zp[s2 * wpset + v][u];
      zz[0] += bias;
      const int rl = s2 * rows_set + st * kOneRows + u, r = r0 + rl;
      float dl[1] = {0.f}, loss = 0.f;
      if (r < g.B) {
        const int64_t row = idx ? (int64_t)idx[(int64_t)jb.member * g.idx_stride + r] : (int64_t)r;
        loss = row_loss<1>(g.task, 1, zz, yv, row, invB, dl);
        g.logits[(int64_t)jb.member * g.B_cap + r] = zz[0];
      }
      dls[s2][u] = dl[0];
      dlrow[rl] = dl[0];
      lrow[rl] = loss;
    }
    __syncthreads();
    // 2. dZ of the last hidden layer and the weight-gradient partial
#pragma unroll
    for (int u = 0; u < kOneRows; ++u) {
      const float dl = dls[set][u];
      const __nv_bfloat16* b = reinterpret_cast<const __nv_bfloat16*>(&cur[u]);
      float o[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float h = __bfloat162float(b[k]);
        o[k] = h > 0.f ? (dl * Wr[k]) * md.scale : 0.f;
        a[k] = fmaf(dl, h, a[k]);
      }
      uint4 pz;
      __nv_bfloat162* pb = reinterpret_cast<__nv_bfloat162*>(&pz);
#pragma unroll
      for (int k = 0; k < 4; ++k) pb[k] = __floats2bfloat162_rn(o[2 * k], o[2 * k + 1]);
      if (has) *reinterpret_cast<uint4*>(dZ + (int64_t)(st * kOneRows + u) * w) = pz;
      if (jb.colsum) {  // column sums of dZ as stored
        const uint32_t* pw = reinterpret_cast<const uint32_t*>(&pz);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          cz[2 * k] += __uint_as_float(pw[k] << 16);
          cz[2 * k + 1] += __uint_as_float(pw[k] & 0xFFFF0000u);
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kOneRows; ++u) cur[u] = nxt[u];
  }
  float* part = g.head_part + jb.part_off;
  float* dbp = g.dbp && jb.colsum ? g.dbp + jb.dz_off / 32 + (int64_t)jb.blk * w : nullptr;
  if (S == 1) {
    if (has) {
      store8(part + col, a);
      if (dbp) store8(dbp + col, cz);
    }
  } else {  // the sets' partials added in set order
    if (has) {
      store8(red + set * w + col, a);
      store8(redz + set * w + col, cz);
    }
    __syncthreads();
    for (int e = threadIdx.x; e < w; e += blockDim.x) {
      float v = 0.f, vz = 0.f;
      for (int s2 = 0; s2 < S; ++s2) {
        v += red[s2 * w + e];
        vz += redz[s2 * w + e];
      }
      part[e] = v;
      if (dbp) dbp[e] = vz;
    }
  }
  // bias and loss partials of the block (rows in order)
  if (threadIdx.x == 0) {
    float v = 0.f;
    for (int rr = 0; rr < kHeadRows; ++rr) v += dlrow[rr];
    part[w] = v;
  }
  if (threadIdx.x == 32) {
    float v = 0.f;
    for (int rr = 0; rr < kHeadRows; ++rr) v += lrow[rr];
    g.loss_part[(int64_t)jb.member * g.n_blk_cap + jb.blk] = v;
  }
}

// Sum the per-block head partials (fixed order) into the head gradients and
// the per-member mean loss; in update mode apply the member's AdamW to the
// head parameters directly (the gradients are not stored).  Grid: member x
// chunks of 256 head parameters; inactive members report NaN.
__global__ void k_head_reduce(HeadReduceArgs g) {
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x;
  const HeadReduceJob jb = g.jobs[i];
  const int n_blk = g.B_pad / kHeadRows;
  if (!g.active[i]) {
    float* lo = g.dyn ? g.dyn->loss_out : g.loss_out;
    if (blockIdx.y == 0 && threadIdx.x == 0 && lo) lo[i] = __int_as_float(0x7fc00000);
    return;
  }
  const int w = jb.w, d_out = g.d_out;
  const int e0 = blockIdx.y * blockDim.x;
  if (e0 >= d_out * w + d_out) return;
  const int64_t stride = g.part_stride[i];
  float lr = 0.f, wdw = 0.f, wdb = 0.f, ib1 = 1.f, ib2 = 1.f;
  if (g.update) {
    const MemberDev md = g.adam.mem[i];
    const float2 bc = g.adam.bias_corr[i];
    lr = md.lr;
    wdw = md.wd;
    wdb = g.adam.wd_on_bias ? md.wd : 0.f;
    ib1 = 1.f / bc.x;
    ib2 = 1.f / bc.y;
  }
  for (int e = e0 + threadIdx.x; e < min(e0 + (int)blockDim.x, d_out * w + d_out); e += blockDim.x) {
    float s = 0.f;
#pragma unroll 8
    for (int b = 0; b < n_blk; ++b) s += g.head_part[jb.part_off + b * stride + e];
    const bool is_b = e >= d_out * w;
    const int64_t o = is_b ? jb.gb_off + (e - d_out * w) : jb.gw_off + e;
    if (g.update) {
      float p = g.adam.params[o], m = g.adam.m[o], v = g.adam.v[o];
      adamw_elem(p, m, v, s, lr, is_b ? wdb : wdw, g.adam.beta1, g.adam.beta2, g.adam.eps, ib1, ib2);
      g.adam.params[o] = p;
      g.adam.m[o] = m;
      g.adam.v[o] = v;
      if (g.adam.wq_out) g.adam.wq_out[o] = __float2bfloat16_rn(p);
    } else {
      g.grads[o] = s;
    }
  }
  if (blockIdx.y == 0 && threadIdx.x == 0) {
    float s = 0.f;
    for (int b = 0; b < n_blk; ++b) s += g.loss_part[(int64_t)i * g.n_blk_cap + b];
    const float loss = s / (float)g.B;
    float* lo = g.dyn ? g.dyn->loss_out : g.loss_out;
    if (lo) lo[i] = loss;
    g.loss_last[i] = loss;
  }
}

// ------------------------------------------------------------------ AdamW
// Stand-alone AdamW over chunks of the arena (unless AdamW is fused into the
// weight-gradient epilogue), with the member's lr and wd and its step's bias
// corrections; float4 body, scalar tail.  In bf16 mode the same threads
// first fill the dropout mask arena for the next step.
__global__ void __launch_bounds__(256) k_adamw(AdamArgs g) {
  pdl_trigger();
  pdl_wait();
  const Chunk ch = g.chunks[blockIdx.x];
  const Segment s = g.segs[ch.seg];
  const MemberDev md = g.mem[s.member];
  const float2 bc = g.bias_corr[s.member];
  const float lr = md.lr;
  const float wd = (s.is_bias && !g.wd_on_bias) ? 0.f : md.wd;
  const float b1 = g.beta1, b2 = g.beta2, eps = g.eps;
  const float ib1 = 1.f / bc.x, ib2 = 1.f / bc.y;
  const int n4 = ch.len >> 2;  // chunk offsets are multiples of 4 elements
  float4* P4 = reinterpret_cast<float4*>(g.params + ch.off);
  const float4* G4 = reinterpret_cast<const float4*>(g.grads + ch.off);
  float4* M4 = reinterpret_cast<float4*>(g.m + ch.off);
  float4* V4 = reinterpret_cast<float4*>(g.v + ch.off);
  for (int e = threadIdx.x; e < n4; e += blockDim.x) {
    float4 p = P4[e], m = M4[e], v = V4[e];
    const float4 gr = __ldcs(G4 + e);
    adamw_elem(p.x, m.x, v.x, gr.x, lr, wd, b1, b2, eps, ib1, ib2);
    adamw_elem(p.y, m.y, v.y, gr.y, lr, wd, b1, b2, eps, ib1, ib2);
    adamw_elem(p.z, m.z, v.z, gr.z, lr, wd, b1, b2, eps, ib1, ib2);
    adamw_elem(p.w, m.w, v.w, gr.w, lr, wd, b1, b2, eps, ib1, ib2);
    P4[e] = p;
    M4[e] = m;
    V4[e] = v;
    if (g.wq) {
      __nv_bfloat162 lo = __floats2bfloat162_rn(p.x, p.y), hi = __floats2bfloat162_rn(p.z, p.w);
      uint2 u;
      u.x = *reinterpret_cast<uint32_t*>(&lo);
      u.y = *reinterpret_cast<uint32_t*>(&hi);
      *reinterpret_cast<uint2*>(g.wq + ch.off + 4 * e) = u;
    }
  }
  for (int e = 4 * n4 + threadIdx.x; e < ch.len; e += blockDim.x) {
    const int64_t o = ch.off + e;
    float p = g.params[o], m = g.m[o], v = g.v[o];
    adamw_elem(p, m, v, g.grads[o], lr, wd, b1, b2, eps, ib1, ib2);
    g.params[o] = p;
    g.m[o] = m;
    g.v[o] = v;
    if (g.wq) g.wq[o] = __float2bfloat16_rn(p);
  }
  // the next step's dropout masks: ALU work that other blocks' HBM streaming
  // overlaps (after this block's own stores have left, so that it does not
  // delay them)
  fill_masks(g.mg, (int64_t)blockIdx.x * blockDim.x + threadIdx.x, (int64_t)gridDim.x * blockDim.x);
}

// ------------------------------------------------------------------- init
// Element of the padded arena -> the element index within the layer
// (weights row-major unpadded, then biases) -> Philox word -> U(-b, b), fp32.
__global__ void k_init(InitArgs g) {
  const Chunk ch = g.chunks[blockIdx.x];
  const Segment s = g.segs[ch.seg];
  for (int e = threadIdx.x; e < ch.len; e += blockDim.x) {
    const int64_t o = ch.off + e;
    const int64_t local = o - s.off;
    float val = 0.f;
    bool real = true;
    uint32_t idx;
    if (s.is_bias) {
      idx = (uint32_t)(s.w_elems + local);
    } else {
      const int64_t row = local / s.cols_pad, col = local % s.cols_pad;
      real = col < s.cols;
      idx = (uint32_t)(row * s.cols + col);
    }
    if (real) {
      U4 r4 = philox10(idx >> 2, 0u, 0u, (1u << 28) | ((uint32_t)s.member << 4) | (uint32_t)s.layer,
                       (uint32_t)g.seed, (uint32_t)(g.seed >> 32));
      const uint32_t q = idx & 3u;
      const uint32_t r = q == 0 ? r4.x : q == 1 ? r4.y : q == 2 ? r4.z : r4.w;
      const double u = ((double)(r >> 8) + 0.5) * 5.9604644775390625e-08;  // 2^-24
      const double bound = 1.0 / sqrt((double)s.fan_in);
      val = (float)((2.0 * u - 1.0) * bound);
    }
    g.params[o] = val;
    g.grads[o] = 0.f;
    g.m[o] = 0.f;
    g.v[o] = 0.f;
    if (g.wq0) {
      g.wq0[o] = __float2bfloat16_rn(val);
      g.wq1[o] = __float2bfloat16_rn(val);
    }
  }
}

// bf16 copies of the whole arena (after pack_set_params / pack_set_active).
__global__ void k_refresh_wq(const float* __restrict__ p, __nv_bfloat16* __restrict__ wq0,
                             __nv_bfloat16* __restrict__ wq1, int64_t n) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n; e += (int64_t)gridDim.x * blockDim.x) {
    const __nv_bfloat16 b = __float2bfloat16_rn(p[e]);
    wq0[e] = b;
    wq1[e] = b;
  }
}

// ----------------------------------------------------------- predict head
// Forward-only head: probabilities (softmax / sigmoid) or values into
// out[member, n0 + r, :] for r < rows.
template <typename T, int DO>
__global__ void __launch_bounds__(256) k_predict_head(PredictHeadArgs<T> g) {
  constexpr int R = DO <= 10 ? 4 : 2;
  pdl_wait();
  const HeadJob jb = g.jobs[blockIdx.x];
  const int r0 = jb.blk * kHeadRows;
  if (r0 >= g.rows) return;
  const MemberDev md = g.mem[jb.member];
  const int w = md.w, d_out = g.d_out, ldh = jb.h_ld;
  const T* H = g.act + jb.h_off + (int64_t)r0 * ldh;
  const float* Wh = g.params + jb.w_off;
  const float* bh = g.params + jb.b_off;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const HeadLogits<T, DO, R> hl(w, lane);
  for (int p0 = 0; p0 < HeadLogits<T, DO, R>::kRowsPerWarp; p0 += hl.step()) {
    const int rl0 = warp * HeadLogits<T, DO, R>::kRowsPerWarp + p0 + hl.grp * R;
    const bool live = hl.grp < hl.groups && r0 + rl0 < g.rows;
    float acc[R][DO];
    hl.run(H, ldh, Wh, bh, w, d_out, rl0, live, acc);
    if (!live) continue;
    // the group's lanes write its R rows in turn
    for (int q = hl.gl; q < R; q += hl.lpr) {
      const int r = r0 + rl0 + q;
      if (r >= g.rows) break;
      float z[DO];
#pragma unroll
      for (int c = 0; c < DO; ++c) z[c] = acc[0][c];
#pragma unroll
      for (int qq = 1; qq < R; ++qq)
        if (q == qq)
#pragma unroll
          for (int c = 0; c < DO; ++c) z[c] = acc[qq][c];
      float* o = g.out + ((int64_t)jb.member * g.N + g.n0 + r) * d_out;
      if (g.task == 1) {
        float mx = z[0];
#pragma unroll
        for (int c = 1; c < DO; ++c) if (c < d_out) mx = fmaxf(mx, z[c]);
        float sum = 0.f;
#pragma unroll
        for (int c = 0; c < DO; ++c) if (c < d_out) sum += expf(z[c] - mx);
        const float inv = 1.f / sum;
#pragma unroll
        for (int c = 0; c < DO; ++c)
          if (c < d_out) o[c] = expf(z[c] - mx) * inv;
      } else {
        o[0] = g.task == 0 ? 1.f / (1.f + expf(-z[0])) : z[0];
      }
    }
  }
}

// ------------------------------------------------------------- mask dump
__global__ void k_debug_masks(uint8_t* __restrict__ out, int32_t B, int32_t w, uint64_t seed,
                              uint32_t member, uint32_t layer, uint32_t step, uint32_t T) {
  const int64_t n4 = (int64_t)B * (w / 4);
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n4; e += (int64_t)gridDim.x * blockDim.x) {
    const int r = (int)(e / (w / 4)), c4 = (int)(e % (w / 4));
    const uint32_t k = keep_bits4(seed, member, layer, step, (uint32_t)r, (uint32_t)c4, T);
#pragma unroll
    for (int q = 0; q < 4; ++q) out[(int64_t)r * w + c4 * 4 + q] = (uint8_t)((k >> q) & 1u);
  }
}

// ------------------------------------------------------------- Philox words
// in [n, 6]: counter c0..c3 then key k0, k1; out [n, 4]: the four words.
__global__ void k_debug_philox(const uint32_t* __restrict__ in, uint32_t* __restrict__ out, int32_t n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const uint32_t* c = in + (int64_t)i * 6;
  const U4 r = philox10(c[0], c[1], c[2], c[3], c[4], c[5]);
  uint32_t* o = out + (int64_t)i * 4;
  o[0] = r.x;
  o[1] = r.y;
  o[2] = r.z;
  o[3] = r.w;
}

// ------------------------------------------------------------- launchers
template <typename T>
void launch_gather(cudaStream_t st, const float* X, const int32_t* idx, const StepDyn* dyn, int B, int B_pad,
                   int d_in, int d_in_pad, int ldx, T* xb, int advance, int32_t* t_dev, float2* bias_corr,
                   const int32_t* active_ids, int n_active, float beta1, float beta2, int* zero, int n_zero,
                   int stacked, int64_t xb_stride) {
  const int blocks = std::max(1, (int)ceil_div(B_pad, 8));  // 8 rows (warps) per block
  const unsigned gy = stacked ? (unsigned)std::max(n_active, 1) : 1u;
  const float ln_b1 = (float)std::log((double)beta1), ln_b2 = (float)std::log((double)beta2);
  launch_pdl(k_gather<T>, dim3(blocks, gy), dim3(256), 0, st, X, idx, dyn, B, B_pad, d_in, d_in_pad, ldx, xb, advance,
             t_dev, bias_corr, active_ids, n_active, ln_b1, ln_b2, zero, n_zero, stacked, xb_stride);
}

template <typename T>
void launch_fill_ones(cudaStream_t st, const OnesJob* jobs, int n_jobs, T* xb, T* act, T* ex) {
  if (n_jobs > 0) k_fill_ones<T><<<n_jobs, 256, 0, st>>>(jobs, xb, act, ex);
}

template <typename T>
void launch_gemm_simt(cudaStream_t st, const GemmArgs<T>& g, int tile_base, int n_tiles) {
  if (n_tiles > 0) launch_pdl(k_gemm_simt<T>, dim3(n_tiles), dim3(256), 0, st, g, tile_base);
}

template <int DO>
static bool launch_head_stage(cudaStream_t st, const HeadArgs<__nv_bfloat16>& g, int n_jobs) {
  const int64_t bytes = head_stage_smem(g.w_max, DO);
  if (bytes > kHeadStageSmemMax) return false;
  launch_pdl(k_head_stage<DO>, dim3(n_jobs), dim3(256), (size_t)bytes, st, g);
  return true;
}

void head_stage_prepare() {
  cudaFuncSetAttribute(k_head_stage<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, kHeadStageSmemMax);
  cudaFuncSetAttribute(k_head_stage<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, kHeadStageSmemMax);
  cudaFuncSetAttribute(k_head_stage<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, kHeadStageSmemMax);
  cudaFuncSetAttribute(k_head_stage<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, kHeadStageSmemMax);
  cudaFuncSetAttribute(k_head_stage<10>, cudaFuncAttributeMaxDynamicSharedMemorySize, kHeadStageSmemMax);
  cudaFuncSetAttribute(k_head_stage<16>, cudaFuncAttributeMaxDynamicSharedMemorySize, kHeadStageSmemMax);
}

template <typename T>
void launch_head(cudaStream_t st, const HeadArgs<T>& g, int n_jobs) {
  if (n_jobs <= 0) return;
  if constexpr (std::is_same_v<T, __nv_bfloat16>) {
    // one output on members wider than 512: the one-pass kernel (the staged
    // block would run one per SM)
    if (g.d_out == 1 && g.w_max > 512 && g.w_max <= 2048) {
      launch_pdl(k_head_one, dim3(n_jobs), dim3(256), 0, st, g);
      return;
    }
    if (g.stage && !(g.d_out == 1 && g.w_max > 512)) {
      bool done = false;
      switch (head_bucket(g.d_out)) {
        case 1: done = launch_head_stage<1>(st, g, n_jobs); break;
        case 2: done = launch_head_stage<2>(st, g, n_jobs); break;
        case 4: done = launch_head_stage<4>(st, g, n_jobs); break;
        case 8: done = launch_head_stage<8>(st, g, n_jobs); break;
        case 10: done = launch_head_stage<10>(st, g, n_jobs); break;
        case 16: done = launch_head_stage<16>(st, g, n_jobs); break;
        default: break;
      }
      if (done) return;
    }
  }
  switch (head_bucket(g.d_out)) {
    case 1: launch_pdl(k_head<T, 1>, dim3(n_jobs), dim3(256), 0, st, g); break;
    case 2: launch_pdl(k_head<T, 2>, dim3(n_jobs), dim3(256), 0, st, g); break;
    case 4: launch_pdl(k_head<T, 4>, dim3(n_jobs), dim3(256), 0, st, g); break;
    case 8: launch_pdl(k_head<T, 8>, dim3(n_jobs), dim3(256), 0, st, g); break;
    case 10: launch_pdl(k_head<T, 10>, dim3(n_jobs), dim3(256), 0, st, g); break;
    case 16: launch_pdl(k_head<T, 16>, dim3(n_jobs), dim3(256), 0, st, g); break;
    default: launch_pdl(k_head<T, kMaxDout>, dim3(n_jobs), dim3(256), 0, st, g); break;
  }
}

void launch_head_reduce(cudaStream_t st, const HeadReduceArgs& g, int m, int max_elems) {
  launch_pdl(k_head_reduce, dim3(m, (unsigned)ceil_div(max_elems, 256)), dim3(256), 0, st, g);
}

void launch_adamw(cudaStream_t st, const AdamArgs& g, int n_chunks) {
  if (n_chunks > 0) launch_pdl(k_adamw, dim3(n_chunks), dim3(256), 0, st, g);
}

void launch_init(cudaStream_t st, const InitArgs& g, int n_chunks) {
  if (n_chunks > 0) k_init<<<n_chunks, 256, 0, st>>>(g);
}

// ---------------------------------------------------- periodic embeddings
// E_i[b, q] (q = j d + k) = alpha_q f_q(x_bj) + beta_q with f_0(x) = x and
// f_k(x) = cos(w_j,k-1 x + b_j,k-1).  Both kernels tile a member's columns
// in groups of 32 (lane = column: each thread keeps its column's feature,
// component and parameters in registers) and spread the rows over the
// block's 8 warps.
constexpr int kEmbRows = 128;  // rows per forward block

struct EmbCol {
  int j, k;
  float w, b, alpha, beta;
};

__device__ __forceinline__ EmbCol emb_col(const EmbMember& em, const float* params, int d_in, int q) {
  const int d = em.d, dm = d - 1;
  const float* w = params + em.p_off;
  const float* bb = w + (int64_t)d_in * dm;
  const float* al = bb + (int64_t)d_in * dm;
  const float* be = al + (int64_t)d_in * d;
  EmbCol c;
  c.j = q / d;
  c.k = q - c.j * d;
  c.alpha = al[q];
  c.beta = be[q];
  c.w = c.k ? w[c.j * dm + c.k - 1] : 0.f;
  c.b = c.k ? bb[c.j * dm + c.k - 1] : 0.f;
  return c;
}

// Forward: block (32-column group, 128-row group, active member); rows >= B
// and the pad columns up to in0_pad are written as zero.
template <typename T>
__global__ void __launch_bounds__(256) k_emb_fwd(EmbArgs<T> a) {
  pdl_trigger();
  pdl_wait();
  const int member = a.active_ids[blockIdx.z];
  const EmbMember em = a.em[member];
  const int q = blockIdx.x * 32 + (threadIdx.x & 31);
  if (q >= em.in0_pad) return;
  const float* X = a.dyn ? a.dyn->X : a.X;
  const int32_t* idx = a.dyn ? a.dyn->idx : a.idx;
  if (idx) idx += (int64_t)member * a.idx_stride;
  const bool col = q < em.in0;
  const EmbCol c = col ? emb_col(em, a.params, a.d_in, q) : EmbCol{0, 0, 0.f, 0.f, 0.f, 0.f};
  const int64_t ld = em.in0_pad + kOnesCols;
  T* E = a.ex + em.e_off + q;
  const int r1 = min(a.B_pad, (int)(blockIdx.y + 1) * kEmbRows);
  for (int b = blockIdx.y * kEmbRows + (threadIdx.x >> 5); b < r1; b += 8) {
    float e = 0.f;
    if (col && b < a.B) {
      const int64_t row = idx ? (int64_t)idx[b] : (int64_t)b;
      const float x = X[row * a.d_in + c.j];
      const float f = c.k == 0 ? x : cosf(fmaf(c.w, x, c.b));
      e = fmaf(c.alpha, f, c.beta);
    }
    E[(int64_t)b * ld] = Elem<T>::from_f(e);
  }
}

// Backward: block (32-column group, active member), warp r takes rows r,
// r + 8, ...; with dE = the first layer's input gradient,
//   d alpha_q = sum_b dE f_q,  d beta_q = sum_b dE,
//   d w = -alpha_q sum_b dE sin(u) x,  d b = -alpha_q sum_b dE sin(u)
// (u = w x + b, cosine components).  Each thread sums up to 32 of its rows
// in fp32 and adds that partial to fp64 sums; the 8 warps' fp64 sums are
// added in warp order.
template <typename T>
__global__ void __launch_bounds__(256, 6) k_emb_bwd(EmbArgs<T> a) {
  pdl_trigger();
  pdl_wait();
  const int member = a.active_ids[blockIdx.y];
  const EmbMember em = a.em[member];
  if ((int)blockIdx.x * 32 >= em.in0) return;   // block-uniform
  const int lane = threadIdx.x & 31, wp = threadIdx.x >> 5;
  const int q = blockIdx.x * 32 + lane;
  const bool col = q < em.in0;
  const int qc = col ? q : em.in0 - 1;          // in-range column for the loads of idle lanes
  const float* X = a.dyn ? a.dyn->X : a.X;
  const int32_t* idx = a.dyn ? a.dyn->idx : a.idx;
  if (idx) idx += (int64_t)member * a.idx_stride;
  const EmbCol c = emb_col(em, a.params, a.d_in, qc);
  const T* dE = a.dz + em.de_off + qc;
  double s_a = 0.0, s_be = 0.0, s_w = 0.0, s_b = 0.0;
  for (int b0 = wp; b0 < a.B; b0 += 8 * 32) {
    float p_a = 0.f, p_be = 0.f, p_w = 0.f, p_b = 0.f;
    const int b1 = min(a.B, b0 + 8 * 32);
#pragma unroll 4
    for (int b = b0; b < b1; b += 8) {
      const float g = Elem<T>::to_f(dE[(int64_t)b * em.in0_pad]);
      const int64_t row = idx ? (int64_t)idx[b] : (int64_t)b;
      const float x = X[row * a.d_in + c.j];
      p_be += g;
      if (c.k == 0) {
        p_a = fmaf(g, x, p_a);
      } else {
        float sn, cs;
        sincosf(fmaf(c.w, x, c.b), &sn, &cs);
        p_a = fmaf(g, cs, p_a);
        const float gs = g * sn;
        p_w = fmaf(gs, x, p_w);
        p_b += gs;
      }
    }
    s_a += p_a;
    s_be += p_be;
    s_w += p_w;
    s_b += p_b;
  }
  __shared__ double red[4][8][32];
  red[0][wp][lane] = s_a;
  red[1][wp][lane] = s_be;
  red[2][wp][lane] = s_w;
  red[3][wp][lane] = s_b;
  __syncthreads();
  if (wp != 0 || !col) return;
  double t[4] = {0.0, 0.0, 0.0, 0.0};
  for (int r = 0; r < 8; ++r)
    for (int u = 0; u < 4; ++u) t[u] += red[u][r][lane];
  const int d = em.d, dm = d - 1;
  float* gw = a.grads + em.p_off;
  float* gb = gw + (int64_t)a.d_in * dm;
  float* ga = gb + (int64_t)a.d_in * dm;
  float* gbt = ga + (int64_t)a.d_in * d;
  ga[q] = (float)t[0];
  gbt[q] = (float)t[1];
  if (c.k) {
    gw[c.j * dm + c.k - 1] = (float)(-(double)c.alpha * t[2]);
    gb[c.j * dm + c.k - 1] = (float)(-(double)c.alpha * t[3]);
  }
}

template <typename T>
void launch_emb_fwd(cudaStream_t st, const EmbArgs<T>& a, int n_active, int cols_max) {
  if (n_active > 0 && a.B_pad > 0)
    launch_pdl(k_emb_fwd<T>, dim3((unsigned)ceil_div(cols_max, 32), (unsigned)ceil_div(a.B_pad, kEmbRows),
                                  (unsigned)n_active), dim3(256), 0, st, a);
}
template <typename T>
void launch_emb_bwd(cudaStream_t st, const EmbArgs<T>& a, int n_active, int cols_max) {
  if (n_active > 0)
    launch_pdl(k_emb_bwd<T>, dim3((unsigned)ceil_div(cols_max, 32), (unsigned)n_active), dim3(256), 0, st, a);
}

// ------------------------------------------------------------------ Muon
// One block of 256 threads per chunk of a Muon matrix (row-major [rows,
// cols] in the arena): kMuonChunk consecutive elements, or for a transposed
// matrix a 32 x 128 tile of W (muon_chunks).  Widths are multiples of 16 and
// padded input widths multiples of 8, and arena blocks start 32-element
// aligned, so 4 consecutive elements of a chunk share a row and start at a
// 16-byte boundary: the kernels move float4 and 4-element vectors, each
// thread kMuonV of them, all loads first.  The per-element arithmetic is
// fp32; doubles appear only in the partial sums (GB300's FP64 rate is a
// small fraction of its FP32 rate).
constexpr int kMuonV = kMuonChunk / 4 / 256;
static_assert(kMuonChunk % 1024 == 0, "a Muon chunk is a whole number of float4 per thread");

template <typename T>
struct MuonChunk {
  MuonMat mt;
  int mat;     // its index in the matrix list
  int e0, n4;  // flat chunk: its first element within the matrix and its float4 count
  int i0, j0;  // tile of a transposed matrix: its first row and column of W
  __device__ __forceinline__ MuonChunk(const MuonArgs<T>& a, int blk) {
    mat = a.chunk_mat[blk];
    mt = a.mats[mat];
    const int k = blk - mt.chunk0;
    if (!mt.tr) {
      e0 = k * kMuonChunk;
      n4 = (min(e0 + kMuonChunk, mt.rows * mt.cols) - e0) >> 2;
      i0 = j0 = 0;
    } else {
      const int tpr = (mt.cols + kMuonTileC - 1) / kMuonTileC;
      i0 = (k / tpr) * kMuonTileR;
      j0 = (k % tpr) * kMuonTileC;
      e0 = n4 = 0;
    }
  }
  // Element offset in W (from w_off) of this chunk's float4 q (0 <= q <
  // kMuonChunk / 4), or -1 outside the matrix.  Tiles: row q / 32, columns
  // 4 (q % 32) .. + 3 of the tile, so a warp reads 512 contiguous bytes.
  __device__ __forceinline__ int w_elem(int q) const {
    if (!mt.tr) return q < n4 ? e0 + 4 * q : -1;
    const int row = i0 + (q >> 5), col = j0 + 4 * (q & 31);
    return row < mt.rows && col < mt.cols ? row * mt.cols + col : -1;
  }
  // Tiles: piece p (0 <= p < kMuonChunk / 4) of X's rows -- row j0 + p / 8,
  // columns i0 + 4 (p % 8) .. + 3, i.e. W's column j0 + p / 8 at its rows
  // i0 + 4 (p % 8) .. + 3 -- as an element offset in X, or -1 outside.
  __device__ __forceinline__ int x_piece(int p) const {
    const int j = j0 + (p >> 3), i = i0 + 4 * (p & 7);
    return j < mt.cols && i < mt.rows ? j * mt.c + i : -1;
  }
};

__device__ __forceinline__ float4 load4f(const float* p) { return *reinterpret_cast<const float4*>(p); }
__device__ __forceinline__ float4 load4f(const __nv_bfloat16* p) {
  const uint2 u = *reinterpret_cast<const uint2*>(p);
  const float2 lo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
  const float2 hi = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
  return make_float4(lo.x, lo.y, hi.x, hi.y);
}

// A tile's X values staged in shared memory as [tile row][tile column] of W
// (pitch kMuonTileC + 2: the column reads of x_piece order touch distinct
// banks).
template <typename T>
using MuonStage = T[kMuonTileR][kMuonTileC + 2];

// the momentum update of one element; returns U's element
__device__ __forceinline__ float muon_mom(float g, float& m, float mu) {
  m = mu * m + (1.f - mu) * g;
  return (1.f - mu) * g + mu * m;
}

// 1 / max(|U|_F, 1e-7) of a matrix from its chunks' sums of squares, by one
// warp in a fixed order (lane j sums chunks j, j + 32, ...; then a butterfly):
// the same value wherever it is computed.
__device__ __forceinline__ float muon_inv_norm(const double* part, int chunk0, int n_chunks, int lane) {
  double ss = 0.0;
  for (int k = lane; k < n_chunks; k += 32) ss += __ldcg(part + chunk0 + k);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  return (float)(1.0 / fmax(sqrt(ss), 1e-7));
}

// momentum M <- mu M + (1 - mu) G; U = (1 - mu) G + mu M; the chunk's sum of
// squares of U (fp32 per thread, then fp64 in a fixed-order tree).  Also
// clears the counters of the Newton-Schulz launch that follows.  x0_fused:
// U is also written as X0 (a transposed matrix's tile through shared memory,
// as whole row segments of X), and the last chunk of a matrix to finish
// stores the matrix's scale.
template <typename T>
__global__ void __launch_bounds__(256) k_muon_momentum(MuonArgs<T> a) {
  pdl_trigger();
  pdl_wait();
  for (int i = blockIdx.x * 256 + threadIdx.x; i < a.n_ns_cnt; i += gridDim.x * 256) a.ns_cnt[i] = 0;
  const MuonChunk<T> ck(a, blockIdx.x);
  const float mu = a.mu;
  const float* G = a.grads + ck.mt.w_off;
  float* M = a.mom + ck.mt.w_off;
  T* X = a.ns + ck.mt.x_off[0];
  __shared__ MuonStage<T> st;
  float4 g[kMuonV], m[kMuonV];
  int ev[kMuonV];
#pragma unroll
  for (int k = 0; k < kMuonV; ++k) {
    ev[k] = ck.w_elem(threadIdx.x + 256 * k);
    if (ev[k] >= 0) {
      g[k] = *reinterpret_cast<const float4*>(G + ev[k]);
      m[k] = *reinterpret_cast<const float4*>(M + ev[k]);
    }
  }
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < kMuonV; ++k) {
    if (ev[k] < 0) continue;
    const float u0 = muon_mom(g[k].x, m[k].x, mu), u1 = muon_mom(g[k].y, m[k].y, mu);
    const float u2 = muon_mom(g[k].z, m[k].z, mu), u3 = muon_mom(g[k].w, m[k].w, mu);
    *reinterpret_cast<float4*>(M + ev[k]) = m[k];
    ss = fmaf(u0, u0, ss);
    ss = fmaf(u1, u1, ss);
    ss = fmaf(u2, u2, ss);
    ss = fmaf(u3, u3, ss);
    if (a.x0_fused) {
      if (!ck.mt.tr) {
        store4(X + ev[k], make_float4(u0, u1, u2, u3));
      } else {
        const int q = threadIdx.x + 256 * k, r = q >> 5, c = 4 * (q & 31);
        st[r][c] = Elem<T>::from_f(u0);
        st[r][c + 1] = Elem<T>::from_f(u1);
        st[r][c + 2] = Elem<T>::from_f(u2);
        st[r][c + 3] = Elem<T>::from_f(u3);
      }
    }
  }
  if (a.x0_fused && ck.mt.tr) {  // block-uniform
    __syncthreads();
#pragma unroll
    for (int k = 0; k < kMuonV; ++k) {
      const int p = threadIdx.x + 256 * k, xo = ck.x_piece(p);
      if (xo < 0) continue;
      const int jj = p >> 3, i4 = 4 * (p & 7);
      store4(X + xo, make_float4(Elem<T>::to_f(st[i4][jj]), Elem<T>::to_f(st[i4 + 1][jj]),
                                 Elem<T>::to_f(st[i4 + 2][jj]), Elem<T>::to_f(st[i4 + 3][jj])));
    }
  }
  double s = (double)ss;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  __shared__ double red[8];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  __shared__ int last;
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < 8; ++w) t += red[w];
    a.part[blockIdx.x] = t;
    if (a.x0_fused) {
      __threadfence();  // the partial before the arrival
      last = atomicAdd(a.mat_done + ck.mat, 1) == ck.mt.n_chunks - 1;
    }
  }
  if (!a.x0_fused) return;
  __syncthreads();
  if (last && threadIdx.x < 32) {
    __threadfence();  // every arrival before the partials' reads
    const float inv = muon_inv_norm(a.part, ck.mt.chunk0, ck.mt.n_chunks, threadIdx.x);
    if (threadIdx.x == 0) {
      a.ns_scale[ck.mat] = inv;
      a.mat_done[ck.mat] = 0;
    }
  }
}

// X0 = U / max(||U||_F, 1e-7), transposed when rows > cols (element by
// element: this pass serves the fp32 mode).  Chunks in reverse order: the
// momentum pass's last chunks are still in L2.
template <typename T>
__global__ void __launch_bounds__(256) k_muon_x0(MuonArgs<T> a) {
  pdl_trigger();
  pdl_wait();
  const MuonChunk<T> ck(a, gridDim.x - 1 - blockIdx.x);
  __shared__ float inv_s;
  if (threadIdx.x < 32) {  // the matrix's norm from its chunks' partials, one warp
    const float inv = muon_inv_norm(a.part, ck.mt.chunk0, ck.mt.n_chunks, threadIdx.x);
    if (threadIdx.x == 0) inv_s = inv;
  }
  const float mu = a.mu;
  const float* G = a.grads + ck.mt.w_off;
  const float* M = a.mom + ck.mt.w_off;
  float4 g[kMuonV], m[kMuonV];
  int ev[kMuonV];
#pragma unroll
  for (int k = 0; k < kMuonV; ++k) {
    ev[k] = ck.w_elem(threadIdx.x + 256 * k);
    if (ev[k] >= 0) {
      g[k] = __ldcs(reinterpret_cast<const float4*>(G + ev[k]));
      m[k] = *reinterpret_cast<const float4*>(M + ev[k]);
    }
  }
  __syncthreads();
  const float inv = inv_s;
  T* X = a.ns + ck.mt.x_off[0];
#pragma unroll
  for (int k = 0; k < kMuonV; ++k) {
    const int e = ev[k];
    if (e < 0) continue;
    const float4 u = make_float4(((1.f - mu) * g[k].x + mu * m[k].x) * inv, ((1.f - mu) * g[k].y + mu * m[k].y) * inv,
                                 ((1.f - mu) * g[k].z + mu * m[k].z) * inv, ((1.f - mu) * g[k].w + mu * m[k].w) * inv);
    if (!ck.mt.tr) {
      store4(X + e, u);
    } else {  // the 4 elements share a row i of W: entries (j .. j + 3, i) of X
      const int i = e / ck.mt.cols, j = e - i * ck.mt.cols;
      const int x0 = j * ck.mt.c + i;
      X[x0] = Elem<T>::from_f(u.x);
      X[x0 + ck.mt.c] = Elem<T>::from_f(u.y);
      X[x0 + 2 * ck.mt.c] = Elem<T>::from_f(u.z);
      X[x0 + 3 * ck.mt.c] = Elem<T>::from_f(u.w);
    }
  }
}

// W <- W - lr wd W; W <- W - lr scale O, O = the final X (transposed back: a
// transposed matrix's tile reads whole row segments of X into shared memory)
template <typename T>
__global__ void __launch_bounds__(256) k_muon_apply(MuonArgs<T> a) {
  pdl_trigger();
  pdl_wait();
  const MuonChunk<T> ck(a, blockIdx.x);
  const float lr = ck.mt.lr, wd = a.mem[ck.mt.member].wd, sc = ck.mt.scale;
  const T* X = a.ns + (a.x_final ? ck.mt.x_off[1] : ck.mt.x_off[0]);  // no runtime index into the record
  float* P = a.params + ck.mt.w_off;
  __shared__ MuonStage<T> st;
  if (ck.mt.tr) {  // block-uniform
#pragma unroll
    for (int k = 0; k < kMuonV; ++k) {
      const int p = threadIdx.x + 256 * k, xo = ck.x_piece(p);
      if (xo < 0) continue;
      const float4 v = load4f(X + xo);
      const int jj = p >> 3, i4 = 4 * (p & 7);
      st[i4][jj] = Elem<T>::from_f(v.x);
      st[i4 + 1][jj] = Elem<T>::from_f(v.y);
      st[i4 + 2][jj] = Elem<T>::from_f(v.z);
      st[i4 + 3][jj] = Elem<T>::from_f(v.w);
    }
    __syncthreads();
  }
  float4 p[kMuonV], x[kMuonV];
  int ev[kMuonV];
#pragma unroll
  for (int k = 0; k < kMuonV; ++k) {
    const int q = threadIdx.x + 256 * k, r = q >> 5, c = 4 * (q & 31);
    ev[k] = ck.w_elem(q);
    p[k] = x[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (ev[k] >= 0) {
      p[k] = *reinterpret_cast<const float4*>(P + ev[k]);
      x[k] = ck.mt.tr ? make_float4(Elem<T>::to_f(st[r][c]), Elem<T>::to_f(st[r][c + 1]),
                                    Elem<T>::to_f(st[r][c + 2]), Elem<T>::to_f(st[r][c + 3]))
                      : load4f(X + ev[k]);
    }
  }
#pragma unroll
  for (int k = 0; k < kMuonV; ++k) {
    if (ev[k] < 0) continue;
    float4 q = p[k];
    q.x = q.x - lr * wd * q.x;
    q.y = q.y - lr * wd * q.y;
    q.z = q.z - lr * wd * q.z;
    q.w = q.w - lr * wd * q.w;
    q.x = q.x - lr * sc * x[k].x;
    q.y = q.y - lr * sc * x[k].y;
    q.z = q.z - lr * sc * x[k].z;
    q.w = q.w - lr * sc * x[k].w;
    *reinterpret_cast<float4*>(P + ev[k]) = q;
    if (a.wq_out) store4(a.wq_out + ck.mt.w_off + ev[k], q);
  }
}

template <typename T>
void launch_muon(cudaStream_t st, const MuonArgs<T>& a, int n_chunks, int phase) {
  if (n_chunks <= 0) return;
  if (phase == 0) launch_pdl(k_muon_momentum<T>, dim3(n_chunks), dim3(256), 0, st, a);
  else if (phase == 1) launch_pdl(k_muon_x0<T>, dim3(n_chunks), dim3(256), 0, st, a);
  else launch_pdl(k_muon_apply<T>, dim3(n_chunks), dim3(256), 0, st, a);
}

__global__ void __launch_bounds__(256) k_masks(MaskGen mg) {
  pdl_trigger();
  pdl_wait();
  fill_masks(mg, (int64_t)blockIdx.x * blockDim.x + threadIdx.x, (int64_t)gridDim.x * blockDim.x);
}

void launch_masks(cudaStream_t st, const MaskGen& mg) {
  const int64_t total = (int64_t)mg.n_chunks * mg.rows;
  if (total <= 0) return;
  launch_pdl(k_masks, dim3((unsigned)std::min<int64_t>(ceil_div(total, 256), 152 * 8)), dim3(256), 0, st, mg);
}

void launch_refresh_wq(cudaStream_t st, const float* p, __nv_bfloat16* wq0, __nv_bfloat16* wq1, int64_t n) {
  k_refresh_wq<<<152 * 4, 256, 0, st>>>(p, wq0, wq1, n);
}

template <typename T>
void launch_predict_head(cudaStream_t st, const PredictHeadArgs<T>& g, int n_jobs) {
  if (n_jobs <= 0) return;
  switch (head_bucket(g.d_out)) {
    case 1: k_predict_head<T, 1><<<n_jobs, 256, 0, st>>>(g); break;
    case 2: k_predict_head<T, 2><<<n_jobs, 256, 0, st>>>(g); break;
    case 4: k_predict_head<T, 4><<<n_jobs, 256, 0, st>>>(g); break;
    case 8: k_predict_head<T, 8><<<n_jobs, 256, 0, st>>>(g); break;
    case 10: k_predict_head<T, 10><<<n_jobs, 256, 0, st>>>(g); break;
    case 16: k_predict_head<T, 16><<<n_jobs, 256, 0, st>>>(g); break;
    default: k_predict_head<T, kMaxDout><<<n_jobs, 256, 0, st>>>(g); break;
  }
}

void launch_debug_masks(cudaStream_t st, uint8_t* out, int B, int w, uint64_t seed, uint32_t member,
                        uint32_t layer, uint32_t step, uint32_t T) {
  k_debug_masks<<<64, 256, 0, st>>>(out, B, w, seed, member, layer, step, T);
}

void launch_debug_philox(cudaStream_t st, const uint32_t* in, uint32_t* out, int n) {
  k_debug_philox<<<(int)ceil_div(n, 128), 128, 0, st>>>(in, out, n);
}

#define TP_INSTANTIATE(T)                                                                              \
  template void launch_gather<T>(cudaStream_t, const float*, const int32_t*, const StepDyn*, int, int, int, int, \
                                 int, T*, int, int32_t*, float2*, const int32_t*, int, float, float,    \
                                 int*, int, int, int64_t);                                              \
  template void launch_fill_ones<T>(cudaStream_t, const OnesJob*, int, T*, T*, T*);                    \
  template void launch_gemm_simt<T>(cudaStream_t, const GemmArgs<T>&, int, int);                       \
  template void launch_head<T>(cudaStream_t, const HeadArgs<T>&, int);                                 \
  template void launch_predict_head<T>(cudaStream_t, const PredictHeadArgs<T>&, int);           \
  template void launch_muon<T>(cudaStream_t, const MuonArgs<T>&, int, int);                      \
  template void launch_emb_fwd<T>(cudaStream_t, const EmbArgs<T>&, int, int);                     \
  template void launch_emb_bwd<T>(cudaStream_t, const EmbArgs<T>&, int, int);

TP_INSTANTIATE(float)
TP_INSTANTIATE(__nv_bfloat16)

}  // namespace tp
