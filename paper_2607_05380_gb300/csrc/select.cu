// select.cu -- greedy ensemble selection on the device (Sec. 3.5 "Greedy
// ensembling").  Each iteration scores every unused candidate c as the
// ensemble S + {c}, picks the best (lowest index on ties), and stops when the
// best addition does not strictly improve the current score.  The running sum
// S of the selected candidates' predictions is fp64; the ensemble value of a
// row is (S + p_c) * (1 / (n + 1)) in fp64, each row's loss / squared-error
// term is then taken in fp32, and terms are summed in fp64 in a fixed order
// (per-thread rows, then a shuffle tree, then blocks in index order).  The
// accuracy decision (argmax) is taken on the fp64 ensemble values.
#include "kernels.cuh"

namespace tp {

constexpr int kSelThreads = 256;
constexpr int kSelRowsPerThread = 4;
constexpr int kSelRowsPerBlock = kSelThreads * kSelRowsPerThread;

enum { kStN = 0, kStDone = 1, kStLast = 2, kStHdr = 4 };
constexpr int kScoreAuc = 3;      // TP_SCORE_AUC
constexpr int kAucThreads = 1024;

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__global__ void k_sel_init(double* __restrict__ S, int64_t n_S, int32_t* __restrict__ state, int32_t n_state,
                           double* __restrict__ cur, const uint8_t* __restrict__ excl, int32_t m_ens) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n_S; e += (int64_t)gridDim.x * blockDim.x)
    S[e] = 0.0;
  if (blockIdx.x == 0) {
    const int used0 = kStHdr + m_ens;  // used[c] starts as excl[c]
    for (int e = threadIdx.x; e < n_state; e += blockDim.x)
      state[e] = (excl != nullptr && e >= used0) ? (excl[e - used0] != 0) : 0;
    if (threadIdx.x == 0) {
      state[kStLast] = -1;
      cur[0] = __longlong_as_double(0x7ff0000000000000LL);  // +inf
    }
  }
}

__device__ __forceinline__ double row_term(const double* __restrict__ S, const float* __restrict__ p,
                                           const void* __restrict__ y, int64_t b, int32_t d_out,
                                           int32_t task, int32_t score, double inv) {
  const double* s = S + b * d_out;
  const float* q = p + b * d_out;
  if (score == 1) {  // accuracy
    int pred;
    if (task == 1) {
      pred = 0;
      double best = (s[0] + (double)q[0]) * inv;
      for (int c = 1; c < d_out; ++c) {
        double e = (s[c] + (double)q[c]) * inv;
        if (e > best) { best = e; pred = c; }
      }
    } else {
      pred = (s[0] + (double)q[0]) * inv > 0.5 ? 1 : 0;
    }
    return pred == ((const int32_t*)y)[b] ? 1.0 : 0.0;
  }
  if (task == 2) {
    float e = (float)((s[0] + (double)q[0]) * inv);
    float d = e - ((const float*)y)[b];
    return (double)(d * d);
  }
  const int yv = ((const int32_t*)y)[b];
  const int k = task == 1 ? yv : 0;
  if (k < 0 || k >= d_out) return __longlong_as_double(0x7ff8000000000000LL);  // invalid label: NaN score
  float e = (float)((s[k] + (double)q[k]) * inv);
  e = fminf(fmaxf(e, 1e-7f), 1.0f - 1e-7f);
  float t = (task == 1 || yv == 1) ? -logf(e) : -logf(1.0f - e);
  return (double)t;
}

__global__ void __launch_bounds__(kSelThreads) k_sel_score(const double* __restrict__ S, const float* __restrict__ preds,
                                                           const void* __restrict__ y, int64_t N, int32_t d_out,
                                                           int32_t task, int32_t score, const int32_t* __restrict__ state,
                                                           double* __restrict__ partial, int32_t n_blk, int32_t m_ens) {
  const int c = blockIdx.y;
  const int32_t* used = state + kStHdr + m_ens;
  if (state[kStDone] || used[c]) return;
  const double inv = 1.0 / (double)(state[kStN] + 1);
  const float* p = preds + (int64_t)c * N * d_out;
  const int64_t r0 = (int64_t)blockIdx.x * kSelRowsPerBlock;
  double acc = 0.0;
#pragma unroll
  for (int q = 0; q < kSelRowsPerThread; ++q) {
    const int64_t b = r0 + q * kSelThreads + threadIdx.x;
    if (b < N) acc += row_term(S, p, y, b, d_out, task, score, inv);
  }
  acc = warp_sum_d(acc);
  __shared__ double ws[kSelThreads / 32];
  if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int w = 0; w < kSelThreads / 32; ++w) s += ws[w];
    partial[(int64_t)c * n_blk + blockIdx.x] = s;
  }
}

// Score of candidate c from its per-block partial sums: blocks in index
// order, then the mean over N rows and the score's transform (the ROC-AUC
// kernel writes the candidate's score itself, -AUC, as its first partial).
__device__ __forceinline__ double cand_score(const double* __restrict__ partial, int c, int32_t n_blk, int64_t N,
                                             int32_t score) {
  if (score == kScoreAuc) return partial[(int64_t)c * n_blk];
  double s = 0.0;
  for (int b = 0; b < n_blk; ++b) s += partial[(int64_t)c * n_blk + b];
  const double mean = s / (double)N;
  return score == 1 ? -mean : (score == 2 ? sqrt(mean) : mean);
}

// Every candidate's score on its own, from the first iteration's partials.
__global__ void k_sel_solo(const double* __restrict__ partial, int32_t P, int32_t n_blk, int64_t N, int32_t score,
                           const int32_t* __restrict__ state, int32_t m_ens, double* __restrict__ solo) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= P) return;
  const int32_t* used = state + kStHdr + m_ens;
  solo[c] = used[c] ? __longlong_as_double(0x7ff8000000000000LL) : cand_score(partial, c, n_blk, N, score);
}

// ROC-AUC score of candidate c (one block per candidate): the ensemble's
// scores (S + p_c) / (n + 1), rounded to fp32, sorted with their labels by a
// stable 4-pass radix sort of order-preserving keys (8-bit digits; within a
// 1024-key tile a key's place among equal digits comes from its warp's
// match mask and the warps before it), then each positive's mid-rank among
// equal scores by binary search: AUC = (sum of the positives' ranks -
// n_pos (n_pos + 1) / 2) / (n_pos n_neg).  Rank sums are half-integers, exact
// in fp64, so the result does not depend on the order of the sum.
// two blocks per SM (32 registers a thread), so that a pool of up to two
// candidates per SM sorts in one wave
__global__ void __launch_bounds__(kAucThreads, 2) k_sel_auc(const double* __restrict__ S,
                                                         const float* __restrict__ preds,
                                                         const int32_t* __restrict__ y, int64_t N,
                                                         const int32_t* __restrict__ state,
                                                         double* __restrict__ partial, int32_t n_blk,
                                                         int32_t m_ens, uint32_t* __restrict__ keys,
                                                         uint8_t* __restrict__ lab) {
  const int c = blockIdx.x;
  const int32_t* used = state + kStHdr + m_ens;
  if (state[kStDone] || used[c]) return;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const double inv = 1.0 / (double)(state[kStN] + 1);
  const float* p = preds + (int64_t)c * N;
  uint32_t* const k0 = keys + (int64_t)(2 * c) * N;
  uint32_t* const k1 = k0 + N;
  uint8_t* const l0 = lab + (int64_t)(2 * c) * N;
  uint8_t* const l1 = l0 + N;
  for (int64_t b = tid; b < N; b += kAucThreads) {
    const float f = (float)((S[b] + (double)p[b]) * inv);
    const uint32_t u = __float_as_uint(f);
    k0[b] = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
    l0[b] = y[b] == 1 ? 1 : 0;
  }
  __shared__ uint32_t hist[256], base[256], tot[256];
  __shared__ uint32_t wcnt[kAucThreads / 32][256];
  for (int e = tid; e < (kAucThreads / 32) * 256; e += kAucThreads) (&wcnt[0][0])[e] = 0;
  __syncthreads();
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 8 * pass;
    const bool odd = pass & 1;
    const uint32_t* src = odd ? k1 : k0;
    const uint8_t* srcl = odd ? l1 : l0;
    uint32_t* dst = odd ? k0 : k1;
    uint8_t* dstl = odd ? l0 : l1;
    if (tid < 256) hist[tid] = 0;
    __syncthreads();
    for (int64_t b = tid; b < N; b += kAucThreads) atomicAdd(&hist[(src[b] >> shift) & 255u], 1u);
    __syncthreads();
    if (tid == 0) {
      uint32_t run = 0;
      for (int d = 0; d < 256; ++d) {
        base[d] = run;
        run += hist[d];
      }
    }
    __syncthreads();
    for (int64_t t0 = 0; t0 < N; t0 += kAucThreads) {
      const int64_t b = t0 + tid;
      const bool valid = b < N;
      const uint32_t key = valid ? src[b] : 0u;
      const uint8_t l = valid ? srcl[b] : 0;
      const int d = valid ? (int)((key >> shift) & 255u) : 256;
      const uint32_t peers = __match_any_sync(0xffffffffu, d);
      const int rank = __popc(peers & ((1u << lane) - 1u));
      if (valid && rank == 0) wcnt[warp][d] = __popc(peers);
      __syncthreads();
      if (tid < 256) {   // per digit: exclusive prefix over warps, then the tile's total
        uint32_t run = 0;
        for (int w = 0; w < kAucThreads / 32; ++w) {
          const uint32_t v = wcnt[w][tid];
          wcnt[w][tid] = run;
          run += v;
        }
        tot[tid] = run;
      }
      __syncthreads();
      if (valid) {
        const uint32_t off = base[d] + wcnt[warp][d] + (uint32_t)rank;
        dst[off] = key;
        dstl[off] = l;
      }
      __syncthreads();
      if (tid < 256) {
        base[tid] += tot[tid];
        for (int w = 0; w < kAucThreads / 32; ++w) wcnt[w][tid] = 0;
      }
      __syncthreads();
    }
  }
  // sorted: k0, l0 (four passes).  Mid-ranks of the positives.
  const uint32_t* sk = k0;
  const uint8_t* sl = l0;
  double rs = 0.0;
  int64_t np = 0;
  for (int64_t i = tid; i < N; i += kAucThreads) {
    if (!sl[i]) continue;
    const uint32_t key = sk[i];
    int64_t lo = 0, hi = i;              // first index with this key
    while (lo < hi) {
      const int64_t mid = (lo + hi) >> 1;
      if (sk[mid] < key) lo = mid + 1; else hi = mid;
    }
    const int64_t first = lo;
    lo = i + 1;
    hi = N;                              // one past the last index with this key
    while (lo < hi) {
      const int64_t mid = (lo + hi) >> 1;
      if (sk[mid] <= key) lo = mid + 1; else hi = mid;
    }
    rs += 0.5 * (double)(first + 1 + lo);
    ++np;
  }
  __shared__ double rsum[kAucThreads / 32];
  __shared__ long long pcnt[kAucThreads / 32];
  for (int o = 16; o > 0; o >>= 1) {
    rs += __shfl_xor_sync(0xffffffffu, rs, o);
    np += __shfl_xor_sync(0xffffffffu, np, o);
  }
  if (lane == 0) {
    rsum[warp] = rs;
    pcnt[warp] = np;
  }
  __syncthreads();
  if (tid == 0) {
    double r = 0.0;
    long long n_pos = 0;
    for (int w = 0; w < kAucThreads / 32; ++w) {
      r += rsum[w];
      n_pos += pcnt[w];
    }
    const long long n_neg = (long long)N - n_pos;
    double auc = __longlong_as_double(0x7ff8000000000000LL);
    if (n_pos > 0 && n_neg > 0)
      auc = (r - 0.5 * (double)n_pos * (double)(n_pos + 1)) / ((double)n_pos * (double)n_neg);
    partial[(int64_t)c * n_blk] = -auc;
  }
}

__global__ void __launch_bounds__(1024) k_sel_pick(const double* __restrict__ partial, int32_t P, int32_t n_blk,
                                                   int64_t N, int32_t score, int32_t* __restrict__ state,
                                                   double* __restrict__ cur, int32_t m_ens) {
  if (state[kStDone]) {
    if (threadIdx.x == 0) state[kStLast] = -1;  // nothing to add this iteration
    return;
  }
  int32_t* selected = state + kStHdr;
  int32_t* used = state + kStHdr + m_ens;
  double best = __longlong_as_double(0x7ff0000000000000LL);
  int best_c = -1;
  for (int c = threadIdx.x; c < P; c += blockDim.x) {
    if (used[c]) continue;
    const double sc = cand_score(partial, c, n_blk, N, score);
    if (sc < best) { best = sc; best_c = c; }   // ascending c per thread: lowest index wins ties
  }
  // block argmin, ties to the lowest index
  __shared__ double sb[1024];
  __shared__ int sc_[1024];
  sb[threadIdx.x] = best;
  sc_[threadIdx.x] = best_c;
  __syncthreads();
  for (int o = blockDim.x / 2; o > 0; o >>= 1) {
    if (threadIdx.x < o) {
      double ob = sb[threadIdx.x + o];
      int oc = sc_[threadIdx.x + o];
      double mb = sb[threadIdx.x];
      int mc = sc_[threadIdx.x];
      bool take = oc >= 0 && (mc < 0 || ob < mb || (ob == mb && oc < mc));
      if (take) { sb[threadIdx.x] = ob; sc_[threadIdx.x] = oc; }
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const int c = sc_[0];
    const double b = sb[0];
    const int n = state[kStN];
    if (c < 0 || (n > 0 && !(b < cur[0]))) {
      state[kStDone] = 1;
      state[kStLast] = -1;
    } else {
      selected[n] = c;
      used[c] = 1;
      state[kStN] = n + 1;
      state[kStLast] = c;
      cur[0] = b;
      if (n + 1 >= m_ens) state[kStDone] = 1;
    }
  }
}

__global__ void k_sel_add(double* __restrict__ S, const float* __restrict__ preds, int64_t n_S,
                          const int32_t* __restrict__ state) {
  const int c = state[kStLast];
  if (c < 0) return;
  const float* p = preds + (int64_t)c * n_S;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n_S; e += (int64_t)gridDim.x * blockDim.x)
    S[e] += (double)p[e];
}

int64_t select_scratch_bytes(int32_t P, int64_t N, int32_t d_out, int32_t m_ens, int32_t score) {
  const int64_t n_blk = ceil_div(N, kSelRowsPerBlock);
  int64_t bytes = round_up(N * d_out * 8, 256) + round_up((int64_t)P * n_blk * 8, 256) + 256 +
                  round_up((int64_t)(kStHdr + m_ens + P) * 4, 256);
  if (score == kScoreAuc) bytes += round_up((int64_t)P * 2 * N * 4, 256) + round_up((int64_t)P * 2 * N, 256);
  return bytes;
}

SelectScratch select_carve(void* base, int32_t P, int64_t N, int32_t d_out, int32_t m_ens, int32_t score) {
  const int64_t n_blk = ceil_div(N, kSelRowsPerBlock);
  char* p = (char*)base;
  SelectScratch s;
  s.S = (double*)p;
  p += round_up(N * d_out * 8, 256);
  s.partial = (double*)p;
  p += round_up((int64_t)P * n_blk * 8, 256);
  s.cur = (double*)p;
  p += 256;
  s.state = (int32_t*)p;
  p += round_up((int64_t)(kStHdr + m_ens + P) * 4, 256);
  s.keys = nullptr;
  s.lab = nullptr;
  if (score == kScoreAuc) {
    s.keys = (uint32_t*)p;
    p += round_up((int64_t)P * 2 * N * 4, 256);
    s.lab = (uint8_t*)p;
  }
  return s;
}

// Enqueue the whole selection (m_ens iterations) on `st`; no host sync.
// Returns the number of the state words to copy back (header + selection).
int select_enqueue(cudaStream_t st, const SelectScratch& s, const float* preds, int32_t P, int64_t N,
                   int32_t d_out, const void* y, int32_t task, int32_t score, int32_t m_ens,
                   const uint8_t* excl, double* solo, int64_t* launches) {
  const int32_t n_blk = (int32_t)ceil_div(N, kSelRowsPerBlock);
  const int64_t n_S = N * d_out;
  const int32_t n_state = kStHdr + m_ens + P;
  const int add_blocks = (int)std::min<int64_t>(ceil_div(n_S, 256), 152 * 8);
  k_sel_init<<<add_blocks, 256, 0, st>>>(s.S, n_S, s.state, n_state, s.cur, excl, m_ens);
  int64_t nl = 1;
  for (int it = 0; it < m_ens; ++it) {
    if (score == kScoreAuc)
      k_sel_auc<<<P, kAucThreads, 0, st>>>(s.S, preds, (const int32_t*)y, N, s.state, s.partial, n_blk, m_ens,
                                           s.keys, s.lab);
    else
      k_sel_score<<<dim3(n_blk, P), kSelThreads, 0, st>>>(s.S, preds, y, N, d_out, task, score, s.state,
                                                          s.partial, n_blk, m_ens);
    if (it == 0 && solo != nullptr) {
      k_sel_solo<<<(int)ceil_div(P, 256), 256, 0, st>>>(s.partial, P, n_blk, N, score, s.state, m_ens, solo);
      ++nl;
    }
    k_sel_pick<<<1, 1024, 0, st>>>(s.partial, P, n_blk, N, score, s.state, s.cur, m_ens);
    k_sel_add<<<add_blocks, 256, 0, st>>>(s.S, preds, n_S, s.state);
    nl += 3;
  }
  if (launches) *launches += nl;
  return kStHdr + m_ens;
}

}  // namespace tp
