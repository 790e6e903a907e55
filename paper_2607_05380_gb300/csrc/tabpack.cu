// tabpack.cu -- host side of the C ABI declared in include/tabpack.h: pack
// layout, schedule construction (which member/layer/tile runs in which
// launch), the step orchestration on the pack's stream, and error handling.
#include <cuda_runtime.h>

#include <algorithm>
#include <array>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "kernels.cuh"
#include "tabpack.h"
#include "tc_gemm.cuh"

using namespace tp;

namespace {

thread_local std::string g_thread_error;

struct PhaseEvents {
  std::vector<cudaEvent_t> pool;
  std::vector<std::pair<int, int>> pending;  // (phase, event index of start; stop = +1)
  double ms[TP_PH_COUNT] = {0};
  int64_t launches[TP_PH_COUNT] = {0};
};

}  // namespace

struct tabpack {
  tp_config cfg{};
  int d_in_pad = 0, ldx = 0, B_cap = 0, n_blk_cap = 0, Lmax = 0;
  cudaStream_t st = nullptr;
  bool bf16 = true;
  bool bias_colsums = false;  // bf16: bias gradients from dZ column sums where bias_from_colsums
  std::vector<int32_t> depth, width;
  std::vector<float> dropout, lr, wd;
  std::vector<std::array<int64_t, kMaxDepth + 1>> W_off, b_off;
  std::vector<std::array<int64_t, kMaxDepth>> act_off, dz_off;
  std::vector<uint8_t> active;
  std::vector<Segment> segs;
  std::vector<MemberDev> mem;
  std::vector<int64_t> part_off, part_stride;
  int64_t n_params = 0, act_elems = 0, dz_elems = 0, xb_elems = 0, head_part_elems = 0;
  size_t elem = 2;

  // device memory
  float *params = nullptr, *grads = nullptr, *adam_m = nullptr, *adam_v = nullptr;
  __nv_bfloat16* wq[2] = {nullptr, nullptr};
  int wcur = 0;  // the bf16 weight copy the next step reads
  bool fuse_adamw = false;  // bf16: AdamW in the wgrad epilogue (else a stand-alone pass)
  void *xb = nullptr, *act = nullptr, *dz = nullptr;
  float *logits = nullptr, *head_part = nullptr, *loss_part = nullptr, *loss_last = nullptr;
  // bf16: column sums of dZ over 32-row groups (64-row blocks for the last
  // hidden layer's, written by the head), element dz_off / 32 + g * w + j,
  // for the layers whose bias gradient comes from them (bias_from_colsums)
  float* dbp = nullptr;
  int32_t* t_dev = nullptr;
  float2* bias_corr = nullptr;
  uint8_t* active_dev = nullptr;
  int32_t* active_ids_dev = nullptr;
  MemberDev* mem_dev = nullptr;
  Segment* segs_dev = nullptr;
  Chunk* chunks_dev = nullptr;
  GemmProblem* probs_dev = nullptr;
  GemmTile* tiles_dev = nullptr;
  HeadJob* head_jobs_dev = nullptr;
  HeadReduceJob* hred_dev = nullptr;
  int64_t* part_stride_dev = nullptr;
  TcPlan tc;  // tensor-core GEMM plan (bf16 mode)

  // bf16 prediction runs in chunks of P_cap rows (up to kPredictRows, built
  // on first use) with its own forward-only tile plan over its own arenas:
  // p_xb [P_cap, ldx] and, per member, two activation buffers
  // [P_cap, w + 16] that consecutive layers use in turn (layer l writes
  // buffer l & 1; a row block of layer l + 2 starts only after every tile of
  // layer l + 1 on that row block has finished reading it).
  TcPlan tcp;
  int P_cap = 0;
  void *p_xb = nullptr, *p_act = nullptr;
  std::vector<std::array<int64_t, kMaxDepth>> p_act_off;
  HeadJob* p_head_dev = nullptr;
  int n_p_head = 0;
  bool p_stale = true;      // active set changed since the prediction plan was built

  // Muon for the hidden-layer weights (pack_set_muon): one MuonMat per (member,
  // hidden layer), its X0, X1, A, Bm in the Newton-Schulz arena `ns` (the
  // product precision), the flat list of the element chunks (muon_chunks) of
  // the active members' matrices and a sum-of-squares partial per chunk.  The
  // momentum buffers are the AdamW first-moment arena (AdamW skips these
  // matrices).
  bool muon = false;
  float muon_mu = 0.95f;
  int ns_steps = 5;
  std::vector<MuonMat> mmats;
  void* ns = nullptr;
  MuonMat* mmats_dev = nullptr;
  int32_t* mchunk_mat_dev = nullptr;
  double* mpart_dev = nullptr;
  float* mscale_dev = nullptr;   // per matrix: 1 / |U|_F (bf16 mode)
  int* mdone_dev = nullptr;      // per matrix: momentum chunks done (bf16 mode)
  int n_muon_chunks = 0;
  std::pair<int, int> ns_simt_rng[5] = {};  // CUDA-core Newton-Schulz tiles (fp32 mode)

  // Periodic feature embeddings (pack_create_emb; App. "Feature Embeddings"):
  // member i's first layer reads E_i [B_cap, in0_pad[i] + 16] (bf16 / fp32,
  // column in0_pad[i] = 1) in the `ex` arena at e_off[i], E_i[b, j d + k] =
  // alpha_jk [x_bj, cos(w_j x_bj + b_j)]_k + beta_jk; the first layer's
  // input gradient dE_i [B_cap, in0_pad[i]] lives in the dz arena at
  // de_off[i]; the embedding parameters [w, b, alpha, beta]
  // (d_in (4 d_emb - 2) values) follow the member's head in its run at
  // emb_off[i].  Without embeddings in0 = d_in and in0_pad = d_in_pad.
  bool emb = false;
  std::vector<int32_t> d_emb, in0, in0_pad;
  std::vector<int64_t> e_off, de_off, emb_off, n_emb;
  int64_t ex_elems = 0;
  void* ex = nullptr;
  int emb_cols_max = 0;     // max in0 over members (grid of the embedding kernels)
  EmbMember* embm_dev = nullptr;
  // the prediction arena's embedding matrices (bf16 prediction plan)
  void* p_ex = nullptr;
  std::vector<int64_t> p_e_off;
  EmbMember* embm_p_dev = nullptr;

  // Stacked batches (Sec. 3.6: a batch per member), built on first use:
  // xbs holds member i's gathered batch at i * xb_elems ([B_cap, ldx] each,
  // its column d_in_pad = 1), and tcs is the tensor-core plan whose layer-0
  // tiles read member i's matrix.
  void* xbs = nullptr;
  TcPlan tcs;
  bool s_stale = true;      // active set changed since tcs was built

  // Dropout keep words of one step (bf16 mode): per (member, layer) with
  // p > 0, [ceil(w / 32), B_cap] words from mask_off[i][l] (-1: none).  The
  // AdamW pass of a training step fills them for step + 1; masks_for is the
  // step they hold (-1: none), and a step whose masks are not there runs
  // k_masks first.
  std::vector<std::array<int64_t, kMaxDepth>> mask_off;
  int64_t mask_words = 0;
  uint32_t* masks = nullptr;
  MaskSeg* mseg_dev = nullptr;
  int32_t* mchunk_dev = nullptr;
  int n_mchunks = 0;
  int64_t masks_for = -1;

  // schedule (active members)
  int n_active = 0, n_chunks = 0, n_head_jobs = 0;
  std::vector<std::pair<int, int>> fwd_rng, bwd_rng;  // CUDA-core tile ranges per depth index
  int cap_chunks = 0, cap_probs = 0, cap_tiles = 0, cap_head = 0;

  // CUDA graphs of the training step, one per (B, update, weight copy); the
  // per-call arguments travel through dyn_dev, filled from a pinned ring
  struct GraphEntry {
    int B, update, wcur, stacked;
    cudaGraphExec_t exec;
    int64_t n_launch;
  };
  std::vector<GraphEntry> graphs;
  bool use_graphs = true;
  cudaStream_t st_cap = nullptr;  // graphs are captured here (the legacy stream cannot capture)
  StepDyn* dyn_dev = nullptr;
  static constexpr int kRing = 16;
  StepDyn* dyn_host = nullptr;    // pinned [kRing]
  cudaEvent_t dyn_ev[kRing] = {};
  bool dyn_used[kRing] = {};
  int dyn_next = 0;

  int last_B = 0;
  int64_t launches = 0;
  size_t dev_bytes = 0;
  std::vector<void*> allocs;
  std::string err;
  bool profiling = false;
  PhaseEvents prof;
};

namespace {

tp_status fail(tabpack* h, tp_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  if (h) h->err = buf;
  else g_thread_error = buf;
  return s;
}

#define TP_CUDA(h, call)                                                                   \
  do {                                                                                     \
    cudaError_t e_ = (call);                                                               \
    if (e_ != cudaSuccess)                                                                 \
      return fail((h), e_ == cudaErrorMemoryAllocation ? TP_ENOMEM : TP_ECUDA, "%s: %s (%s:%d)", \
                  #call, cudaGetErrorString(e_), __FILE__, __LINE__);                      \
  } while (0)

#define TP_LAUNCHED(h)                                                                     \
  do {                                                                                     \
    cudaError_t e_ = cudaGetLastError();                                                   \
    if (e_ != cudaSuccess)                                                                 \
      return fail((h), TP_ECUDA, "kernel launch: %s (%s:%d)", cudaGetErrorString(e_), __FILE__, __LINE__); \
  } while (0)

#define TP_TRY(expr)                 \
  do {                               \
    tp_status s_ = (expr);           \
    if (s_ != TP_OK) return s_;      \
  } while (0)

template <typename P>
tp_status dalloc(tabpack* h, P** ptr, size_t bytes) {
  void* p = nullptr;
  if (bytes == 0) bytes = 16;
  cudaError_t e = cudaMalloc(&p, bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(h, TP_ENOMEM, "cudaMalloc(%zu bytes): %s", bytes, cudaGetErrorString(e));
  }
  h->allocs.push_back(p);
  h->dev_bytes += bytes;
  *ptr = (P*)p;
  return TP_OK;
}

void prof_begin(tabpack* h, int phase, int* slot) {
  *slot = -1;
  if (!h->profiling) return;
  auto& P = h->prof;
  int idx = (int)P.pending.size() * 2;
  while ((int)P.pool.size() < idx + 2) {
    cudaEvent_t e;
    cudaEventCreate(&e);
    P.pool.push_back(e);
  }
  cudaEventRecord(P.pool[idx], h->st);
  P.pending.push_back({phase, idx});
  *slot = idx;
}

void prof_end(tabpack* h, int slot, int n_launch, int phase) {
  if (slot < 0) return;
  cudaEventRecord(h->prof.pool[slot + 1], h->st);
  h->prof.launches[phase] += n_launch;
}

void prof_flush(tabpack* h) {
  auto& P = h->prof;
  if (P.pending.empty()) return;
  cudaStreamSynchronize(h->st);
  for (auto& pr : P.pending) {
    float ms = 0.f;
    cudaEventElapsedTime(&ms, P.pool[pr.second], P.pool[pr.second + 1]);
    P.ms[pr.first] += ms;
  }
  P.pending.clear();
}

int ldh_of(const tabpack* h, int i) { return h->width[i] + kOnesCols; }

void drop_graphs(tabpack* h);
void free_predict(tabpack* h);

// ------------------------------------------------------------------ layout
// Column sums of dZ save a weight-gradient column tile of every layer whose
// input width is a multiple of 256, but add work to the head and to the
// dgrad epilogues, which lie on the backward launch's dependency chain.
// They pay where the backward is bound by tensor throughput, taken as an
// ideal backward tensor time (nominal 2 PFLOP/s) of 300 us or more.
bool auto_bias_colsums(const tabpack* h) {
  if (!h->bf16) return false;
  double flops = 0.0;
  for (int i = 0; i < h->cfg.m; ++i) {
    const double w = h->width[i], L = h->depth[i];
    flops += 2.0 * h->B_cap * (w * h->in0_pad[i] + 2.0 * (L - 1.0) * w * w);
  }
  return flops / 2.0e15 >= 300e-6;
}

tp_status build_layout(tabpack* h) {
  const auto& c = h->cfg;
  const int m = c.m;
  h->d_in_pad = (int)round_up(c.d_in, 8);
  h->ldx = h->d_in_pad + kOnesCols;
  h->in0.assign(m, c.d_in);
  h->in0_pad.assign(m, h->d_in_pad);
  h->e_off.assign(m, 0);
  h->de_off.assign(m, 0);
  h->emb_off.assign(m, 0);
  h->n_emb.assign(m, 0);
  if (h->emb)
    for (int i = 0; i < m; ++i) {
      h->in0[i] = c.d_in * h->d_emb[i];
      h->in0_pad[i] = (int)round_up(h->in0[i], 8);
      h->n_emb[i] = (int64_t)c.d_in * (4 * h->d_emb[i] - 2);
      h->emb_cols_max = std::max(h->emb_cols_max, h->in0_pad[i]);
    }
  h->B_cap = (int)round_up(c.max_batch, kRowTile);
  h->n_blk_cap = h->B_cap / kHeadRows;
  h->bias_colsums = auto_bias_colsums(h);
  h->W_off.resize(m);
  h->b_off.resize(m);
  h->act_off.resize(m);
  h->dz_off.resize(m);
  h->mem.resize(m);
  h->part_off.resize(m);
  h->part_stride.resize(m);
  int64_t off = 0, aoff = 0, zoff = 0, hoff = 0;
  h->Lmax = 0;
  for (int i = 0; i < m; ++i) {
    const int L = h->depth[i], w = h->width[i];
    h->Lmax = std::max(h->Lmax, L);
    for (int l = 0; l <= L; ++l) {
      const int in = l == 0 ? h->in0[i] : w, in_pad = l == 0 ? h->in0_pad[i] : w;
      const int out = l == L ? c.d_out : w;
      off = round_up(off, kSegAlign);
      h->W_off[i][l] = off;
      h->segs.push_back(Segment{off, i, l, out, in, in_pad, 0, in, out * in});
      off += (int64_t)out * in_pad;
      off = round_up(off, kSegAlign);
      h->b_off[i][l] = off;
      h->segs.push_back(Segment{off, i, l, out, 1, 1, 1, in, out * in});
      off += out;
    }
    if (h->emb) {  // the embedding parameters, stepped by AdamW like biases
      off = round_up(off, kSegAlign);
      h->emb_off[i] = off;
      h->segs.push_back(Segment{off, i, L + 1, (int32_t)h->n_emb[i], 1, 1, 1, c.d_in, 0});
      off += h->n_emb[i];
    }
    for (int l = 0; l < L; ++l) {
      h->act_off[i][l] = aoff;
      aoff += round_up((int64_t)h->B_cap * ldh_of(h, i), 128);
      h->dz_off[i][l] = zoff;
      zoff += round_up((int64_t)h->B_cap * w, 128);
    }
    if (h->emb) {
      h->de_off[i] = zoff;
      zoff += round_up((int64_t)h->B_cap * h->in0_pad[i], 128);
      h->e_off[i] = h->ex_elems;
      h->ex_elems += round_up((int64_t)h->B_cap * (h->in0_pad[i] + kOnesCols), 128);
    }
    const float p = h->dropout[i];
    double T = std::floor((double)p * 4294967296.0);
    if (T > 4294967295.0) T = 4294967295.0;
    MemberDev md;
    md.L = L;
    md.w = w;
    md.p = p;
    md.scale = 1.f / (1.f - p);
    md.lr = h->lr[i];
    md.wd = h->wd[i];
    md.drop_T = (uint32_t)T;
    md._pad = 0;
    h->mem[i] = md;
    h->part_stride[i] = round_up((int64_t)c.d_out * (w + 1), 32);
    h->part_off[i] = hoff;
    hoff += h->part_stride[i] * h->n_blk_cap;
  }
  h->n_params = round_up(off, kSegAlign);
  h->mask_off.assign(m, {});
  h->mask_words = 0;
  for (int i = 0; i < m; ++i)
    for (int l = 0; l < kMaxDepth; ++l) {
      h->mask_off[i][l] = -1;
      if (!h->bf16 || l >= h->depth[i] || h->mem[i].drop_T == 0) continue;
      h->mask_off[i][l] = h->mask_words;
      h->mask_words += ceil_div(h->width[i], 32) * (int64_t)h->B_cap;
    }
  if (h->mask_words >= (int64_t)1 << 31) return fail(h, TP_EINVAL, "dropout mask arena too large");
  h->act_elems = std::max<int64_t>(aoff, 128);
  h->dz_elems = std::max<int64_t>(zoff, 128);
  h->xb_elems = (int64_t)h->B_cap * h->ldx;
  h->head_part_elems = std::max<int64_t>(hoff, 32);
  return TP_OK;
}

// --------------------------------------------------------------- schedule
// Rebuilt whenever the active set changes: per depth index the forward and
// backward GEMM work of the active members, the head and AdamW work lists.
tp_status build_schedule(tabpack* h) {
  const auto& c = h->cfg;
  const int m = c.m;
  std::vector<int32_t> ids;
  for (int i = 0; i < m; ++i)
    if (h->active[i]) ids.push_back(i);
  h->n_active = (int)ids.size();

  // CUDA-core products (fp32 mode)
  std::vector<GemmProblem> probs;
  std::vector<GemmTile> tiles;
  h->fwd_rng.assign(h->Lmax, {0, 0});
  h->bwd_rng.assign(h->Lmax, {0, 0});
  if (!h->bf16) {
    auto add_tiles = [&](int prob, int M_rows, int N) {
      for (int m0 = 0; m0 < M_rows; m0 += 64)
        for (int n0 = 0; n0 < N; n0 += 64) tiles.push_back(GemmTile{prob, m0, n0, std::min(64, N - n0)});
    };
    for (int l = 0; l < h->Lmax; ++l) {
      const int base = (int)tiles.size();
      for (int i : ids) {
        if (h->depth[i] <= l) continue;
        const int w = h->width[i];
        GemmProblem P{};
        P.kind = kFwd; P.member = i; P.layer = l;
        P.M = 0; P.N = w; P.K = l == 0 ? h->in0_pad[i] : w;
        P.a_src = l == 0 ? (h->emb ? kSrcEmb : kSrcXb) : kSrcAct;
        P.a_off = l == 0 ? (h->emb ? h->e_off[i] : 0) : h->act_off[i][l - 1];
        P.lda = l == 0 ? (h->emb ? h->in0_pad[i] + kOnesCols : h->ldx) : ldh_of(h, i);
        P.b_src = kSrcWq; P.b_off = h->W_off[i][l]; P.ldb = P.K;
        P.c_off = h->act_off[i][l]; P.ldc = ldh_of(h, i);
        P.aux_off = h->b_off[i][l];
        probs.push_back(P);
        add_tiles((int)probs.size() - 1, h->B_cap, w);
      }
      h->fwd_rng[l] = {base, (int)tiles.size() - base};
    }
    for (int l = h->Lmax - 1; l >= 0; --l) {
      const int base = (int)tiles.size();
      for (int i : ids) {
        if (h->depth[i] <= l) continue;
        const int w = h->width[i];
        const int in_pad = l == 0 ? h->in0_pad[i] : w;
        if (l == 0 && h->emb) {   // the input gradient of the first layer, for the embeddings
          GemmProblem P{};
          P.kind = kDgrad; P.member = i; P.layer = 0;
          P.M = 0; P.N = in_pad; P.K = w;
          P.a_src = kSrcDz; P.a_off = h->dz_off[i][0]; P.lda = w;
          P.b_src = kSrcWq; P.b_off = h->W_off[i][0]; P.ldb = in_pad;
          P.c_off = h->de_off[i]; P.ldc = in_pad;
          P.aux_off = -1;
          probs.push_back(P);
          add_tiles((int)probs.size() - 1, h->B_cap, in_pad);
        }
        if (l > 0) {
          GemmProblem P{};
          P.kind = kDgrad; P.member = i; P.layer = l;
          P.M = 0; P.N = w; P.K = w;
          P.a_src = kSrcDz; P.a_off = h->dz_off[i][l]; P.lda = w;
          P.b_src = kSrcWq; P.b_off = h->W_off[i][l]; P.ldb = w;
          P.c_off = h->dz_off[i][l - 1]; P.ldc = w;
          P.aux_off = h->act_off[i][l - 1]; P.ld_aux = ldh_of(h, i);
          probs.push_back(P);
          add_tiles((int)probs.size() - 1, h->B_cap, w);
        }
        GemmProblem Q{};
        Q.kind = kWgrad; Q.member = i; Q.layer = l;
        Q.M = w; Q.N = in_pad + 1; Q.K = 0;  // the last column is the bias gradient
        Q.a_src = kSrcDz; Q.a_off = h->dz_off[i][l]; Q.lda = w;
        Q.b_src = l == 0 ? (h->emb ? kSrcEmb : kSrcXb) : kSrcAct;
        Q.b_off = l == 0 ? (h->emb ? h->e_off[i] : 0) : h->act_off[i][l - 1];
        Q.ldb = l == 0 ? (h->emb ? h->in0_pad[i] + kOnesCols : h->ldx) : ldh_of(h, i);
        Q.c_off = h->W_off[i][l]; Q.ldc = in_pad;
        Q.aux_off = h->b_off[i][l];
        probs.push_back(Q);
        add_tiles((int)probs.size() - 1, w, in_pad + 1);
      }
      h->bwd_rng[l] = {base, (int)tiles.size() - base};
    }
    for (auto& r : h->ns_simt_rng) r = {(int)tiles.size(), 0};
    if (h->muon)
      for (int which = 0; which < 5; ++which) {
        const int base = (int)tiles.size();
        const int p = which == 0 || which == 3 ? 0 : 1;
        for (const MuonMat& mt : h->mmats) {
          if (!h->active[mt.member]) continue;
          GemmProblem P{};
          P.member = mt.member; P.layer = mt.layer;
          P.M = mt.r;
          P.a_src = kSrcNs; P.b_src = kSrcNs;
          if (which < 2) {
            P.kind = kNsGram; P.N = mt.r; P.K = mt.c;
            P.a_off = P.b_off = mt.x_off[p]; P.lda = P.ldb = mt.c;
            P.c_off = mt.a_off; P.ldc = mt.r;
          } else if (which == 2) {
            P.kind = kNsPoly; P.N = mt.r; P.K = mt.r;
            P.a_off = P.b_off = mt.a_off; P.lda = P.ldb = mt.r;
            P.c_off = mt.bm_off; P.ldc = mt.r;
            P.aux_off = mt.a_off; P.ld_aux = mt.r;
          } else {
            P.kind = kNsApply; P.N = mt.c; P.K = mt.r;
            P.a_off = mt.bm_off; P.lda = mt.r;
            P.b_off = mt.x_off[p]; P.ldb = mt.c;
            P.c_off = mt.x_off[1 - p]; P.ldc = mt.c;
            P.aux_off = mt.x_off[p]; P.ld_aux = mt.c;
          }
          probs.push_back(P);
          add_tiles((int)probs.size() - 1, mt.r, P.N);
        }
        h->ns_simt_rng[which] = {base, (int)tiles.size() - base};
      }
  }

  std::vector<HeadJob> hj;
  std::vector<HeadReduceJob> hr(m);
  for (int i = 0; i < m; ++i) {
    const int L = h->depth[i];
    hr[i] = HeadReduceJob{i, h->n_blk_cap, h->part_off[i], h->W_off[i][L], h->b_off[i][L], h->width[i], 0};
  }
  for (int i : ids) {
    const int L = h->depth[i];
    for (int b = 0; b < h->n_blk_cap; ++b) {
      HeadJob j{};
      j.member = i;
      j.blk = b;
      j.h_ld = ldh_of(h, i);
      j.split = head_split(h->width[i], h->cfg.d_out);
      j.colsum = h->bias_colsums && bias_from_colsums(L == 1 ? h->in0_pad[i] : h->width[i]) ? 1 : 0;
      j.h_off = h->act_off[i][L - 1];
      j.dz_off = h->dz_off[i][L - 1];
      j.w_off = h->W_off[i][L];
      j.b_off = h->b_off[i][L];
      j.part_off = h->part_off[i] + (int64_t)b * h->part_stride[i];
      hj.push_back(j);
    }
  }
  // widest members' blocks first (a block's cost grows with the width), so
  // that the blocks left for the last wave are the cheapest
  std::stable_sort(hj.begin(), hj.end(),
                   [h](const HeadJob& x, const HeadJob& y) { return h->width[x.member] > h->width[y.member]; });
  // element-wise chunks of the active members (init, fp32-mode AdamW)
  std::vector<Chunk> ch;
  for (int s = 0; s < (int)h->segs.size(); ++s) {
    const Segment& S = h->segs[s];
    if (!h->active[S.member]) continue;
    if (h->muon && !S.is_bias && S.layer < h->depth[S.member]) continue;  // Muon's
    const int64_t len = S.is_bias ? S.rows : (int64_t)S.rows * S.cols_pad;
    for (int64_t o = 0; o < len; o += 4096)
      ch.push_back(Chunk{S.off + o, (int32_t)std::min<int64_t>(4096, len - o), s});
  }

  // capacities are fixed at create (all members active)
  if (h->head_jobs_dev == nullptr) {
    h->cap_probs = (int)probs.size() + 1;
    h->cap_tiles = (int)tiles.size() + 1;
    h->cap_head = (int)hj.size() + 1;
    h->cap_chunks = (int)ch.size() + 1;
    TP_TRY(dalloc(h, &h->probs_dev, sizeof(GemmProblem) * h->cap_probs));
    TP_TRY(dalloc(h, &h->tiles_dev, sizeof(GemmTile) * h->cap_tiles));
    TP_TRY(dalloc(h, &h->head_jobs_dev, sizeof(HeadJob) * h->cap_head));
    TP_TRY(dalloc(h, &h->hred_dev, sizeof(HeadReduceJob) * m));
    TP_TRY(dalloc(h, &h->chunks_dev, sizeof(Chunk) * h->cap_chunks));
    TP_TRY(dalloc(h, &h->active_ids_dev, sizeof(int32_t) * m));
  }
  // Muon adds Newton-Schulz problems: grow those two lists once
  if ((int)probs.size() > h->cap_probs) {
    h->cap_probs = (int)probs.size() + 1;
    TP_TRY(dalloc(h, &h->probs_dev, sizeof(GemmProblem) * h->cap_probs));
  }
  if ((int)tiles.size() > h->cap_tiles) {
    h->cap_tiles = (int)tiles.size() + 1;
    TP_TRY(dalloc(h, &h->tiles_dev, sizeof(GemmTile) * h->cap_tiles));
  }
  if ((int)probs.size() > h->cap_probs || (int)tiles.size() > h->cap_tiles || (int)hj.size() > h->cap_head ||
      (int)ch.size() > h->cap_chunks)
    return fail(h, TP_ESTATE, "schedule grew beyond its capacity");
  TP_CUDA(h, cudaStreamSynchronize(h->st));
  drop_graphs(h);  // captured launches carry the old work-list sizes
  if (!probs.empty()) TP_CUDA(h, cudaMemcpy(h->probs_dev, probs.data(), sizeof(GemmProblem) * probs.size(), cudaMemcpyHostToDevice));
  if (!tiles.empty()) TP_CUDA(h, cudaMemcpy(h->tiles_dev, tiles.data(), sizeof(GemmTile) * tiles.size(), cudaMemcpyHostToDevice));
  if (!hj.empty()) TP_CUDA(h, cudaMemcpy(h->head_jobs_dev, hj.data(), sizeof(HeadJob) * hj.size(), cudaMemcpyHostToDevice));
  TP_CUDA(h, cudaMemcpy(h->hred_dev, hr.data(), sizeof(HeadReduceJob) * m, cudaMemcpyHostToDevice));
  if (!ch.empty()) TP_CUDA(h, cudaMemcpy(h->chunks_dev, ch.data(), sizeof(Chunk) * ch.size(), cudaMemcpyHostToDevice));
  if (!ids.empty()) TP_CUDA(h, cudaMemcpy(h->active_ids_dev, ids.data(), sizeof(int32_t) * ids.size(), cudaMemcpyHostToDevice));
  TP_CUDA(h, cudaMemcpy(h->active_dev, h->active.data(), m, cudaMemcpyHostToDevice));
  // dropout mask segments of the active members
  h->n_mchunks = 0;
  h->masks_for = -1;
  if (h->mask_words > 0) {
    std::vector<MaskSeg> ms;
    std::vector<int32_t> mc;
    for (int i : ids)
      for (int l = 0; l < h->depth[i]; ++l) {
        if (h->mask_off[i][l] < 0) continue;
        const int nck = (int)ceil_div(h->width[i], 32);
        ms.push_back(MaskSeg{h->mask_off[i][l], i, l, h->mem[i].drop_T, (int32_t)mc.size()});
        for (int k = 0; k < nck; ++k) mc.push_back((int32_t)ms.size() - 1);
      }
    if (!ms.empty()) {
      TP_CUDA(h, cudaMemcpy(h->mseg_dev, ms.data(), sizeof(MaskSeg) * ms.size(), cudaMemcpyHostToDevice));
      TP_CUDA(h, cudaMemcpy(h->mchunk_dev, mc.data(), sizeof(int32_t) * mc.size(), cudaMemcpyHostToDevice));
    }
    h->n_mchunks = (int)mc.size();
  }
  // Muon: flat chunk list of the active members' matrices
  h->n_muon_chunks = 0;
  if (h->muon) {
    std::vector<int32_t> cm;
    for (size_t j = 0; j < h->mmats.size(); ++j) {
      MuonMat& mt = h->mmats[j];
      mt.chunk0 = (int32_t)cm.size();
      mt.n_chunks = h->active[mt.member] ? (int32_t)muon_chunks(mt) : 0;
      for (int k = 0; k < mt.n_chunks; ++k) cm.push_back((int32_t)j);
    }
    TP_CUDA(h, cudaMemcpy(h->mmats_dev, h->mmats.data(), sizeof(MuonMat) * h->mmats.size(), cudaMemcpyHostToDevice));
    if (!cm.empty())
      TP_CUDA(h, cudaMemcpy(h->mchunk_mat_dev, cm.data(), sizeof(int32_t) * cm.size(), cudaMemcpyHostToDevice));
    h->n_muon_chunks = (int)cm.size();
  }
  h->n_head_jobs = (int)hj.size();
  h->n_chunks = (int)ch.size();
  h->p_stale = true;
  h->s_stale = true;
  if (h->bf16) {
    TcLayout lay;
    lay.depth = &h->depth;
    lay.width = &h->width;
    lay.active = &h->active;
    lay.W_off = &h->W_off;
    lay.b_off = &h->b_off;
    lay.act_off = &h->act_off;
    lay.dz_off = &h->dz_off;
    lay.m = m;
    lay.d_in_pad = h->d_in_pad;
    lay.ldx = h->ldx;
    lay.B_cap = h->B_cap;
    lay.wq[0] = h->wq[0];
    lay.wq[1] = h->wq[1];
    lay.xb = h->xb;
    lay.act = h->act;
    lay.dz = h->dz;
    lay.bias_colsums = h->bias_colsums;
    lay.mask_off = h->mask_words > 0 ? &h->mask_off : nullptr;
    lay.muon = h->muon ? &h->mmats : nullptr;
    lay.ns = h->ns;
    lay.ns_steps = h->ns_steps;
    lay.in0_pad = &h->in0_pad;
    if (h->emb) {
      lay.xb = h->ex;
      lay.x0_off = &h->e_off;
      lay.de_off = &h->de_off;
    }
    TP_TRY(tc_build_plan(h->tc, lay, h->err));
  }
  return TP_OK;
}

// Column in_pad of xb and column w of every act matrix := 1 (all rows).
template <typename T>
tp_status fill_ones(tabpack* h) {
  std::vector<OnesJob> jobs;
  jobs.push_back(OnesJob{0, h->ldx, h->d_in_pad, h->B_cap, 0});
  if (h->emb)
    for (int i = 0; i < h->cfg.m; ++i) jobs.push_back(OnesJob{h->e_off[i], h->in0_pad[i] + kOnesCols, h->in0_pad[i], h->B_cap, 2});
  for (int i = 0; i < h->cfg.m; ++i)
    for (int l = 0; l < h->depth[i]; ++l)
      jobs.push_back(OnesJob{h->act_off[i][l], ldh_of(h, i), h->width[i], h->B_cap, 1});
  OnesJob* d = nullptr;
  TP_CUDA(h, cudaMalloc(&d, sizeof(OnesJob) * jobs.size()));
  cudaError_t e = cudaMemcpy(d, jobs.data(), sizeof(OnesJob) * jobs.size(), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) {
    launch_fill_ones<T>(h->st, d, (int)jobs.size(), (T*)h->xb, (T*)h->act, (T*)h->ex);
    h->launches++;
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
  cudaFree(d);
  if (e != cudaSuccess) return fail(h, TP_ECUDA, "fill ones: %s", cudaGetErrorString(e));
  return TP_OK;
}

tp_status alloc_all(tabpack* h) {
  const int m = h->cfg.m;
  h->elem = h->bf16 ? 2 : 4;
  TP_TRY(dalloc(h, &h->params, sizeof(float) * h->n_params));
  TP_TRY(dalloc(h, &h->grads, sizeof(float) * h->n_params));
  TP_TRY(dalloc(h, &h->adam_m, sizeof(float) * h->n_params));
  TP_TRY(dalloc(h, &h->adam_v, sizeof(float) * h->n_params));
  if (h->bf16) {
    TP_TRY(dalloc(h, &h->wq[0], sizeof(__nv_bfloat16) * h->n_params));
    TP_TRY(dalloc(h, &h->wq[1], sizeof(__nv_bfloat16) * h->n_params));
  }
  TP_TRY(dalloc(h, &h->xb, h->elem * h->xb_elems));
  TP_TRY(dalloc(h, &h->act, h->elem * h->act_elems));
  TP_TRY(dalloc(h, &h->dz, h->elem * h->dz_elems));
  TP_TRY(dalloc(h, &h->logits, sizeof(float) * (size_t)m * h->B_cap * h->cfg.d_out));
  TP_TRY(dalloc(h, &h->head_part, sizeof(float) * h->head_part_elems));
  if (h->bf16) TP_TRY(dalloc(h, &h->dbp, sizeof(float) * (size_t)(h->dz_elems / 32 + 32)));
  TP_TRY(dalloc(h, &h->loss_part, sizeof(float) * (size_t)m * h->n_blk_cap));
  TP_TRY(dalloc(h, &h->loss_last, sizeof(float) * m));
  TP_TRY(dalloc(h, &h->t_dev, sizeof(int32_t) * m));
  TP_TRY(dalloc(h, &h->bias_corr, sizeof(float2) * m));
  TP_TRY(dalloc(h, &h->active_dev, m));
  TP_TRY(dalloc(h, &h->mem_dev, sizeof(MemberDev) * m));
  TP_TRY(dalloc(h, &h->segs_dev, sizeof(Segment) * h->segs.size()));
  TP_TRY(dalloc(h, &h->part_stride_dev, sizeof(int64_t) * m));
  TP_TRY(dalloc(h, &h->dyn_dev, sizeof(StepDyn)));
  if (h->mask_words > 0) {
    int64_t n_mc = 0;
    for (int i = 0; i < m; ++i)
      if (h->mask_off[i][0] >= 0) n_mc += h->depth[i] * ceil_div(h->width[i], 32);
    TP_TRY(dalloc(h, &h->masks, sizeof(uint32_t) * h->mask_words));
    TP_TRY(dalloc(h, &h->mseg_dev, sizeof(MaskSeg) * (size_t)m * kMaxDepth));
    TP_TRY(dalloc(h, &h->mchunk_dev, sizeof(int32_t) * n_mc));
  }
  TP_CUDA(h, cudaHostAlloc((void**)&h->dyn_host, sizeof(StepDyn) * tabpack::kRing, cudaHostAllocDefault));
  for (int k = 0; k < tabpack::kRing; ++k) TP_CUDA(h, cudaEventCreateWithFlags(&h->dyn_ev[k], cudaEventDisableTiming));
  TP_CUDA(h, cudaStreamCreateWithFlags(&h->st_cap, cudaStreamNonBlocking));
  TP_CUDA(h, cudaMemset(h->t_dev, 0, sizeof(int32_t) * m));
  TP_CUDA(h, cudaMemset(h->bias_corr, 0, sizeof(float2) * m));
  TP_CUDA(h, cudaMemset(h->xb, 0, h->elem * h->xb_elems));
  if (h->emb) {
    TP_CUDA(h, cudaMalloc(&h->ex, h->elem * (size_t)h->ex_elems));
    TP_CUDA(h, cudaMemset(h->ex, 0, h->elem * (size_t)h->ex_elems));
  }
  TP_CUDA(h, cudaMemset(h->act, 0, h->elem * h->act_elems));
  TP_CUDA(h, cudaMemset(h->dz, 0, h->elem * h->dz_elems));
  TP_CUDA(h, cudaMemset(h->logits, 0, sizeof(float) * (size_t)m * h->B_cap * h->cfg.d_out));
  TP_CUDA(h, cudaMemcpy(h->mem_dev, h->mem.data(), sizeof(MemberDev) * m, cudaMemcpyHostToDevice));
  TP_CUDA(h, cudaMemcpy(h->segs_dev, h->segs.data(), sizeof(Segment) * h->segs.size(), cudaMemcpyHostToDevice));
  TP_CUDA(h, cudaMemcpy(h->part_stride_dev, h->part_stride.data(), sizeof(int64_t) * m, cudaMemcpyHostToDevice));
  return TP_OK;
}

void free_predict(tabpack* h) {
  tc_free_plan(h->tcp);
  for (void* p : {h->p_xb, h->p_act, (void*)h->p_head_dev, h->p_ex, (void*)h->embm_p_dev})
    if (p) cudaFree(p);
  h->p_xb = h->p_act = h->p_ex = nullptr;
  h->p_head_dev = nullptr;
  h->embm_p_dev = nullptr;
  h->P_cap = 0;
  h->n_p_head = 0;
  h->p_stale = true;
}

void drop_graphs(tabpack* h) {
  for (auto& ge : h->graphs) cudaGraphExecDestroy(ge.exec);
  h->graphs.clear();
}

void free_all(tabpack* h) {
  if (h->st) cudaStreamSynchronize(h->st);
  drop_graphs(h);
  if (h->st_cap) cudaStreamDestroy(h->st_cap);
  h->st_cap = nullptr;
  for (auto& e : h->dyn_ev)
    if (e) cudaEventDestroy(e);
  if (h->dyn_host) cudaFreeHost(h->dyn_host);
  h->dyn_host = nullptr;
  tc_free_plan(h->tc);
  free_predict(h);
  tc_free_plan(h->tcs);
  if (h->xbs) cudaFree(h->xbs);
  h->xbs = nullptr;
  if (h->ex) cudaFree(h->ex);
  h->ex = nullptr;
  if (h->embm_dev) cudaFree(h->embm_dev);
  h->embm_dev = nullptr;
  for (void* p : {h->ns, (void*)h->mmats_dev, (void*)h->mchunk_mat_dev, (void*)h->mpart_dev, (void*)h->mscale_dev,
                  (void*)h->mdone_dev})
    if (p) cudaFree(p);
  h->ns = nullptr;
  h->mmats_dev = nullptr;
  h->mchunk_mat_dev = nullptr;
  h->mpart_dev = nullptr;
  h->mscale_dev = nullptr;
  h->mdone_dev = nullptr;
  for (void* p : h->allocs) cudaFree(p);
  h->allocs.clear();
  for (auto e : h->prof.pool) cudaEventDestroy(e);
  h->prof.pool.clear();
}

template <typename T>
GemmArgs<T> gemm_args(tabpack* h, int B, int B_pad, uint32_t step, int train, bool stacked = false) {
  GemmArgs<T> g;
  g.probs = h->probs_dev;
  g.tiles = h->tiles_dev;
  g.xb = (const T*)(stacked ? h->xbs : h->xb);
  g.xb_stride = stacked ? h->xb_elems : 0;
  g.act = (T*)h->act;
  g.dz = (T*)h->dz;
  g.wq = (const T*)h->params;  // the CUDA-core path runs in fp32 mode only
  g.params = h->params;
  g.grads = h->grads;
  g.mem = h->mem_dev;
  g.B = B;
  g.B_pad = B_pad;
  g.step = step;
  g.train = train;
  g.seed = h->cfg.seed;
  g.dyn = nullptr;
  g.ns = (T*)h->ns;
  g.ex = (const T*)h->ex;
  return g;
}

AdamDev adam_dev(tabpack* h, __nv_bfloat16* wq_out) {
  AdamDev a;
  a.params = h->params;
  a.m = h->adam_m;
  a.v = h->adam_v;
  a.wq_out = wq_out;
  a.bias_corr = h->bias_corr;
  a.mem = h->mem_dev;
  a.beta1 = h->cfg.beta1;
  a.beta2 = h->cfg.beta2;
  a.eps = h->cfg.eps;
  a.wd_on_bias = h->cfg.wd_on_bias;
  return a;
}

template <typename T>
tp_status run_forward(tabpack* h, int B, int B_pad, uint32_t step, const StepDyn* dyn, int train,
                      bool stacked = false) {
  if (h->bf16) {  // every layer in one launch
    int slot;
    prof_begin(h, train ? TP_PH_FWD : TP_PH_PREDICT, &slot);
    TP_TRY(tc_run_fwd(stacked ? h->tcs : h->tc, h->st, B, B_pad, h->wcur, train, h->masks, h->B_cap, h->params, h->mem_dev, h->act,
                      h->err));
    TP_LAUNCHED(h);
    h->launches++;
    prof_end(h, slot, 1, train ? TP_PH_FWD : TP_PH_PREDICT);
    return TP_OK;
  }
  for (int l = 0; l < h->Lmax; ++l) {  // CUDA-core path: one launch per depth
    int slot;
    prof_begin(h, train ? TP_PH_FWD : TP_PH_PREDICT, &slot);
    auto g = gemm_args<T>(h, B, B_pad, step, train, stacked);
    g.dyn = dyn;
    launch_gemm_simt<T>(h->st, g, h->fwd_rng[l].first, h->fwd_rng[l].second);
    TP_LAUNCHED(h);
    h->launches++;
    prof_end(h, slot, 1, train ? TP_PH_FWD : TP_PH_PREDICT);
  }
  return TP_OK;
}

template <typename T>
EmbArgs<T> emb_args(tabpack* h, const float* X, const int32_t* idx, const StepDyn* dyn, bool stacked, int B,
                    int B_pad) {
  EmbArgs<T> a;
  a.em = h->embm_dev;
  a.active_ids = h->active_ids_dev;
  a.X = X;
  a.idx = idx;
  a.dyn = dyn;
  a.params = h->params;
  a.grads = h->grads;
  a.ex = (T*)h->ex;
  a.dz = (const T*)h->dz;
  a.idx_stride = stacked ? B : 0;
  a.B = B;
  a.B_pad = B_pad;
  a.d_in = h->cfg.d_in;
  return a;
}

// Filling the mask arena for a step (dyn non-NULL: dyn->step + step_add).
MaskGen mask_gen(tabpack* h, uint32_t step, const StepDyn* dyn, uint32_t step_add) {
  MaskGen mg{};
  mg.masks = h->masks;
  mg.segs = h->mseg_dev;
  mg.chunk_seg = h->mchunk_dev;
  mg.n_chunks = h->bf16 ? h->n_mchunks : 0;
  mg.rows = h->B_cap;
  mg.seed = h->cfg.seed;
  mg.step = step;
  mg.step_add = step_add;
  mg.dyn = dyn;
  return mg;
}

// One step on the pack's stream (enqueue only; the caller flips the weight
// copy for the next step):
//   gather -> forward (per depth) -> head + loss -> head reduce (+ head AdamW)
//   -> backward (per depth, deepest first; bias gradients from the ones
//   column; AdamW fused into the wgrad epilogue or) -> one AdamW pass.
// dyn non-NULL: X, idx, y, loss_out and step are read from it on the device.
template <typename T>
tp_status run_step(tabpack* h, const float* X, int64_t n_rows, const int32_t* idx, const void* y, int B,
                   uint32_t step, float* loss_out, bool update, const StepDyn* dyn, bool stacked) {
  // with embeddings every member has its own first-layer matrix already: the
  // main plan serves stacked batches too (the rows enter through idx)
  const bool st_x = stacked && !h->emb;
  TcPlan& plan = st_x ? h->tcs : h->tc;
  const int B_pad = (int)round_up(B, kRowTile);
  const bool fused = update && h->bf16 && h->fuse_adamw;
  __nv_bfloat16* wq_next = h->bf16 ? h->wq[h->wcur ^ 1] : nullptr;
  int slot;
  prof_begin(h, TP_PH_GATHER, &slot);
  launch_gather<T>(h->st, X, idx, dyn, B, B_pad, h->cfg.d_in, h->d_in_pad, h->ldx, (T*)(st_x ? h->xbs : h->xb),
                   update ? 1 : 0, h->t_dev, h->bias_corr, h->active_ids_dev, h->n_active, h->cfg.beta1, h->cfg.beta2,
                   plan.cnt_dev, plan.n_cnt, st_x ? 1 : 0, h->xb_elems);
  if (h->emb) {   // the members' first-layer inputs: their periodic embeddings
    launch_emb_fwd<T>(h->st, emb_args<T>(h, X, idx, dyn, stacked, B, B_pad), h->n_active, h->emb_cols_max);
    TP_LAUNCHED(h);
    h->launches++;
  }
  TP_LAUNCHED(h);
  h->launches++;
  prof_end(h, slot, h->emb ? 2 : 1, TP_PH_GATHER);
  TP_TRY(run_forward<T>(h, B, B_pad, step, dyn, 1, st_x));
  // head + loss
  prof_begin(h, TP_PH_HEAD, &slot);
  HeadArgs<T> hg;
  hg.jobs = h->head_jobs_dev;
  hg.mem = h->mem_dev;
  hg.act = (const T*)h->act;
  hg.dz = (T*)h->dz;
  hg.params = h->params;
  hg.head_part = h->head_part;
  hg.loss_part = h->loss_part;
  hg.logits = h->logits;
  hg.idx = idx;
  hg.y = y;
  hg.B = B;
  hg.B_pad = B_pad;
  hg.B_cap = h->B_cap;
  hg.d_out = h->cfg.d_out;
  hg.task = h->cfg.task;
  hg.n_blk_cap = h->n_blk_cap;
  hg.dyn = dyn;
  hg.idx_stride = stacked ? B : 0;
  hg.w_max = *std::max_element(h->width.begin(), h->width.end());
  hg.stage = h->bf16 ? 1 : 0;
  hg.err = h->bf16 && h->tc.enabled ? h->tc.err_dev : nullptr;
  hg.dbp = h->bf16 ? h->dbp : nullptr;   // the tensor-core backward sums them into the bias gradients
  launch_head<T>(h->st, hg, h->n_head_jobs);
  TP_LAUNCHED(h);
  h->launches++;
  // head gradients (sum of the per-block partials), losses, head AdamW
  HeadReduceArgs rg;
  rg.jobs = h->hred_dev;
  rg.active = h->active_dev;
  rg.part_stride = h->part_stride_dev;
  rg.head_part = h->head_part;
  rg.loss_part = h->loss_part;
  rg.grads = h->grads;
  rg.loss_out = loss_out;
  rg.loss_last = h->loss_last;
  rg.B = B;
  rg.B_pad = B_pad;
  rg.d_out = h->cfg.d_out;
  rg.n_blk_cap = h->n_blk_cap;
  rg.update = fused ? 1 : 0;
  rg.adam = adam_dev(h, wq_next);
  rg.dyn = dyn;
  int w_max = 0;
  for (int w : h->width) w_max = std::max(w_max, w);
  launch_head_reduce(h->st, rg, h->cfg.m, h->cfg.d_out * (w_max + 1));
  TP_LAUNCHED(h);
  h->launches++;
  prof_end(h, slot, 2, TP_PH_HEAD);
  // backward products: tensor cores, every layer in one launch; CUDA cores,
  // one launch per depth, deepest first
  const AdamDev ad = adam_dev(h, wq_next);
  if (h->bf16) {
    prof_begin(h, TP_PH_BWD, &slot);
    TP_TRY(tc_run_bwd(plan, h->st, B, B_pad, h->wcur, h->mem_dev, h->act, h->dz, h->grads, h->dbp, fused ? 1 : 0,
                      ad, h->err));
    TP_LAUNCHED(h);
    h->launches++;
    prof_end(h, slot, 1, TP_PH_BWD);
  } else {
    for (int l = h->Lmax - 1; l >= 0; --l) {
      prof_begin(h, TP_PH_BWD, &slot);
      auto g = gemm_args<T>(h, B, B_pad, step, 1, st_x);
      launch_gemm_simt<T>(h->st, g, h->bwd_rng[l].first, h->bwd_rng[l].second);
      TP_LAUNCHED(h);
      h->launches++;
      prof_end(h, slot, 1, TP_PH_BWD);
    }
  }
  if (h->emb) {   // the embedding parameters' gradients from the first layer's input gradient
    prof_begin(h, TP_PH_BWD, &slot);
    launch_emb_bwd<T>(h->st, emb_args<T>(h, X, idx, dyn, stacked, B, B_pad), h->n_active, h->emb_cols_max);
    TP_LAUNCHED(h);
    h->launches++;
    prof_end(h, slot, 1, TP_PH_BWD);
  }
  if (update && h->muon && h->n_muon_chunks > 0) {
    // Muon on the hidden-layer weights: momentum and |U|, X0, the
    // Newton-Schulz iterations, the update (and the bf16 copy for the next step)
    prof_begin(h, TP_PH_MUON, &slot);
    MuonArgs<T> ma;
    ma.mats = h->mmats_dev;
    ma.chunk_mat = h->mchunk_mat_dev;
    ma.grads = h->grads;
    ma.mom = h->adam_m;
    ma.params = h->params;
    ma.ns = (T*)h->ns;
    ma.part = h->mpart_dev;
    ma.wq_out = wq_next;
    ma.mem = h->mem_dev;
    ma.mu = h->muon_mu;
    ma.x_final = h->ns_steps & 1;
    ma.ns_cnt = h->bf16 ? h->tc.ns_cnt_dev : nullptr;
    ma.n_ns_cnt = h->bf16 ? h->tc.n_ns_cnt : 0;
    // bf16: the momentum kernel writes U as X0 and 1 / |U|_F, which the
    // first iteration's products apply; fp32: k_muon_x0 normalises X0
    ma.x0_fused = h->bf16 ? 1 : 0;
    ma.ns_scale = h->mscale_dev;
    ma.mat_done = h->mdone_dev;
    int nl = 0;
    for (int phase = 0; phase < (h->bf16 ? 1 : 2); ++phase) {
      launch_muon<T>(h->st, ma, h->n_muon_chunks, phase);
      TP_LAUNCHED(h);
      ++nl;
    }
    if (h->bf16) {  // every iteration in one tensor-core launch
      TP_TRY(tc_run_ns(h->tc, h->st, h->ns, h->mscale_dev, h->mem_dev, h->err));
      TP_LAUNCHED(h);
      ++nl;
    } else {
      for (int it = 0; it < h->ns_steps; ++it) {
        const int p = it & 1;
        const int which[3] = {p, 2, 3 + p};
        for (int q = 0; q < 3; ++q) {
          auto g = gemm_args<T>(h, B, B_pad, step, 0);
          launch_gemm_simt<T>(h->st, g, h->ns_simt_rng[which[q]].first, h->ns_simt_rng[which[q]].second);
          TP_LAUNCHED(h);
          ++nl;
        }
      }
    }
    launch_muon<T>(h->st, ma, h->n_muon_chunks, 2);
    TP_LAUNCHED(h);
    ++nl;
    h->launches += nl;
    prof_end(h, slot, nl, TP_PH_MUON);
  }
  if (update && !fused && h->n_chunks > 0) {
    prof_begin(h, TP_PH_ADAMW, &slot);
    AdamArgs ag;
    ag.chunks = h->chunks_dev;
    ag.segs = h->segs_dev;
    ag.mem = h->mem_dev;
    ag.bias_corr = h->bias_corr;
    ag.params = h->params;
    ag.grads = h->grads;
    ag.m = h->adam_m;
    ag.v = h->adam_v;
    ag.wq = wq_next;
    ag.beta1 = h->cfg.beta1;
    ag.beta2 = h->cfg.beta2;
    ag.eps = h->cfg.eps;
    ag.wd_on_bias = h->cfg.wd_on_bias;
    ag.mg = mask_gen(h, step + 1u, dyn, 1u);  // the next step's dropout masks
    launch_adamw(h->st, ag, h->n_chunks);
    TP_LAUNCHED(h);
    h->launches++;
    prof_end(h, slot, 1, TP_PH_ADAMW);
  }
  (void)n_rows;
  return TP_OK;
}

// A training (update) or forward-backward step: replay the captured graph
// of this (B, update, weight copy) after copying the per-call arguments to
// the device, or launch the kernels directly while profiling.
template <typename T>
tp_status step_entry(tabpack* h, const float* X, int64_t n_rows, const int32_t* idx, const void* y, int B,
                     uint32_t step, float* loss_out, bool update, bool stacked = false) {
  // the forward reads the step's dropout masks from the arena: fill it now
  // unless the previous step's AdamW pass did
  const bool masks_next = update && h->bf16 && !h->fuse_adamw && h->n_chunks > 0;
  if (h->bf16 && h->n_mchunks > 0 && h->masks_for != (int64_t)step) {
    launch_masks(h->st, mask_gen(h, step, nullptr, 0));
    TP_LAUNCHED(h);
    h->launches++;
  }
  if (!h->use_graphs || h->profiling) {
    TP_TRY(run_step<T>(h, X, n_rows, idx, y, B, step, loss_out, update, nullptr, stacked));
  } else {
    // per-call arguments: pinned ring slot -> dyn_dev, ordered before the graph
    const int k = h->dyn_next;
    h->dyn_next = (k + 1) % tabpack::kRing;
    if (h->dyn_used[k]) TP_CUDA(h, cudaEventSynchronize(h->dyn_ev[k]));
    h->dyn_host[k] = StepDyn{X, idx, y, loss_out, step, 0};
    TP_CUDA(h, cudaMemcpyAsync(h->dyn_dev, &h->dyn_host[k], sizeof(StepDyn), cudaMemcpyHostToDevice, h->st));
    TP_CUDA(h, cudaEventRecord(h->dyn_ev[k], h->st));
    h->dyn_used[k] = true;
    tabpack::GraphEntry* ge = nullptr;
    for (auto& e : h->graphs)
      if (e.B == B && e.update == (int)update && e.wcur == h->wcur && e.stacked == (int)stacked) ge = &e;
    if (!ge) {
      cudaStream_t user = h->st;
      h->st = h->st_cap;
      const int64_t l0 = h->launches;
      cudaError_t e = cudaStreamBeginCapture(h->st, cudaStreamCaptureModeThreadLocal);
      tp_status s = e == cudaSuccess ? run_step<T>(h, X, n_rows, idx, y, B, step, loss_out, update, h->dyn_dev, stacked)
                                     : fail(h, TP_ECUDA, "cudaStreamBeginCapture: %s", cudaGetErrorString(e));
      cudaGraph_t graph = nullptr;
      cudaError_t e2 = e == cudaSuccess ? cudaStreamEndCapture(h->st, &graph) : cudaSuccess;
      h->st = user;
      const int64_t n_launch = h->launches - l0;
      h->launches = l0;
      if (s != TP_OK) {
        if (graph) cudaGraphDestroy(graph);
        return s;
      }
      if (e2 != cudaSuccess) return fail(h, TP_ECUDA, "cudaStreamEndCapture: %s", cudaGetErrorString(e2));
      cudaGraphExec_t exec = nullptr;
      e = cudaGraphInstantiate(&exec, graph, 0);
      cudaGraphDestroy(graph);
      if (e != cudaSuccess) return fail(h, TP_ECUDA, "cudaGraphInstantiate: %s", cudaGetErrorString(e));
      h->graphs.push_back(tabpack::GraphEntry{B, (int)update, h->wcur, (int)stacked, exec, n_launch});
      ge = &h->graphs.back();
    }
    TP_CUDA(h, cudaGraphLaunch(ge->exec, h->st));
    h->launches += ge->n_launch;
  }
  if (update && h->bf16) h->wcur ^= 1;
  h->masks_for = masks_next ? (int64_t)(uint32_t)(step + 1u) : (int64_t)step;
  h->last_B = B;
  return TP_OK;
}

// The stacked-batch arena and (bf16) its tile plan, on first use and after an
// active-set change.
template <typename T>
tp_status ensure_stacked(tabpack* h) {
  const int m = h->cfg.m;
  if (!h->xbs) {
    TP_CUDA(h, cudaStreamSynchronize(h->st));
    const size_t bytes = h->elem * (size_t)m * h->xb_elems;
    TP_CUDA(h, cudaMalloc(&h->xbs, bytes));
    TP_CUDA(h, cudaMemset(h->xbs, 0, bytes));
    std::vector<OnesJob> jobs;
    for (int i = 0; i < m; ++i) jobs.push_back(OnesJob{(int64_t)i * h->xb_elems, h->ldx, h->d_in_pad, h->B_cap, 0});
    OnesJob* d = nullptr;
    TP_CUDA(h, cudaMalloc(&d, sizeof(OnesJob) * jobs.size()));
    cudaError_t e = cudaMemcpy(d, jobs.data(), sizeof(OnesJob) * jobs.size(), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) {
      launch_fill_ones<T>(h->st, d, (int)jobs.size(), (T*)h->xbs, (T*)h->act, nullptr);
      h->launches++;
      e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    cudaFree(d);
    if (e != cudaSuccess) return fail(h, TP_ECUDA, "stacked batch arena: %s", cudaGetErrorString(e));
    h->s_stale = true;
  }
  if (h->bf16 && h->s_stale) {
    TcLayout lay;
    lay.depth = &h->depth;
    lay.width = &h->width;
    lay.active = &h->active;
    lay.W_off = &h->W_off;
    lay.b_off = &h->b_off;
    lay.act_off = &h->act_off;
    lay.dz_off = &h->dz_off;
    lay.m = m;
    lay.d_in_pad = h->d_in_pad;
    lay.ldx = h->ldx;
    lay.B_cap = h->B_cap;
    lay.wq[0] = h->wq[0];
    lay.wq[1] = h->wq[1];
    lay.xb = h->xbs;
    lay.act = h->act;
    lay.dz = h->dz;
    lay.bias_colsums = h->bias_colsums;
    lay.mask_off = h->mask_words > 0 ? &h->mask_off : nullptr;
    lay.xb_stride = h->xb_elems;
    TP_CUDA(h, cudaStreamSynchronize(h->st));
    TP_TRY(tc_build_plan(h->tcs, lay, h->err));
  }
  h->s_stale = false;
  return TP_OK;
}

constexpr int kPredictRows = 8192;
constexpr int64_t kPredictEmbBytes = int64_t(1) << 30;   // cap of the prediction embedding arena

// Rows of one prediction chunk for N rows: at most kPredictRows, and with
// embeddings at most what keeps the embedding arena under kPredictEmbBytes.
int predict_rows(const tabpack* h, int64_t N) {
  int64_t rows = std::min<int64_t>(round_up(N, kRowTile), kPredictRows);
  if (h->emb) {
    int64_t per_row = 0;
    for (int i = 0; i < h->cfg.m; ++i) per_row += h->in0_pad[i] + kOnesCols;
    const int64_t fit = kPredictEmbBytes / ((int64_t)sizeof(__nv_bfloat16) * per_row) / kRowTile * kRowTile;
    rows = std::min(rows, std::max<int64_t>(fit, kRowTile));
  }
  return (int)rows;
}

// (Re)build the bf16 prediction plan for chunks of at least P_need rows.
tp_status build_predict(tabpack* h, int P_need) {
  if (h->tcp.enabled && !h->p_stale && h->P_cap >= P_need) return TP_OK;
  const int m = h->cfg.m;
  if (h->P_cap < P_need) {
    TP_CUDA(h, cudaStreamSynchronize(h->st));
    free_predict(h);
    h->P_cap = P_need;
    h->p_act_off.assign(m, {});
    int64_t off = 0;
    for (int i = 0; i < m; ++i) {
      const int64_t buf = round_up((int64_t)h->P_cap * ldh_of(h, i), 128);
      for (int l = 0; l < h->depth[i]; ++l) h->p_act_off[i][l] = off + (l & 1) * buf;
      off += std::min(h->depth[i], 2) * buf;
    }
    const size_t xb_bytes = sizeof(__nv_bfloat16) * (size_t)h->P_cap * h->ldx;
    const size_t act_bytes = sizeof(__nv_bfloat16) * (size_t)std::max<int64_t>(off, 128);
    TP_CUDA(h, cudaMalloc(&h->p_xb, xb_bytes));
    TP_CUDA(h, cudaMalloc(&h->p_act, act_bytes));
    TP_CUDA(h, cudaMalloc(&h->p_head_dev, sizeof(HeadJob) * (size_t)m * (h->P_cap / kHeadRows)));
    // columns the forward never writes (ones / pad columns) stay zero
    TP_CUDA(h, cudaMemset(h->p_xb, 0, xb_bytes));
    TP_CUDA(h, cudaMemset(h->p_act, 0, act_bytes));
    if (h->emb) {
      // the members' embedding matrices for a chunk, with their ones column
      h->p_e_off.assign(m, 0);
      int64_t eoff = 0;
      for (int i = 0; i < m; ++i) {
        h->p_e_off[i] = eoff;
        eoff += round_up((int64_t)h->P_cap * (h->in0_pad[i] + kOnesCols), 128);
      }
      TP_CUDA(h, cudaMalloc(&h->p_ex, sizeof(__nv_bfloat16) * (size_t)eoff));
      TP_CUDA(h, cudaMemset(h->p_ex, 0, sizeof(__nv_bfloat16) * (size_t)eoff));
      std::vector<EmbMember> em(m);
      std::vector<OnesJob> jobs;
      for (int i = 0; i < m; ++i) {
        em[i] = EmbMember{h->d_emb[i], h->in0[i], h->in0_pad[i], 0, h->p_e_off[i], 0, h->emb_off[i]};
        jobs.push_back(OnesJob{h->p_e_off[i], h->in0_pad[i] + kOnesCols, h->in0_pad[i], h->P_cap, 2});
      }
      TP_CUDA(h, cudaMalloc((void**)&h->embm_p_dev, sizeof(EmbMember) * m));
      TP_CUDA(h, cudaMemcpy(h->embm_p_dev, em.data(), sizeof(EmbMember) * m, cudaMemcpyHostToDevice));
      OnesJob* d = nullptr;
      TP_CUDA(h, cudaMalloc(&d, sizeof(OnesJob) * jobs.size()));
      cudaError_t e = cudaMemcpy(d, jobs.data(), sizeof(OnesJob) * jobs.size(), cudaMemcpyHostToDevice);
      if (e == cudaSuccess) {
        launch_fill_ones<__nv_bfloat16>(h->st, d, (int)jobs.size(), nullptr, nullptr, (__nv_bfloat16*)h->p_ex);
        h->launches++;
        e = cudaGetLastError();
      }
      if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
      cudaFree(d);
      if (e != cudaSuccess) return fail(h, TP_ECUDA, "prediction embedding arena: %s", cudaGetErrorString(e));
    }
  }
  TcLayout lay;
  lay.depth = &h->depth;
  lay.width = &h->width;
  lay.active = &h->active;
  lay.W_off = &h->W_off;
  lay.b_off = &h->b_off;
  lay.act_off = &h->p_act_off;
  lay.dz_off = &h->dz_off;
  lay.m = m;
  lay.d_in_pad = h->d_in_pad;
  lay.ldx = h->ldx;
  lay.B_cap = h->P_cap;
  lay.wq[0] = h->wq[0];
  lay.wq[1] = h->wq[1];
  lay.xb = h->p_xb;
  lay.act = h->p_act;
  lay.dz = nullptr;
  lay.fwd_only = true;
  lay.in0_pad = &h->in0_pad;
  if (h->emb) {
    lay.xb = h->p_ex;
    lay.x0_off = &h->p_e_off;
  }
  TP_CUDA(h, cudaStreamSynchronize(h->st));
  TP_TRY(tc_build_plan(h->tcp, lay, h->err));
  std::vector<HeadJob> hj;
  for (int i = 0; i < m; ++i) {
    if (!h->active[i]) continue;
    const int L = h->depth[i];
    for (int b = 0; b < h->P_cap / kHeadRows; ++b) {
      HeadJob j{};
      j.member = i;
      j.blk = b;
      j.h_ld = ldh_of(h, i);
      j.split = 1;
      j.h_off = h->p_act_off[i][L - 1];
      j.w_off = h->W_off[i][L];
      j.b_off = h->b_off[i][L];
      hj.push_back(j);
    }
  }
  if (!hj.empty()) TP_CUDA(h, cudaMemcpy(h->p_head_dev, hj.data(), sizeof(HeadJob) * hj.size(), cudaMemcpyHostToDevice));
  h->n_p_head = (int)hj.size();
  h->p_stale = false;
  return TP_OK;
}

// bf16 prediction: chunks of P_cap rows through the forward-only plan.
tp_status run_predict_tc(tabpack* h, const float* X, int64_t N, float* out) {
  TP_TRY(build_predict(h, predict_rows(h, N)));
  for (int64_t n0 = 0; n0 < N; n0 += h->P_cap) {
    const int rows = (int)std::min<int64_t>(h->P_cap, N - n0);
    const int B_pad = (int)round_up(rows, kRowTile);
    int slot;
    prof_begin(h, TP_PH_PREDICT, &slot);
    launch_gather<__nv_bfloat16>(h->st, X + n0 * h->cfg.d_in, nullptr, nullptr, rows, B_pad, h->cfg.d_in, h->d_in_pad,
                                 h->ldx, (__nv_bfloat16*)h->p_xb, 0, h->t_dev, h->bias_corr, h->active_ids_dev, 0,
                                 h->cfg.beta1, h->cfg.beta2, h->tcp.cnt_dev, h->tcp.n_cnt);
    TP_LAUNCHED(h);
    int nl = 3;
    if (h->emb) {
      EmbArgs<__nv_bfloat16> ea = emb_args<__nv_bfloat16>(h, X + n0 * h->cfg.d_in, nullptr, nullptr, false, rows, B_pad);
      ea.em = h->embm_p_dev;
      ea.ex = (__nv_bfloat16*)h->p_ex;
      launch_emb_fwd<__nv_bfloat16>(h->st, ea, h->n_active, h->emb_cols_max);
      TP_LAUNCHED(h);
      ++nl;
    }
    TP_TRY(tc_run_fwd(h->tcp, h->st, rows, B_pad, h->wcur, 0, nullptr, 0, h->params, h->mem_dev, h->p_act, h->err));
    TP_LAUNCHED(h);
    PredictHeadArgs<__nv_bfloat16> pg;
    pg.jobs = h->p_head_dev;
    pg.mem = h->mem_dev;
    pg.act = (const __nv_bfloat16*)h->p_act;
    pg.params = h->params;
    pg.out = out;
    pg.N = N;
    pg.n0 = n0;
    pg.rows = rows;
    pg.d_out = h->cfg.d_out;
    pg.task = h->cfg.task;
    pg._pad = 0;
    launch_predict_head<__nv_bfloat16>(h->st, pg, h->n_p_head);
    TP_LAUNCHED(h);
    h->launches += nl;
    prof_end(h, slot, nl, TP_PH_PREDICT);
  }
  return TP_OK;
}

template <typename T>
tp_status run_predict(tabpack* h, const float* X, int64_t N, float* out) {
  if (h->bf16) return run_predict_tc(h, X, N, out);
  for (int64_t n0 = 0; n0 < N; n0 += h->B_cap) {
    const int rows = (int)std::min<int64_t>(h->B_cap, N - n0);
    const int B_pad = (int)round_up(rows, kRowTile);
    int slot;
    prof_begin(h, TP_PH_PREDICT, &slot);
    launch_gather<T>(h->st, X + n0 * h->cfg.d_in, nullptr, nullptr, rows, B_pad, h->cfg.d_in, h->d_in_pad, h->ldx,
                     (T*)h->xb,
                     0, h->t_dev, h->bias_corr, h->active_ids_dev, 0, h->cfg.beta1, h->cfg.beta2, h->tc.cnt_dev,
                     h->tc.n_cnt);
    TP_LAUNCHED(h);
    h->launches++;
    if (h->emb) {
      launch_emb_fwd<T>(h->st, emb_args<T>(h, X + n0 * h->cfg.d_in, nullptr, nullptr, false, rows, B_pad),
                        h->n_active, h->emb_cols_max);
      TP_LAUNCHED(h);
      h->launches++;
    }
    prof_end(h, slot, h->emb ? 2 : 1, TP_PH_PREDICT);
    TP_TRY(run_forward<T>(h, rows, B_pad, 0u, nullptr, 0));
    prof_begin(h, TP_PH_PREDICT, &slot);
    PredictHeadArgs<T> pg;
    pg.jobs = h->head_jobs_dev;
    pg.mem = h->mem_dev;
    pg.act = (const T*)h->act;
    pg.params = h->params;
    pg.out = out;
    pg.N = N;
    pg.n0 = n0;
    pg.rows = rows;
    pg.d_out = h->cfg.d_out;
    pg.task = h->cfg.task;
    pg._pad = 0;
    launch_predict_head<T>(h->st, pg, h->n_head_jobs);
    TP_LAUNCHED(h);
    h->launches++;
    prof_end(h, slot, 1, TP_PH_PREDICT);
  }
  return TP_OK;
}

// both bf16 copies := bf16(params) (after a host write or an active-set change)
tp_status refresh_copies(tabpack* h) {
  if (!h->bf16) return TP_OK;
  launch_refresh_wq(h->st, h->params, h->wq[0], h->wq[1], h->n_params);
  TP_LAUNCHED(h);
  h->launches++;
  TP_CUDA(h, cudaStreamSynchronize(h->st));
  return TP_OK;
}

tp_status check_step_args(tabpack* h, const float* X, int64_t n_rows, const int32_t* idx, const void* y, int B) {
  if (!h) return fail(nullptr, TP_EINVAL, "null pack");
  if (!X || !idx || !y) return fail(h, TP_EINVAL, "X, idx and y must be device pointers");
  if (B < 1 || B > h->cfg.max_batch) return fail(h, TP_EINVAL, "B=%d outside [1, max_batch=%d]", B, h->cfg.max_batch);
  if (n_rows < 1) return fail(h, TP_EINVAL, "n_rows=%lld", (long long)n_rows);
  return TP_OK;
}

// Member i's contiguous run of the parameter arena: (first element, length).
std::pair<int64_t, int64_t> member_run(const tabpack* h, int i) {
  const int L = h->depth[i];
  const int64_t first = h->W_off[i][0];
  const int64_t last = h->emb ? h->emb_off[i] + h->n_emb[i] : h->b_off[i][L] + h->cfg.d_out;
  return {first, last - first};
}

tp_status check_ml(tabpack* h, int member, int layer) {
  if (!h) return fail(nullptr, TP_EINVAL, "null pack");
  if (member < 0 || member >= h->cfg.m) return fail(h, TP_EINVAL, "member %d out of range", member);
  if (layer < 0 || layer > h->depth[member]) return fail(h, TP_EINVAL, "layer %d out of range", layer);
  return TP_OK;
}

// synchronise and surface a bounded-wait timeout of the tensor-core pipeline
tp_status sync_check(tabpack* h) {
  TP_CUDA(h, cudaStreamSynchronize(h->st));
  if (h->bf16 && h->tc.enabled) TP_TRY(tc_check(h->tc, h->st, h->err));
  if (h->bf16 && h->tcp.enabled) TP_TRY(tc_check(h->tcp, h->st, h->err));
  if (h->bf16 && h->tcs.enabled) TP_TRY(tc_check(h->tcs, h->st, h->err));
  return TP_OK;
}

}  // namespace

void tp::record_thread_error(const char* msg) { g_thread_error = msg; }

// ====================================================================== ABI
extern "C" {

static tp_status create_impl(const tp_config* cfg, const int32_t* depth, const int32_t* width, const float* dropout,
                             const float* lr, const float* wd, const int32_t* d_emb, const float* freq,
                             void* cuda_stream, tabpack_t** out) {
  if (out) *out = nullptr;
  if (!cfg || !depth || !width || !dropout || !lr || !wd || !out)
    return fail(nullptr, TP_EINVAL, "null argument");
  if (cfg->m < 1 || cfg->d_in < 1 || cfg->max_batch < 1) return fail(nullptr, TP_EINVAL, "m, d_in, max_batch must be >= 1");
  if (cfg->task < 0 || cfg->task > 2) return fail(nullptr, TP_EINVAL, "unknown task %d", cfg->task);
  if (cfg->precision != TP_BF16 && cfg->precision != TP_FP32) return fail(nullptr, TP_EINVAL, "unknown precision");
  if (cfg->task == TP_MULTICLASS ? (cfg->d_out < 2 || cfg->d_out > kMaxDout) : cfg->d_out != 1)
    return fail(nullptr, TP_EINVAL, "d_out=%d invalid for task %d", cfg->d_out, cfg->task);
  if (!(cfg->beta1 >= 0.f && cfg->beta1 < 1.f && cfg->beta2 >= 0.f && cfg->beta2 < 1.f && cfg->eps >= 0.f))
    return fail(nullptr, TP_EINVAL, "AdamW constants out of range");
  for (int i = 0; i < cfg->m; ++i) {
    if (depth[i] < 1 || depth[i] > kMaxDepth) return fail(nullptr, TP_EINVAL, "depth[%d]=%d not in 1..%d", i, depth[i], kMaxDepth);
    if (width[i] < 16 || width[i] > 4096 || width[i] % 16)
      return fail(nullptr, TP_EINVAL, "width[%d]=%d must be a multiple of 16 in [16, 4096]", i, width[i]);
    if (!(dropout[i] >= 0.f && dropout[i] < 1.f)) return fail(nullptr, TP_EINVAL, "dropout[%d] not in [0, 1)", i);
    if (!(lr[i] >= 0.f) || !(wd[i] >= 0.f)) return fail(nullptr, TP_EINVAL, "lr/wd[%d] must be >= 0", i);
  }
  if (cfg->m >= (1 << 24)) return fail(nullptr, TP_EINVAL, "too many members");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(nullptr, TP_ECUDA, "no CUDA device: %s", cudaGetErrorString(e));
  cudaDeviceProp prop;
  e = cudaGetDeviceProperties(&prop, dev);
  if (e != cudaSuccess) return fail(nullptr, TP_ECUDA, "cudaGetDeviceProperties: %s", cudaGetErrorString(e));
  if (prop.major != 10) return fail(nullptr, TP_ENOTSUP, "needs a Blackwell (sm_10x) GPU, found sm_%d%d", prop.major, prop.minor);

  tabpack* h = new tabpack();
  h->cfg = *cfg;
  h->st = (cudaStream_t)cuda_stream;
  h->bf16 = cfg->precision == TP_BF16;
  h->fuse_adamw = h->bf16 && cfg->fuse_optimizer != 0;
  h->depth.assign(depth, depth + cfg->m);
  h->width.assign(width, width + cfg->m);
  h->dropout.assign(dropout, dropout + cfg->m);
  h->lr.assign(lr, lr + cfg->m);
  h->wd.assign(wd, wd + cfg->m);
  h->active.assign(cfg->m, 1);
  if (d_emb) {
    h->emb = true;
    h->d_emb.assign(d_emb, d_emb + cfg->m);
    h->fuse_adamw = false;   // the embedding parameters take the stand-alone AdamW pass
  }
  if (h->bf16) head_stage_prepare();   // the staged head kernel's shared-memory limit (outside any capture)
  tp_status s = build_layout(h);
  if (s == TP_OK) s = alloc_all(h);
  if (s == TP_OK) s = build_schedule(h);
  if (s == TP_OK) s = h->bf16 ? fill_ones<__nv_bfloat16>(h) : fill_ones<float>(h);
  if (s == TP_OK) {
    // Philox init of every parameter (all members active here)
    InitArgs ig{h->chunks_dev, h->segs_dev, h->params, h->grads, h->adam_m, h->adam_v, h->wq[0], h->wq[1], cfg->seed};
    launch_init(h->st, ig, h->n_chunks);
    h->launches++;
    cudaError_t le = cudaGetLastError();
    if (le == cudaSuccess) le = cudaStreamSynchronize(h->st);
    if (le != cudaSuccess) s = fail(h, TP_ECUDA, "init: %s", cudaGetErrorString(le));
  }
  if (s == TP_OK && h->emb) {
    // embedding parameters: the caller's frequencies, zero phases and scales
    std::vector<EmbMember> em(cfg->m);
    const float* fr = freq;
    for (int i = 0; i < cfg->m && s == TP_OK; ++i) {
      std::vector<float> v((size_t)h->n_emb[i], 0.f);
      const int64_t nf = (int64_t)cfg->d_in * (h->d_emb[i] - 1);
      std::copy(fr, fr + nf, v.begin());
      fr += nf;
      if (cudaMemcpy(h->params + h->emb_off[i], v.data(), v.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess)
        s = fail(h, TP_ECUDA, "embedding init copy failed");
      em[i] = EmbMember{h->d_emb[i], h->in0[i], h->in0_pad[i], 0, h->e_off[i], h->de_off[i], h->emb_off[i]};
    }
    if (s == TP_OK && cudaMalloc((void**)&h->embm_dev, sizeof(EmbMember) * cfg->m) != cudaSuccess)
      s = fail(h, TP_ENOMEM, "cudaMalloc(embedding records) failed");
    if (s == TP_OK &&
        cudaMemcpy(h->embm_dev, em.data(), sizeof(EmbMember) * cfg->m, cudaMemcpyHostToDevice) != cudaSuccess)
      s = fail(h, TP_ECUDA, "embedding records copy failed");
  }
  if (s != TP_OK) {
    g_thread_error = h->err;
    free_all(h);
    delete h;
    return s;
  }
  *out = h;
  return TP_OK;
}

tp_status pack_create(const tp_config* cfg, const int32_t* depth, const int32_t* width, const float* dropout,
                      const float* lr, const float* wd, void* cuda_stream, tabpack_t** out) {
  return create_impl(cfg, depth, width, dropout, lr, wd, nullptr, nullptr, cuda_stream, out);
}

tp_status pack_create_emb(const tp_config* cfg, const int32_t* depth, const int32_t* width, const float* dropout,
                          const float* lr, const float* wd, const int32_t* d_emb, const float* freq,
                          void* cuda_stream, tabpack_t** out) {
  if (out) *out = nullptr;
  if (!cfg || !d_emb || !freq) return fail(nullptr, TP_EINVAL, "null argument");
  for (int i = 0; i < cfg->m; ++i)
    if (d_emb[i] < 1 || d_emb[i] > 64) return fail(nullptr, TP_EINVAL, "d_emb[%d]=%d not in 1..64", i, d_emb[i]);
  return create_impl(cfg, depth, width, dropout, lr, wd, d_emb, freq, cuda_stream, out);
}

tp_status pack_get_emb(tabpack_t* h, int32_t member, int32_t grads, float* out) {
  TP_TRY(check_ml(h, member, 0));
  if (!h->emb || !out) return fail(h, TP_EINVAL, "the pack has no embeddings");
  TP_TRY(sync_check(h));
  TP_CUDA(h, cudaMemcpy(out, (grads ? h->grads : h->params) + h->emb_off[member], h->n_emb[member] * 4,
                        cudaMemcpyDeviceToHost));
  return TP_OK;
}

tp_status pack_set_emb(tabpack_t* h, int32_t member, const float* in) {
  TP_TRY(check_ml(h, member, 0));
  if (!h->emb || !in) return fail(h, TP_EINVAL, "the pack has no embeddings");
  TP_TRY(sync_check(h));
  TP_CUDA(h, cudaMemcpy(h->params + h->emb_off[member], in, h->n_emb[member] * 4, cudaMemcpyHostToDevice));
  return TP_OK;
}

tp_status pack_member_emb(const tabpack_t* h, int32_t member, int32_t* d_emb) {
  if (!h || !d_emb) return fail(const_cast<tabpack_t*>(h), TP_EINVAL, "null argument");
  if (member < 0 || member >= h->cfg.m) return fail(const_cast<tabpack_t*>(h), TP_EINVAL, "member %d out of range", member);
  *d_emb = h->emb ? h->d_emb[member] : 0;
  return TP_OK;
}

void pack_destroy(tabpack_t* h) {
  if (!h) return;
  free_all(h);
  delete h;
}

tp_status pack_set_stream(tabpack_t* h, void* cuda_stream) {
  if (!h) return fail(nullptr, TP_EINVAL, "null pack");
  TP_CUDA(h, cudaStreamSynchronize(h->st));
  h->st = (cudaStream_t)cuda_stream;
  return TP_OK;
}

tp_status pack_train_step(tabpack_t* h, const float* X, int64_t n_rows, const int32_t* idx, const void* y,
                          int32_t B, uint32_t step, float* loss_out) {
  TP_TRY(check_step_args(h, X, n_rows, idx, y, B));
  if (h->n_active == 0) return fail(h, TP_ESTATE, "no active member");
  return h->bf16 ? step_entry<__nv_bfloat16>(h, X, n_rows, idx, y, B, step, loss_out, true)
                 : step_entry<float>(h, X, n_rows, idx, y, B, step, loss_out, true);
}

tp_status pack_forward_backward(tabpack_t* h, const float* X, int64_t n_rows, const int32_t* idx, const void* y,
                                int32_t B, uint32_t step, float* loss_out) {
  TP_TRY(check_step_args(h, X, n_rows, idx, y, B));
  if (h->n_active == 0) return fail(h, TP_ESTATE, "no active member");
  return h->bf16 ? step_entry<__nv_bfloat16>(h, X, n_rows, idx, y, B, step, loss_out, false)
                 : step_entry<float>(h, X, n_rows, idx, y, B, step, loss_out, false);
}

tp_status pack_train_step_stacked(tabpack_t* h, const float* X, int64_t n_rows, const int32_t* idx, const void* y,
                                  int32_t B, uint32_t step, float* loss_out) {
  TP_TRY(check_step_args(h, X, n_rows, idx, y, B));
  if (h->n_active == 0) return fail(h, TP_ESTATE, "no active member");
  if (h->bf16) {
    if (!h->emb) TP_TRY(ensure_stacked<__nv_bfloat16>(h));
    return step_entry<__nv_bfloat16>(h, X, n_rows, idx, y, B, step, loss_out, true, true);
  }
  if (!h->emb) TP_TRY(ensure_stacked<float>(h));
  return step_entry<float>(h, X, n_rows, idx, y, B, step, loss_out, true, true);
}

tp_status pack_forward_backward_stacked(tabpack_t* h, const float* X, int64_t n_rows, const int32_t* idx,
                                        const void* y, int32_t B, uint32_t step, float* loss_out) {
  TP_TRY(check_step_args(h, X, n_rows, idx, y, B));
  if (h->n_active == 0) return fail(h, TP_ESTATE, "no active member");
  if (h->bf16) {
    if (!h->emb) TP_TRY(ensure_stacked<__nv_bfloat16>(h));
    return step_entry<__nv_bfloat16>(h, X, n_rows, idx, y, B, step, loss_out, false, true);
  }
  if (!h->emb) TP_TRY(ensure_stacked<float>(h));
  return step_entry<float>(h, X, n_rows, idx, y, B, step, loss_out, false, true);
}

tp_status pack_set_muon(tabpack_t* h, const float* lr_muon, float momentum, int32_t ns_steps) {
  if (!h || !lr_muon) return fail(h, TP_EINVAL, "null argument");
  if (!(momentum >= 0.f && momentum < 1.f) || ns_steps < 1 || ns_steps > 32)
    return fail(h, TP_EINVAL, "momentum must be in [0, 1) and ns_steps in 1..32");
  for (int i = 0; i < h->cfg.m; ++i)
    if (!(lr_muon[i] >= 0.f)) return fail(h, TP_EINVAL, "lr_muon[%d] must be >= 0", i);
  for (int i = 0; i < h->cfg.m; ++i) {
    const int64_t in_max = std::max<int64_t>(h->in0_pad[i], h->width[i]);
    if ((int64_t)h->width[i] * in_max > (int64_t)INT32_MAX)
      return fail(h, TP_EINVAL, "member %d: a Muon matrix would have 2^31 elements or more", i);
  }
  TP_TRY(sync_check(h));
  const int m = h->cfg.m;
  if (!h->muon) {
    // the matrices and their Newton-Schulz buffers (128-element aligned)
    int64_t off = 0, n_chunks = 0;
    for (int i = 0; i < m; ++i)
      for (int l = 0; l < h->depth[i]; ++l) {
        MuonMat mt{};
        mt.member = i;
        mt.layer = l;
        mt.rows = h->width[i];
        mt.cols = l == 0 ? h->in0_pad[i] : h->width[i];
        const int real_cols = l == 0 ? h->in0[i] : h->width[i];
        mt.tr = mt.rows > mt.cols;
        mt.r = std::min(mt.rows, mt.cols);
        mt.c = std::max(mt.rows, mt.cols);
        mt.w_off = h->W_off[i][l];
        auto take = [&](int64_t n) { const int64_t o = off; off = round_up(off + n, 128); return o; };
        mt.x_off[0] = take((int64_t)mt.r * mt.c);
        mt.x_off[1] = take((int64_t)mt.r * mt.c);
        mt.a_off = take((int64_t)mt.r * mt.r);
        mt.bm_off = take((int64_t)mt.r * mt.r);
        mt.scale = (float)std::sqrt(std::max(1.0, (double)mt.rows / (double)real_cols));
        n_chunks += muon_chunks(mt);
        h->mmats.push_back(mt);
      }
    TP_CUDA(h, cudaMalloc(&h->ns, h->elem * (size_t)std::max<int64_t>(off, 128)));
    TP_CUDA(h, cudaMemset(h->ns, 0, h->elem * (size_t)std::max<int64_t>(off, 128)));
    TP_CUDA(h, cudaMalloc((void**)&h->mmats_dev, sizeof(MuonMat) * h->mmats.size()));
    TP_CUDA(h, cudaMalloc((void**)&h->mchunk_mat_dev, sizeof(int32_t) * std::max<int64_t>(n_chunks, 1)));
    TP_CUDA(h, cudaMalloc((void**)&h->mpart_dev, sizeof(double) * std::max<int64_t>(n_chunks, 1)));
    const size_t n_mat = std::max<size_t>(h->mmats.size(), 1);
    TP_CUDA(h, cudaMalloc((void**)&h->mscale_dev, sizeof(float) * n_mat));
    TP_CUDA(h, cudaMalloc((void**)&h->mdone_dev, sizeof(int) * n_mat));
    TP_CUDA(h, cudaMemset(h->mdone_dev, 0, sizeof(int) * n_mat));
    // Muon's momentum starts at zero in the first-moment arena
    for (const MuonMat& mt : h->mmats)
      TP_CUDA(h, cudaMemset(h->adam_m + mt.w_off, 0, sizeof(float) * (size_t)mt.rows * mt.cols));
  }
  for (MuonMat& mt : h->mmats) mt.lr = lr_muon[mt.member];
  h->muon = true;
  h->muon_mu = momentum;
  h->ns_steps = ns_steps;
  h->fuse_adamw = false;   // the weight-gradient epilogue would apply AdamW to Muon's matrices
  // the tensor-core plan's map table gains the Newton-Schulz buffers
  tc_free_plan(h->tc);
  drop_graphs(h);
  TP_TRY(build_schedule(h));
  return sync_check(h);
}

tp_status pack_debug_muon_dir(tabpack_t* h, int32_t member, int32_t layer, float* out) {
  TP_TRY(check_ml(h, member, layer));
  if (!h->muon || layer >= h->depth[member] || !out) return fail(h, TP_EINVAL, "no Muon matrix there");
  TP_TRY(sync_check(h));
  const MuonMat* mt = nullptr;
  for (const MuonMat& x : h->mmats)
    if (x.member == member && x.layer == layer) mt = &x;
  const int64_t n = (int64_t)mt->r * mt->c;
  const int xf = h->ns_steps & 1;
  std::vector<float> X(n);
  if (h->bf16) {
    std::vector<__nv_bfloat16> xb(n);
    TP_CUDA(h, cudaMemcpy(xb.data(), (__nv_bfloat16*)h->ns + mt->x_off[xf], n * 2, cudaMemcpyDeviceToHost));
    for (int64_t e = 0; e < n; ++e) X[e] = __bfloat162float(xb[e]);
  } else {
    TP_CUDA(h, cudaMemcpy(X.data(), (float*)h->ns + mt->x_off[xf], n * 4, cudaMemcpyDeviceToHost));
  }
  const int in = layer == 0 ? h->in0[member] : h->width[member];
  for (int i = 0; i < mt->rows; ++i)
    for (int j = 0; j < in; ++j) out[(int64_t)i * in + j] = X[mt->tr ? (int64_t)j * mt->c + i : (int64_t)i * mt->c + j];
  return TP_OK;
}

tp_status pack_predict(tabpack_t* h, const float* X, int64_t N, float* out) {
  if (!h) return fail(nullptr, TP_EINVAL, "null pack");
  if (!X || !out || N < 1) return fail(h, TP_EINVAL, "X/out null or N < 1");
  if (h->n_active == 0) return fail(h, TP_ESTATE, "no active member");
  return h->bf16 ? run_predict<__nv_bfloat16>(h, X, N, out) : run_predict<float>(h, X, N, out);
}

tp_status pack_set_active(tabpack_t* h, const uint8_t* active) {
  if (!h || !active) return fail(h, TP_EINVAL, "null argument");
  TP_TRY(sync_check(h));
  for (int i = 0; i < h->cfg.m; ++i) h->active[i] = active[i] ? 1 : 0;
  TP_TRY(build_schedule(h));
  // a member that stops keeps its latest weights in both bf16 copies
  return refresh_copies(h);
}

static tp_status copy_layer(tabpack_t* h, int member, int layer, float* W, float* b, const float* src) {
  TP_TRY(check_ml(h, member, layer));
  TP_TRY(sync_check(h));
  const int L = h->depth[member], w = h->width[member];
  const int in = layer == 0 ? h->in0[member] : w, in_pad = layer == 0 ? h->in0_pad[member] : w;
  const int out = layer == L ? h->cfg.d_out : w;
  if (W) {
    std::vector<float> tmp((size_t)out * in_pad);
    TP_CUDA(h, cudaMemcpy(tmp.data(), src + h->W_off[member][layer], tmp.size() * 4, cudaMemcpyDeviceToHost));
    for (int r = 0; r < out; ++r) std::memcpy(W + (size_t)r * in, tmp.data() + (size_t)r * in_pad, (size_t)in * 4);
  }
  if (b) TP_CUDA(h, cudaMemcpy(b, src + h->b_off[member][layer], (size_t)out * 4, cudaMemcpyDeviceToHost));
  return TP_OK;
}

tp_status pack_get_params(tabpack_t* h, int32_t member, int32_t layer, float* W, float* b) {
  if (!h) return fail(nullptr, TP_EINVAL, "null pack");
  return copy_layer(h, member, layer, W, b, h->params);
}

tp_status pack_get_grads(tabpack_t* h, int32_t member, int32_t layer, float* W, float* b) {
  if (!h) return fail(nullptr, TP_EINVAL, "null pack");
  return copy_layer(h, member, layer, W, b, h->grads);
}

tp_status pack_set_params(tabpack_t* h, int32_t member, int32_t layer, const float* W, const float* b) {
  TP_TRY(check_ml(h, member, layer));
  TP_TRY(sync_check(h));
  const int L = h->depth[member], w = h->width[member];
  const int in = layer == 0 ? h->in0[member] : w, in_pad = layer == 0 ? h->in0_pad[member] : w;
  const int out = layer == L ? h->cfg.d_out : w;
  if (W) {
    std::vector<float> tmp((size_t)out * in_pad, 0.f);
    for (int r = 0; r < out; ++r) std::memcpy(tmp.data() + (size_t)r * in_pad, W + (size_t)r * in, (size_t)in * 4);
    TP_CUDA(h, cudaMemcpy(h->params + h->W_off[member][layer], tmp.data(), tmp.size() * 4, cudaMemcpyHostToDevice));
  }
  if (b) TP_CUDA(h, cudaMemcpy(h->params + h->b_off[member][layer], b, (size_t)out * 4, cudaMemcpyHostToDevice));
  return refresh_copies(h);
}

tp_status pack_member_size(const tabpack_t* h, int32_t member, int64_t* n_elems) {
  if (!h || !n_elems) return fail(const_cast<tabpack_t*>(h), TP_EINVAL, "null argument");
  if (member < 0 || member >= h->cfg.m) return fail(const_cast<tabpack_t*>(h), TP_EINVAL, "member %d out of range", member);
  *n_elems = member_run(h, member).second;
  return TP_OK;
}

tp_status pack_snapshot(tabpack_t* h, int32_t member, float* dst) {
  TP_TRY(check_ml(h, member, 0));
  if (!dst) return fail(h, TP_EINVAL, "null dst");
  const auto run = member_run(h, member);
  TP_CUDA(h, cudaMemcpyAsync(dst, h->params + run.first, (size_t)run.second * 4, cudaMemcpyDeviceToDevice, h->st));
  return TP_OK;
}

tp_status pack_restore(tabpack_t* h, int32_t member, const float* src) {
  TP_TRY(check_ml(h, member, 0));
  if (!src) return fail(h, TP_EINVAL, "null src");
  TP_TRY(sync_check(h));
  const auto run = member_run(h, member);
  TP_CUDA(h, cudaMemcpyAsync(h->params + run.first, src, (size_t)run.second * 4, cudaMemcpyDeviceToDevice, h->st));
  return refresh_copies(h);
}

tp_status pack_get_config(const tabpack_t* h, tp_config* cfg) {
  if (!h || !cfg) return fail(const_cast<tabpack_t*>(h), TP_EINVAL, "null argument");
  *cfg = h->cfg;
  return TP_OK;
}

tp_status pack_member_hparams(const tabpack_t* h, int32_t member, int32_t* depth, int32_t* width, float* dropout,
                              float* lr, float* wd) {
  if (!h) return fail(nullptr, TP_EINVAL, "null pack");
  if (member < 0 || member >= h->cfg.m) return fail(const_cast<tabpack_t*>(h), TP_EINVAL, "member %d out of range", member);
  if (depth) *depth = h->depth[member];
  if (width) *width = h->width[member];
  if (dropout) *dropout = h->dropout[member];
  if (lr) *lr = h->lr[member];
  if (wd) *wd = h->wd[member];
  return TP_OK;
}

tp_status pack_get_active(const tabpack_t* h, uint8_t* active) {
  if (!h || !active) return fail(const_cast<tabpack_t*>(h), TP_EINVAL, "null argument");
  for (int i = 0; i < h->cfg.m; ++i) active[i] = h->active[i];
  return TP_OK;
}

void* pack_get_stream(const tabpack_t* h) { return h ? (void*)h->st : nullptr; }

tp_status pack_get_logits(tabpack_t* h, int32_t member, float* out) {
  TP_TRY(check_ml(h, member, 0));
  if (!out) return fail(h, TP_EINVAL, "null out");
  TP_TRY(sync_check(h));
  TP_CUDA(h, cudaMemcpy(out, h->logits + (size_t)member * h->B_cap * h->cfg.d_out,
                        sizeof(float) * (size_t)h->last_B * h->cfg.d_out, cudaMemcpyDeviceToHost));
  return TP_OK;
}

tp_status pack_debug_masks(tabpack_t* h, int32_t member, int32_t layer, uint32_t step, int32_t B, uint8_t* keep) {
  TP_TRY(check_ml(h, member, layer));
  if (layer >= h->depth[member]) return fail(h, TP_EINVAL, "layer %d is the head", layer);
  if (B < 1 || !keep) return fail(h, TP_EINVAL, "bad B or null keep");
  const int w = h->width[member];
  uint8_t* d = nullptr;
  TP_CUDA(h, cudaMalloc(&d, (size_t)B * w));
  launch_debug_masks(h->st, d, B, w, h->cfg.seed, (uint32_t)member, (uint32_t)layer, step, h->mem[member].drop_T);
  h->launches++;
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
  if (e == cudaSuccess) e = cudaMemcpy(keep, d, (size_t)B * w, cudaMemcpyDeviceToHost);
  cudaFree(d);
  if (e != cudaSuccess) return fail(h, TP_ECUDA, "debug masks: %s", cudaGetErrorString(e));
  return TP_OK;
}

tp_status pack_debug_mask_arena(tabpack_t* h, int32_t member, int32_t layer, int32_t B, uint8_t* keep,
                                int64_t* step_held) {
  TP_TRY(check_ml(h, member, layer));
  if (layer >= h->depth[member]) return fail(h, TP_EINVAL, "layer %d is the head", layer);
  if (B < 1 || B > h->B_cap || !keep || !step_held) return fail(h, TP_EINVAL, "bad B or null output");
  if (!h->bf16) return fail(h, TP_ESTATE, "fp32 mode evaluates dropout in the epilogue: no mask arena");
  TP_TRY(sync_check(h));
  const int w = h->width[member];
  *step_held = h->masks_for;
  const int64_t off = h->mask_off[member][layer];
  if (off < 0) {  // p = 0: the forward applies no mask
    memset(keep, 1, (size_t)B * w);
    return TP_OK;
  }
  const int n_chunk = (int)ceil_div(w, 32);
  std::vector<uint32_t> words((size_t)n_chunk * h->B_cap);
  TP_CUDA(h, cudaMemcpy(words.data(), h->masks + off, sizeof(uint32_t) * words.size(), cudaMemcpyDeviceToHost));
  for (int r = 0; r < B; ++r)
    for (int c = 0; c < w; ++c)
      keep[(size_t)r * w + c] = (uint8_t)((words[(size_t)(c >> 5) * h->B_cap + r] >> (c & 31)) & 1u);
  return TP_OK;
}

tp_status pack_debug_gemm_timeout(tabpack_t* h, double wait_s, int32_t poison) {
  if (!h) return fail(nullptr, TP_EINVAL, "null pack");
  if (!h->bf16 || !h->tc.enabled) return fail(h, TP_ESTATE, "the tensor-core plan runs in bf16 mode only");
  if (!(wait_s > 0.0) || wait_s > 60.0) return fail(h, TP_EINVAL, "wait budget must be in (0, 60] s");
  TP_CUDA(h, cudaStreamSynchronize(h->st));
  const uint64_t ns = (uint64_t)(wait_s * 1e9);
  h->tc.wait_ns = ns;
  h->tcs.wait_ns = ns;
  h->tcp.wait_ns = ns;
  // captured graphs hold the old launch arguments
  for (auto& e : h->graphs) cudaGraphExecDestroy(e.exec);
  h->graphs.clear();
  if (poison) TP_TRY(tc_debug_poison(h->tc, h->st, h->err));
  return TP_OK;
}

tp_status pack_debug_bias_path(tabpack_t* h, int32_t mode) {
  if (!h) return fail(nullptr, TP_EINVAL, "null pack");
  if (mode < -1 || mode > 1) return fail(h, TP_EINVAL, "mode must be -1, 0 or 1");
  if (!h->bf16) return fail(h, TP_ESTATE, "the bias path choice exists in bf16 mode only");
  TP_TRY(sync_check(h));
  h->bias_colsums = mode < 0 ? auto_bias_colsums(h) : mode == 1;
  h->s_stale = true;
  return build_schedule(h);
}

tp_status pack_debug_philox(const uint32_t* ctr, const uint32_t* key, int32_t n, uint32_t* out) {
  if (n < 1 || !ctr || !key || !out) return fail(nullptr, TP_EINVAL, "bad n or null pointer");
  std::vector<uint32_t> in((size_t)n * 6);
  for (int32_t i = 0; i < n; ++i) {
    for (int q = 0; q < 4; ++q) in[(size_t)i * 6 + q] = ctr[(size_t)i * 4 + q];
    in[(size_t)i * 6 + 4] = key[(size_t)i * 2];
    in[(size_t)i * 6 + 5] = key[(size_t)i * 2 + 1];
  }
  uint32_t* d = nullptr;
  cudaError_t e = cudaMalloc(&d, sizeof(uint32_t) * (size_t)n * 10);
  if (e != cudaSuccess) return fail(nullptr, TP_ECUDA, "debug philox: %s", cudaGetErrorString(e));
  e = cudaMemcpy(d, in.data(), sizeof(uint32_t) * in.size(), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) {
    tp::launch_debug_philox(0, d, d + (size_t)n * 6, n);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaMemcpy(out, d + (size_t)n * 6, sizeof(uint32_t) * (size_t)n * 4, cudaMemcpyDeviceToHost);
  cudaFree(d);
  if (e != cudaSuccess) return fail(nullptr, TP_ECUDA, "debug philox: %s", cudaGetErrorString(e));
  return TP_OK;
}

tp_status pack_debug_activations(tabpack_t* h, int32_t member, int32_t layer, float* out) {
  TP_TRY(check_ml(h, member, layer));
  if (layer >= h->depth[member]) return fail(h, TP_EINVAL, "layer %d is the head", layer);
  if (!out) return fail(h, TP_EINVAL, "null out");
  TP_TRY(sync_check(h));
  const int w = h->width[member], ldh = ldh_of(h, member);
  const size_t n = (size_t)h->last_B * ldh;
  if (h->bf16) {
    std::vector<__nv_bfloat16> tmp(n);
    TP_CUDA(h, cudaMemcpy(tmp.data(), (const __nv_bfloat16*)h->act + h->act_off[member][layer], n * 2,
                          cudaMemcpyDeviceToHost));
    for (int r = 0; r < h->last_B; ++r)
      for (int c = 0; c < w; ++c) out[(size_t)r * w + c] = __bfloat162float(tmp[(size_t)r * ldh + c]);
  } else {
    std::vector<float> tmp(n);
    TP_CUDA(h, cudaMemcpy(tmp.data(), (const float*)h->act + h->act_off[member][layer], n * 4, cudaMemcpyDeviceToHost));
    for (int r = 0; r < h->last_B; ++r) std::memcpy(out + (size_t)r * w, tmp.data() + (size_t)r * ldh, (size_t)w * 4);
  }
  return TP_OK;
}

tp_status pack_select_greedy(const float* preds, int32_t P, int64_t N, int32_t d_out, const void* y, int32_t task,
                             int32_t score, int32_t m_ens, void* cuda_stream, int32_t* selected,
                             int32_t* n_selected, double* final_score) {
  if (!preds || !y || !selected || !n_selected) return fail(nullptr, TP_EINVAL, "null argument");
  if (P < 1 || N < 1 || m_ens < 1) return fail(nullptr, TP_EINVAL, "P, N, m_ens must be >= 1");
  if (task < 0 || task > 2 || score < 0 || score > 3) return fail(nullptr, TP_EINVAL, "unknown task/score");
  if (score == TP_SCORE_AUC && task != TP_BINARY) return fail(nullptr, TP_EINVAL, "auc needs a binary task");
  if (score == TP_SCORE_ACCURACY && task == TP_REGRESSION) return fail(nullptr, TP_EINVAL, "accuracy needs classification");
  if (score == TP_SCORE_RMSE && task != TP_REGRESSION) return fail(nullptr, TP_EINVAL, "rmse needs regression");
  if (task == TP_MULTICLASS ? (d_out < 2 || d_out > kMaxDout) : d_out != 1) return fail(nullptr, TP_EINVAL, "bad d_out");
  if (P > 65535) return fail(nullptr, TP_EINVAL, "P > 65535");
  cudaStream_t st = (cudaStream_t)cuda_stream;
  const int64_t bytes = select_scratch_bytes(P, N, d_out, m_ens, score);
  void* scratch = nullptr;
  cudaError_t e = cudaMallocAsync(&scratch, (size_t)bytes, st);
  if (e != cudaSuccess) return fail(nullptr, TP_ENOMEM, "cudaMallocAsync(%lld): %s", (long long)bytes, cudaGetErrorString(e));
  SelectScratch s = select_carve(scratch, P, N, d_out, m_ens, score);
  const int n_words = select_enqueue(st, s, preds, P, N, d_out, y, task, score, m_ens, nullptr, nullptr, nullptr);
  std::vector<int32_t> host(n_words);
  double cur = 0.0;
  e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaMemcpyAsync(host.data(), s.state, sizeof(int32_t) * n_words, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&cur, s.cur, sizeof(double), cudaMemcpyDeviceToHost, st);
  cudaError_t fe = cudaFreeAsync(scratch, st);
  if (e == cudaSuccess) e = fe;
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return fail(nullptr, TP_ECUDA, "select: %s", cudaGetErrorString(e));
  const int n = host[0];
  *n_selected = n;
  for (int k = 0; k < n; ++k) selected[k] = host[4 + k];
  if (final_score) *final_score = cur;
  return TP_OK;
}

tp_status pack_profile_enable(tabpack_t* h, int32_t enable) {
  if (!h) return fail(nullptr, TP_EINVAL, "null pack");
  h->profiling = enable != 0;
  return TP_OK;
}

tp_status pack_profile_read(tabpack_t* h, double* ms, int64_t* launches, int32_t reset) {
  if (!h) return fail(nullptr, TP_EINVAL, "null pack");
  prof_flush(h);
  TP_TRY(sync_check(h));
  for (int p = 0; p < TP_PH_COUNT; ++p) {
    if (ms) ms[p] = h->prof.ms[p];
    if (launches) launches[p] = h->prof.launches[p];
    if (reset) {
      h->prof.ms[p] = 0;
      h->prof.launches[p] = 0;
    }
  }
  return TP_OK;
}

int64_t pack_launch_count(const tabpack_t* h) { return h ? h->launches : -1; }

tp_status pack_sizes(const tabpack_t* h, int64_t* n_params, int64_t* device_bytes) {
  if (!h) return fail(nullptr, TP_EINVAL, "null pack");
  if (n_params) *n_params = h->n_params;
  if (device_bytes) *device_bytes = (int64_t)h->dev_bytes;
  return TP_OK;
}

const char* pack_last_error(const tabpack_t* h) { return h ? h->err.c_str() : g_thread_error.c_str(); }

}  // extern "C"
