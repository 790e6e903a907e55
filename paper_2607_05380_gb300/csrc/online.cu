// online.cu -- the online ensemble (Sec. 3.5 "Online ensemble") with the
// ensemble and base-model early stopping of Sec. 3.6.
//
// Once per epoch the ensemble is rebuilt from scratch by greedy selection
// over a pool of the active members' current states and the previous
// epoch's ensemble members.  Everything on the device goes through the
// pack's public entry points (predict, snapshot, set_active) and the
// selection kernels of select.cu; this file holds the bookkeeping.
//
// Device memory of one object:
//   pool   [m + m_ens, n_val, d_out] fp32: rows 0..m-1 the members' current
//          predictions (written by pack_predict), rows m.. the previous
//          ensemble's predictions in its selection order;
//   tmp    [m_ens, n_val, d_out] fp32: the new ensemble's rows, gathered
//          before they replace rows m..;
//   slots  [2 m_ens, slot_elems] fp32: parameter snapshots.  The instances
//          of the last ensemble and of the best ensemble each hold one
//          slot (an instance in both holds one), so 2 m_ens always suffice.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <limits>
#include <string>
#include <vector>

#include "kernels.cuh"
#include "tabpack.h"

using namespace tp;

namespace {

struct Instance {
  int32_t member, epoch, slot;
};

// out[e] = (sum_j p[j, e] in fp64, j ascending) * inv, rounded to fp32
__global__ void k_ens_mean(const float* __restrict__ p, int32_t n, int64_t n_e, double inv, float* __restrict__ out) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n_e; e += (int64_t)gridDim.x * blockDim.x) {
    double s = 0.0;
    for (int j = 0; j < n; ++j) s += (double)p[(int64_t)j * n_e + e];
    out[e] = (float)(s * inv);
  }
}

}  // namespace

struct tabpack_online {
  tabpack_t* pack = nullptr;
  tp_config cfg{};
  int64_t n_val = 0;
  int32_t score = 0, m_ens = 0, p_base = 0, p_ens = 0;
  int64_t slot_elems = 0, row_elems = 0;  // row_elems = n_val * d_out
  int n_slots = 0;

  float* pool = nullptr;
  float* tmp = nullptr;
  float* slots = nullptr;
  void* scratch = nullptr;
  uint8_t* excl_dev = nullptr;
  double* solo_dev = nullptr;

  std::vector<Instance> last, best;
  std::vector<uint8_t> slot_busy;
  std::vector<double> m_score, m_best;
  std::vector<int32_t> m_bad;
  double best_score = std::numeric_limits<double>::infinity();
  double last_score = std::numeric_limits<double>::quiet_NaN();
  int32_t epoch = 0, best_epoch = 0, ens_bad = 0, stop = 0, n_pool = 0;

  tabpack_t* ens_pack = nullptr;  // the best ensemble's instances as members
  int32_t ens_pack_epoch = -1;    // best_epoch it was built for
  float* ens_out = nullptr;
  int64_t ens_out_cap = 0;

  std::string err;
};

namespace {

tp_status ofail(tabpack_online* o, tp_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  if (o) o->err = buf;
  else record_thread_error(buf);
  return s;
}

// a failed pack call: keep the pack's message
tp_status pack_fail(tabpack_online* o, tabpack_t* pack, tp_status s, const char* what) {
  return ofail(o, s, "%s: %s", what, pack_last_error(pack));
}

#define O_CUDA(o, call)                                                                           \
  do {                                                                                            \
    cudaError_t e_ = (call);                                                                      \
    if (e_ != cudaSuccess)                                                                        \
      return ofail((o), e_ == cudaErrorMemoryAllocation ? TP_ENOMEM : TP_ECUDA, "%s: %s (%s:%d)", \
                   #call, cudaGetErrorString(e_), __FILE__, __LINE__);                            \
  } while (0)

#define O_PACK(o, pk, call, what)            \
  do {                                       \
    tp_status s_ = (call);                   \
    if (s_ != TP_OK) return pack_fail((o), (pk), s_, (what)); \
  } while (0)

void free_online(tabpack_online* o) {
  if (o->ens_pack) pack_destroy(o->ens_pack);
  for (void* p : {(void*)o->pool, (void*)o->tmp, (void*)o->slots, o->scratch, (void*)o->excl_dev,
                  (void*)o->solo_dev, (void*)o->ens_out})
    if (p) cudaFree(p);
}

float* slot_ptr(tabpack_online* o, int slot) { return o->slots + (int64_t)slot * o->slot_elems; }

// (Re)build the pack whose members are the best ensemble's instances.
tp_status build_ens_pack(tabpack_online* o) {
  if (o->ens_pack && o->ens_pack_epoch == o->best_epoch) return TP_OK;
  if (o->ens_pack) {
    pack_destroy(o->ens_pack);
    o->ens_pack = nullptr;
  }
  const int n = (int)o->best.size();
  std::vector<int32_t> depth(n), width(n);
  std::vector<float> drop(n), lr(n), wd(n);
  for (int j = 0; j < n; ++j)
    O_PACK(o, o->pack, pack_member_hparams(o->pack, o->best[j].member, &depth[j], &width[j], &drop[j], &lr[j], &wd[j]),
           "pack_member_hparams");
  tp_config c = o->cfg;
  c.m = n;
  c.fuse_optimizer = 0;
  // members with periodic embeddings: the same sizes (the frequencies are
  // placeholders, every parameter comes from the snapshot)
  std::vector<int32_t> d_emb(n);
  int64_t n_freq = 0;
  for (int j = 0; j < n; ++j) {
    O_PACK(o, o->pack, pack_member_emb(o->pack, o->best[j].member, &d_emb[j]), "pack_member_emb");
    n_freq += (int64_t)c.d_in * std::max(d_emb[j] - 1, 0);
  }
  tabpack_t* ep = nullptr;
  tp_status s;
  if (n > 0 && d_emb[0] > 0) {
    std::vector<float> freq((size_t)std::max<int64_t>(n_freq, 1), 0.f);
    s = pack_create_emb(&c, depth.data(), width.data(), drop.data(), lr.data(), wd.data(), d_emb.data(), freq.data(),
                        pack_get_stream(o->pack), &ep);
  } else {
    s = pack_create(&c, depth.data(), width.data(), drop.data(), lr.data(), wd.data(), pack_get_stream(o->pack), &ep);
  }
  if (s != TP_OK) return pack_fail(o, nullptr, s, "pack_create (ensemble)");
  o->ens_pack = ep;
  for (int j = 0; j < n; ++j)
    O_PACK(o, ep, pack_restore(ep, j, slot_ptr(o, o->best[j].slot)), "pack_restore (ensemble)");
  o->ens_pack_epoch = o->best_epoch;
  return TP_OK;
}

}  // namespace

extern "C" {

tp_status pack_online_create(tabpack_t* pack, int64_t n_val, int32_t score, int32_t m_ens, int32_t p_base,
                             int32_t p_ens, tabpack_online_t** out) {
  if (out) *out = nullptr;
  if (!pack || !out) return ofail(nullptr, TP_EINVAL, "null argument");
  tp_config cfg;
  if (pack_get_config(pack, &cfg) != TP_OK) return ofail(nullptr, TP_EINVAL, "bad pack");
  if (n_val < 1 || m_ens < 1 || p_base < 0 || p_ens < 0)
    return ofail(nullptr, TP_EINVAL, "n_val, m_ens must be >= 1 and p_base, p_ens >= 0");
  if (score < 0 || score > 3) return ofail(nullptr, TP_EINVAL, "unknown score %d", score);
  if (score == TP_SCORE_AUC && cfg.task != TP_BINARY) return ofail(nullptr, TP_EINVAL, "auc needs a binary task");
  if (score == TP_SCORE_ACCURACY && cfg.task == TP_REGRESSION) return ofail(nullptr, TP_EINVAL, "accuracy needs classification");
  if (score == TP_SCORE_RMSE && cfg.task != TP_REGRESSION) return ofail(nullptr, TP_EINVAL, "rmse needs regression");
  const int64_t P_max = (int64_t)cfg.m + m_ens;
  if (P_max > 65535) return ofail(nullptr, TP_EINVAL, "m + m_ens > 65535");

  tabpack_online* o = new tabpack_online();
  o->pack = pack;
  o->cfg = cfg;
  o->n_val = n_val;
  o->score = score;
  o->m_ens = m_ens;
  o->p_base = p_base;
  o->p_ens = p_ens;
  o->row_elems = n_val * cfg.d_out;
  o->n_slots = 2 * m_ens;
  for (int i = 0; i < cfg.m; ++i) {
    int64_t n = 0;
    pack_member_size(pack, i, &n);
    o->slot_elems = std::max(o->slot_elems, round_up(n, 64));  // 256-byte aligned slots
  }
  o->slot_busy.assign(o->n_slots, 0);
  o->m_score.assign(cfg.m, std::numeric_limits<double>::quiet_NaN());
  o->m_best.assign(cfg.m, std::numeric_limits<double>::infinity());
  o->m_bad.assign(cfg.m, 0);

  auto alloc = [&](void** p, size_t bytes) -> tp_status {
    cudaError_t e = cudaMalloc(p, bytes);
    if (e != cudaSuccess) {
      *p = nullptr;
      return ofail(nullptr, TP_ENOMEM, "cudaMalloc(%zu): %s", bytes, cudaGetErrorString(e));
    }
    return TP_OK;
  };
  tp_status s = alloc((void**)&o->pool, (size_t)(P_max * o->row_elems) * 4);
  if (s == TP_OK) s = alloc((void**)&o->tmp, (size_t)((int64_t)m_ens * o->row_elems) * 4);
  if (s == TP_OK) s = alloc((void**)&o->slots, (size_t)((int64_t)o->n_slots * o->slot_elems) * 4);
  if (s == TP_OK) s = alloc(&o->scratch, (size_t)select_scratch_bytes((int32_t)P_max, n_val, cfg.d_out, m_ens, score));
  if (s == TP_OK) s = alloc((void**)&o->excl_dev, (size_t)P_max);
  if (s == TP_OK) s = alloc((void**)&o->solo_dev, (size_t)P_max * 8);
  if (s != TP_OK) {
    free_online(o);
    delete o;
    return s;
  }
  *out = o;
  return TP_OK;
}

void pack_online_destroy(tabpack_online_t* o) {
  if (!o) return;
  cudaStreamSynchronize((cudaStream_t)pack_get_stream(o->pack));
  free_online(o);
  delete o;
}

tp_status pack_online_epoch(tabpack_online_t* o, const float* X_val, const void* y_val, int32_t* stop) {
  if (!o) return ofail(nullptr, TP_EINVAL, "null online ensemble");
  if (!X_val || !y_val) return ofail(o, TP_EINVAL, "X_val and y_val must be device pointers");
  if (o->stop) return ofail(o, TP_ESTATE, "training has stopped (epoch %d)", o->epoch);
  tabpack_t* pk = o->pack;
  const int m = o->cfg.m;
  cudaStream_t st = (cudaStream_t)pack_get_stream(pk);
  std::vector<uint8_t> active(m);
  O_PACK(o, pk, pack_get_active(pk, active.data()), "pack_get_active");
  if (std::count(active.begin(), active.end(), 1) == 0) return ofail(o, TP_ESTATE, "no active member");
  const int32_t e = o->epoch + 1;
  const int n_prev = (int)o->last.size();
  const int32_t P = m + n_prev;

  // 1. current predictions of the active members: pool rows 0..m-1
  O_PACK(o, pk, pack_predict(pk, X_val, o->n_val, o->pool), "pack_predict");
  // 2. the pool: inactive members take no part
  std::vector<uint8_t> excl(P, 0);
  int n_pool = n_prev;
  for (int i = 0; i < m; ++i) {
    excl[i] = active[i] ? 0 : 1;
    n_pool += active[i] ? 1 : 0;
  }
  O_CUDA(o, cudaMemcpyAsync(o->excl_dev, excl.data(), (size_t)P, cudaMemcpyHostToDevice, st));
  // 3. greedy selection, with every candidate's own score on the side
  SelectScratch ss = select_carve(o->scratch, P, o->n_val, o->cfg.d_out, o->m_ens, o->score);
  const int n_words = select_enqueue(st, ss, o->pool, P, o->n_val, o->cfg.d_out, y_val, o->cfg.task, o->score,
                                     o->m_ens, o->excl_dev, o->solo_dev, nullptr);
  O_CUDA(o, cudaGetLastError());
  std::vector<int32_t> state(n_words);
  std::vector<double> solo(P);
  double fin = 0.0;
  O_CUDA(o, cudaMemcpyAsync(state.data(), ss.state, sizeof(int32_t) * n_words, cudaMemcpyDeviceToHost, st));
  O_CUDA(o, cudaMemcpyAsync(&fin, ss.cur, sizeof(double), cudaMemcpyDeviceToHost, st));
  O_CUDA(o, cudaMemcpyAsync(solo.data(), o->solo_dev, sizeof(double) * P, cudaMemcpyDeviceToHost, st));
  O_CUDA(o, cudaStreamSynchronize(st));
  const int n_sel = state[0];
  const int32_t* sel = state.data() + 4;

  // 4. base-model early stopping on each active member's own score
  std::vector<int> removed;
  for (int i = 0; i < m; ++i) {
    if (!active[i]) {
      o->m_score[i] = std::numeric_limits<double>::quiet_NaN();
      continue;
    }
    const double sc = solo[i];
    o->m_score[i] = sc;
    if (sc < o->m_best[i]) {
      o->m_best[i] = sc;
      o->m_bad[i] = 0;
    } else {
      o->m_bad[i] += 1;
    }
    if (o->m_bad[i] >= o->p_base + 1) removed.push_back(i);
  }

  // 5. the new ensemble as instances; earlier instances keep their slots
  std::vector<Instance> now(n_sel);
  for (int k = 0; k < n_sel; ++k) {
    const int c = sel[k];
    now[k] = c < m ? Instance{c, e, -1} : o->last[c - m];
  }
  const bool improved = n_sel > 0 && fin < o->best_score;
  std::fill(o->slot_busy.begin(), o->slot_busy.end(), 0);
  for (const Instance& in : now)
    if (in.slot >= 0) o->slot_busy[in.slot] = 1;
  if (!improved)
    for (const Instance& in : o->best) o->slot_busy[in.slot] = 1;
  for (Instance& in : now) {
    if (in.slot >= 0) continue;
    int s = 0;
    while (s < o->n_slots && o->slot_busy[s]) ++s;
    if (s == o->n_slots) return ofail(o, TP_ESTATE, "no free snapshot slot (internal)");
    o->slot_busy[s] = 1;
    in.slot = s;
    O_PACK(o, pk, pack_snapshot(pk, in.member, slot_ptr(o, s)), "pack_snapshot");
  }
  // 6. the new ensemble's predictions become pool rows m.. for the next epoch
  const size_t row_bytes = (size_t)o->row_elems * 4;
  for (int k = 0; k < n_sel; ++k)
    O_CUDA(o, cudaMemcpyAsync(o->tmp + (int64_t)k * o->row_elems, o->pool + (int64_t)sel[k] * o->row_elems, row_bytes,
                              cudaMemcpyDeviceToDevice, st));
  if (n_sel > 0)
    O_CUDA(o, cudaMemcpyAsync(o->pool + (int64_t)m * o->row_elems, o->tmp, row_bytes * n_sel, cudaMemcpyDeviceToDevice, st));

  // 7. ensemble early stopping
  if (improved) {
    o->best = now;
    o->best_score = fin;
    o->best_epoch = e;
    o->ens_bad = 0;
  } else {
    o->ens_bad += 1;
  }
  o->last = now;
  o->last_score = n_sel > 0 ? fin : std::numeric_limits<double>::quiet_NaN();
  o->epoch = e;
  o->n_pool = n_pool;

  // 8. members that stopped improving leave the pack
  int n_active = 0;
  for (int i : removed) active[i] = 0;
  for (int i = 0; i < m; ++i) n_active += active[i];
  if (!removed.empty()) O_PACK(o, pk, pack_set_active(pk, active.data()), "pack_set_active");
  O_CUDA(o, cudaStreamSynchronize(st));
  o->stop = (o->ens_bad >= o->p_ens + 1 || n_active == 0) ? 1 : 0;
  if (stop) *stop = o->stop;
  return TP_OK;
}

tp_status pack_online_info(const tabpack_online_t* o, tp_online_info* info) {
  if (!o || !info) return ofail(const_cast<tabpack_online_t*>(o), TP_EINVAL, "null argument");
  std::vector<uint8_t> active(o->cfg.m);
  pack_get_active(o->pack, active.data());
  info->epoch = o->epoch;
  info->stop = o->stop;
  info->n_active = (int32_t)std::count(active.begin(), active.end(), 1);
  info->ens_bad = o->ens_bad;
  info->best_epoch = o->best_epoch;
  info->n_best = (int32_t)o->best.size();
  info->n_last = (int32_t)o->last.size();
  info->n_pool = o->n_pool;
  info->best_score = o->best_score;
  info->last_score = o->last_score;
  return TP_OK;
}

tp_status pack_online_members(const tabpack_online_t* o, double* score, double* best, int32_t* bad) {
  if (!o) return ofail(nullptr, TP_EINVAL, "null online ensemble");
  for (int i = 0; i < o->cfg.m; ++i) {
    if (score) score[i] = o->m_score[i];
    if (best) best[i] = o->m_best[i];
    if (bad) bad[i] = o->m_bad[i];
  }
  return TP_OK;
}

tp_status pack_online_ensemble(const tabpack_online_t* o, int32_t which, int32_t* member, int32_t* epoch, int32_t* n,
                               double* score) {
  if (!o || !n) return ofail(const_cast<tabpack_online_t*>(o), TP_EINVAL, "null argument");
  if (which != 0 && which != 1) return ofail(const_cast<tabpack_online_t*>(o), TP_EINVAL, "which must be 0 or 1");
  const std::vector<Instance>& v = which == 0 ? o->best : o->last;
  for (size_t k = 0; k < v.size(); ++k) {
    if (member) member[k] = v[k].member;
    if (epoch) epoch[k] = v[k].epoch;
  }
  *n = (int32_t)v.size();
  if (score) *score = which == 0 ? o->best_score : o->last_score;
  return TP_OK;
}

tp_status pack_online_snapshot(tabpack_online_t* o, int32_t j, float* dst) {
  if (!o || !dst) return ofail(o, TP_EINVAL, "null argument");
  if (j < 0 || j >= (int)o->best.size()) return ofail(o, TP_EINVAL, "instance %d out of range (best ensemble has %d)",
                                                      j, (int)o->best.size());
  int64_t n = 0;
  O_PACK(o, o->pack, pack_member_size(o->pack, o->best[j].member, &n), "pack_member_size");
  cudaStream_t st = (cudaStream_t)pack_get_stream(o->pack);
  O_CUDA(o, cudaMemcpyAsync(dst, slot_ptr(o, o->best[j].slot), (size_t)n * 4, cudaMemcpyDeviceToDevice, st));
  O_CUDA(o, cudaStreamSynchronize(st));
  return TP_OK;
}

tp_status pack_online_predict(tabpack_online_t* o, const float* X, int64_t N, float* out) {
  if (!o) return ofail(nullptr, TP_EINVAL, "null online ensemble");
  if (!X || !out || N < 1) return ofail(o, TP_EINVAL, "X/out null or N < 1");
  if (o->best.empty()) return ofail(o, TP_ESTATE, "no ensemble yet");
  cudaStream_t st = (cudaStream_t)pack_get_stream(o->pack);
  if (tp_status s = build_ens_pack(o); s != TP_OK) return s;
  O_PACK(o, o->ens_pack, pack_set_stream(o->ens_pack, st), "pack_set_stream");
  const int n = (int)o->best.size();
  const int64_t n_e = N * o->cfg.d_out;
  if (o->ens_out_cap < (int64_t)n * n_e) {
    O_CUDA(o, cudaStreamSynchronize(st));
    if (o->ens_out) cudaFree(o->ens_out);
    o->ens_out = nullptr;
    o->ens_out_cap = 0;
    O_CUDA(o, cudaMalloc((void**)&o->ens_out, (size_t)n * n_e * 4));
    o->ens_out_cap = (int64_t)n * n_e;
  }
  O_PACK(o, o->ens_pack, pack_predict(o->ens_pack, X, N, o->ens_out), "pack_predict (ensemble)");
  const int blocks = (int)std::min<int64_t>(ceil_div(n_e, 256), 152 * 8);
  k_ens_mean<<<blocks, 256, 0, st>>>(o->ens_out, n, n_e, 1.0 / (double)n, out);
  O_CUDA(o, cudaGetLastError());
  return TP_OK;
}

const char* pack_online_last_error(const tabpack_online_t* o) { return o ? o->err.c_str() : pack_last_error(nullptr); }

}  // extern "C"
