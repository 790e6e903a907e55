// select_static.cu -- greedy ensemble selection that allocates no memory.
//
// pack_select_greedy obtains its scratch (the running ensemble sum, the
// per-block partial scores and the selection state) with cudaMallocAsync.
// Some callers cannot allocate device memory at the moment they select: a
// host process running under a fixed device-memory budget that has already
// been handed out, code inside an allocator callback or a memory-pool
// teardown, or an embedding runtime that forbids allocation calls after its
// start-up.  pack_select_greedy_static serves them: it runs the same kernels
// on a fixed scratch array that the library places in device memory when it
// is loaded (kStaticScratchBytes on every GPU the process uses, held until
// the process exits).
#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>

#include "kernels.cuh"
#include "tabpack.h"

namespace tp {

constexpr int64_t kStaticScratchBytes = 16ll << 20;   // 16 MiB
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_select_scratch[kStaticScratchBytes];

// Device address of g_select_scratch per device.  In host code the symbol
// names a host-side stand-in, never the device array, so the address is
// looked up with the device current and cached.  The cache entry remembers
// the context it was taken in: after a device reset (or the primary context
// being released and created again) the module is loaded anew, the context
// handle changes and the address is looked up again.
typedef int (*PFN_ctxGetCurrent)(void**);   // CUresult cuCtxGetCurrent(CUcontext*)

struct ScratchAddr {
  void* ctx = nullptr;
  void* addr = nullptr;
};
static ScratchAddr g_scratch_addr[kMaxDevices];
static std::mutex g_scratch_mu;

static void* current_context() {
  static PFN_ctxGetCurrent fn = nullptr;
  static bool looked = false;
  if (!looked) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (PFN_ctxGetCurrent)p;
    looked = true;
  }
  void* ctx = nullptr;
  if (fn == nullptr || fn(&ctx) != 0) return nullptr;
  return ctx;
}

static cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  void* ctx = current_context();
  ScratchAddr& c = g_scratch_addr[dev];
  if (c.addr == nullptr || ctx == nullptr || c.ctx != ctx) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_select_scratch);
    if (e != cudaSuccess) return e;
    c.addr = p;
    c.ctx = ctx;
  }
  *out = c.addr;
  return cudaSuccess;
}

}  // namespace tp

using namespace tp;

namespace {
tp_status static_fail(tp_status s, const char* msg, cudaError_t e = cudaSuccess) {
  char buf[256];
  if (e != cudaSuccess)
    snprintf(buf, sizeof buf, "%s: %s", msg, cudaGetErrorString(e));
  else
    snprintf(buf, sizeof buf, "%s", msg);
  record_thread_error(buf);
  return s;
}
}  // namespace

extern "C" {

tp_status pack_select_greedy_static(const float* preds, int32_t P, int64_t N, int32_t d_out, const void* y,
                                    int32_t task, int32_t score, int32_t m_ens, void* cuda_stream,
                                    int32_t* selected, int32_t* n_selected, double* final_score) {
  if (!preds || !y || !selected || !n_selected) return static_fail(TP_EINVAL, "null argument");
  if (P < 1 || N < 1 || m_ens < 1) return static_fail(TP_EINVAL, "P, N, m_ens must be >= 1");
  if (task < 0 || task > 2 || score < 0 || score > 3) return static_fail(TP_EINVAL, "unknown task/score");
  if (score == TP_SCORE_AUC && task != TP_BINARY) return static_fail(TP_EINVAL, "auc needs a binary task");
  if (score == TP_SCORE_ACCURACY && task == TP_REGRESSION)
    return static_fail(TP_EINVAL, "accuracy needs classification");
  if (score == TP_SCORE_RMSE && task != TP_REGRESSION) return static_fail(TP_EINVAL, "rmse needs regression");
  if (task == TP_MULTICLASS ? (d_out < 2 || d_out > kMaxDout) : d_out != 1) return static_fail(TP_EINVAL, "bad d_out");
  if (P > 65535) return static_fail(TP_EINVAL, "P > 65535");
  const int64_t need = select_scratch_bytes(P, N, d_out, m_ens, score);
  if (need > kStaticScratchBytes) {
    char buf[320];
    snprintf(buf, sizeof buf,
             "problem needs %lld bytes of scratch, the static array holds %lld (N * d_out * 8 + P * ceil(N/1024) * 8 "
             "+ (4 + m_ens + P) * 4 + 1024, plus P * N * 10 + 512 for the ROC-AUC score, must fit)",
             (long long)need, (long long)kStaticScratchBytes);
    return static_fail(TP_EINVAL, buf);
  }
  void* base = nullptr;
  cudaError_t e = scratch_address(&base);
  if (e != cudaSuccess) return static_fail(TP_ECUDA, "cudaGetSymbolAddress(scratch)", e);
  cudaStream_t st = (cudaStream_t)cuda_stream;
  SelectScratch s = select_carve(base, P, N, d_out, m_ens, score);
  // select_enqueue's first kernel zeroes the running sum and the state, so the
  // previous call's contents do not leak into this one.
  select_enqueue(st, s, preds, P, N, d_out, y, task, score, m_ens, nullptr, nullptr, nullptr);
  int32_t hdr[4] = {0, 0, 0, 0};
  double cur = 0.0;
  e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaMemcpyAsync(hdr, s.state, sizeof hdr, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&cur, s.cur, sizeof(double), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  // only the n selected slots reach the caller, as with pack_select_greedy
  const int32_t n = hdr[0] < 0 ? 0 : (hdr[0] > m_ens ? m_ens : hdr[0]);
  if (e == cudaSuccess && n > 0)
    e = cudaMemcpyAsync(selected, s.state + 4, sizeof(int32_t) * n, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess && n > 0) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return static_fail(TP_ECUDA, "select (static scratch)", e);
  *n_selected = n;
  if (final_score) *final_score = cur;
  return TP_OK;
}

}  // extern "C"
