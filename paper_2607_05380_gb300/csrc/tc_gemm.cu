// tc_gemm.cu -- persistent warp-specialised grouped GEMM on tcgen05 (sm_103a).
//
// One launch runs every forward product of the step (all members, all
// depths), another every backward product: a list of 128 x N output tiles
// (N <= 256, a multiple of 16) that each persistent CTA (one per SM) walks
// with stride gridDim.x.  The list is ordered by dependency level (forward:
// the layer; backward: the distance from the head, with each level's wgrad
// tiles moved beside the next level's dgrad tiles) and by cost, largest
// first, within a level.  A tile whose A operand is produced in the same
// launch waits for a row-block completion counter (the producer polls it
// with acquire loads, bounded); every epilogue warp publishes its stores
// with a release add when it finishes a tile.  All CTAs are resident at once
// (grid <= SMs, one CTA per SM), and a tile only waits on tiles earlier in
// the list, so the waits always end.  Warp roles:
//   warp 0     TMA producer: per 64-wide K block, loads the A tile
//              (2 boxes of 64 x 64 bf16) and the B tile (N/64 boxes) into a
//              4-stage shared-memory ring, 128-byte swizzled.
//   warp 1     MMA issuer: one thread issues tcgen05.mma (M=128, K=16 per
//              instruction) into one of two TMEM accumulators (2 x 256
//              fp32 columns) and commits each stage back to the producer.
//   warp 10    publisher: per stored tile, the release count that tiles in
//              other CTAs wait on (so that the epilogue warps do not wait for
//              their stores to drain before starting the next tile)
//   warps 2-9  epilogue: tcgen05.ld of the accumulator (warp w reads TMEM
//              lanes 32 (w % 4) .. +31, i.e. those output rows; the two
//              warps of a lane quarter take alternate 32-column chunks) and
//              the fused epilogue of the product kind:
//                kFwd   z = acc + b; h = dropout(relu(z)) / (1 - p)   -> bf16
//                kDgrad dz_prev = acc * [H_prev > 0] / (1 - p)          -> bf16
//                       (and, where the layer's wgrad wants them, its column
//                       sums over each warp's 32 rows)
//                kWgrad dW, db = acc (the bias column) or the sum of dZ's
//                       column sums (store), or AdamW(p, m, v; dW, db) with
//                       the fp32 master, the moments and the bf16 copy
// Ragged K (member widths that are multiples of 16 but not of 64) issues
// only the K=16 steps that exist; out-of-range operand rows and columns are
// zero-filled by TMA.  Operands are read K-major or MN-major straight from
// their row-major arrays through the descriptor's major-ness bits, so no
// transposed copies are kept.  Because the weight-gradient reduction runs
// over the whole batch inside one tile, the fused AdamW sees final gradients
// and they never travel through HBM.
//
// Every mbarrier wait is bounded (2 s): a role that gives up sets the
// pack's device error word and an abort flag in shared memory; the other
// roles then stop, the producer waits (bounded) for its own copies in
// flight, the MMA thread for its own MMAs, TMEM is freed and the CTA exits.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstdio>
#include <cstdlib>

#include "tc_gemm.cuh"

namespace tp {
namespace {

constexpr int kBoxBytes = 64 * 64 * 2;  // one 64 x 64 bf16 TMA box
constexpr int kABytes = 2 * kBoxBytes;  // 128 rows of A per CTA
// Epilogue warps: one or two per TMEM lane quarter.  Eight (the default)
// halve each warp's share of a tile's columns; four keep every SM
// sub-partition at two warps (a 255-register cap, and the MMA issuer shares
// its sub-partition with one epilogue warp) but were measured slower: the
// longer epilogue of a tile delays the next accumulator.
#ifndef TP_EPI_WARPS
#define TP_EPI_WARPS 8
#endif
constexpr int kEpiWarps = TP_EPI_WARPS;
static_assert(kEpiWarps == 4 || kEpiWarps == 8, "one or two epilogue warps per TMEM lane quarter");
constexpr int kEpiPerQ = kEpiWarps / 4;         // epilogue warps per lane quarter
constexpr int kChunks = 8 / kEpiPerQ;           // 32-column chunks per warp of a 256-column tile
constexpr int kThreads = 96 + 32 * kEpiWarps;   // producer warp, MMA warp, epilogue warps, publisher warp
constexpr int kPubWarp = 2 + kEpiWarps;
constexpr int kPubSlots = 4;                    // tiles in flight between the epilogue and the publisher
constexpr uint32_t kTmemCols = 512;
constexpr int kAccCols = 256;
constexpr uint64_t kWaitNs = 2000000000ull;
// per epilogue warp a 32 x 32 fp32 transpose buffer (wgrad epilogue)
constexpr int kTrBytes = kEpiWarps * 32 * 32 * 4;

// Pipeline geometry for tiles of kCta CTAs.  kCta = 1: a CTA computes
// 128 x N and stages 128 rows of A and up to 256 rows / columns of B per K
// block (48 KB, 4 stages).  kCta = 2: a CTA pair computes 256 x N with
// cta_group::2 MMAs; each CTA stages its own 128 rows of A and half of B
// (32 KB, 6 stages), so a CTA streams two thirds of the bytes per FLOP and
// keeps half again as many K blocks in flight.
template <int kCta>
struct Geo {
  static constexpr int kStages = kCta == 2 ? 6 : 4;
  static constexpr int kBBytes = (kCta == 2 ? 2 : 4) * kBoxBytes;
  static constexpr int kStageBytes = kABytes + kBBytes;
};
template <int kStages>
struct SmemTail {
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t stored[kPubSlots];    // the epilogue warps have stored a tile (one arrival each)
  uint64_t pub_free[kPubSlots];  // the publisher has counted it
  uint64_t done;
  uint32_t tmem_base;
  int abort;
};
template <int kCta>
constexpr int smem_bytes() {
  return Geo<kCta>::kStages * Geo<kCta>::kStageBytes + kTrBytes + 1024 +
         (int)sizeof(SmemTail<Geo<kCta>::kStages>) + 64;
}
static_assert(smem_bytes<1>() <= 232448 && smem_bytes<2>() <= 232448, "shared memory per CTA");

struct TcArgs {
  const TcTile* tiles;
  int32_t n_tiles;
  int32_t B, B_pad;
  int32_t train;
  int32_t mask_rows;  // rows of a chunk of keep words in the mask arena
  int32_t w_shift;  // added to the weight-map index of kFwd / kDgrad tiles (weight copy)
  int32_t update;   // kWgrad: 1 = fused AdamW, 0 = store gradients
  const uint32_t* masks;  // dropout keep words of the step (train)
  const CUtensorMap* maps;
  const float* params;
  const MemberDev* mem;
  __nv_bfloat16* act;
  __nv_bfloat16* dz;
  float* grads;
  AdamDev adam;
  int* err;
  int* cnt;            // row-block completion counters
  int32_t kmaj_off;    // index distance to the same matrix's map with 128-row boxes (K-major loads)
  __nv_bfloat16* ns;   // Newton-Schulz arena (kNs launches)
  const float* ns_scale;  // per Muon matrix: 1 / |U|_F (kNs launches)
  uint64_t wait_ns;    // budget of every wait that can give up (TcPlan::wait_ns)
  float* dbp;          // column-sum partials of dZ (kDgrad writes them, kWgrad reads them)
};

// ------------------------------------------------------------ PTX helpers
__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait: false if the abort flag is raised or the budget runs out
// (then the flag and the device error word are set).
// A wait that gives up records its site code in the error word (the first
// one wins): 1 producer stage empty, 3 producer dependency, 5 MMA
// accumulator free, 6 MMA stage full, 7 epilogue accumulator full, 10 final
// copy drain, 12 final MMA drain, 8 epilogue publish slot, 9 publisher,
// 13 epilogue Newton-Schulz dependency, 14 epilogue bias-partial dependency.
// The MMA and epilogue waits (5, 6, 7, 8) wait on another role of the same
// CTA and take twice the budget of the producer's, the publisher's (9) four
// times, so a stalled dependency is reported as its own site.
__device__ __noinline__ bool mbar_wait_slow(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* err,
                                            uint64_t budget_ns, int site) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (global_ns() - t0 > budget_ns) {
      *abort_flag = 1;
      atomicCAS(err, 0, site);
      return false;
    }
  }
}

__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* err,
                                          uint64_t budget_ns, int site) {
  return mbar_try_wait(bar, parity) || mbar_wait_slow(bar, parity, abort_flag, err, budget_ns, site);
}

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void red_release_add(int* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
// Generic-proxy writes of other CTAs, acquired through a counter, become
// visible to this thread's subsequent TMA (async-proxy) reads.
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Bounded wait, by the whole warp, until counters p[0 .. n-1] each reach
// `need`.  Lane j polls counters j, j + 32, ...: a weight-gradient tile waits
// on every row block of its operand (16 counters for 2048 rows), and one
// lane reading them in turn paid 16 acquire round trips to L2 per tile even
// when all were long complete.  The warp barrier orders every lane after all
// lanes' acquires; the caller's proxy fence follows it.
__device__ __noinline__ bool dep_wait(const int* p, int n, int need, volatile int* abort_flag, int* err,
                                      uint64_t budget_ns, int site, int lane) {
  bool mine = true;
  for (int j = lane; mine && j < n; j += 32) {
    if (ld_acquire(p + j) >= need) continue;
    const uint64_t t0 = global_ns();
    while (ld_acquire(p + j) < need) {
      if (*abort_flag) {
        mine = false;
        break;
      }
      if (global_ns() - t0 > budget_ns) {
        *abort_flag = 1;
        atomicCAS(err, 0, site);
        mine = false;
        break;
      }
      __nanosleep(32);
    }
  }
  __syncwarp();
  return __all_sync(0xffffffffu, mine);
}

// Column sums of a warp's 32 x 32 chunk (lane = row, c[j] = column j):
// halving exchanges (16 + 8 + 4 + 2 + 1 shuffles), after which lane l
// holds column l's sum in c[0].  The order of the additions is fixed.
template <int W>
__device__ __forceinline__ void colsum_halve(float (&c)[32], int lane) {
  const bool up = (lane & W) != 0;
#pragma unroll
  for (int k = 0; k < W; ++k) {
    const float keep = up ? c[W + k] : c[k];
    const float send = up ? c[k] : c[W + k];
    c[k] = keep + __shfl_xor_sync(0xffffffffu, send, W);
  }
}
__device__ __forceinline__ float colsum32(float (&c)[32], int lane) {
  colsum_halve<16>(c, lane);
  colsum_halve<8>(c, lane);
  colsum_halve<4>(c, lane);
  colsum_halve<2>(c, lane);
  colsum_halve<1>(c, lane);
  return c[0];
}

// p[0] + p[ld] + ... + p[(n - 1) ld], added in that order (kept out of line:
// inlined, its loop state raised the epilogue's register spills).
__device__ __noinline__ float sum_strided(const float* p, int n, int ld) {
  float s = 0.f;
#pragma unroll 8
  for (int i = 0; i < n; ++i) s += p[(int64_t)i * ld];
  return s;
}

// Bulk prefetch of `bytes` (a multiple of 16; 16-byte aligned address) into L2.
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint64_t* bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
      "l"(map), "r"(smem_u32(bar)), "r"(x), "r"(y)
      : "memory");
}
// Copy of a box into this CTA's shared memory whose completion is counted on
// the mbarrier at shared::cluster address `bar`, which may belong to the
// peer CTA of the pair (cta_group::2).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], "
      "[%2];" ::"r"(dst),
      "l"(map), "r"(bar), "r"(x), "r"(y)
      : "memory");
}
// shared::cluster address of this CTA's shared variable at `addr` in CTA `rank`
__device__ __forceinline__ uint32_t mapa(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar) : "memory");
}
// Arrivals that order no memory accesses of the arriving thread.  A release
// arrival waits until the thread's earlier global stores are performed at its
// scope; the epilogue's accumulator hand-back follows tcgen05.wait::ld, which
// has already completed every TMEM read it covers, so it needs no release.
__device__ __forceinline__ void mbar_arrive_relaxed(uint64_t* bar) {
  asm volatile("mbarrier.arrive.relaxed.cta.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_cluster_relaxed(uint32_t bar) {
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor: start, leading / stride byte offsets,
// version 1 (bits 46-48), 128-byte swizzle (layout 2, bits 61-63).
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = (uint64_t)((addr >> 4) & 0x3FFFu);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Instruction descriptor of kind::f16: fp32 accumulate, bf16 A and B.
__device__ __forceinline__ uint32_t instr_desc(int m, int n, int a_mn, int b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)a_mn << 15) | ((uint32_t)b_mn << 16) |
         ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

template <int kCta>
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  if constexpr (kCta == 2)
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(
            d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
  else
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(
            d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}
// Arrive on `bar` once this thread's MMAs so far have completed; for a CTA
// pair on the mbarrier at `bar`'s offset in both CTAs.
template <int kCta>
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  if constexpr (kCta == 2)
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
            smem_u32(bar)),
        "h"((uint16_t)3)
        : "memory");
  else
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
        "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]),
        "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
        "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  __nv_bfloat162 t = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&t);
}

// One chunk of an epilogue warp's bf16 output -- its 32 rows (lane = row)
// by 32 columns -- written as row segments: each lane puts its row's four
// 16-byte groups into the warp's transpose buffer (XOR-swizzled by row, so
// that both the row-wise write and the segment-wise read are free of bank
// conflicts; stage_group), and flush_chunk reads them back four lanes per row,
// so that every store instruction writes eight whole 64-byte row segments
// instead of 32 half sectors of 32 different rows.
__device__ __forceinline__ void stage_group(uint8_t* buf, int lane, int s, uint32_t a, uint32_t b, uint32_t c,
                                            uint32_t d) {
  *reinterpret_cast<uint4*>(buf + lane * 64 + 16 * (s ^ ((lane >> 1) & 3))) = make_uint4(a, b, c, d);
}
// out: the warp's first row at the chunk's first column; rows from rbase on
// are valid below m_lim, columns below ncols.  kAhead: the four shared
// loads first, then the four stores (16 more registers, no load-to-store
// round trip per row group).
template <bool kAhead = false>
__device__ __forceinline__ void flush_chunk(uint8_t* buf, int lane, __nv_bfloat16* out, int64_t ldc, int rbase,
                                            int m_lim, int ncols) {
  __syncwarp();
  const int seg = lane & 3;
  if constexpr (kAhead) {
    uint4 val[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int rl = 8 * j + (lane >> 2);
      val[j] = *reinterpret_cast<const uint4*>(buf + rl * 64 + 16 * (seg ^ ((rl >> 1) & 3)));
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int rl = 8 * j + (lane >> 2);
      if (rbase + rl < m_lim && 8 * seg < ncols) *reinterpret_cast<uint4*>(out + (int64_t)rl * ldc + 8 * seg) = val[j];
    }
  } else {
#pragma unroll 1
    for (int j = 0; j < 4; ++j) {
      const int rl = 8 * j + (lane >> 2);
      const uint4 val = *reinterpret_cast<const uint4*>(buf + rl * 64 + 16 * (seg ^ ((rl >> 1) & 3)));
      if (rbase + rl < m_lim && 8 * seg < ncols) *reinterpret_cast<uint4*>(out + (int64_t)rl * ldc + 8 * seg) = val;
    }
  }
  __syncwarp();  // the buffer is reused by the next chunk
}

// The transpose of a chunk staged by stage_group in `src`, staged the same
// way in `dst`: per group S of source columns, ldmatrix .trans reads the four
// 8 x 8 blocks of rows 8 k .. 8 k + 7 (k = 0..3) transposed and stmatrix
// writes them as rows 8 S .. 8 S + 7, group k, of dst.  Lane l addresses row
// l % 8 of block l / 8; the XOR swizzle keeps both conflict-free.  The
// caller orders the staging before (warp barrier) and the reads after.
__device__ __forceinline__ void stage_transpose(const uint8_t* src, uint8_t* dst, int lane) {
  const int rr = lane & 7, blk = lane >> 3;
#pragma unroll
  for (int S = 0; S < 4; ++S) {
    const int ri = 8 * blk + rr;
    const uint32_t a = smem_u32(src + ri * 64 + 16 * (S ^ ((ri >> 1) & 3)));
    uint32_t r0, r1, r2, r3;
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(a)
                 : "memory");
    const int ro = 8 * S + rr;
    const uint32_t d = smem_u32(dst + ro * 64 + 16 * (blk ^ ((ro >> 1) & 3)));
    asm volatile("stmatrix.sync.aligned.m8n8.x4.shared.b16 [%0], {%1, %2, %3, %4};" ::"r"(d), "r"(r0), "r"(r1),
                 "r"(r2), "r"(r3)
                 : "memory");
  }
}

// Element (row, col) of a chunk staged by stage_group (16-bit).
__device__ __forceinline__ uint32_t staged_elem(const uint8_t* buf, int row, int col) {
  return *reinterpret_cast<const uint16_t*>(buf + row * 64 + 16 * ((col >> 3) ^ ((row >> 1) & 3)) + 2 * (col & 7));
}

// a[i] for a runtime i < N (N = 4 or 8) without indexing (keeps a[] in registers)
template <typename V, int N>
__device__ __forceinline__ V pick(const V (&a)[N], int i) {
  V r = a[0];
#pragma unroll
  for (int k = 1; k < N; ++k) r = i == k ? a[k] : r;
  return r;
}

__device__ __forceinline__ bool tile_live(const TcTile& t, int B_pad) {
  return t.kind == kWgrad || t.kind >= kNsGram || t.m0 < B_pad;
}
// Operand major-ness of a product kind: A is MN-major only for kWgrad; B is
// K-major for kFwd, kNsGram and kNsPoly.  Only kFwd and kDgrad read the
// weight copies (w_shift applies to their B maps).
__device__ __forceinline__ bool b_kmajor(int kind) { return kind == kFwd || kind == kNsGram || kind == kNsPoly; }
__device__ __forceinline__ bool reads_weights(int kind) { return kind == kFwd || kind == kDgrad; }

// This CTA's rows of a tile: row block `mi` of the tile (rows m0 .. m0 + 127).
// Rows beyond the product still load their share of the operands for the
// peer CTA but store nothing.
struct SubTile {
  int m0;
  bool rows_live;
};
__device__ __forceinline__ SubTile sub_tile(const TcTile& t, int mi, int B_pad) {
  SubTile u;
  u.m0 = t.m0 + kRowTile * mi;
  u.rows_live = u.m0 < (t.m_real ? t.m_real : B_pad);
  return u;
}

// Fused-AdamW weight-gradient tile: epilogue warp e of this CTA asks L2 for
// 128 / kEpiWarps of the CTA's 128 weight rows of the tile's fp32 master, first and
// second moments (one bulk prefetch per row and array), so that the
// epilogue's loads of the tile hit L2.  Weight rows are 16-byte aligned and
// the weight columns of a tile a multiple of 8 (n0 a multiple of 16, in_pad of 8).
__device__ __forceinline__ void prefetch_adam_rows(const TcArgs& g, const TcTile& t, int rank, int e, int lane) {
  const SubTile u = sub_tile(t, rank, g.B_pad);
  const int cols = min(t.n_len, (t.db_off >= 0 ? t.n_real : t.n_real - 1) - t.n0);
  if (!u.rows_live || cols <= 0) return;
  constexpr int kR = 128 / kEpiWarps;
  for (int k = lane; k < 3 * kR; k += 32) {
    const int r = u.m0 + kR * e + (k % kR);
    if (r >= t.m_real) continue;
    const float* base = k < kR ? g.adam.params : k < 2 * kR ? g.adam.m : g.adam.v;
    prefetch_l2(base + t.c_off + (int64_t)r * t.ldc + t.n0, (uint32_t)cols * 4u);
  }
}

// Prefetch of the tensor map of a tile's A (which = 0) or B (which = 1)
// operand, as the producer selects it below.
__device__ __forceinline__ void prefetch_tile_map(const TcArgs& g, const TcTile& t, int which) {
  const bool a_k = t.kind != kWgrad, b_k = b_kmajor(t.kind);
  const CUtensorMap* m = which == 0 ? g.maps + t.map_a + (a_k ? g.kmaj_off : 0)
                                    : g.maps + t.map_b + (reads_weights(t.kind) ? g.w_shift : 0) + (b_k ? g.kmaj_off : 0);
  asm volatile("prefetch.tensormap [%0];" ::"l"(m) : "memory");
}

// ------------------------------------------------------------------ kernel
// kNs: the Newton-Schulz products of Muon (their own instantiation, so that
// their epilogue adds nothing to the training products' registers).
template <int kCta, bool kNs>
__global__ void __launch_bounds__(kThreads, 1) k_tc_gemm(const TcArgs g) {
  using G = Geo<kCta>;
  constexpr int kStages = G::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  float* tr_all = (float*)(smem + kStages * G::kStageBytes);
  SmemTail<kStages>* tl = (SmemTail<kStages>*)(smem + kStages * G::kStageBytes + kTrBytes);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rank = kCta == 2 ? (int)cluster_rank() : 0;  // row block of the tile this CTA holds
  const bool leader = rank == 0;                         // issues the pair's MMAs
  const int clu = blockIdx.x / kCta, n_clu = gridDim.x / kCta;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&tl->full[s], 1);
      mbar_init(&tl->empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tl->tfull[b], 1);
      mbar_init(&tl->tempty[b], kEpiWarps * kCta);  // one arrival per epilogue warp of the pair
    }
    for (int b = 0; b < kPubSlots; ++b) {
      mbar_init(&tl->stored[b], kEpiWarps);
      mbar_init(&tl->pub_free[b], 1);
    }
    mbar_init(&tl->done, 1);
    tl->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    // one warp of each CTA of the pair allocates collectively
    if constexpr (kCta == 2) {
      asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tl->tmem_base)),
                   "r"(kTmemCols)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    } else {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tl->tmem_base)),
                   "r"(kTmemCols)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (kCta == 2) cluster_sync();  // the peer's barriers exist before any copy or arrival targets them
  // The set-up above overlaps the previous kernel; data reads start here.  The
  // GEMM itself never triggers its dependents early: CTAs of the next kernel
  // parked beside a running GEMM measurably slow it down.
  pdl_wait();
  const uint32_t tmem = tl->tmem_base;
  volatile int* abort_flag = &tl->abort;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    // The whole warp walks the tiles; lane 0 waits for free stages and posts
    // the expected bytes, then lane j issues TMA box j of the K block, so the
    // boxes of a stage leave in parallel instead of one after another.  In a
    // CTA pair both CTAs' copies complete on the leader's full barrier, which
    // the leader expects for both.
    uint32_t stage = 0, phase = 0;
    uint32_t issued_mask = 0, last_parity = 0;  // per stage: ever issued, parity of the last issue
    bool ok = true;
    // A tile's descriptor is read while the previous tile's copies stream,
    // and its tensor maps reach the descriptor cache from the middle of that
    // tile: at a tile boundary the producer goes straight to the dependency
    // check and the copies (a global read there cost a round trip in which
    // the ring drained).
    TcTile tile{}, nxt{};
    if (clu < g.n_tiles) tile = g.tiles[clu];
    if (lane < 2 && clu < g.n_tiles) prefetch_tile_map(g, tile, lane);
    for (int t = clu; ok && t < g.n_tiles; t += n_clu, tile = nxt) {
      const bool has_next = t + n_clu < g.n_tiles;
      if (has_next) nxt = g.tiles[t + n_clu];
      if (!tile_live(tile, g.B_pad)) continue;
      const SubTile u = sub_tile(tile, rank, g.B_pad);
      const int K = tile.k_len ? tile.k_len : g.B_pad;
      // K-major operands (A of kFwd / kDgrad, B of kFwd) load 128-row boxes,
      // MN-major ones 64 x 64 boxes.  This CTA's B: all n_len rows / columns
      // (kCta 1) or its half of them (kCta 2).
      const bool a_k = tile.kind != kWgrad, b_k = b_kmajor(tile.kind);
      const int nbA = a_k ? 1 : 2;
      const int nh = tile.n_len / kCta;
      const int bn0 = tile.n0 + rank * nh;
      const int nbB = b_k ? (nh + 127) >> 7 : (nh + 63) >> 6;
      const uint32_t boxB = b_k ? 2 * kBoxBytes : kBoxBytes;
      const uint32_t bytes = (uint32_t)kCta * (2 * kBoxBytes + (uint32_t)nbB * boxB);
      // lane bl < nbA: A box bl; then B box bl - nbA
      const int bl = lane;
      const bool is_a = bl < nbA;
      const int qb = bl - nbA;
      const bool mine = is_a || qb < nbB;
      const CUtensorMap* map =
          is_a ? g.maps + tile.map_a + (a_k ? g.kmaj_off : 0)
               : g.maps + tile.map_b + (reads_weights(tile.kind) ? g.w_shift : 0) + (b_k ? g.kmaj_off : 0);
      const bool mn = is_a ? !a_k : !b_k;  // MN-major box: x = row / column, y = k
      const int xy0 = is_a ? u.m0 + 64 * bl : bn0 + (b_k ? 128 : 64) * qb;
      const uint32_t off = is_a ? (uint32_t)bl * kBoxBytes : (uint32_t)kABytes + (uint32_t)qb * boxB;
      // Newton-Schulz tiles count on one counter per matrix and product,
      // shared by the CTAs of a pair, and both CTAs wait: each loads half of
      // B, which earlier tiles of the launch wrote.
      bool dep_ok = true;
      if ((u.rows_live || kNs) && tile.dep >= 0)
        dep_ok = dep_wait(g.cnt + tile.dep + (tile.dep_n && !kNs ? rank : 0),
                          tile.dep_n ? tile.dep_n : g.B_pad / kRowTile, tile.dep_need, abort_flag, g.err, g.wait_ns, 3,
                          lane);
      if (!dep_ok) {
        ok = false;
        break;
      }
      if (tile.dep >= 0) fence_proxy_async_global();  // every issuing lane, after the warp's acquires
      const int k_mid = (((K + 63) >> 6) >> 1) << 6;
      for (int k0 = 0; k0 < K; k0 += 64) {
        if (k0 == k_mid && lane < 2 && has_next) prefetch_tile_map(g, nxt, lane);
        bool got = true;
        if (lane == 0) {
          got = mbar_wait(&tl->empty[stage], phase ^ 1u, abort_flag, g.err, g.wait_ns, 1);
          if (got && leader) mbar_expect_tx(&tl->full[stage], bytes);
        }
        if (!__shfl_sync(0xffffffffu, got, 0)) {
          ok = false;
          break;
        }
        if (mine) {
          const uint32_t dst = smem_u32(smem + stage * G::kStageBytes) + off;
          const int x = mn ? xy0 : k0, y = mn ? k0 : xy0;
          if constexpr (kCta == 2) tma_load_2d_pair(dst, map, mapa(smem_u32(&tl->full[stage]), 0), x, y);
          else tma_load_2d(dst, map, &tl->full[stage], x, y);
        }
        issued_mask |= 1u << stage;
        last_parity = (last_parity & ~(1u << stage)) | (phase << stage);
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    // wait (bounded) until every copy counted on this CTA's full barriers has
    // landed (in a pair the leader's barriers count both CTAs' copies)
    if (lane == 0 && leader)
      for (int s = 0; s < kStages; ++s)
        if (issued_mask & (1u << s)) {
          int dummy_abort = 0;
          mbar_wait(&tl->full[s], (last_parity >> s) & 1u, &dummy_abort, g.err, kWaitNs, 10);
        }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // --------------------------------------------------------------- MMA
      // The issue loop is kept short: it shares its sub-partition's issue
      // slots with two epilogue warps, and every instruction it spends
      // between MMAs delays the tensor pipe.  Descriptors are formed once:
      // stage s adds s * kStageBytes / 16 to the start-address field and K
      // step kk adds 32 bytes (K-major) or 2048 bytes (MN-major) / 16; the
      // field (address / 16 < 2^14) never carries into the next field.
      const uint32_t s0 = smem_u32(smem);
      const uint64_t dA_k = smem_desc(s0, 16, 1024), dA_mn = smem_desc(s0, kBoxBytes, 1024);
      const uint64_t dB_k = smem_desc(s0 + kABytes, 16, 1024), dB_mn = smem_desc(s0 + kABytes, kBoxBytes, 1024);
      constexpr uint32_t kStageStep = G::kStageBytes >> 4;
      uint32_t stage = 0, phase = 0, acc = 0, acc_phase = 0;
      bool ok = true;
      // the next tile's descriptor is read while this tile's MMAs issue
      TcTile tile{}, nxt{};
      if (clu < g.n_tiles) tile = g.tiles[clu];
      for (int t = clu; ok && t < g.n_tiles; t += n_clu, tile = nxt) {
        if (t + n_clu < g.n_tiles) nxt = g.tiles[t + n_clu];
        if (!tile_live(tile, g.B_pad)) continue;
        const int K = tile.k_len ? tile.k_len : g.B_pad;
        if (!mbar_wait(&tl->tempty[acc], acc_phase ^ 1u, abort_flag, g.err, 2 * g.wait_ns, 5)) break;
        tc_fence_after();
        const uint32_t d = tmem + acc * kAccCols;
        const int a_mn = tile.kind == kWgrad, b_mn = !b_kmajor(tile.kind);
        const uint32_t idesc = instr_desc(128 * kCta, tile.n_len, a_mn, b_mn);
        const uint64_t ta = a_mn ? dA_mn : dA_k, tb = b_mn ? dB_mn : dB_k;
        const uint32_t ka = a_mn ? 2048 >> 4 : 32 >> 4, kb = b_mn ? 2048 >> 4 : 32 >> 4;
        uint32_t accum = 0;
        for (int k0 = 0; k0 < K; k0 += 64) {
          if (!mbar_wait(&tl->full[stage], phase, abort_flag, g.err, 2 * g.wait_ns, 6)) {
            ok = false;
            break;
          }
          const uint64_t sa = ta + stage * kStageStep, sb = tb + stage * kStageStep;
          if (K - k0 >= 64) {
            umma_bf16<kCta>(d, sa, sb, idesc, accum);
            umma_bf16<kCta>(d, sa + ka, sb + kb, idesc, 1u);
            umma_bf16<kCta>(d, sa + 2 * ka, sb + 2 * kb, idesc, 1u);
            umma_bf16<kCta>(d, sa + 3 * ka, sb + 3 * kb, idesc, 1u);
          } else {
            const int nk = (K - k0 + 15) >> 4;
            for (int kk = 0; kk < nk; ++kk) umma_bf16<kCta>(d, sa + kk * ka, sb + kk * kb, idesc, kk ? 1u : accum);
          }
          accum = 1u;
          umma_commit<kCta>(&tl->empty[stage]);  // the stage is free in every CTA of the tile
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit<kCta>(&tl->tfull[acc]);
        acc ^= 1u;
        if (acc == 0) acc_phase ^= 1u;
      }
      // all MMAs this thread issued have completed before TMEM is freed
      umma_commit<kCta>(&tl->done);
      int dummy_abort = 0;
      mbar_wait(&tl->done, 0, &dummy_abort, g.err, kWaitNs, 12);
    }
  } else if (warp < kPubWarp) {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;             // TMEM lane quarter this warp may access
    const int half = (warp - 2) >> 2;   // 0 for warps 2-5, 1 for warps 6-9
    const int row = 32 * q + lane;
    uint32_t acc = 0, acc_phase = 0;
    int n_pub = 0;   // tiles handed to the publisher
    // Fused AdamW: the parameter rows of the CTA's next weight-gradient tile
    // stream into L2 while this tile's products run and its epilogue works.
    if (g.update && clu < g.n_tiles && g.tiles[clu].kind == kWgrad)
      prefetch_adam_rows(g, g.tiles[clu], rank, warp - 2, lane);
    for (int t = clu; t < g.n_tiles; t += n_clu) {
      const TcTile tile = g.tiles[t];
      if (g.update && t + n_clu < g.n_tiles) {
        const TcTile nx = g.tiles[t + n_clu];
        if (nx.kind == kWgrad) prefetch_adam_rows(g, nx, rank, warp - 2, lane);
      }
      if (!tile_live(tile, g.B_pad)) continue;
      const SubTile u = sub_tile(tile, rank, g.B_pad);
      const MemberDev md = g.mem[tile.member];
      const int m_lim = tile.m_real ? tile.m_real : g.B_pad;
      const int r = u.m0 + row;
      const bool row_ok = r < m_lim;
      // the two warps of a lane quarter take alternate 32-column chunks:
      // chunk ci covers columns 32 * half + 32 * kEpiPerQ * ci .. + 31 of the tile
      const int n_end = u.rows_live ? tile.n_len : 0;
      // last output column of this tile plus one: a chunk may reach past the
      // tile (n_len is a multiple of 16, chunks are 32 wide), and the columns
      // past it belong to the next column tile
      const int n_hi = min(tile.n_real, tile.n0 + tile.n_len);
      // Inputs that do not depend on the accumulator are prepared while the
      // tile's MMAs run: forward, this lane's bias value of each chunk
      // (column = lane; later broadcast through shared memory) and the 32
      // dropout keep bits of its row; dgrad, the 32 ReLU-mask bits of its row.
      float bias_l[kChunks];
      uint32_t bits[kChunks];
#pragma unroll
      for (int ci = 0; ci < kChunks; ++ci) {
        const int c = 32 * half + 32 * kEpiPerQ * ci;
        const int col0 = tile.n0 + c;
        const int ncols = min(32, n_hi - col0);
        bias_l[ci] = 0.f;
        bits[ci] = 0xFFFFFFFFu;
        if (c >= n_end || ncols <= 0) continue;
        if (tile.kind == kFwd) {
          if (lane < ncols) bias_l[ci] = __ldg(g.params + tile.aux_off + col0 + lane);
          // tile origins and chunks are 32-column aligned for forward tiles
          if (row_ok && g.train && tile.mask_off >= 0)
            bits[ci] = __ldg(g.masks + tile.mask_off + (int64_t)(col0 >> 5) * g.mask_rows + r);
        } else if (tile.kind == kDgrad && row_ok && tile.aux_off >= 0) {
          const __nv_bfloat16* hm = g.act + tile.aux_off + (int64_t)r * tile.ld_aux + col0;
          uint32_t mb = 0;
#pragma unroll
          for (int s = 0; s < 4; ++s) {
            if (8 * s >= ncols) break;
            const uint4 hv = *reinterpret_cast<const uint4*>(hm + 8 * s);
            const __nv_bfloat16* hb = reinterpret_cast<const __nv_bfloat16*>(&hv);
#pragma unroll
            for (int e = 0; e < 8; ++e) mb |= (uint32_t)(__bfloat162float(hb[e]) > 0.f) << (8 * s + e);
          }
          bits[ci] = mb;
        }
      }
      // Newton-Schulz: the epilogue reads `aux` (A or X), which earlier
      // tiles of the launch wrote, with plain loads; its own acquire of the
      // tile's dependency orders them (and, through this tile's count, the
      // later tiles that overwrite a buffer after it).
      if constexpr (kNs) {
        if (tile.dep >= 0 &&
            !dep_wait(g.cnt + tile.dep, 1, tile.dep_need, abort_flag, g.err, 2 * g.wait_ns, 13, lane))
          break;
      }
      // Newton-Schulz: this lane's 32 values of the aux term in chunk ci of
      // its warp (zeros where the chunk is not written), loaded one chunk
      // ahead -- the first while the tile's products run.
      auto ns_aux = [&](int ci, uint4(&a)[4]) {
        const int c = 32 * half + 32 * kEpiPerQ * ci;
        const int col0 = tile.n0 + c;
        const int ncols = min(32, n_hi - col0);
        const bool need = tile.kind != kNsGram && row_ok && c < n_end && ncols > 0 &&
                          (tile.kind == kNsApply || col0 >= u.m0 + 32 * q);
        const __nv_bfloat16* p = g.ns + tile.aux_off + (int64_t)r * tile.ld_aux + col0;
#pragma unroll
        for (int s = 0; s < 4; ++s)
          a[s] = need && 8 * s < ncols ? *reinterpret_cast<const uint4*>(p + 8 * s) : make_uint4(0u, 0u, 0u, 0u);
      };
      // Weight-gradient tiles of column 0: the bias gradient sums dZ's
      // column-sum partials with plain loads.  Row blocks of dZ written in
      // this launch are acquired here (their counts were reached before the
      // tile's operands were loaded, so this does not wait).
      const bool bias_tile = !kNs && tile.kind == kWgrad && tile.n0 == 0 && half == 0 && g.dbp != nullptr &&
                             tile.db_off >= 0 && u.rows_live;
      if (bias_tile && tile.dep >= 0 &&
          !dep_wait(g.cnt + tile.dep, g.B_pad / kRowTile, tile.dep_need, abort_flag, g.err, 2 * g.wait_ns, 14, lane))
        break;
      uint4 axn[4];
      if constexpr (kNs) ns_aux(0, axn);
      if (!mbar_wait(&tl->tfull[acc], acc_phase, abort_flag, g.err, 2 * g.wait_ns, 7)) break;
      tc_fence_after();
      const uint32_t taddr = tmem + ((uint32_t)(32 * q) << 16) + acc * kAccCols;
      float lr = 0.f, wd_w = 0.f, wd_b = 0.f, ib1 = 1.f, ib2 = 1.f;
      if (tile.kind == kWgrad && g.update) {
        const float2 bc = g.adam.bias_corr[tile.member];
        lr = md.lr;
        wd_w = md.wd;
        wd_b = g.adam.wd_on_bias ? md.wd : 0.f;
        ib1 = 1.f / bc.x;
        ib2 = 1.f / bc.y;
      }
#pragma unroll 1
      for (int ci = 0; ci < kChunks; ++ci) {
        const int c = 32 * half + 32 * kEpiPerQ * ci;
        if (c >= n_end) break;
        const int col0 = tile.n0 + c;
        const int ncols = min(32, n_hi - col0);
        const bool live = row_ok && ncols > 0;
        uint32_t v[32];
        tmem_ld32(taddr + c, v);
        if constexpr (kNs) {
          // Newton-Schulz: out = alpha acc + beta aux, bf16 (kNsGram: A;
          // kNsPoly: Bm = c (A A) + b A; kNsApply: X' = (Bm X) + a X).  The
          // warp's 32 x 32 chunk is staged in its buffer and leaves as whole
          // 64-byte row segments.  A and Bm are symmetric and only the tiles
          // on or above the diagonal run; chunk origins are 32-aligned, so a
          // chunk lies wholly above, on or below the diagonal.  Above: the
          // chunk, and its transpose (staged by ldmatrix / stmatrix in the
          // buffer's second half) at the mirror position.  On: the chunk
          // with its upper triangle mirrored into the lower.  Below (on a
          // diagonal tile): nothing, its mirror writes it.
          uint4 axc[4];
#pragma unroll
          for (int s = 0; s < 4; ++s) axc[s] = axn[s];
          if (ci + 1 < kChunks) ns_aux(ci + 1, axn);
          if (ncols <= 0) continue;  // warp-uniform
          const bool sym = tile.kind != kNsApply;
          const int rbase = u.m0 + 32 * q;
          if (sym && col0 < rbase) continue;  // warp-uniform
          // the first iteration reads U = |U|_F X0: A = s^2 (U U^T), X' = s (Bm U + a U)
          const float sc = tile.ns_scale ? g.ns_scale[tile.ns_scale - 1] : 1.f;
          const float al = tile.kind == kNsPoly ? kNsC : (tile.kind == kNsGram ? sc * sc : sc);
          const float be = tile.kind == kNsPoly ? kNsB : (tile.kind == kNsApply ? kNsA * sc : 0.f);
          uint32_t pk[16];
#pragma unroll
          for (int s = 0; s < 4; ++s) {
            const __nv_bfloat16* ab = reinterpret_cast<const __nv_bfloat16*>(&axc[s]);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const int j = 8 * s + 2 * e;
              pk[4 * s + e] = pack_bf16x2(al * __uint_as_float(v[j]) + be * __bfloat162float(ab[2 * e]),
                                          al * __uint_as_float(v[j + 1]) + be * __bfloat162float(ab[2 * e + 1]));
            }
          }
          uint8_t* buf = reinterpret_cast<uint8_t*>(tr_all + (warp - 2) * 32 * 32);
          __nv_bfloat16* out = g.ns + tile.c_off + (int64_t)rbase * tile.ldc + col0;
#pragma unroll
          for (int s = 0; s < 4; ++s) stage_group(buf, lane, s, pk[4 * s], pk[4 * s + 1], pk[4 * s + 2], pk[4 * s + 3]);
          if (!sym || col0 > rbase) {
            flush_chunk<true>(buf, lane, out, tile.ldc, rbase, m_lim, ncols);
            if (sym) {  // rows col0 .. col0 + 31 of the output at columns rbase .. rbase + 31
              stage_transpose(buf, buf + 2048, lane);
              flush_chunk<true>(buf + 2048, lane, g.ns + tile.c_off + (int64_t)col0 * tile.ldc + rbase, tile.ldc, col0,
                                col0 + ncols, min(32, m_lim - rbase));
            }
          } else {
            // on the diagonal: row i keeps its columns j >= i and takes
            // element (j, i) of the chunk for j < i
            __syncwarp();
            uint32_t t2[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
              const int j0 = 2 * e, j1 = 2 * e + 1;
              const uint32_t lo = j0 >= lane ? (pk[e] & 0xFFFFu) : staged_elem(buf, j0, lane);
              const uint32_t hi = j1 >= lane ? (pk[e] >> 16) : staged_elem(buf, j1, lane);
              t2[e] = lo | (hi << 16);
            }
            __syncwarp();
#pragma unroll
            for (int s = 0; s < 4; ++s) stage_group(buf, lane, s, t2[4 * s], t2[4 * s + 1], t2[4 * s + 2], t2[4 * s + 3]);
            flush_chunk<true>(buf, lane, out, tile.ldc, rbase, m_lim, ncols);
          }
        } else if (tile.kind == kWgrad) {
          // Transpose the warp's 32 rows x 32 columns through shared memory
          // (float4 groups XOR-swizzled by row, so that both the row-wise
          // write and the group-wise read are free of bank conflicts).  Then
          // lane (rsub, gc) = (lane / 8, lane % 8) takes columns col0 + 4 gc ..
          // + 3 of rows 4 i + rsub, i = 0..7: every warp access covers four
          // 128-byte row segments.
          float* tr = tr_all + (warp - 2) * 32 * 32;
#pragma unroll
          for (int gi = 0; gi < 8; ++gi)
            *reinterpret_cast<float4*>(tr + lane * 32 + 4 * (gi ^ (lane & 7))) =
                make_float4(__uint_as_float(v[4 * gi]), __uint_as_float(v[4 * gi + 1]),
                            __uint_as_float(v[4 * gi + 2]), __uint_as_float(v[4 * gi + 3]));
          __syncwarp();
          // in_pad: a multiple of 8, so a float4 group is all weights or
          // starts at the bias column (when the bias comes from the ones column)
          const int in_pad = tile.db_off >= 0 ? tile.n_real : tile.n_real - 1;
          const int gc = lane & 7, rsub = lane >> 3;
          const int col = col0 + 4 * gc;
          const bool is_w = col < in_pad && col < n_hi;
          const int rbase = u.m0 + 32 * q;
          const int nrows = min(32, m_lim - rbase);
          if (g.update) {
            const AdamDev& ad = g.adam;
            if (is_w) {
              // rounds of three row groups: nine float4 loads in flight per
              // lane (the 10-warp CTA allows 168 registers per thread)
#pragma unroll 1
              for (int i0 = 0; i0 < 8; i0 += 3) {
                float4 P[3], M[3], V[3];
#pragma unroll
                for (int i = 0; i < 3; ++i) {
                  const int rr = 4 * (i0 + i) + rsub;
                  if (i0 + i < 8 && rr < nrows) {
                    const int64_t o = tile.c_off + (int64_t)(rbase + rr) * tile.ldc + col;
                    P[i] = *reinterpret_cast<const float4*>(ad.params + o);
                    M[i] = *reinterpret_cast<const float4*>(ad.m + o);
                    V[i] = *reinterpret_cast<const float4*>(ad.v + o);
                  }
                }
#pragma unroll
                for (int i = 0; i < 3; ++i) {
                  const int rr = 4 * (i0 + i) + rsub;
                  if (i0 + i >= 8 || rr >= nrows) break;
                  const float4 G = *reinterpret_cast<const float4*>(tr + rr * 32 + 4 * (gc ^ (rr & 7)));
                  adamw_elem(P[i].x, M[i].x, V[i].x, G.x, lr, wd_w, ad.beta1, ad.beta2, ad.eps, ib1, ib2);
                  adamw_elem(P[i].y, M[i].y, V[i].y, G.y, lr, wd_w, ad.beta1, ad.beta2, ad.eps, ib1, ib2);
                  adamw_elem(P[i].z, M[i].z, V[i].z, G.z, lr, wd_w, ad.beta1, ad.beta2, ad.eps, ib1, ib2);
                  adamw_elem(P[i].w, M[i].w, V[i].w, G.w, lr, wd_w, ad.beta1, ad.beta2, ad.eps, ib1, ib2);
                  const int64_t o = tile.c_off + (int64_t)(rbase + rr) * tile.ldc + col;
                  *reinterpret_cast<float4*>(ad.params + o) = P[i];
                  *reinterpret_cast<float4*>(ad.m + o) = M[i];
                  *reinterpret_cast<float4*>(ad.v + o) = V[i];
                  *reinterpret_cast<uint2*>(ad.wq_out + o) =
                      make_uint2(pack_bf16x2(P[i].x, P[i].y), pack_bf16x2(P[i].z, P[i].w));
                }
              }
            }
          } else {
            if (is_w) {
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                const int rr = 4 * i + rsub;
                if (rr >= nrows) break;
                *reinterpret_cast<float4*>(g.grads + tile.c_off + (int64_t)(rbase + rr) * tile.ldc + col) =
                    *reinterpret_cast<const float4*>(tr + rr * 32 + 4 * (gc ^ (rr & 7)));
              }
            }
          }
          // db_j, lane = row j: from the bias column when this chunk holds it,
          // or from dZ's column sums (partials of column j in batch order)
          const int cb = in_pad - col0;
          const bool col_b = tile.db_off < 0 && cb >= 0 && cb < 32 && in_pad < n_hi;
          if ((col_b || (bias_tile && ci == 0)) && lane < nrows) {
            const float gb = col_b ? tr[lane * 32 + 4 * ((cb >> 2) ^ (lane & 7)) + (cb & 3)]
                                   : sum_strided(g.dbp + tile.db_off + rbase + lane, g.B_pad / tile.db_rows, tile.m_real);
            const int64_t o = tile.aux_off + rbase + lane;
            if (g.update) {
              const AdamDev& ad = g.adam;
              float pb = ad.params[o], mb = ad.m[o], vb = ad.v[o];
              adamw_elem(pb, mb, vb, gb, lr, wd_b, ad.beta1, ad.beta2, ad.eps, ib1, ib2);
              ad.params[o] = pb;
              ad.m[o] = mb;
              ad.v[o] = vb;
              ad.wq_out[o] = __float2bfloat16_rn(pb);
            } else {
              g.grads[o] = gb;
            }
          }
          __syncwarp();  // the buffer is reused by the next chunk
          continue;
        }
        if (tile.kind == kFwd) {  // ncols: a multiple of 8 (widths are multiples of 16)
          const float bl = pick(bias_l, ci);
          if (ncols <= 0) continue;   // warp-uniform: every lane takes part in the store below
          const uint32_t keep = pick(bits, ci);
          const float sc = g.train ? md.scale : 1.f;
          uint8_t* buf = reinterpret_cast<uint8_t*>(tr_all + (warp - 2) * 32 * 32);
          // the chunk's 32 bias values sit past the 2 KB of staged rows and
          // reach every lane as broadcast reads (8 shared loads instead of 32
          // shuffles); the flush's closing warp barrier orders their reuse
          float* bsm = reinterpret_cast<float*>(buf + 2048);
          bsm[lane] = bl;
          __syncwarp();
#pragma unroll
          for (int sg = 0; sg < 4; ++sg) {
            const float4 b0 = *reinterpret_cast<const float4*>(bsm + 8 * sg);
            const float4 b1 = *reinterpret_cast<const float4*>(bsm + 8 * sg + 4);
            const float bv[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
            uint32_t pk[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              float h2[2];
#pragma unroll
              for (int u2 = 0; u2 < 2; ++u2) {
                const int j = 8 * sg + 2 * e + u2;
                const float z = __uint_as_float(v[j]) + bv[2 * e + u2];
                const float a = z > 0.f ? z : 0.f;
                h2[u2] = ((keep >> j) & 1u) ? a * sc : 0.f;
              }
              pk[e] = pack_bf16x2(h2[0], h2[1]);
            }
            stage_group(buf, lane, sg, pk[0], pk[1], pk[2], pk[3]);
          }
          const int rbase = u.m0 + 32 * q;
          flush_chunk(buf, lane, g.act + tile.c_off + (int64_t)rbase * tile.ldc + col0, tile.ldc, rbase, m_lim, ncols);
        } else if (tile.kind == kDgrad) {
          if (ncols <= 0) continue;
          const uint32_t mb = row_ok ? pick(bits, ci) : 0u;
          const float dsc = tile.aux_off >= 0 ? md.scale : 1.f;   // the first layer's input gradient: 1
          uint8_t* buf = reinterpret_cast<uint8_t*>(tr_all + (warp - 2) * 32 * 32);
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const int j = 2 * e;
            const float x0 = ((mb >> j) & 1u) ? __uint_as_float(v[j]) * dsc : 0.f;
            const float x1 = ((mb >> (j + 1)) & 1u) ? __uint_as_float(v[j + 1]) * dsc : 0.f;
            pk[e] = pack_bf16x2(x0, x1);
          }
#pragma unroll
          for (int sg = 0; sg < 4; ++sg) stage_group(buf, lane, sg, pk[4 * sg], pk[4 * sg + 1], pk[4 * sg + 2], pk[4 * sg + 3]);
          const int rbase = u.m0 + 32 * q;
          flush_chunk(buf, lane, g.dz + tile.c_off + (int64_t)rbase * tile.ldc + col0, tile.ldc, rbase, m_lim, ncols);
          // the column sums of the stored values over this warp's 32 rows,
          // where the layer's weight-gradient tiles take db from them
          if (tile.db_rows > 0 && g.dbp != nullptr) {
            float x[32];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
              x[2 * e] = __uint_as_float(pk[e] << 16);
              x[2 * e + 1] = __uint_as_float(pk[e] & 0xFFFF0000u);
            }
            const float cs = colsum32(x, lane);
            if (lane < ncols) g.dbp[tile.c_off / 32 + (int64_t)(rbase >> 5) * tile.ldc + col0 + lane] = cs;
          }
        }
      }
      // this warp has read its part of the accumulator: release it to the
      // MMA issuer (the leader CTA's barrier in a pair)
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if constexpr (kCta == 2) mbar_arrive_cluster_relaxed(mapa(smem_u32(&tl->tempty[acc]), 0));
        else mbar_arrive_relaxed(&tl->tempty[acc]);
      }
      acc ^= 1u;
      if (acc == 0) acc_phase ^= 1u;
      if (tile.sig >= 0 && u.rows_live) {
        // hand this warp's part of the tile to the publisher: the arrival
        // (a release at CTA scope after the warp barrier) orders every
        // lane's stores before the publisher's count.  A slot is reused
        // once the publisher has counted its previous tile.
        const int slot = n_pub % kPubSlots;
        bool got = true;
        if (n_pub >= kPubSlots && lane == 0)
          got = mbar_wait(&tl->pub_free[slot], (uint32_t)((n_pub / kPubSlots) - 1) & 1u, abort_flag, g.err,
                          2 * g.wait_ns, 8);
        if (!__shfl_sync(0xffffffffu, got, 0)) break;
        __syncwarp();
        if (lane == 0) mbar_arrive(&tl->stored[slot]);
        ++n_pub;
      }
    }
  } else {
    // ------------------------------------------------------------ publisher
    // Per stored tile (the epilogue's order), once every epilogue warp has
    // arrived: the count that other CTAs' tiles wait on.  The release is
    // cumulative over the stores the arrivals ordered before it; the proxy
    // fence serves the readers' tensor-map loads.
    if (lane == 0) {
      int n_pub = 0;
      for (int t = clu; t < g.n_tiles; t += n_clu) {
        const TcTile tile = g.tiles[t];
        if (!tile_live(tile, g.B_pad)) continue;
        const SubTile u = sub_tile(tile, rank, g.B_pad);
        if (tile.sig < 0 || !u.rows_live) continue;
        const int slot = n_pub % kPubSlots;
        if (!mbar_wait(&tl->stored[slot], (uint32_t)(n_pub / kPubSlots) & 1u, abort_flag, g.err, 4 * g.wait_ns, 9))
          break;
        fence_proxy_async_global();
        red_release_add(g.cnt + tile.sig + (kNs ? 0 : rank), kEpiWarps);
        mbar_arrive(&tl->pub_free[slot]);
        ++n_pub;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (kCta == 2) cluster_sync();  // the pair's MMAs, copies and arrivals are over
  if (warp == 1) {
    if constexpr (kCta == 2)
      asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    else
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

// ------------------------------------------------------------------- host
PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
  }
  return fn;
}

// 2-D bf16 row-major matrix [rows, cols] with row pitch `ld` elements,
// boxes of 64 columns x box_rows rows, 128-byte swizzle.
bool encode_map(CUtensorMap* m, const void* base, int64_t cols, int64_t rows, int64_t ld, int box_rows,
                std::string& err) {
  auto fn = get_encode();
  if (!fn) {
    err = "cuTensorMapEncodeTiled unavailable";
    return false;
  }
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    err = "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")";
    return false;
  }
  return true;
}

// Balanced split of n columns into tiles of at most 256 (multiples of 16),
// every tile starting at a multiple of `align` (16 or 32).
void split_n(int n, std::vector<std::pair<int, int>>& out, int align = 16) {
  out.clear();
  const int nt = (int)ceil_div(n, 256);
  const int len = (int)round_up(ceil_div(n, nt), align);
  for (int n0 = 0; n0 < n; n0 += len) out.push_back({n0, std::min(len, (int)round_up(n - n0, 16))});
}

}  // namespace

tp_status tc_build_plan(TcPlan& plan, const TcLayout& lay, std::string& err) {
  const int m = lay.m;
  auto in0p = [&](int i) { return lay.in0_pad ? (*lay.in0_pad)[i] : lay.d_in_pad; };
  const auto& depth = *lay.depth;
  const auto& width = *lay.width;
  const auto& active = *lay.active;
  if (plan.maps_dev == nullptr) {
    // tensor maps, twice (64-row boxes for MN-major loads, then 128-row
    // boxes for K-major loads, kmaj_off apart): 0 = gathered batch
    // [B_cap, d_in_pad + 16]; per (member, layer) act [B_cap, w + 16],
    // dz [B_cap, w]; then the weights of copy 0, then the weights of copy 1
    // (w_shift apart)
    std::vector<CUtensorMap> maps;
    plan.map_act.assign((size_t)m * kMaxDepth, -1);
    plan.map_dz.assign((size_t)m * kMaxDepth, -1);
    plan.map_w.assign((size_t)m * kMaxDepth, -1);
    CUtensorMap mp;
    const __nv_bfloat16* actb = (const __nv_bfloat16*)lay.act;
    const __nv_bfloat16* dzb = (const __nv_bfloat16*)lay.dz;
    for (int set = 0; set < 2; ++set) {
      const int br = set ? 128 : 64;
      const int base = (int)maps.size();
      // the first layer's input: one batch matrix, or one per member
      // (stacked batches, embeddings: map index = member)
      for (int i = 0; i < (lay.xb_stride || lay.x0_off ? m : 1); ++i) {
        if (lay.x0_off) {
          const int ld = (*lay.in0_pad)[i] + kOnesCols;
          if (!encode_map(&mp, (const __nv_bfloat16*)lay.xb + (*lay.x0_off)[i], ld, lay.B_cap, ld, br, err))
            return TP_ECUDA;
        } else {
          const __nv_bfloat16* xbi = (const __nv_bfloat16*)lay.xb + (int64_t)i * lay.xb_stride;
          if (!encode_map(&mp, xbi, lay.ldx, lay.B_cap, lay.ldx, br, err)) return TP_ECUDA;
        }
        maps.push_back(mp);
      }
      for (int i = 0; i < m; ++i)
        for (int l = 0; l < depth[i]; ++l) {
          const int w = width[i];
          if (!encode_map(&mp, actb + (*lay.act_off)[i][l], w + kOnesCols, lay.B_cap, w + kOnesCols, br, err))
            return TP_ECUDA;
          if (set == 0) plan.map_act[(size_t)i * kMaxDepth + l] = (int)maps.size();
          maps.push_back(mp);
          if (lay.fwd_only) continue;
          if (!encode_map(&mp, dzb + (*lay.dz_off)[i][l], w, lay.B_cap, w, br, err)) return TP_ECUDA;
          if (set == 0) plan.map_dz[(size_t)i * kMaxDepth + l] = (int)maps.size();
          maps.push_back(mp);
        }
      const int w_base = (int)maps.size();
      for (int copy = 0; copy < 2; ++copy)
        for (int i = 0; i < m; ++i)
          for (int l = 0; l < depth[i]; ++l) {
            const int w = width[i], in_pad = l == 0 ? in0p(i) : w;
            if (!encode_map(&mp, lay.wq[copy] + (*lay.W_off)[i][l], in_pad, w, in_pad, br, err)) return TP_ECUDA;
            if (set == 0 && copy == 0) plan.map_w[(size_t)i * kMaxDepth + l] = (int)maps.size();
            maps.push_back(mp);
          }
      plan.w_shift = ((int)maps.size() - w_base) / 2;
      if (set == 1) plan.kmaj_off = base;
      // Muon: X0, X1 [r, c] and A, Bm [r, r] of every Muon matrix
      if (lay.muon && lay.ns) {
        const __nv_bfloat16* nsb = (const __nv_bfloat16*)lay.ns;
        if (set == 0) plan.map_ns.assign(lay.muon->size() * 4, -1);
        for (size_t j = 0; j < lay.muon->size(); ++j) {
          const MuonMat& mt = (*lay.muon)[j];
          const int64_t offs[4] = {mt.x_off[0], mt.x_off[1], mt.a_off, mt.bm_off};
          for (int q = 0; q < 4; ++q) {
            const int cols = q < 2 ? mt.c : mt.r;
            if (!encode_map(&mp, nsb + offs[q], cols, mt.r, cols, br, err)) return TP_ECUDA;
            if (set == 0) plan.map_ns[j * 4 + q] = (int)maps.size();
            maps.push_back(mp);
          }
        }
        plan.ns_maps = true;
      }
    }
    plan.n_maps = (int)maps.size();
    if (cudaMalloc(&plan.maps_dev, sizeof(CUtensorMap) * maps.size()) != cudaSuccess) {
      err = "cudaMalloc(tensor maps) failed";
      return TP_ENOMEM;
    }
    if (cudaMemcpy(plan.maps_dev, maps.data(), sizeof(CUtensorMap) * maps.size(), cudaMemcpyHostToDevice) !=
        cudaSuccess) {
      err = "cudaMemcpy(tensor maps) failed";
      return TP_ECUDA;
    }
    if (cudaMalloc(&plan.err_dev, sizeof(int)) != cudaSuccess || cudaMemset(plan.err_dev, 0, sizeof(int)) != cudaSuccess) {
      err = "cudaMalloc(error word) failed";
      return TP_ENOMEM;
    }
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&plan.n_sm, cudaDevAttrMultiProcessorCount, dev);
    if (cudaFuncSetAttribute(k_tc_gemm<1, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<1>()) !=
            cudaSuccess ||
        cudaFuncSetAttribute(k_tc_gemm<2, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<2>()) !=
            cudaSuccess ||
        cudaFuncSetAttribute(k_tc_gemm<1, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<1>()) !=
            cudaSuccess ||
        cudaFuncSetAttribute(k_tc_gemm<2, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<2>()) !=
            cudaSuccess) {
      err = "cudaFuncSetAttribute(smem) failed";
      return TP_ECUDA;
    }
    // CTAs per tile.  A CTA pair (256-row tiles, cta_group::2) streams two
    // thirds of the operand bytes per FLOP and keeps more K blocks in flight;
    // it pays when every SM has many K blocks to stream (wide members, large
    // batches) and costs idle halves and a few resident CTAs otherwise.
    // TP_GEMM_CTAS=1|2 overrides the choice.
    int64_t fwd_kblocks = 0;
    for (int i = 0; i < m; ++i)
      for (int l = 0; l < depth[i]; ++l) {
        const int in_pad = l == 0 ? in0p(i) : width[i];
        fwd_kblocks += (lay.B_cap / kRowTile) * ceil_div(width[i], 256) * ceil_div(in_pad, 64);
      }
    plan.cta = fwd_kblocks >= 100 * (int64_t)plan.n_sm ? 2 : 1;
    if (const char* e = getenv("TP_GEMM_CTAS")) {
      const int v = atoi(e);
      if (v == 1 || v == 2) plan.cta = v;
    }
    plan.max_clusters = plan.n_sm;
    if (plan.cta == 2) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(2 * plan.n_sm);
      cfg.blockDim = dim3(kThreads);
      cfg.dynamicSmemBytes = smem_bytes<2>();
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = 2;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, (void*)k_tc_gemm<2, false>, &cfg) == cudaSuccess && n >= 1) {
        plan.max_clusters = n;
      } else {
        cudaGetLastError();
        plan.cta = 1;
      }
    }
  }

  // Tiles of the active members.  Forward: level = layer.  Backward: level
  // = distance from the head (each member's top hidden layer first); the
  // dgrad tiles of a level (which the next level waits for) and its wgrad
  // tiles are each sorted largest first, and the wgrad tiles are interleaved
  // with the next level's dgrad tiles (below).
  const int nrb = lay.B_cap / kRowTile;
  if (plan.cnt_dev == nullptr) {
    plan.n_cnt = (lay.fwd_only ? 1 : 2) * m * kMaxDepth * nrb;
    if (cudaMalloc(&plan.cnt_dev, sizeof(int) * plan.n_cnt) != cudaSuccess ||
        cudaMemset(plan.cnt_dev, 0, sizeof(int) * plan.n_cnt) != cudaSuccess) {
      err = "cudaMalloc(tc counters) failed";
      return TP_ENOMEM;
    }
  }
  auto cnt_act = [&](int i, int l) { return (i * kMaxDepth + l) * nrb; };
  auto cnt_dz = [&](int i, int l) { return ((m + i) * kMaxDepth + l) * nrb; };
  int Lmax = 0;
  for (int i = 0; i < m; ++i) Lmax = std::max(Lmax, depth[i]);
  std::vector<TcTile> all;
  auto cost = [&](const TcTile& t) { return (int64_t)(t.k_len ? t.k_len : lay.B_cap) * t.n_len; };
  // Within a level, tiles whose member has the longest chain of dependent
  // products still ahead go first (list scheduling by remaining chain), then
  // the costlier tiles.  Forward: layers above; dgrad: layers below.
  auto chain = [&](const TcTile& t) {
    return t.kind == kFwd ? depth[t.member] - 1 - t.layer : t.kind == kDgrad ? t.layer : 0;
  };
  auto by_chain_cost = [&](const TcTile& a, const TcTile& b) {
    const int ca = chain(a), cb = chain(b);
    return ca != cb ? ca > cb : cost(a) > cost(b);
  };
  auto sorted_append = [&](std::vector<TcTile>& v) {
    std::stable_sort(v.begin(), v.end(), by_chain_cost);
    all.insert(all.end(), v.begin(), v.end());
  };
  // The tiles of one product: R row blocks (plan.cta at a time) by the
  // column tiles ns; proto.dep / proto.sig are the counters of row block 0.
  const int cta = plan.cta;
  auto emit = [&](std::vector<TcTile>& v, const TcTile& proto, int R, const std::vector<std::pair<int, int>>& ns) {
    for (int rb = 0; rb < R; rb += cta)
      for (const auto& nn : ns) {
        TcTile t = proto;
        t.m0 = rb * kRowTile;
        t.n0 = nn.first;
        t.n_len = nn.second;
        if (proto.dep >= 0 && proto.dep_n == 1) t.dep = proto.dep + rb;
        if (proto.sig >= 0) t.sig = proto.sig + rb;
        v.push_back(t);
      }
  };
  std::vector<std::pair<int, int>> ns;
  for (int l = 0; l < Lmax; ++l) {
    std::vector<TcTile> v;
    for (int i = 0; i < m; ++i) {
      if (!active[i] || depth[i] <= l) continue;
      const int w = width[i];
      split_n(w, ns, 32);  // 32-column aligned: one keep word per chunk of the epilogue
      TcTile t{};
      t.kind = kFwd; t.member = i; t.layer = l;
      t.mask_off = lay.mask_off ? (int32_t)(*lay.mask_off)[i][l] : -1;
      t.m_real = 0; t.n_real = w;
      t.k_len = l == 0 ? in0p(i) : w;
      t.map_a = l == 0 ? (lay.xb_stride || lay.x0_off ? i : 0) : plan.map_act[(size_t)i * kMaxDepth + l - 1];
      t.map_b = plan.map_w[(size_t)i * kMaxDepth + l];
      t.ldc = w + kOnesCols;
      t.ld_aux = 0;
      t.dep = l == 0 ? -1 : cnt_act(i, l - 1);
      t.dep_n = 1;
      t.dep_need = kEpiWarps * (int)ns.size();  // every epilogue warp of every column tile of a row block
      t.sig = l + 1 < depth[i] ? cnt_act(i, l) : -1;
      t.c_off = (*lay.act_off)[i][l];
      t.aux_off = (*lay.b_off)[i][l];
      emit(v, t, lay.B_cap / kRowTile, ns);
    }
    sorted_append(v);
  }
  plan.fwd_rng = {0, (int)all.size()};
  if (lay.fwd_only) Lmax = 0;  // no backward tiles
  std::vector<std::vector<TcTile>> VD(Lmax), VW(Lmax);
  for (int lev = 0; lev < Lmax; ++lev) {
    std::vector<TcTile>& vd = VD[lev];
    std::vector<TcTile>& vw = VW[lev];
    for (int i = 0; i < m; ++i) {
      if (!active[i] || depth[i] <= lev) continue;
      const int l = depth[i] - 1 - lev;
      const int w = width[i], in_pad = l == 0 ? in0p(i) : w;
      split_n(w, ns);
      const int need = kEpiWarps * (int)ns.size();  // dgrad column tiles of layer l + 1 per row block of dz_l
      const bool from_head = l == depth[i] - 1;
      if (l == 0 && lay.de_off) {   // the first layer's input gradient (embeddings): no mask, no scale
        std::vector<std::pair<int, int>> ne;
        split_n(in_pad, ne);
        TcTile t{};
        t.kind = kDgrad; t.member = i; t.layer = 0;
        t.mask_off = -1;
        t.m_real = 0; t.n_real = in_pad;
        t.k_len = w;
        t.map_a = plan.map_dz[(size_t)i * kMaxDepth + 0];
        t.map_b = plan.map_w[(size_t)i * kMaxDepth + 0];
        t.ldc = in_pad;
        t.ld_aux = 0;
        t.dep = from_head ? -1 : cnt_dz(i, 0);
        t.dep_n = 1;
        t.dep_need = need;
        t.sig = -1;
        t.c_off = (*lay.de_off)[i];
        t.aux_off = -1;
        emit(vd, t, lay.B_cap / kRowTile, ne);
      }
      if (l > 0) {
        TcTile t{};
        t.kind = kDgrad; t.member = i; t.layer = l;
        t.mask_off = -1;
        t.m_real = 0; t.n_real = w;
        t.k_len = w;
        t.map_a = plan.map_dz[(size_t)i * kMaxDepth + l];
        t.map_b = plan.map_w[(size_t)i * kMaxDepth + l];
        t.ldc = w;
        t.ld_aux = w + kOnesCols;
        t.dep = from_head ? -1 : cnt_dz(i, l);
        t.dep_n = 1;
        t.dep_need = need;
        t.sig = cnt_dz(i, l - 1);
        t.c_off = (*lay.dz_off)[i][l - 1];
        t.aux_off = (*lay.act_off)[i][l - 1];
        t.db_rows = lay.bias_colsums && bias_from_colsums(l - 1 == 0 ? in0p(i) : w) ? 32 : 0;  // dz_{l-1}'s column sums
        emit(vd, t, lay.B_cap / kRowTile, ns);
      }
      // the weight columns, and the bias column unless the bias gradient
      // comes from dZ's column sums (bias_from_colsums)
      const bool cs = lay.bias_colsums && bias_from_colsums(in_pad);
      std::vector<std::pair<int, int>> nw;
      split_n(cs ? in_pad : in_pad + 1, nw);
      TcTile t{};
      t.kind = kWgrad; t.member = i; t.layer = l;
      t.mask_off = -1;
      t.m_real = w; t.n_real = cs ? in_pad : in_pad + 1;
      t.db_rows = from_head ? kHeadRows : 32;
      t.db_off = cs ? (*lay.dz_off)[i][l] / 32 : -1;
      t.k_len = 0;
      t.map_a = plan.map_dz[(size_t)i * kMaxDepth + l];
      t.map_b = l == 0 ? (lay.xb_stride || lay.x0_off ? i : 0) : plan.map_act[(size_t)i * kMaxDepth + l - 1];
      t.ldc = in_pad;
      t.ld_aux = 0;
      t.dep = from_head ? -1 : cnt_dz(i, l);  // every row block of dz_l
      t.dep_n = 0;
      t.dep_need = need;
      t.sig = -1;
      t.c_off = (*lay.W_off)[i][l];
      t.aux_off = (*lay.b_off)[i][l];
      emit(vw, t, (int)ceil_div(w, kRowTile), nw);
    }
    auto by_cost = [&](const TcTile& a, const TcTile& b) { return cost(a) > cost(b); };
    std::stable_sort(vd.begin(), vd.end(), by_chain_cost);
    std::stable_sort(vw.begin(), vw.end(), by_cost);
  }
  // Nothing waits for a weight-gradient tile, so the wgrad tiles of level
  // lev move back beside the dgrad tiles of level lev + 1: in blocks of one
  // tile per resident CTA (pair), taken from the two lists in proportion to
  // their lengths, every CTA alternates between tiles whose epilogue streams
  // parameters (fused AdamW) and tiles whose time goes to the tensor cores.
  // A level starts with a block of wgrad tiles, which wait for nothing,
  // while the previous level's last dgrad rows finish.  Each tile still only
  // waits for tiles earlier in the list.
  auto interleave = [&](const std::vector<TcTile>& a, const std::vector<TcTile>& b) {
    const size_t blk = (size_t)std::max(1, plan.max_clusters);
    size_t ia = 0, ib = 0;
    while (ia < a.size() || ib < b.size()) {
      const bool take_a = ib >= b.size() || (ia < a.size() && ia * b.size() < ib * a.size());
      if (take_a) {
        const size_t e = std::min(a.size(), ia + blk);
        all.insert(all.end(), a.begin() + ia, a.begin() + e);
        ia = e;
      } else {
        const size_t e = std::min(b.size(), ib + blk);
        all.insert(all.end(), b.begin() + ib, b.begin() + e);
        ib = e;
      }
    }
  };
  if (Lmax > 0) {
    all.insert(all.end(), VD[0].begin(), VD[0].end());
    for (int lev = 1; lev < Lmax; ++lev) interleave(VD[lev], VW[lev - 1]);
    all.insert(all.end(), VW[Lmax - 1].begin(), VW[Lmax - 1].end());
  }
  plan.bwd_rng = {plan.fwd_rng.second, (int)all.size() - plan.fwd_rng.second};
  // Muon: every Newton-Schulz iteration's three products of the active
  // members' matrices in one launch, product after product (costliest tiles
  // first within each).  Counters, per matrix j: 3 j + 0 / 1 / 2 count the
  // stored X X^T / polynomial / update tiles (kEpiWarps per CTA with live
  // rows), cumulatively over the iterations.  Iteration it's X X^T tiles
  // wait for every update tile of iteration it - 1, its polynomial tiles for
  // every X X^T tile of it, its update tiles for every polynomial tile of it.
  // Every dependency lies in an earlier product of the list, and the chain
  // orders each buffer's rewrite after the last reads of its previous
  // contents (A and Bm each iteration, X every other).  Buffer 0 holds U
  // unnormalised: the first iteration's X X^T and update tiles carry the
  // matrix's 1 / |U|_F (ns_scale).
  plan.ns_rng = {(int)all.size(), 0};
  if (lay.muon && plan.ns_maps && lay.ns_steps > 0) {
    const int n_mat = (int)lay.muon->size();
    if (plan.n_ns_cnt != 3 * n_mat) {
      if (plan.ns_cnt_dev) cudaFree(plan.ns_cnt_dev);
      plan.ns_cnt_dev = nullptr;
      plan.n_ns_cnt = 3 * n_mat;
      if (cudaMalloc(&plan.ns_cnt_dev, sizeof(int) * plan.n_ns_cnt) != cudaSuccess ||
          cudaMemset(plan.ns_cnt_dev, 0, sizeof(int) * plan.n_ns_cnt) != cudaSuccess) {
        plan.n_ns_cnt = 0;
        err = "cudaMalloc(Newton-Schulz counters) failed";
        return TP_ENOMEM;
      }
    }
    // the tiles of one product of every active matrix (X buffer p), with
    // per matrix the number of CTAs with live rows
    std::vector<int> live[3];
    auto product = [&](int kind, int p) {
      std::vector<TcTile> v;
      for (int j = 0; j < n_mat; ++j) {
        const MuonMat& mt = (*lay.muon)[j];
        if (!active[mt.member]) continue;
        TcTile t{};
        t.member = mt.member;
        t.layer = mt.layer;
        t.m0 = 0;
        t.m_real = mt.r;
        t.dep = -1;
        t.sig = -1;
        t.mask_off = -1;
        if (kind == kNsGram) {        // A = X X^T
          t.n_real = mt.r;
          t.k_len = mt.c;
          t.map_a = t.map_b = plan.map_ns[j * 4 + p];
          t.c_off = mt.a_off;
          t.ldc = mt.r;
        } else if (kind == kNsPoly) { // Bm = b A + c A A
          t.n_real = mt.r;
          t.k_len = mt.r;
          t.map_a = t.map_b = plan.map_ns[j * 4 + 2];
          t.c_off = mt.bm_off;
          t.ldc = mt.r;
          t.aux_off = mt.a_off;
          t.ld_aux = mt.r;
        } else {                      // X' = a X + Bm X
          t.n_real = mt.c;
          t.k_len = mt.r;
          t.map_a = plan.map_ns[j * 4 + 3];
          t.map_b = plan.map_ns[j * 4 + p];
          t.c_off = mt.x_off[1 - p];
          t.ldc = mt.c;
          t.aux_off = mt.x_off[p];
          t.ld_aux = mt.c;
        }
        t.kind = kind;
        split_n(t.n_real, ns, 32);
        const size_t first = v.size();
        emit(v, t, (int)ceil_div(mt.r, kRowTile), ns);
        // A and Bm are symmetric: a tile whose elements all lie below the
        // diagonal (every column < every row) is left out; the epilogue of the
        // tiles on and above it writes each upper element and its mirror
        if (kind != kNsApply)
          v.erase(std::remove_if(v.begin() + first, v.end(),
                                 [](const TcTile& x) { return x.n0 + x.n_len <= x.m0; }),
                  v.end());
        int n_live = 0;
        for (size_t e = first; e < v.size(); ++e) {
          v[e].dep_n = 1;
          v[e].sig = 3 * j + (kind - kNsGram);
          for (int q = 0; q < cta; ++q) n_live += v[e].m0 + kRowTile * q < mt.r;
        }
        live[kind - kNsGram].resize(n_mat);
        live[kind - kNsGram][j] = kEpiWarps * n_live;
      }
      std::stable_sort(v.begin(), v.end(), [](const TcTile& a, const TcTile& b) {
        return (int64_t)a.k_len * a.n_len > (int64_t)b.k_len * b.n_len;
      });
      return v;
    };
    static_assert(kNsPoly == kNsGram + 1 && kNsApply == kNsGram + 2, "Newton-Schulz kinds are consecutive");
    for (int it = 0; it < lay.ns_steps; ++it) {
      const int p = it & 1;  // the X buffer read by this iteration
      for (int kind = kNsGram; kind <= kNsApply; ++kind) {
        std::vector<TcTile> v = product(kind, kind == kNsPoly ? 0 : p);
        for (TcTile& t : v) {
          const int j = t.sig / 3;
          const int prev = kind == kNsGram ? 2 : kind - kNsGram - 1;  // the product waited for
          const int done = kind == kNsGram ? it : it + 1;              // its iterations completed
          t.dep = done > 0 ? 3 * j + prev : -1;
          t.dep_need = done > 0 ? done * live[prev][j] : 0;
          if (it == 0 && kind != kNsPoly) t.ns_scale = j + 1;
          if (kind == kNsApply && it + 1 == lay.ns_steps) t.sig = -1;  // nothing waits for the last update
        }
        all.insert(all.end(), v.begin(), v.end());
      }
    }
    plan.ns_rng = {plan.ns_rng.first, (int)all.size() - plan.ns_rng.first};
  }
  if ((int)all.size() + 1 > plan.cap_tiles) {
    if (plan.tiles_dev) cudaFree(plan.tiles_dev);
    plan.cap_tiles = (int)all.size() + 1;
    if (cudaMalloc(&plan.tiles_dev, sizeof(TcTile) * plan.cap_tiles) != cudaSuccess) {
      err = "cudaMalloc(tc tiles) failed";
      return TP_ENOMEM;
    }
  }
  if (!all.empty() &&
      cudaMemcpy(plan.tiles_dev, all.data(), sizeof(TcTile) * all.size(), cudaMemcpyHostToDevice) != cudaSuccess) {
    err = "cudaMemcpy(tc tiles) failed";
    return TP_ECUDA;
  }
  plan.enabled = true;
  return TP_OK;
}

static tp_status launch(TcPlan& plan, cudaStream_t st, const std::pair<int, int>& rng, const TcArgs& base,
                        std::string& err, bool ns = false) {
  if (rng.second <= 0) return TP_OK;
  TcArgs a = base;
  a.tiles = plan.tiles_dev + rng.first;
  a.n_tiles = rng.second;
  a.maps = plan.maps_dev;
  a.err = plan.err_dev;
  a.cnt = ns ? plan.ns_cnt_dev : plan.cnt_dev;
  a.kmaj_off = plan.kmaj_off;
  a.wait_ns = plan.wait_ns;
  const int cta = plan.cta;
  // every CTA resident at once (the dataflow waits rely on it)
  const int n_clu = std::max(1, std::min(rng.second, plan.max_clusters));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_clu * cta);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = cta == 2 ? smem_bytes<2>() : smem_bytes<1>();
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = cta;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = cta == 2 ? 2 : 1;
  cudaError_t e = ns ? (cta == 2 ? cudaLaunchKernelEx(&cfg, k_tc_gemm<2, true>, a)
                                 : cudaLaunchKernelEx(&cfg, k_tc_gemm<1, true>, a))
                     : (cta == 2 ? cudaLaunchKernelEx(&cfg, k_tc_gemm<2, false>, a)
                                 : cudaLaunchKernelEx(&cfg, k_tc_gemm<1, false>, a));
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) {
    err = std::string("tcgen05 GEMM launch: ") + cudaGetErrorString(e);
    return TP_ECUDA;
  }
  return TP_OK;
}

tp_status tc_run_fwd(TcPlan& plan, cudaStream_t st, int B, int B_pad, int wcur, int train, const uint32_t* masks,
                     int mask_rows, const float* params, const MemberDev* mem, void* act, std::string& err) {
  TcArgs a{};
  a.B = B;
  a.B_pad = B_pad;
  a.train = train;
  a.masks = masks;
  a.mask_rows = mask_rows;
  a.w_shift = wcur ? plan.w_shift : 0;
  a.update = 0;
  a.params = params;
  a.mem = mem;
  a.act = (__nv_bfloat16*)act;
  return launch(plan, st, plan.fwd_rng, a, err);
}

tp_status tc_run_bwd(TcPlan& plan, cudaStream_t st, int B, int B_pad, int wcur, const MemberDev* mem, void* act,
                     void* dz, float* grads, float* dbp, int update, const AdamDev& adam, std::string& err) {
  TcArgs a{};
  a.B = B;
  a.B_pad = B_pad;
  a.w_shift = wcur ? plan.w_shift : 0;
  a.update = update;
  a.mem = mem;
  a.act = (__nv_bfloat16*)act;
  a.dz = (__nv_bfloat16*)dz;
  a.grads = grads;
  a.dbp = dbp;
  a.adam = adam;
  return launch(plan, st, plan.bwd_rng, a, err);
}

tp_status tc_run_ns(TcPlan& plan, cudaStream_t st, void* ns, const float* ns_scale, const MemberDev* mem,
                    std::string& err) {
  TcArgs a{};
  a.B = 0;
  a.B_pad = 0;
  a.mem = mem;  // the epilogue reads every tile's member record
  a.ns = (__nv_bfloat16*)ns;
  a.ns_scale = ns_scale;
  return launch(plan, st, plan.ns_rng, a, err, true);
}

tp_status tc_check(TcPlan& plan, cudaStream_t st, std::string& err) {
  if (!plan.err_dev) return TP_OK;
  int v = 0;
  if (cudaMemcpyAsync(&v, plan.err_dev, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess) {
    err = "reading the tcgen05 error word failed";
    return TP_ECUDA;
  }
  if (v) {
    cudaMemsetAsync(plan.err_dev, 0, sizeof(int), st);
    err = "a tcgen05 GEMM pipeline wait timed out (wait site " + std::to_string(v) + ")";
    return TP_ETIMEOUT;
  }
  return TP_OK;
}

tp_status tc_debug_poison(TcPlan& plan, cudaStream_t st, std::string& err) {
  const int n = plan.fwd_rng.second;
  if (!plan.tiles_dev || n <= 0) {
    err = "no forward tiles to poison";
    return TP_ESTATE;
  }
  std::vector<TcTile> t((size_t)n);
  if (cudaStreamSynchronize(st) != cudaSuccess ||
      cudaMemcpy(t.data(), plan.tiles_dev + plan.fwd_rng.first, sizeof(TcTile) * n, cudaMemcpyDeviceToHost) !=
          cudaSuccess) {
    err = "reading the tile list failed";
    return TP_ECUDA;
  }
  for (int i = 0; i < n; ++i)
    if (t[i].dep >= 0) {
      // a count the launch never reaches: the producer of this tile waits
      // before it issues any copy, gives up after wait_ns and aborts its CTA
      t[i].dep_need = 1 << 30;
      if (cudaMemcpy(plan.tiles_dev + plan.fwd_rng.first + i, &t[i], sizeof(TcTile), cudaMemcpyHostToDevice) !=
          cudaSuccess) {
        err = "writing the tile list failed";
        return TP_ECUDA;
      }
      return TP_OK;
    }
  err = "no forward tile waits on a dependency (a pack of depth-1 members)";
  return TP_ESTATE;
}

void tc_free_plan(TcPlan& plan) {
  if (plan.maps_dev) cudaFree(plan.maps_dev);
  if (plan.tiles_dev) cudaFree(plan.tiles_dev);
  if (plan.err_dev) cudaFree(plan.err_dev);
  if (plan.cnt_dev) cudaFree(plan.cnt_dev);
  plan.cnt_dev = nullptr;
  plan.n_cnt = 0;
  if (plan.ns_cnt_dev) cudaFree(plan.ns_cnt_dev);
  plan.ns_cnt_dev = nullptr;
  plan.n_ns_cnt = 0;
  plan.maps_dev = nullptr;
  plan.tiles_dev = nullptr;
  plan.cap_tiles = 0;
  plan.err_dev = nullptr;
  plan.enabled = false;
  plan.ns_maps = false;
  plan.map_ns.clear();
}

}  // namespace tp
