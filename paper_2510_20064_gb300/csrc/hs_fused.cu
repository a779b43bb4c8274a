// hs_fused.cu -- single-read stochastic feedback (Thm 1) on thread-block
// clusters.
//
// alpha = sum_v min(p_v, q_v) needs each drafter row's normaliser before the
// min, so a row has to stay on chip between its sum pass and its overlap
// pass.  A vocabulary row (up to ~300 KB of bf16) does not fit one SM, so a
// cluster of C CTAs takes one (b,k) tile, each CTA a V/C slice, and loops
// persistently over tiles:
//   * the CTA's slice of every row of its tiles -- the target row, then the
//     N drafter rows -- streams into a 3-stage shared-memory ring with
//     cp.async.bulk (TMA; each CTA reads its own slice, no multicast); a
//     coordinator warp refills a stage as soon as every consumer has read it;
//   * 15 consumer warps load a row from the ring into registers, form
//     e_v = 2^{z_v c - o_w} with o_w = c * (the warp's max), c = log2e/T,
//     and their sum (one ex2 per logit, values kept in registers);
//   * the cluster merges the per-CTA (offset, sum) pairs through distributed
//     shared memory: every CTA stores its pair into each peer and arrives on
//     the peer's mbarrier; then every thread knows the row's offset O and
//     normaliser Z, and p_v or q_v = e_v 2^{o_t - O} / Z;
//   * the target's p stays in shared memory (fp32) for the tile's N drafters;
//     a drafter row adds sum_v min(p_v, q_v) to its per-warp partial;
//   * at the end of a tile the coordinator sums the warps' N partials and
//     sends them to the cluster's rank 0, whose coordinator sums them in rank
//     order and writes alpha[:, b, k] one tile later.  The coordinator never
//     blocks: its waits poll, servicing ring refills meanwhile, and no
//     consumer warp waits for another warp of its CTA.
// Rows are software-pipelined: the pass over row g+1's logits runs while
// row g's cluster exchange is in flight, so each thread holds two rows of
// exponentials (eA / eB).  Every wait is bounded; on expiry the kernel
// records HS_ERR_TIMEOUT and finishes without waiting further.
#include <math.h>
#include <stdint.h>

#include <mutex>

#include "hs_common.cuh"
#include "hs_fused.h"
#include "hs_twopass.h"

namespace hs {
namespace fused {
namespace {

// 15 consumer warps + 1 load warp: 16 warps put 4 on each SM sub-partition,
// which leaves 128 registers per thread for the two rows of exponentials a
// consumer thread keeps.
constexpr int kConsumerWarps = 15;
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kThreads = kConsumers + 32;
constexpr int kStages = 4;
constexpr int kXSlots = 8;  // rows whose exchange may be in flight at once
constexpr int kXArm = 4;    // the xbar phase of row g + kXArm is armed at row g
constexpr int kASlots = 8;  // tiles whose alpha partials may be in flight (rank 0)
constexpr int kTSlots = 4;  // tiles whose per-warp partials await the coordinator
constexpr int kMaxU = 5;    // 16-byte vectors per consumer thread and row

// TMEM row slots of exponentials per consumer thread: the 512 columns of a
// lane quadrant hold, for each of its 4 consumer warps, the tile's p and the
// slots, 8U columns each.  (Three slots fit when U <= 4, for rows pipelined
// four deep; measured, that was no faster: the row rate is not set by the
// exchange latency the depth would hide.)
constexpr int kSlots = 2;
constexpr int kMaxRanks = 16;  // CTAs per cluster (above 8: a non-portable size)
constexpr long long kTimeoutCycles = 1LL << 31;  // about a second
constexpr uint32_t kNegInfBf16x2 = 0xFF80FF80u;
constexpr uint32_t kNegInfF16x2 = 0xFC00FC00u;

struct __align__(16) Shared {
  uint64_t full[kStages];          // ring stage loaded (TMA complete_tx)
  uint64_t redbar[kXSlots];        // every consumer warp posted its row pair
  uint64_t xbar[kXSlots];          // every rank's pair of a row arrived
  uint64_t accbar[kTSlots];        // every consumer warp posted a tile's partials
  uint64_t abar[kASlots];          // every rank's tile partials arrived (rank 0)
  float2 red[kXSlots][16];                // per-warp (offset, sum) of a row
  float2 xch[kXSlots][kMaxRanks];         // per-rank (offset, sum) of a row
  float acc[kTSlots][kMaxN][kConsumerWarps];  // per-warp alpha partials of a tile
  uint64_t rowbar[kXSlots];               // a row's per-warp scales are published
  float rowf[kXSlots][16];                // per-warp scale f: p or q = f * exponential
  uint32_t tval[kASlots];                 // tile's target row is usable
  uint32_t dval[kASlots];                 // bit i: tile's drafter i row is usable
  float clacc[kASlots][kMaxRanks][kMaxN];  // per-rank alpha partials (rank 0)
  int error;
  uint32_t tmem_base;  // tensor memory: p and two rows of exponentials per thread
};

struct Params {
  const void* target;
  const int32_t* path;
  int M;
  const void* drafter;
  int N, B, P, V;
  float c;     // log2(e) / T
  int S;       // slice length in elements (multiple of 8)
  int ntiles;  // B * P
  float* alpha;
  int* dev_status;
};

// ---- PTX wrappers -----------------------------------------------------------

__device__ __forceinline__ uint32_t saddr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_id() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_count() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t mapa(uint32_t a, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
               :: "r"(bar), "r"(bytes) : "memory");
}
// try_wait suspends the thread until the phase completes or a system-chosen
// time limit passes, so a waiting warp does not spin through the issue slots.
// (Without a time-limit operand: on the two-pass kernel that form measured
// fewer instructions and 3% less time than a 1 ms limit.)
__device__ __forceinline__ bool mbar_test_cta(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile("{\n\t.reg .pred p;\n\t"
               "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
               "selp.u32 %0, 1, 0, p;\n\t}"
               : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile("{\n\t.reg .pred p;\n\t"
               "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
               "selp.u32 %0, 1, 0, p;\n\t}"
               : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
  return ok != 0;
}
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes,
                                          uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes "
               "[%0], [%1], %2, [%3];"
               :: "r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}
// Store a pair into another CTA of the cluster; the store itself completes 8
// bytes of the transaction count of that CTA's mbarrier (no fence needed).
__device__ __forceinline__ void st_async_f2(uint32_t a, float x, float y, uint32_t bar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];"
               :: "r"(a), "f"(x), "f"(y), "r"(bar) : "memory");
}
__device__ __forceinline__ void st_async_f(uint32_t a, float x, uint32_t bar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.f32 [%0], %1, [%2];"
               :: "r"(a), "f"(x), "r"(bar) : "memory");
}
__device__ __forceinline__ uint4 lds128(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
  return v;
}

// Bounded wait on an mbarrier phase (the slow path of wait_phase).  Returns false (and records a timeout
// once per CTA) when the phase did not complete in time or an earlier wait
// of this CTA already timed out.
// The exit drain passes fast_fail = false: it must see in-flight copies land
// even after another wait has given up.
__device__ __noinline__ bool wait_slow(uint32_t bar, uint32_t parity, Shared& sh,
                                       int* dev_status, bool fast_fail) {
  const long long t0 = clock64();
  while (true) {
    if (fast_fail && *reinterpret_cast<volatile int*>(&sh.error)) return false;
    if (mbar_test(bar, parity)) return true;
    if (clock64() - t0 > kTimeoutCycles) {
      *reinterpret_cast<volatile int*>(&sh.error) = 1;
      report(dev_status, HS_ERR_TIMEOUT);
      return false;
    }
  }
}

__device__ __forceinline__ bool wait_phase(uint32_t bar, uint32_t parity, Shared& sh,
                                           int* dev_status, bool fast_fail = true) {
  if (mbar_test(bar, parity)) return true;
  return wait_slow(bar, parity, sh, dev_status, fast_fail);
}
// The same for a barrier that only this CTA's own threads complete: the
// fast path acquires at CTA scope.
__device__ __forceinline__ bool wait_local(uint32_t bar, uint32_t parity, Shared& sh,
                                           int* dev_status) {
  if (mbar_test_cta(bar, parity)) return true;
  return wait_slow(bar, parity, sh, dev_status, true);
}

// ---- per-element helpers ----------------------------------------------------

template <int DT>
__device__ __forceinline__ uint32_t pmax(uint32_t a, uint32_t b) {
  uint32_t r;
  if (DT == HS_BF16)
    asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  else
    asm("max.NaN.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
template <int DT>
__device__ __forceinline__ float lo(uint32_t w) {
  if (DT == HS_BF16) return __uint_as_float(w << 16);
  return __half2float(__ushort_as_half(static_cast<unsigned short>(w & 0xffffu)));
}
template <int DT>
__device__ __forceinline__ float hi(uint32_t w) {
  if (DT == HS_BF16) return __uint_as_float(w & 0xffff0000u);
  return __half2float(__ushort_as_half(static_cast<unsigned short>(w >> 16)));
}

// Packed fp32 pairs (sm_100+ f32x2 arithmetic: one instruction, two lanes).
typedef unsigned long long f2_t;
__device__ __forceinline__ f2_t pk(float a, float b) {
  f2_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void upk(f2_t v, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(v));
}
__device__ __forceinline__ f2_t ffma2(f2_t a, f2_t b, f2_t c) {
  f2_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
__device__ __forceinline__ f2_t fadd2(f2_t a, f2_t b) {
  f2_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ f2_t fmul2(f2_t a, f2_t b) {
  f2_t r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}

// ---- tensor memory ------------------------------------------------------------
// Each consumer thread keeps, in its own TMEM lane, the target's p for its
// positions and the exponentials of two rows (one 32-bit column per value):
// the register file then only holds the row being computed.
__device__ __forceinline__ void tmem_alloc512(uint32_t dst_smem) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;"
               :: "r"(dst_smem) : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc512(uint32_t taddr) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" :: "r"(taddr) : "memory");
}
__device__ __forceinline__ void tmem_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tmem_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
// 8 or 16 consecutive columns of this thread's lane, as packed pairs.
template <int NV>
__device__ __forceinline__ void tmem_st(uint32_t taddr, const f2_t* v) {
  float f[2 * NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) upk(v[i], f[2 * i], f[2 * i + 1]);
  if (NV == 4)
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};"
                 :: "r"(taddr), "f"(f[0]), "f"(f[1]), "f"(f[2]), "f"(f[3]), "f"(f[4]),
                    "f"(f[5]), "f"(f[6]), "f"(f[7]) : "memory");
  else
    asm volatile("tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, "
                 "%9, %10, %11, %12, %13, %14, %15, %16};"
                 :: "r"(taddr), "f"(f[0]), "f"(f[1]), "f"(f[2]), "f"(f[3]), "f"(f[4]),
                    "f"(f[5]), "f"(f[6]), "f"(f[7]), "f"(f[8]), "f"(f[9]), "f"(f[10]),
                    "f"(f[11]), "f"(f[12]), "f"(f[13]), "f"(f[14]), "f"(f[15]) : "memory");
}
template <int NV>
__device__ __forceinline__ void tmem_ld(uint32_t taddr, f2_t* v) {
  float f[2 * NV];
  if (NV == 4)
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                 : "=f"(f[0]), "=f"(f[1]), "=f"(f[2]), "=f"(f[3]), "=f"(f[4]), "=f"(f[5]),
                   "=f"(f[6]), "=f"(f[7]) : "r"(taddr) : "memory");
  else
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, "
                 "%9, %10, %11, %12, %13, %14, %15}, [%16];"
                 : "=f"(f[0]), "=f"(f[1]), "=f"(f[2]), "=f"(f[3]), "=f"(f[4]), "=f"(f[5]),
                   "=f"(f[6]), "=f"(f[7]), "=f"(f[8]), "=f"(f[9]), "=f"(f[10]), "=f"(f[11]),
                   "=f"(f[12]), "=f"(f[13]), "=f"(f[14]), "=f"(f[15]) : "r"(taddr) : "memory");
#pragma unroll
  for (int i = 0; i < NV; ++i) v[i] = pk(f[2 * i], f[2 * i + 1]);
}

__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
// Warp maximum, NaN if any lane holds a NaN (sm_100+ redux on f32).
__device__ __forceinline__ float warp_max_f(float f) {
  float r;
  asm volatile("redux.sync.max.NaN.f32 %0, %1, 0xffffffff;" : "=f"(r) : "f"(f));
  return r;
}
__device__ __forceinline__ float fmax_nan(float a, float b) {
  float r;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}

// ---- the kernel ---------------------------------------------------------------

// The coordinator's walk over the global addresses of this CTA's slices of
// its rows, in stream order: per tile, the target row, then the N drafter
// rows.  One division per tile; the tree path index of the next tile is
// fetched a tile ahead.
struct RowWalk {
  int r = 0;             // row within the tile
  int64_t tile = 0;      // global tile index b * P + k
  const char* tsrc;      // target row slice of the current tile
  const char* dsrc;      // drafter 0's row slice of the current tile
  int64_t dstride;       // bytes from drafter i's row to drafter i+1's
  int next_path = 0;     // path index of the next tile (tree targets)

  __device__ void start_tile(const Params& p, int64_t slice0, int nd) {
    const int64_t b = tile / p.P, k = tile - b * p.P;
    const int64_t trow = p.path ? b * p.M + ((nd < 0 || nd >= p.M) ? 0 : nd) : tile;
    tsrc = static_cast<const char*>(p.target) + (trow * p.V + slice0) * 2;
    dsrc = static_cast<const char*>(p.drafter) + ((b * p.P + k) * p.V + slice0) * 2;
  }
  __device__ void init(const Params& p, uint32_t cid, uint32_t ncl, int64_t slice0) {
    tile = cid;
    dstride = int64_t(p.B) * p.P * p.V * 2;
    const int nd = (p.path && tile < p.ntiles) ? p.path[tile] : 0;
    if (p.path && tile + ncl < p.ntiles) next_path = p.path[tile + ncl];
    if (tile < p.ntiles) start_tile(p, slice0, nd);
  }
  // source of the current row; then advance
  __device__ const char* next(const Params& p, uint32_t ncl, int64_t slice0) {
    const char* src = r == 0 ? tsrc : dsrc + (r - 1) * dstride;
    if (++r == p.N + 1) {
      r = 0;
      tile += ncl;
      if (tile < p.ntiles) {
        const int nd = next_path;
        if (p.path && tile + ncl < p.ntiles) next_path = p.path[tile + ncl];
        start_tile(p, slice0, nd);
      }
    }
    return src;
  }
};

// Stream one row slice into `stage` (one thread).
__device__ __forceinline__ void issue(Shared& sh, unsigned char* stage, int g, const char* src,
                                      uint32_t bytes) {
  const uint32_t full = saddr(&sh.full[g % kStages]);
  if (bytes) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    mbar_arrive_tx(full, bytes);
    bulk_load(saddr(stage), src, bytes, full);
  } else {
    mbar_arrive(full);
  }
}

template <int DT, int U>
__global__ void __launch_bounds__(kThreads, 1) fused_kernel(const Params p) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  Shared& sh = *reinterpret_cast<Shared*>(smem_raw);
  // every ring stage holds SU = U * kConsumers * 8 >= S elements so that
  // each consumer thread always handles U whole 16-byte vectors; the part
  // past the CTA's slice is -inf (set once, below)
  constexpr int SU = U * kConsumers * 8;
  constexpr uint32_t stage_bytes = SU * 2;
  // TMEM: the consumer warps of one lane quadrant (warps w, w+4, ...) each
  // take 3 * 8U columns (p and two row slots) of the 512
  constexpr int kDepth = kSlots + 1;  // rows in flight per consumer warp
  static_assert(((kConsumerWarps + 3) / 4) * (1 + kSlots) * U * 8 <= 512, "TMEM columns");
  static_assert(kDepth <= kXArm, "a row's exchange slot is re-armed kXArm rows later");
  unsigned char* ring = smem_raw + ((sizeof(Shared) + 127) & ~size_t(127));

  pdl_trigger();  // the small e_len kernel may take the SMs no cluster uses
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = cluster_rank();
  uint32_t C;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(C));
  const uint32_t cid = cluster_id(), ncl = cluster_count();
  const int N = p.N, B = p.B, P = p.P, V = p.V;
  const int my_tiles = cid < uint32_t(p.ntiles) ? int((p.ntiles - 1 - cid) / ncl) + 1 : 0;
  const int R = N + 1;        // rows per tile: the target, then the N drafters
  const int G = my_tiles * R;  // rows this CTA streams
  const int64_t slice0 = int64_t(rank) * p.S;
  const int64_t rest = int64_t(V) - slice0;
  const int len = rest <= 0 ? 0 : (rest < p.S ? int(rest) : p.S);
  const uint32_t bytes = uint32_t(len) * 2u;

  {
    const uint32_t neg = (DT == HS_BF16) ? kNegInfBf16x2 : kNegInfF16x2;
    for (int e = len / 2 + tid; e < SU / 2; e += kThreads)
      for (int s = 0; s < kStages; ++s)
        reinterpret_cast<uint32_t*>(ring + s * stage_bytes)[e] = neg;
  }
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(saddr(&sh.full[s]), 1);
    for (int x = 0; x < kXSlots; ++x) {
      mbar_init(saddr(&sh.redbar[x]), kConsumerWarps);
      mbar_init(saddr(&sh.xbar[x]), 1);
      mbar_init(saddr(&sh.rowbar[x]), 1);
    }
    for (int a = 0; a < kTSlots; ++a) mbar_init(saddr(&sh.accbar[a]), kConsumerWarps);
    for (int a = 0; a < kASlots; ++a) mbar_init(saddr(&sh.abar[a]), 1);
    sh.error = 0;
    // each row's xbar phase: one local arrival (the arm) plus 8 bytes from
    // every rank; the first kXArm rows are armed before any rank can send
    for (int g = 0; g < kXArm && g < G; ++g) mbar_arrive_tx(saddr(&sh.xbar[g]), 8u * C);
    // rank 0's abar phase of tile j: one local arrival (the arm) plus 4 bytes
    // per drafter from every rank; tiles 0..kASlots-1 are armed here, tile
    // j + kASlots once tile j is finished
    for (int a = 0; a < kASlots && a < my_tiles; ++a)
      mbar_arrive_tx(saddr(&sh.abar[a]), 4u * N * C);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) tmem_alloc512(saddr(&sh.tmem_base));
  tmem_fence_before();
  cluster_sync_all();
  tmem_fence_after();
  pdl_wait();  // the set-up above overlaps the previous kernel of the stream

  if (warp == kConsumerWarps) {
    // ---------------------------- coordinator -----------------------------
    // Per row g: waits until every consumer warp posted its pass-1 pair (so
    // the row's ring stage has been read), refills that stage with row
    // g + kStages, merges the warps' pairs and sends the CTA's pair to every
    // rank.  Tile j's per-warp alpha partials are complete once row
    // (j+1)(N+1) + 2 is posted (the consumers run pass 1 two rows ahead of
    // pass 2); they are then summed and sent to rank 0, which writes alpha
    // one tile late.  Every wait sleeps in mbarrier try_wait (bounded).
    RowWalk walk;
    if (lane == 0) {
      walk.init(p, cid, ncl, slice0);
      for (int g = 0; g < G && g < kStages; ++g)
        issue(sh, ring + g * stage_bytes, g, walk.next(p, ncl, slice0), bytes);
    }
    auto finish = [&](int j) {  // rank 0: alpha[:, b, k] of tile j
      wait_local(saddr(&sh.abar[j % kASlots]), uint32_t(j / kASlots) & 1u, sh, p.dev_status);
      if (lane < N) {
        const int64_t tile = int64_t(cid) + int64_t(j) * ncl;
        const int64_t b = tile / P, k = tile % P;
        float t = 0.f;
        for (uint32_t rr = 0; rr < C; ++rr) t += sh.clacc[j % kASlots][rr][lane];
        const bool bad_path = p.path && (p.path[tile] < 0 || p.path[tile] >= p.M);
        if (bad_path || !sh.tval[j % kASlots] || !((sh.dval[j % kASlots] >> lane) & 1u)) {
          t = __int_as_float(0x7fc00000);
          report(p.dev_status, bad_path ? HS_ERR_INVALID_ARG : HS_ERR_NONFINITE);
        }
        p.alpha[(int64_t(lane) * B + b) * P + k] = t;
      }
      __syncwarp();
      if (lane == 0 && j + kASlots < my_tiles)
        mbar_arrive_tx(saddr(&sh.abar[j % kASlots]), 4u * N * C);
    };
    auto reduce_tile = [&](int j) {  // tile j's partials -> rank 0
      const int ts = j % kTSlots;
      wait_local(saddr(&sh.accbar[ts]), uint32_t(j / kTSlots) & 1u, sh, p.dev_status);
      if (lane < N) {
        float t = 0.f;
        for (int w = 0; w < kConsumerWarps; ++w) t += sh.acc[ts][lane][w];
        st_async_f(mapa(saddr(&sh.clacc[j % kASlots][rank][lane]), 0), t,
                   mapa(saddr(&sh.abar[j % kASlots]), 0));
      }
      if (rank == 0 && j > 0) finish(j - 1);  // long since complete
    };
    // B(g): every rank's pair of row g -> the row's offset O and normaliser
    // Z (a butterfly over each group of 8 lanes, lane l holding rank l & 7),
    // then each consumer warp's scale f_w = 2^{o_w - O} / Z and the row's
    // validity; published through rowbar.
    int rB = 0, jB = 0;  // row within tile and tile of the next B step
    auto publish = [&](int g) {
      const int x = g % kXSlots;
      wait_local(saddr(&sh.xbar[x]), uint32_t(g / kXSlots) & 1u, sh, p.dev_status);
      // every lane merges the C pairs itself, in rank order
      float2 v[kMaxRanks];
#pragma unroll
      for (int rr = 0; rr < kMaxRanks; ++rr)
        v[rr] = rr < int(C) ? sh.xch[x][rr] : make_float2(-INFINITY, 0.f);
      float O = v[0].x;
#pragma unroll
      for (int rr = 1; rr < kMaxRanks; ++rr) O = fmax_nan(O, v[rr].x);
      float Z = 0.f;
#pragma unroll
      for (int rr = 0; rr < kMaxRanks; ++rr)
        Z += (v[rr].x == -INFINITY || O == -INFINITY) ? 0.f : v[rr].y * ex2(v[rr].x - O);
      const bool valid = isfinite(O) && Z > 0.f;
      if (lane < kConsumerWarps) {
        const float o = sh.red[x][lane].x;  // the offset warp `lane` used
        sh.rowf[x][lane] = (!valid || o == -INFINITY) ? 0.f : ex2(o - O) * rcp_approx(Z);
      }
      if (lane == 0) {
        const int a = jB % kASlots;
        if (rB == 0) {
          sh.tval[a] = valid ? 1u : 0u;
          sh.dval[a] = 0u;
        } else if (valid) {
          sh.dval[a] |= 1u << (rB - 1);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(saddr(&sh.rowbar[x]));
      if (++rB == R) {
        rB = 0;
        ++jB;
      }
    };
    int reduced = 0;  // tiles sent to rank 0
    for (int g = 0; g < G; ++g) {
      const int x = g % kXSlots;
      wait_local(saddr(&sh.redbar[x]), uint32_t(g / kXSlots) & 1u, sh, p.dev_status);
      if (lane == 0 && g + kStages < G)
        issue(sh, ring + (g % kStages) * stage_bytes, g + kStages, walk.next(p, ncl, slice0),
              bytes);
      // row g - kXArm's exchange is complete here (the consumers have passed
      // pass 2 of row g - kDepth, kDepth <= kXArm), so its slot can be armed
      // for row g + kXArm,
      // which no rank sends before this CTA has posted row g + 1
      if (lane == 0 && g + kXArm < G)
        mbar_arrive_tx(saddr(&sh.xbar[(g + kXArm) % kXSlots]), 8u * C);
      const float2 v = lane < kConsumerWarps ? sh.red[x][lane] : make_float2(-INFINITY, 0.f);
      const float oc = warp_max_f(v.x);
      float sc = (v.x == -INFINITY || oc == -INFINITY) ? 0.f : v.y * ex2(v.x - oc);
#pragma unroll
      for (int d = 8; d > 0; d >>= 1) sc += __shfl_xor_sync(0xffffffffu, sc, d);
      if (lane < int(C))
        st_async_f2(mapa(saddr(&sh.xch[x][rank]), lane), oc, sc, mapa(saddr(&sh.xbar[x]), lane));
      if (g > 0) publish(g - 1);
      // a tile's alpha partials are complete once the consumers have passed
      // pass 2 of its last row, kDepth rows behind the posts of row g
      while (reduced < my_tiles && (reduced + 1) * R + kDepth - 1 <= g) reduce_tile(reduced++);
    }
    if (G > 0) publish(G - 1);
    while (reduced < my_tiles) reduce_tile(reduced++);
    if (G > 0 && rank == 0) finish(my_tiles - 1);
    // drain: every copy has landed before the CTA may exit
    if (lane == 0)
      for (int g = max(0, G - kStages); g < G; ++g)
        wait_phase(saddr(&sh.full[g % kStages]), uint32_t(g / kStages) & 1u, sh, p.dev_status,
                   false);
  } else if (G > 0) {
    // ------------------------------ consumers -----------------------------
    const float c = p.c;
    // the last vector round holds the slice's tail: warps whose vectors there
    // all lie past the slice skip it (they would only see the -inf padding)
    const bool tail = (U - 1) * kConsumers + warp * 32 < len / 8;
    // this thread's TMEM lane (the warp's quadrant) and columns: [0, 8U) p of
    // the tile's target, [8U (1+s), 8U (2+s)) the exponentials of row slot s
    const uint32_t tbase = sh.tmem_base + (uint32_t(32 * (warp & 3)) << 16) +
                           uint32_t((warp >> 2) * (1 + kSlots) * U * 8);

    // pass 1: load row g from the ring (then release the stage); warp max;
    // exponentials relative to the warp's offset; post the warp's (offset,
    // sum) for the coordinator.  E keeps the exponentials (packed pairs).
    auto pass1 = [&](int g, f2_t (&E)[U * 4]) {
      const int s = g % kStages;
      wait_local(saddr(&sh.full[s]), uint32_t(g / kStages) & 1u, sh, p.dev_status);
      const uint32_t stage = saddr(ring + s * stage_bytes);
      uint32_t w[U * 4];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        uint4 v = make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
        if (DT != HS_BF16) v = make_uint4(kNegInfF16x2, kNegInfF16x2, kNegInfF16x2, kNegInfF16x2);
        if (u < U - 1 || tail) v = lds128(stage + (u * kConsumers + tid) * 16);
        w[4 * u] = v.x; w[4 * u + 1] = v.y; w[4 * u + 2] = v.z; w[4 * u + 3] = v.w;
      }
      uint32_t mx[U * 2];  // pairwise tree: log-depth dependency chain
#pragma unroll
      for (int q = 0; q < U * 2; ++q) mx[q] = pmax<DT>(w[2 * q], w[2 * q + 1]);
#pragma unroll
      for (int d = 1; d < U * 2; d *= 2)
#pragma unroll
        for (int q = 0; q + d < U * 2; q += 2 * d) mx[q] = pmax<DT>(mx[q], mx[q + d]);
      const float m = warp_max_f(fmax_nan(lo<DT>(mx[0]), hi<DT>(mx[0])));
      const float o = (m == -INFINITY) ? -INFINITY : m * c;
      const float o_used = (m == -INFINITY) ? 0.f : o;
      const f2_t cc = pk(c, c), off = pk(-o_used, -o_used);
      f2_t acc[2] = {pk(0.f, 0.f), pk(0.f, 0.f)};
#pragma unroll
      for (int q = 0; q < U * 4; ++q) {
        if (q < (U - 1) * 4 || tail) {
          float a, b;
          upk(ffma2(pk(lo<DT>(w[q]), hi<DT>(w[q])), cc, off), a, b);
          E[q] = pk(ex2(a), ex2(b));
          acc[q & 1] = fadd2(acc[q & 1], E[q]);
        }
      }
      float s0, s1, s2, s3;
      upk(acc[0], s0, s1);
      upk(acc[1], s2, s3);
      const float sum = warp_sum((s0 + s1) + (s2 + s3));
      if (lane == 0) {
        sh.red[g % kXSlots][warp] = make_float2(o, sum);
        mbar_arrive(saddr(&sh.redbar[g % kXSlots]));
      }
    };

    // the exponentials of a row into its TMEM slot, two vectors per store
    auto store_row = [&](int slot, const f2_t (&E)[U * 4]) {
      const uint32_t t = tbase + uint32_t((1 + slot) * U * 8);
#pragma unroll
      for (int u = 0; u < U; u += 2) {
        if (u + 1 < U) {
          if (u + 1 < U - 1 || tail) tmem_st<8>(t + u * 8, &E[4 * u]);
          else tmem_st<4>(t + u * 8, &E[4 * u]);
        } else if (tail) {
          tmem_st<4>(t + u * 8, &E[4 * u]);
        }
      }
    };

    // pass 2 of row g (exponentials in TMEM slot g % kSlots): target -> p into
    // TMEM; drafter i -> alpha partial
    auto pass2 = [&](int g, int j, int r) {
      const int x = g % kXSlots;
      wait_local(saddr(&sh.rowbar[x]), uint32_t(g / kXSlots) & 1u, sh, p.dev_status);
      const float f = sh.rowf[x][warp];
      const f2_t ff = pk(f, f);
      const uint32_t te = tbase + uint32_t((1 + g % kSlots) * U * 8);
      tmem_wait_st();  // this row's exponentials and the tile's p have landed
      if (r == 0) {
#pragma unroll
        for (int u = 0; u < U; u += 2) {
          f2_t e[8];
          if (u + 1 < U && (u + 1 < U - 1 || tail)) {
            tmem_ld<8>(te + u * 8, e);
            tmem_wait_ld();
#pragma unroll
            for (int h = 0; h < 8; ++h) e[h] = fmul2(e[h], ff);
            tmem_st<8>(tbase + u * 8, e);
          } else if (u + 1 < U || tail) {
            tmem_ld<4>(te + u * 8, e);
            tmem_wait_ld();
#pragma unroll
            for (int h = 0; h < 4; ++h) e[h] = fmul2(e[h], ff);
            tmem_st<4>(tbase + u * 8, e);
          }
        }
        return;
      }
      const int i = r - 1;
      f2_t acc[2] = {pk(0.f, 0.f), pk(0.f, 0.f)};
#pragma unroll
      for (int u = 0; u < U; u += 2) {
        f2_t e[8], pv[8];
        int nv = 0;
        if (u + 1 < U && (u + 1 < U - 1 || tail)) {
          tmem_ld<8>(te + u * 8, e);
          tmem_ld<8>(tbase + u * 8, pv);
          nv = 8;
        } else if (u + 1 < U || tail) {
          tmem_ld<4>(te + u * 8, e);
          tmem_ld<4>(tbase + u * 8, pv);
          nv = 4;
        }
        if (nv) {
          tmem_wait_ld();
#pragma unroll
          for (int h = 0; h < 8; ++h) {
            if (h < nv) {
              float xx, yy, pa, pb;
              upk(fmul2(e[h], ff), xx, yy);
              upk(pv[h], pa, pb);
              acc[h & 1] = fadd2(acc[h & 1], pk(fminf(pa, xx), fminf(pb, yy)));
            }
          }
        }
      }
      float a0, a1, a2, a3;
      upk(acc[0], a0, a1);
      upk(acc[1], a2, a3);
      const float a = warp_sum((a0 + a1) + (a2 + a3));
      if (lane == 0) {
        const int ts = j % kTSlots;
        sh.acc[ts][i][warp] = a;
        if (i == N - 1) mbar_arrive(saddr(&sh.accbar[ts]));  // tile end
      }
    };

    // kDepth rows in flight: pass 1 of row g + kDepth - 1 runs before pass 2
    // of row g, so the cluster exchange of a row has kDepth - 1 rows of work
    // to hide behind; row r's exponentials live in TMEM slot r % kSlots (row
    // g + kSlots takes the slot row g frees)
    f2_t E[U * 4];
    int jj = 0, rr = 0;  // tile and row within tile of row g
    for (int g = -kSlots; g < G; ++g) {
      const bool more = g + kSlots < G;
      if (more) pass1(g + kSlots, E);
      if (g >= 0) {
        pass2(g, jj, rr);
        if (++rr == R) {
          rr = 0;
          ++jj;
        }
      }
      if (more) store_row((g + kSlots) % kSlots, E);
    }
  }
  // no CTA may leave while a peer can still write into its shared memory;
  // the tensor memory is released once every warp is done with it
  __syncwarp();
  tmem_fence_before();
  cluster_sync_all();
  tmem_fence_after();
  if (warp == 0) tmem_dealloc512(sh.tmem_base);
}

// ---- host side ------------------------------------------------------------------

// The kernel takes all 512 TMEM columns, so no two of its CTAs may share an
// SM (two clusters each waiting in tcgen05.alloc for the other could never
// finish): every launch asks for more than half of an SM's shared memory.
constexpr size_t kMinSmem = 116 * 1024;

size_t shared_bytes(int U) {
  const size_t SU = size_t(U) * kConsumers * 8;  // padded slice, see the kernel
  const size_t b = ((sizeof(Shared) + 127) & ~size_t(127)) + kStages * SU * 2;
  return b < kMinSmem ? kMinSmem : b;
}

constexpr size_t kSmemLimit = 227 * 1024;

struct Plan {
  int C = 0, S = 0, U = 0;
};

// The slice and vector count for clusters of C CTAs; C = 0 when a slice does
// not fit a CTA.
Plan plan_c(int V, int C) {
  Plan pl;
  const int S = ((V + C - 1) / C + 7) / 8 * 8;
  const int U = (S + kConsumers * 8 - 1) / (kConsumers * 8);
  if (U <= kMaxU && shared_bytes(U) <= kSmemLimit) {
    pl.C = C;
    pl.S = S;
    pl.U = U;
  }
  return pl;
}

// The smallest portable cluster (1, 2, 4 or 8 CTAs) that holds a row.
Plan plan_for(int V) {
  for (int C = 1; C <= kMaxC; C *= 2) {
    const Plan pl = plan_c(V, C);
    if (pl.C) return pl;
  }
  return Plan();
}

template <int DT, int U>
void fill_config(cudaLaunchConfig_t& cfg, cudaLaunchAttribute (&attr)[2], const Plan& pl,
                 size_t smem, cudaStream_t stream) {
  cfg = {};
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = pl.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3(pl.C);
}

// Resident clusters of fused_kernel<DT, U> with clusters of pl.C CTAs (0 when
// none fit) on the current device.  Each (device, cluster size) is queried
// once, on its first call, so that later calls can be captured into CUDA
// graphs; the kernel's attributes (shared memory, non-portable cluster
// sizes) are raised once per device as well.  The cache is keyed by device
// and guarded by a mutex, so host threads driving different GPUs may call
// concurrently.
template <int DT, int U>
int resident_clusters(const Plan& pl) {
  auto kern = fused_kernel<DT, U>;
  const size_t smem = shared_bytes(U);
  struct Cache {
    bool configured;
    int resident[kMaxRanks + 1];  // 0: not queried yet, -1: none fit
  };
  static std::mutex mu;
  static Cache cache[kMaxDevices] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
  std::lock_guard<std::mutex> lock(mu);
  Cache& c = cache[dev];
  if (!c.configured) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)) !=
            cudaSuccess ||
        cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
            cudaSuccess)
      return 0;
    c.configured = true;
  }
  if (c.resident[pl.C] == 0) {
    cudaLaunchConfig_t cfg;
    cudaLaunchAttribute attr[2];
    fill_config<DT, U>(cfg, attr, pl, smem, nullptr);
    int n = 0;
    c.resident[pl.C] = (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) == cudaSuccess && n > 0)
                           ? n
                           : -1;
  }
  return c.resident[pl.C] > 0 ? c.resident[pl.C] : 0;
}

template <int DT>
int clusters_of(const Plan& pl) {
  switch (pl.U) {
    case 1: return resident_clusters<DT, 1>(pl);
    case 2: return resident_clusters<DT, 2>(pl);
    case 3: return resident_clusters<DT, 3>(pl);
    case 4: return resident_clusters<DT, 4>(pl);
    default: return resident_clusters<DT, 5>(pl);
  }
}

// The cluster size, from the smallest one that holds a row up to 16 CTAs,
// that keeps the most SMs busy (ties: the smaller).  On a GB300, clusters of
// 8 CTAs fit 15 times (120 SMs), of 9 CTAs 15 times (135 SMs), of 10 CTAs 13
// times; V = 151 936 and 128 256 take 9.
template <int DT>
Plan choose_plan(int V) {
  Plan best = plan_for(V);
  if (best.C == 0) return best;
  int best_sms = best.C * clusters_of<DT>(best);
  for (int C = best.C + 1; C <= kMaxRanks; ++C) {
    const Plan pl = plan_c(V, C);
    if (pl.C == 0) continue;
    const int sms = C * clusters_of<DT>(pl);
    if (sms > best_sms) {
      best = pl;
      best_sms = sms;
    }
  }
  return best;
}

template <int DT, int U>
hs_status launch_t(const Params& p, const Plan& pl, cudaStream_t stream) {
  const int max_clusters = resident_clusters<DT, U>(pl);
  if (max_clusters < 1) return HS_ERR_UNSUPPORTED;
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[2];
  fill_config<DT, U>(cfg, attr, pl, shared_bytes(U), stream);
  const int nclusters = max(1, min(p.ntiles, max_clusters));
  cfg.gridDim = dim3(unsigned(nclusters * pl.C));
  cfg.numAttrs = 2;  // cluster shape + programmatic dependent launch
  if (cudaLaunchKernelEx(&cfg, fused_kernel<DT, U>, p) != cudaSuccess) return HS_ERR_CUDA;
  return HS_OK;
}

template <int DT>
hs_status launch_dt(const Params& p, const Plan& pl, cudaStream_t s) {
  switch (pl.U) {
    case 1: return launch_t<DT, 1>(p, pl, s);
    case 2: return launch_t<DT, 2>(p, pl, s);
    case 3: return launch_t<DT, 3>(p, pl, s);
    case 4: return launch_t<DT, 4>(p, pl, s);
    default: return launch_t<DT, 5>(p, pl, s);
  }
}

__global__ void elen_kernel(const float* __restrict__ alpha, int64_t NB, int P,
                            float* __restrict__ e_len) {
  pdl_wait();
  const int64_t idx = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (idx >= NB) return;
  const float* a = alpha + idx * P;
  float e = 1.f, prod = 1.f;
  for (int k = 0; k < P - 1; ++k) {
    prod *= a[k];
    e += prod;
  }
  e_len[idx] = e;
}

}  // namespace

int long_row_grid(int N, int B, int P, int V) {
  int dev = 0, sms = 0, l2 = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev) != cudaSuccess)
    return 0;
  return twopass::long_row_grid(V, 2, B * P, N, sms, size_t(l2));
}

hs_status launch_two_pass(const void* target, const int32_t* path, int M, const void* drafter,
                          int dtype, int N, int B, int P, int V, float c, int grid, float* alpha,
                          float* e_len, int* dev_status, cudaStream_t stream) {
  const hs_status st = twopass::launch(target, path, M, drafter, dtype, N, B, P, V, c, 0, grid,
                                       alpha, dev_status, stream);
  if (st != HS_OK) return st;
  if (e_len) {
    const int64_t nb = int64_t(N) * B;
    if (launch_pdl(elen_kernel, dim3(unsigned((nb + 255) / 256)), dim3(256), 0, stream, alpha,
                   nb, P, e_len) != cudaSuccess)
      return HS_ERR_CUDA;
  }
  return HS_OK;
}

bool eligible_sizes(int dtype, int N, int V, int greedy) {
  if (greedy || (dtype != HS_BF16 && dtype != HS_FP16)) return false;
  if (N > kMaxN || V % 8 != 0) return false;
  return plan_for(V).C > 0;
}

bool eligible(const void* target, const void* drafter, int dtype, int N, int V, int greedy) {
  if (reinterpret_cast<uintptr_t>(target) % 16 || reinterpret_cast<uintptr_t>(drafter) % 16)
    return false;
  return eligible_sizes(dtype, N, V, greedy);
}

hs_status launch(const void* target, const int32_t* path, int M, const void* drafter, int dtype,
                 int N, int B, int P, int V, float c, float* alpha, float* e_len,
                 int* dev_status, cudaStream_t stream) {
  const Plan pl = dtype == HS_BF16 ? choose_plan<HS_BF16>(V) : choose_plan<HS_FP16>(V);
  if (pl.C == 0) return HS_ERR_UNSUPPORTED;
  Params p;
  p.target = target;
  p.path = path;
  p.M = M;
  p.drafter = drafter;
  p.N = N;
  p.B = B;
  p.P = P;
  p.V = V;
  p.c = c;
  p.S = pl.S;
  p.ntiles = B * P;
  p.alpha = alpha;
  p.dev_status = dev_status;
  // shapes whose rows the cluster kernel can only spread over part of the
  // GPU, with enough drafter rows and rows small enough for L2 to hold every
  // SM's working set, go to the two-pass kernel on all SMs (measured on
  // llama3_batch: 317 against 394 us per call)
  int dev = 0, sms = 0, l2 = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev) != cudaSuccess)
    return HS_ERR_CUDA;
  const int cluster_sms =
      pl.C * (dtype == HS_BF16 ? clusters_of<HS_BF16>(pl) : clusters_of<HS_FP16>(pl));
  hs_status st;
  const int pairs = twopass::pair_grid(V, 2, B * P, N, sms, size_t(l2));
  if (twopass::preferred(V, 2, B * P, N, sms, cluster_sms, size_t(l2)))
    st = twopass::launch(target, path, M, drafter, dtype, N, B, P, V, c, 0, sms, alpha,
                         dev_status, stream);
  else if (pairs > 0)  // one CTA per drafter pair
    st = twopass::launch(target, path, M, drafter, dtype, N, B, P, V, c, 0, pairs, alpha,
                         dev_status, stream);
  else
    st = dtype == HS_BF16 ? launch_dt<HS_BF16>(p, pl, stream) : launch_dt<HS_FP16>(p, pl, stream);
  if (st != HS_OK) return st;
  if (e_len) {
    const int64_t nb = int64_t(N) * B;
    if (launch_pdl(elen_kernel, dim3(unsigned((nb + 255) / 256)), dim3(256), 0, stream, alpha,
                   nb, P, e_len) != cudaSuccess)
      return HS_ERR_CUDA;
  }
  return HS_OK;
}

}  // namespace fused
}  // namespace hs
