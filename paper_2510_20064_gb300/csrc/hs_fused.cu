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

#include "hs_common.cuh"
#include "hs_fused.h"

namespace hs {
namespace fused {
namespace {

// 15 consumer warps + 1 load warp: 16 warps put 4 on each SM sub-partition,
// which leaves 128 registers per thread for the two rows of exponentials a
// consumer thread keeps.
constexpr int kConsumerWarps = 15;
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kThreads = kConsumers + 32;
constexpr int kStages = 3;
// Rows ahead of the ring whose slice is prefetched into L2 (bulk prefetch,
// no shared memory): the ring's TMA loads then hit L2, which keeps a few
// hundred KB per SM in flight although only ~2 stages fit next to p.
constexpr int kPrefetch = 0;
constexpr int kXSlots = 4;  // rows whose exchange may be in flight at once
constexpr int kASlots = 4;  // tiles whose alpha partials may be in flight
constexpr int kMaxU = 5;    // 16-byte vectors per consumer thread and row
constexpr long long kTimeoutCycles = 1LL << 31;  // about a second
constexpr uint32_t kNegInfBf16x2 = 0xFF80FF80u;
constexpr uint32_t kNegInfF16x2 = 0xFC00FC00u;

struct __align__(16) Shared {
  uint64_t full[kStages];          // ring stage loaded (TMA complete_tx)
  uint64_t empty[kStages];         // ring stage read by every consumer warp
  uint64_t redbar[kXSlots];        // every consumer warp posted its row pair
  uint64_t xbar[kXSlots];          // every rank's pair of a row arrived
  uint64_t accbar[2];              // every consumer warp posted a tile's partials
  uint64_t abar[kASlots];          // every rank's tile partials arrived (rank 0)
  float2 red[kXSlots][16];                // per-warp (offset, sum) of a row
  float2 xch[kXSlots][kMaxC];             // per-rank (offset, sum) of a row
  float acc[2][kMaxN][kConsumerWarps];    // per-warp alpha partials of a tile
  uint32_t tvalid[2];                     // the tile's target row is usable
  uint32_t dvalid[2];                     // bit i: drafter i's row is usable
  float clacc[kASlots][kMaxC][kMaxN];     // per-rank alpha partials (rank 0)
  int error;
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
// try_wait suspends the thread until the phase completes or about 1 ms has
// passed, so a waiting warp does not spin through the issue slots.
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile("{\n\t.reg .pred p;\n\t"
               "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n\t"
               "selp.u32 %0, 1, 0, p;\n\t}"
               : "=r"(ok) : "r"(bar), "r"(parity), "r"(1000000u) : "memory");
  return ok != 0;
}
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes,
                                          uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes "
               "[%0], [%1], %2, [%3];"
               :: "r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_probe(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile("{\n\t.reg .pred p;\n\t"
               "mbarrier.test_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
               "selp.u32 %0, 1, 0, p;\n\t}"
               : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
  return ok != 0;
}
// Arrive on a barrier in another CTA of the cluster, ordering this thread's
// earlier shared::cluster stores before the arrival.
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_bar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];"
               :: "r"(cluster_bar) : "memory");
}
__device__ __forceinline__ void st_cluster_f2(uint32_t a, float x, float y) {
  asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" :: "r"(a), "f"(x), "f"(y) : "memory");
}
__device__ __forceinline__ void st_cluster_f(uint32_t a, float x) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" :: "r"(a), "f"(x) : "memory");
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

// Order-preserving int key of a float (NaN above +inf), so that a warp's
// maximum is one redux.sync.
__device__ __forceinline__ int fkey(float f) {
  const int b = __float_as_int(f);
  return (f != f) ? 0x7fffffff : (b >= 0 ? b : b ^ 0x7fffffff);
}
__device__ __forceinline__ float kfloat(int k) {
  return __int_as_float(k >= 0 ? k : k ^ 0x7fffffff);  // 0x7fffffff is a NaN
}
__device__ __forceinline__ float warp_max_key(float f) {
  return kfloat(__reduce_max_sync(0xffffffffu, fkey(f)));
}

// Merge (offset o, sum s) pairs held by the lanes of a warp: the largest
// offset O (NaN wins, -inf means "no finite logit") and sum_l s_l 2^{o_l - O}.
__device__ __forceinline__ void warp_merge(float& o, float& s) {
  const float O = warp_max_key(o);
  float t = (o == -INFINITY || O == -INFINITY) ? 0.f : s * ex2(o - O);
  t = warp_sum(t);
  o = O;
  s = t;
}

// ---- the kernel ---------------------------------------------------------------

template <int DT, int U>
struct Row {
  f2_t e[U * 4];  // exponentials of the thread's logits, packed in pairs
  float o_used;   // offset the exponentials are relative to (the warp's)
  float o;        // reported offset: -inf when the warp saw no finite logit
};

// Global address of this CTA's slice of its row g: row g % (N+1) of the
// CTA's (g / (N+1))-th tile -- the target row, then the drafter rows.
__device__ __forceinline__ const char* row_slice(const Params& p, int g, uint32_t cid,
                                                 uint32_t ncl, int64_t slice0) {
  const int R = p.N + 1;
  const int j = g / R, r = g % R;
  const int64_t tile = int64_t(cid) + int64_t(j) * ncl;
  const int64_t b = tile / p.P, k = tile % p.P;
  int64_t row;
  const void* base;
  if (r == 0) {
    if (p.path) {
      const int nd = p.path[tile];
      row = b * p.M + ((nd < 0 || nd >= p.M) ? 0 : nd);
    } else {
      row = tile;
    }
    base = p.target;
  } else {
    row = (int64_t(r - 1) * p.B + b) * p.P + k;
    base = p.drafter;
  }
  return static_cast<const char*>(base) + (row * p.V + slice0) * 2;
}

// Stream row g into `stage` (one thread); with kPrefetch > 0 also prefetch
// row g + kPrefetch into L2.
__device__ __forceinline__ void issue(const Params& p, Shared& sh, unsigned char* stage, int g,
                                      int G, uint32_t cid, uint32_t ncl, int64_t slice0,
                                      uint32_t bytes) {
  const uint32_t full = saddr(&sh.full[g % kStages]);
  if (bytes) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    mbar_arrive_tx(full, bytes);
    bulk_load(saddr(stage), row_slice(p, g, cid, ncl, slice0), bytes, full);
    if (kPrefetch > 0 && g + kPrefetch < G)
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;"
                   :: "l"(row_slice(p, g + kPrefetch, cid, ncl, slice0)), "r"(bytes) : "memory");
  } else {
    mbar_arrive(full);
  }
}

template <int DT, int U>
__global__ void __launch_bounds__(kThreads, 1) fused_kernel(const Params p) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  Shared& sh = *reinterpret_cast<Shared*>(smem_raw);
  // every buffer holds SU = U * kConsumers * 8 >= S elements so that each
  // consumer thread always handles U whole 16-byte vectors; the part past
  // the CTA's slice is -inf in the ring and 0 in p (set once, below)
  constexpr int SU = U * kConsumers * 8;
  constexpr uint32_t stage_bytes = SU * 2;
  unsigned char* ring = smem_raw + ((sizeof(Shared) + 127) & ~size_t(127));
  // p of the tile's target, as two planes of float4 so that consecutive
  // threads read consecutive 16 bytes: pA[vi] = p[8vi..8vi+3], pB[vi] = p[8vi+4..8vi+7]
  float4* pA = reinterpret_cast<float4*>(ring + kStages * stage_bytes);
  float4* pB = pA + SU / 8;

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
    for (int vi = len / 8 + tid; vi < SU / 8; vi += kThreads)
      pA[vi] = pB[vi] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(saddr(&sh.full[s]), 1);
      mbar_init(saddr(&sh.empty[s]), kConsumerWarps);
    }
    for (int x = 0; x < kXSlots; ++x) {
      mbar_init(saddr(&sh.redbar[x]), kConsumerWarps);
      mbar_init(saddr(&sh.xbar[x]), C);
    }
    for (int a = 0; a < 2; ++a) mbar_init(saddr(&sh.accbar[a]), kConsumerWarps);
    for (int a = 0; a < kASlots; ++a) mbar_init(saddr(&sh.abar[a]), C * N);
    sh.error = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  cluster_sync_all();

  if (warp == kConsumerWarps) {
    // ---------------------------- coordinator -----------------------------
    // Never blocks: every wait polls its barrier and, while it does, lane 0
    // refills each ring stage as soon as all consumer warps have read it.
    // The warp merges the consumer warps' row pairs and sends the CTA's pair
    // to every rank, and reduces each tile's alpha partials (rank 0 also
    // writes alpha, one tile late).
    int issued = 0;
    auto service = [&]() {
      if (lane != 0) return;
      while (issued < G &&
             (issued < kStages ||
              mbar_probe(saddr(&sh.empty[issued % kStages]),
                         uint32_t((issued / kStages) - 1) & 1u))) {
        issue(p, sh, ring + (issued % kStages) * stage_bytes, issued, G, cid, ncl, slice0, bytes);
        ++issued;
      }
    };
    auto poll = [&](uint32_t bar, uint32_t parity) {
      service();
      const long long t0 = clock64();
      while (!mbar_probe(bar, parity)) {
        service();
        if (*reinterpret_cast<volatile int*>(&sh.error)) return;
        if (clock64() - t0 > kTimeoutCycles) {
          *reinterpret_cast<volatile int*>(&sh.error) = 1;
          report(p.dev_status, HS_ERR_TIMEOUT);
          return;
        }
        __nanosleep(32);
      }
    };
    auto finish = [&](int j) {  // rank 0: alpha[:, b, k] of tile j
      poll(saddr(&sh.abar[j % kASlots]), uint32_t(j / kASlots) & 1u);
      if (lane < N) {
        const int64_t tile = int64_t(cid) + int64_t(j) * ncl;
        const int64_t b = tile / P, k = tile % P;
        float t = 0.f;
        for (uint32_t rr = 0; rr < C; ++rr) t += sh.clacc[j % kASlots][rr][lane];
        const bool bad_path = p.path && (p.path[tile] < 0 || p.path[tile] >= p.M);
        if (bad_path || !sh.tvalid[j & 1] || !((sh.dvalid[j & 1] >> lane) & 1u)) {
          t = __int_as_float(0x7fc00000);
          report(p.dev_status, bad_path ? HS_ERR_INVALID_ARG : HS_ERR_NONFINITE);
        }
        p.alpha[(int64_t(lane) * B + b) * P + k] = t;
      }
    };
    auto reduce_tile = [&](int j) {  // tile j's partials -> rank 0
      poll(saddr(&sh.accbar[j & 1]), uint32_t(j >> 1) & 1u);
      if (lane < N) {
        float t = 0.f;
        for (int w = 0; w < kConsumerWarps; ++w) t += sh.acc[j & 1][lane][w];
        st_cluster_f(mapa(saddr(&sh.clacc[j % kASlots][rank][lane]), 0), t);
        mbar_arrive_remote(mapa(saddr(&sh.abar[j % kASlots]), 0));
      }
      if (rank == 0 && j > 0) finish(j - 1);  // long since complete
    };
    for (int g = 0; g < G; ++g) {
      const int x = g % kXSlots;
      poll(saddr(&sh.redbar[x]), uint32_t(g / kXSlots) & 1u);
      float2 v = lane < kConsumerWarps ? sh.red[x][lane] : make_float2(-INFINITY, 0.f);
      float oc = v.x, sc = v.y;
      warp_merge(oc, sc);
      if (lane < int(C)) {
        st_cluster_f2(mapa(saddr(&sh.xch[x][rank]), lane), oc, sc);
        mbar_arrive_remote(mapa(saddr(&sh.xbar[x]), lane));
      }
      // tile j's partials are posted after the consumers' pass over the
      // first row of tile j+1, so reduce tile j once that row is merged
      if (g % R == 0 && g > 0) reduce_tile(g / R - 1);
    }
    if (G > 0) {
      reduce_tile(my_tiles - 1);
      if (rank == 0) finish(my_tiles - 1);
    }
    // every row was issued (the consumers have read them all); drain: every
    // copy has landed before the CTA may exit
    if (lane == 0)
      for (int g = max(0, G - kStages); g < G; ++g)
        wait_phase(saddr(&sh.full[g % kStages]), uint32_t(g / kStages) & 1u, sh, p.dev_status,
                   false);
  } else if (G > 0) {
    // ------------------------------ consumers -----------------------------
    const float c = p.c;
    uint32_t tvalid = 0, dvalid = 0;  // target row usable; bit i: drafter i usable
    Row<DT, U> A, Bv;

    // pass 1: load row g from the ring (then release the stage); warp max;
    // exponentials relative to the warp's offset, kept in registers; post
    // the warp's (offset, sum) for the coordinator
    auto pass1 = [&](int g, Row<DT, U>& Rw) {
      const int s = g % kStages;
      wait_phase(saddr(&sh.full[s]), uint32_t(g / kStages) & 1u, sh, p.dev_status);
      const uint32_t stage = saddr(ring + s * stage_bytes);
      uint32_t w[U * 4];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const uint4 v = lds128(stage + (u * kConsumers + tid) * 16);
        w[4 * u] = v.x; w[4 * u + 1] = v.y; w[4 * u + 2] = v.z; w[4 * u + 3] = v.w;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(saddr(&sh.empty[s]));
      uint32_t mx[U * 2];  // pairwise tree: log-depth dependency chain
#pragma unroll
      for (int q = 0; q < U * 2; ++q) mx[q] = pmax<DT>(w[2 * q], w[2 * q + 1]);
#pragma unroll
      for (int d = 1; d < U * 2; d *= 2)
#pragma unroll
        for (int q = 0; q + d < U * 2; q += 2 * d) mx[q] = pmax<DT>(mx[q], mx[q + d]);
      const float m = warp_max_key(max_nan(lo<DT>(mx[0]), hi<DT>(mx[0])));
      Rw.o = (m == -INFINITY) ? -INFINITY : m * c;
      Rw.o_used = (m == -INFINITY) ? 0.f : Rw.o;
      const f2_t cc = pk(c, c), off = pk(-Rw.o_used, -Rw.o_used);
      f2_t acc[2] = {pk(0.f, 0.f), pk(0.f, 0.f)};
#pragma unroll
      for (int q = 0; q < U * 4; ++q) {
        float a, b;
        upk(ffma2(pk(lo<DT>(w[q]), hi<DT>(w[q])), cc, off), a, b);
        Rw.e[q] = pk(ex2(a), ex2(b));
        acc[q & 1] = fadd2(acc[q & 1], Rw.e[q]);
      }
      float s0, s1, s2, s3;
      upk(acc[0], s0, s1);
      upk(acc[1], s2, s3);
      const float sum = warp_sum((s0 + s1) + (s2 + s3));
      if (lane == 0) {
        sh.red[g % kXSlots][warp] = make_float2(Rw.o, sum);
        mbar_arrive(saddr(&sh.redbar[g % kXSlots]));
      }
    };

    // all ranks' pairs of row g: the row's offset O and 1/Z
    auto gather = [&](int g, float& O, float& invZ) -> bool {
      const int x = g % kXSlots;
      wait_phase(saddr(&sh.xbar[x]), uint32_t(g / kXSlots) & 1u, sh, p.dev_status);
      float2 v = lane < int(C) ? sh.xch[x][lane] : make_float2(-INFINITY, 0.f);
      float o = v.x, s = v.y;
      warp_merge(o, s);
      O = o;
      invZ = 1.f / s;
      return isfinite(o) && s > 0.f;
    };

    // pass 2: target -> p into shared memory; drafter i -> alpha partial
    auto pass2 = [&](int g, Row<DT, U>& Rw) {
      const int j = g / R, r = g % R;
      float O, invZ;
      const bool ok = gather(g, O, invZ);
      const float f = (Rw.o == -INFINITY || !ok) ? 0.f : ex2(Rw.o_used - O) * invZ;
      const f2_t ff = pk(f, f);
      if (r == 0) {
        tvalid = ok ? 1u : 0u;
        dvalid = 0;
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const int vi = u * kConsumers + tid;
          float q[8];
#pragma unroll
          for (int h = 0; h < 4; ++h) upk(fmul2(Rw.e[4 * u + h], ff), q[2 * h], q[2 * h + 1]);
          pA[vi] = make_float4(q[0], q[1], q[2], q[3]);
          pB[vi] = make_float4(q[4], q[5], q[6], q[7]);
        }
        return;
      }
      const int i = r - 1;
      if (ok) dvalid |= 1u << i;
      f2_t acc[2] = {pk(0.f, 0.f), pk(0.f, 0.f)};
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int vi = u * kConsumers + tid;
        const float4 p0 = pA[vi], p1 = pB[vi];
        const float pv[8] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          float xx, yy;
          upk(fmul2(Rw.e[4 * u + h], ff), xx, yy);
          acc[h & 1] = fadd2(acc[h & 1], pk(fminf(pv[2 * h], xx), fminf(pv[2 * h + 1], yy)));
        }
      }
      float a0, a1, a2, a3;
      upk(acc[0], a0, a1);
      upk(acc[1], a2, a3);
      const float a = warp_sum((a0 + a1) + (a2 + a3));
      if (lane == 0) {
        sh.acc[j & 1][i][warp] = a;
        if (i == N - 1) {  // tile end: hand the partials to the coordinator
          if (warp == 0) {
            sh.tvalid[j & 1] = tvalid;
            sh.dvalid[j & 1] = dvalid;
          }
          mbar_arrive(saddr(&sh.accbar[j & 1]));
        }
      }
    };

    pass1(0, A);
    for (int g = 0; g < G; g += 2) {
      if (g + 1 < G) pass1(g + 1, Bv);
      pass2(g, A);
      if (g + 1 < G) {
        if (g + 2 < G) pass1(g + 2, A);
        pass2(g + 1, Bv);
      }
    }
  }
  // no CTA may leave while a peer can still write into its shared memory
  __syncwarp();
  cluster_sync_all();
}

// ---- host side ------------------------------------------------------------------

size_t shared_bytes(int U) {
  const size_t SU = size_t(U) * kConsumers * 8;  // padded slice, see the kernel
  return ((sizeof(Shared) + 127) & ~size_t(127)) + kStages * SU * 2 + SU * 4;
}

constexpr size_t kSmemLimit = 227 * 1024;

struct Plan {
  int C = 0, S = 0, U = 0;
};

Plan plan_for(int V) {
  Plan pl;
  for (int C = 1; C <= kMaxC; C *= 2) {
    const int S = ((V + C - 1) / C + 7) / 8 * 8;
    const int U = (S + kConsumers * 8 - 1) / (kConsumers * 8);
    if (U <= kMaxU && shared_bytes(U) <= kSmemLimit) {
      pl.C = C;
      pl.S = S;
      pl.U = U;
      return pl;
    }
  }
  return pl;
}

template <int DT, int U>
hs_status launch_t(const Params& p, const Plan& pl, cudaStream_t stream) {
  auto kern = fused_kernel<DT, U>;
  const size_t smem = shared_bytes(pl.U);
  static int configured_smem = 0;  // attribute is per kernel; raise it once
  if (configured_smem < int(smem)) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)) !=
        cudaSuccess)
      return HS_ERR_CUDA;
    configured_smem = int(smem);
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = pl.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3(pl.C);
  // resident clusters for this (cluster size, shared memory); queried once, on
  // the first call, so that later calls can be captured into CUDA graphs
  static int cached_c = 0, cached_smem = 0, max_clusters = 0;
  if (cached_c != pl.C || cached_smem != int(smem)) {
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n < 1)
      return HS_ERR_UNSUPPORTED;
    max_clusters = n;
    cached_c = pl.C;
    cached_smem = int(smem);
  }
  const int nclusters = max(1, min(p.ntiles, max_clusters));
  cfg.gridDim = dim3(unsigned(nclusters * pl.C));
  if (cudaLaunchKernelEx(&cfg, kern, p) != cudaSuccess) return HS_ERR_CUDA;
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
  const Plan pl = plan_for(V);
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
  hs_status st = dtype == HS_BF16 ? launch_dt<HS_BF16>(p, pl, stream)
                                  : launch_dt<HS_FP16>(p, pl, stream);
  if (st != HS_OK) return st;
  if (e_len) {
    const int64_t nb = int64_t(N) * B;
    elen_kernel<<<unsigned((nb + 255) / 256), 256, 0, stream>>>(alpha, nb, P, e_len);
    if (cudaGetLastError() != cudaSuccess) return HS_ERR_CUDA;
  }
  return HS_OK;
}

}  // namespace fused
}  // namespace hs
