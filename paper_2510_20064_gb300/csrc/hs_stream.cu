// hs_stream.cu -- stochastic feedback (Thm 1) by one persistent kernel that
// cuts every row into vocabulary chunks, so that calls with few rows per SM
// (or rows too long for the cluster kernel) still keep every SM busy.
//
// alpha = sum_v min(p_v, q_v) needs each row's normaliser before the min.
// Work items are (tile (b,k), chunk j of kChunk logits), tile-major; CTA c
// (one per SM) takes items c, c + G, c + 2G, ... (G CTAs) in steps.  In step
// s it does
//   * the STATISTICS of item x = sG + c: for the target row and the N drafter
//     rows, the chunk's integer reference R = ceil(c_T m) (m a thread's max,
//     c_T = log2(e)/T) and s = sum 2^{c_T z - R}, merged over the CTA and
//     written to global memory, then counted in on the tile's counter;
//   * the OVERLAP of item y = (s-L)G + c, read L steps earlier: once the
//     tile's counter says every chunk of every row has its statistics (a
//     bounded wait), each row's normaliser is merged from its chunks and the
//     item's chunks are read again -- from L2, one step of items being a few
//     tens of MB -- for sum_v 2^{min(c_T z_t - o_t, c_T z_d - o_d)} per
//     drafter (2^x is increasing: one exp2 per pair), the target's exponents
//     kept in registers for all N drafters; the CTA's partial per drafter
//     goes to global memory.
// A small second kernel adds each tile's chunk partials up in chunk order
// (alpha) and forms e_len.
// One producer warp streams every chunk the consumers take, in their order,
// into a ring of 32 KB shared-memory stages with cp.async.bulk; a chunk is
// one stage, 4 vectors of 16 bytes per consumer thread.
// L = 1 + (chunks per row - 1) / G, so that a tile's items all come at most L
// steps after any one of them: no overlap waits for a later step's
// statistics than the ones its own CTA has passed, and the launch is
// cooperative (all CTAs resident), so the waits always end; each is bounded
// anyway: a wait that gives up reports
// HS_ERR_TIMEOUT and writes its item's partials as NaN, so the tile's
// alphas come out NaN.  HBM reads every logit once; L2 serves the second
// read.
#include <math.h>
#include <stdint.h>

#include <mutex>

#include "hs_common.cuh"
#include "hs_stream.h"

namespace hs {
namespace stream {
namespace {

constexpr int kConsumerWarps = 16;
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kThreads = kConsumers + 32;  // + the producer warp
constexpr int kStages = 6;                 // ring stages (192 KB)
constexpr int kVecsPerThread = 4;          // 16-byte vectors of a stage per consumer
constexpr int kChunkVecs = kVecsPerThread * kConsumers;
constexpr int kChunkBytes = kChunkVecs * 16;  // 32 KB
constexpr int kChunk = kChunkVecs * 8;        // logits per chunk (bf16 / fp16)
constexpr int kMaxN = 32;
constexpr int kMaxRows = kMaxN + 1;
constexpr long long kTimeoutCycles = 1LL << 31;  // about a second
constexpr float kFoldLimit = 64.f;  // |o| below which pass 2 folds R + L into one offset

struct Params {
  const void* target;
  const int32_t* path;
  const void* drafter;
  int M, N, B, P, V;
  float c;      // log2(e) / T
  int nchunk;   // chunks per row
  int ntiles;   // B * P
  int nitems;   // ntiles * nchunk
  int lag;      // steps from an item's statistics to its overlap (1 + (nchunk - 1) / G)
  float2* stats;  // [ntiles][N+1][nchunk]: (R, s) of each row chunk; s NaN: bad
  float* apart;   // [N][ntiles][nchunk]: alpha partials
  int* cnt;       // [ntiles]: row chunks with statistics
  int* dev_status;
  long long wait_limit;  // clock cycles a counter wait may take (kTimeoutCycles)
  int stall_tile;        // test hook: this tile's count never completes (-1: none)
};

// Per-warp posts of one step, double-buffered by step parity: buffer b is
// rewritten two steps later, after a barrier every reader has passed.
struct Shared {
  uint64_t full[kStages], empty[kStages];
  float2 sp[2][kMaxRows][kConsumerWarps];  // per-warp (R, s) of each row (s NaN: bad)
  float ap[2][kMaxN][kConsumerWarps];      // per-warp alpha partials
  float2 norm[kMaxRows];                   // (R, L) of each row of the overlap item
  int error;
};

// ---- PTX wrappers ---------------------------------------------------------------

__device__ __forceinline__ uint32_t saddr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile("{\n\t.reg .pred p;\n\t"
               "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
               "selp.u32 %0, 1, 0, p;\n\t}"
               : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
  return ok != 0;
}
// Bounded wait; false (the CTA's error flag set, a timeout reported) after
// about a second, or at once when another wait of the CTA already gave up.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* error,
                                          int* dev_status) {
  if (mbar_test(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (*error) return false;
    if (mbar_test(bar, parity)) return true;
    if (clock64() - t0 > kTimeoutCycles) {
      *error = 1;
      report(dev_status, HS_ERR_TIMEOUT);
      return false;
    }
  }
}
__device__ __forceinline__ uint64_t make_policy(bool keep) {
  uint64_t p;
  if (keep)
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  else
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// One thread: stream `bytes` (a multiple of 16 from a 16-byte-aligned source)
// into a stage, completing its mbarrier's phase, with an L2 policy.
__device__ __forceinline__ void bulk_fill(uint32_t stage, uint32_t bar, const void* src,
                                          uint32_t bytes, uint64_t pol) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
               :: "r"(bar), "r"(bytes) : "memory");
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint "
               "[%0], [%1], %2, [%3], %4;"
               :: "r"(stage), "l"(src), "r"(bytes), "r"(bar), "l"(pol) : "memory");
}
__device__ __forceinline__ uint4 lds128(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
// Barrier of the consumer warps only (the producer warp never joins).
__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, %0;" :: "n"(kConsumers) : "memory");
}

// ---- arithmetic -------------------------------------------------------------------

// Packed fp32 pairs (two lanes of one 64-bit register pair).
__device__ __forceinline__ uint64_t pack2(float lo, float hi) {
  uint64_t d;
  asm("mov.b64 %0, {%1, %2};" : "=l"(d) : "f"(lo), "f"(hi));
  return d;
}
__device__ __forceinline__ float lo2(uint64_t d) { return __uint_as_float(uint32_t(d)); }
__device__ __forceinline__ float hi2(uint64_t d) { return __uint_as_float(uint32_t(d >> 32)); }
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
// The two logits of a stored 32-bit word as floats (exact widening).
template <int DT>
__device__ __forceinline__ float lo_of(uint32_t w) {
  if (DT == HS_BF16) return __uint_as_float(w << 16);
  return __half2float(__ushort_as_half(static_cast<unsigned short>(w & 0xffffu)));
}
template <int DT>
__device__ __forceinline__ float hi_of(uint32_t w) {
  if (DT == HS_BF16) return __uint_as_float(w & 0xffff0000u);
  return __half2float(__ushort_as_half(static_cast<unsigned short>(w >> 16)));
}
template <int DT>
__device__ __forceinline__ uint64_t pair_of(uint32_t w) {
  return pack2(lo_of<DT>(w), hi_of<DT>(w));
}
// NaN-propagating packed max of two stored words.
template <int DT>
__device__ __forceinline__ uint32_t pmax(uint32_t a, uint32_t b) {
  uint32_t r;
  if (DT == HS_BF16)
    asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  else
    asm("max.NaN.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// Statistics of this thread's 32 logits of a row chunk (-inf past the row's
// end): an integer reference R = ceil(c m), m the max of its logits, and
// s = sum 2^{c z - R} (every term at most 1: no overflow; terms far below the
// max vanish as they would below the row max).  R = -inf, s = 0 when all are
// -inf.  bad: a NaN or +inf logit, or c m above the fp32 range (R, s are then
// -inf, 0 and the flag travels on its own).
template <int DT>
__device__ __forceinline__ void chunk_stat(const uint4 (&v)[kVecsPerThread], float c, uint64_t c2,
                                           float& R, float& s, bool& bad) {
  uint32_t mw = pmax<DT>(pmax<DT>(v[0].x, v[0].y), pmax<DT>(v[0].z, v[0].w));
#pragma unroll
  for (int u = 1; u < kVecsPerThread; ++u)
    mw = pmax<DT>(mw, pmax<DT>(pmax<DT>(v[u].x, v[u].y), pmax<DT>(v[u].z, v[u].w)));
  const float cm = max_nan(lo_of<DT>(mw), hi_of<DT>(mw));
  const float Rn = ceilf(cm * c);  // -inf when every logit is -inf
  bad = !(Rn < INFINITY);           // NaN, or +inf (a +inf logit or an overflowing c m)
  R = bad ? -INFINITY : Rn;
  const float off = R == -INFINITY ? 0.f : -R;
  const uint64_t off2 = pack2(off, off);
  uint64_t a = 0ull, b = 0ull;
#pragma unroll
  for (int u = 0; u < kVecsPerThread; ++u) {
    const uint32_t wd[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint64_t e = fma2(pair_of<DT>(wd[q]), c2, off2);
      const uint64_t x = pack2(ex2(lo2(e)), ex2(hi2(e)));
      if (q & 1)
        b = add2(b, x);
      else
        a = add2(a, x);
    }
  }
  const uint64_t t2 = add2(a, b);
  s = bad ? 0.f : lo2(t2) + hi2(t2);
}

// Every lane: the merge (R, S) of the warp's pairs (R, s), each s relative to
// its integer reference R (or -inf with s = 0): the largest reference first,
// then every sum rescaled to it (by an exact power of 2) and added up.
__device__ __forceinline__ void warp_merge(float& R, float& s) {
  float M;
  asm volatile("redux.sync.max.f32 %0, %1, 0xffffffff;" : "=f"(M) : "f"(R));  // warp-collective
  s = (R == -INFINITY) ? 0.f : s * ex2(R - M);
  R = M;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
}

// Every lane: the merge of the pairs q_l (lane l; s NaN marks a bad part):
// (R, s) with s NaN when any part was bad.
__device__ __forceinline__ void merge_lanes(float2 q, float& R, float& s) {
  const bool bad = __any_sync(0xffffffffu, q.y != q.y);
  R = q.x;
  s = q.y != q.y ? 0.f : q.y;
  warp_merge(R, s);
  if (bad) s = __int_as_float(0x7fc00000);
}

// ---- the kernel -------------------------------------------------------------------

// Row r of tile t: 0 the target (a chain row, or the tree's path node; a
// node out of range reads node 0 and the consumers flag the tile), 1 + i
// drafter i.
template <int DT>
__device__ __forceinline__ const char* row_of(const Params& p, int t, int r) {
  if (r == 0) {
    bool bad = false;
    return static_cast<const char*>(target_row<DT>(p.target, p.path, p.M, p.P, t, p.V, &bad));
  }
  return static_cast<const char*>(row_ptr<DT>(p.drafter, int64_t(r - 1) * p.ntiles + t, p.V));
}

// The consumer warps: step by step, the statistics of item s G + cta, then
// the overlap of item (s - lag) G + cta, each chunk taken from the ring in the
// producer's order.  Every consumer thread runs the same control flow (also
// after a timeout, then on whatever the stages hold), so the barriers always
// meet.
template <int DT>
__device__ __forceinline__ void consumer(const Params& p, Shared& sh, uint32_t ring0, int steps,
                                         volatile int* err) {
  const int t = threadIdx.x, w = t >> 5, l = t & 31;
  const int G = gridDim.x, cta = blockIdx.x;
  const int N = p.N, R = N + 1, nvec = p.V / 8;
  const float c = p.c;
  const uint64_t c2 = pack2(c, c);
  const uint32_t ninf = DT == HS_BF16 ? 0xFF80FF80u : 0xFC00FC00u;
  const float nan = __int_as_float(0x7fc00000);
  uint32_t stage = 0, phase = 0;  // the next stage and its phase parity
  bool ok = true;
  // chunk j of the next row from the ring; the row's last chunk has its
  // vectors past the row's end replaced by -inf
  auto take = [&](int j, uint4 (&v)[kVecsPerThread]) {
    if (!mbar_wait(saddr(&sh.full[stage]), phase, err, p.dev_status)) ok = false;
    const uint32_t base = ring0 + stage * kChunkBytes + uint32_t(t) * 16u;
#pragma unroll
    for (int u = 0; u < kVecsPerThread; ++u) v[u] = lds128(base + uint32_t(u * kConsumers) * 16u);
    if (j == p.nchunk - 1) {
#pragma unroll
      for (int u = 0; u < kVecsPerThread; ++u)
        if (j * kChunkVecs + u * kConsumers + t >= nvec) v[u] = make_uint4(ninf, ninf, ninf, ninf);
    }
    // every consumer thread releases its own part of the stage (the stage's
    // barrier counts kConsumers arrivals)
    mbar_arrive(saddr(&sh.empty[stage]));
    if (++stage == kStages) {
      stage = 0;
      phase ^= 1u;
    }
  };
  int pt = -1, pj = 0, pb = 0;  // the overlap item whose partials await their merge
  for (int s = 0; s < steps; ++s) {
    const int b = s & 1;
    const int x = s * G + cta;        // statistics item
    const int y = (s - p.lag) * G + cta;  // overlap item
    if (x < p.nitems) {
      for (int r = 0; r < R; ++r) {
        uint4 v[kVecsPerThread];
        take(x % p.nchunk, v);
        float Rw, sw;
        bool bad;
        chunk_stat<DT>(v, c, c2, Rw, sw, bad);
        warp_merge(Rw, sw);
        if (__any_sync(0xffffffffu, bad)) sw = nan;
        if (l == 0) sh.sp[b][r][w] = make_float2(Rw, sw);
      }
    }
    consumer_sync();  // this step's statistics posts; the last overlap's partial posts
    if (x < p.nitems) {
      // the CTA's pair of each row chunk to global memory, then counted in
      // (release: the store before the count)
      const int tx = x / p.nchunk, jx = x - tx * p.nchunk;
      for (int r = w; r < R; r += kConsumerWarps) {
        float Rc, sc;
        merge_lanes(l < kConsumerWarps ? sh.sp[b][r][l] : make_float2(-INFINITY, 0.f), Rc, sc);
        if (l == 0) {
          p.stats[(int64_t(tx) * R + r) * p.nchunk + jx] = make_float2(Rc, sc);
          __threadfence();
          atomicAdd(p.cnt + tx, 1);
        }
      }
    }
    if (pt >= 0) {
      // the last overlap item's partials: the 16 warps' posts in warp order
      for (int d = w; d < N; d += kConsumerWarps) {
        const float a = warp_sum(l < kConsumerWarps ? sh.ap[pb][d][l] : 0.f);
        if (l == 0) p.apart[(int64_t(d) * p.ntiles + pt) * p.nchunk + pj] = a;
      }
      pt = -1;
    }
    if (s < p.lag || y >= p.nitems) continue;

    // ---- overlap of item y: the tile's row normalisers first ----
    const int ty = y / p.nchunk, jy = y - ty * p.nchunk;
    if (w < R) {
      // every chunk of every row of the tile has its statistics (bounded; the
      // test hook awaits one count more than exist, so that the wait runs
      // out).  Every lane's own acquire orders its loads of the statistics.
      const int need = R * p.nchunk + (ty == p.stall_tile ? 1 : 0);
      bool got = true;
      const long long t0 = clock64();
      while (!__all_sync(0xffffffffu, ld_acquire(p.cnt + ty) >= need)) {
        if (__shfl_sync(0xffffffffu, int(clock64() - t0 > p.wait_limit), 0)) {
          got = false;
          break;
        }
        __nanosleep(32);
      }
      if (!got && l == 0) report(p.dev_status, HS_ERR_TIMEOUT);
      for (int r = w; r < R; r += kConsumerWarps) {
        // lane l merges chunks l, l + 32, ... in order, then the warp merges
        float Rm = -INFINITY, sm = 0.f;
        bool bad = false;
        for (int q = l; q < p.nchunk; q += 32) {
          const float2 st = __ldcg(p.stats + (int64_t(ty) * R + r) * p.nchunk + q);
          bad |= st.y != st.y;
          if (st.x == -INFINITY) continue;
          if (st.x > Rm) {
            sm = Rm == -INFINITY ? 0.f : sm * ex2(Rm - st.x);
            Rm = st.x;
          }
          sm += st.y * ex2(st.x - Rm);
        }
        float Rr, sr;
        merge_lanes(make_float2(Rm, bad ? nan : sm), Rr, sr);
        // (NaN, NaN) for an unusable row, (NaN, +inf) for a wait that gave up
        const bool fine = !(sr != sr) && Rr != -INFINITY && sr > 0.f && !isinf(sr);
        if (l == 0)
          sh.norm[r] = !got ? make_float2(nan, INFINITY)
                            : (fine ? make_float2(Rr, __log2f(sr)) : make_float2(nan, nan));
      }
    }
    consumer_sync();  // the normalisers

    // ---- pass 2: the target chunk's exponents once, then every drafter ----
    // The folded form takes each row's normaliser as one offset o = R + L,
    // held in fp32 to ulp(o)/2: alpha stays within 2.6e-6 relative while
    // |o| < kFoldLimit.  Otherwise (low temperatures, large logits) R and L
    // stay apart: the target's terms use R_t alone, each drafter's are
    // shifted by L_t - L_d (small, full precision), and the partial is scaled
    // by 2^{-L_t}.  NaN normalisers take the split form and are flagged.
    const float2 nt = sh.norm[0];
    bool split = !(fabsf(nt.x + nt.y) < kFoldLimit);
    for (int d = 0; d < N; ++d) {
      const float2 nd = sh.norm[1 + d];
      split |= !(fabsf(nd.x + nd.y) < kFoldLimit);
    }
    bool bad_path = false;
    (void)target_row<DT>(p.target, p.path, p.M, p.P, ty, p.V, &bad_path);
    const float tofs = split ? nt.x : nt.x + nt.y;
    const uint64_t ot2 = pack2(-tofs, -tofs);
    float xt[8 * kVecsPerThread];  // log2 p of the thread's 32 logits (up to the split scale)
    {
      uint4 v[kVecsPerThread];
      take(jy, v);
#pragma unroll
      for (int u = 0; u < kVecsPerThread; ++u) {
        const uint32_t wd[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const uint64_t e = fma2(pair_of<DT>(wd[q]), c2, ot2);
          xt[8 * u + 2 * q] = lo2(e);
          xt[8 * u + 2 * q + 1] = hi2(e);
        }
      }
    }
    const bool ring_ok = ok && *err == 0;
    for (int d = 0; d < N; ++d) {
      const float2 nd = sh.norm[1 + d];
      const float dofs = split ? nd.x : nd.x + nd.y;
      const float shift = split ? nt.y - nd.y : 0.f;
      const uint64_t od2 = pack2(-dofs, -dofs), sh2 = pack2(shift, shift);
      uint4 v[kVecsPerThread];
      take(jy, v);
      uint64_t acc0 = 0ull, acc1 = 0ull;  // two independent chains
#pragma unroll
      for (int u = 0; u < kVecsPerThread; ++u) {
        const uint32_t wd[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint64_t e = fma2(pair_of<DT>(wd[q]), c2, od2);
          if (split) e = add2(e, sh2);
          const uint64_t m = pack2(ex2(fminf(xt[8 * u + 2 * q], lo2(e))),
                                   ex2(fminf(xt[8 * u + 2 * q + 1], hi2(e))));
          if (q & 1)
            acc1 = add2(acc1, m);
          else
            acc0 = add2(acc0, m);
        }
      }
      const uint64_t a2 = add2(acc0, acc1);
      float a = warp_sum(lo2(a2) + hi2(a2));
      if (split) a *= ex2(-nt.y);
      if (l == 0) {
        const bool good = ring_ok && !bad_path && !(nt.x != nt.x) && !(nd.x != nd.x);
        // a wait that gave up has reported itself (HS_ERR_TIMEOUT)
        const bool timed_out = nt.y == INFINITY || nd.y == INFINITY;
        if (!good && ring_ok && !timed_out)
          report(p.dev_status, bad_path ? HS_ERR_INVALID_ARG : HS_ERR_NONFINITE);
        sh.ap[b][d][w] = good ? a : nan;
      }
    }
    pt = ty;
    pj = jy;
    pb = b;
  }
  consumer_sync();  // the last overlap's partial posts
  if (pt >= 0) {
    for (int d = w; d < N; d += kConsumerWarps) {
      const float a = warp_sum(l < kConsumerWarps ? sh.ap[pb][d][l] : 0.f);
      if (l == 0) p.apart[(int64_t(d) * p.ntiles + pt) * p.nchunk + pj] = a;
    }
  }
}

constexpr size_t kRingOffset = (sizeof(Shared) + 127) & ~size_t(127);
size_t shared_bytes() { return kRingOffset + size_t(kStages) * kChunkBytes; }

template <int DT>
__global__ void __launch_bounds__(kThreads, 1) stream_kernel(const Params p) {
  extern __shared__ __align__(128) unsigned char smem[];
  Shared& sh = *reinterpret_cast<Shared*>(smem);
  const uint32_t ring0 = saddr(smem + kRingOffset);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(saddr(&sh.full[s]), 1);
      mbar_init(saddr(&sh.empty[s]), kConsumers);
    }
    sh.error = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  pdl_wait();  // the set-up above overlaps the previous kernel of the stream
  volatile int* err = &sh.error;
  const int G = gridDim.x, cta = blockIdx.x;
  const int steps = (p.nitems + G - 1) / G + p.lag;
  if (warp == kConsumerWarps) {
    // ------------------------------ producer ---------------------------------
    // Per step: the N+1 row chunks of the statistics item (kept in L2 for
    // the next step's overlap), then those of the overlap item (last use).
    if (lane == 0) {
      const uint64_t keep = make_policy(true), once = make_policy(false);
      const int nvec = p.V / 8, R = p.N + 1;
      uint32_t n = 0;  // chunks issued
      bool ok = true;
      auto put = [&](const char* row, int j, uint64_t pol) {
        if (!ok) return;
        const uint32_t s = n % kStages;
        if (n >= kStages &&
            !mbar_wait(saddr(&sh.empty[s]), ((n / kStages) - 1) & 1u, err, p.dev_status)) {
          ok = false;
          return;
        }
        const int v0 = j * kChunkVecs;
        const int nv = nvec - v0 < kChunkVecs ? nvec - v0 : kChunkVecs;
        bulk_fill(ring0 + s * kChunkBytes, saddr(&sh.full[s]), row + int64_t(v0) * 16,
                  uint32_t(nv) * 16u, pol);
        ++n;
      };
      for (int s = 0; s < steps; ++s) {
        const int x = s * G + cta, y = (s - p.lag) * G + cta;
        if (x < p.nitems) {
          const int tx = x / p.nchunk, jx = x - tx * p.nchunk;
          for (int r = 0; r < R; ++r) put(row_of<DT>(p, tx, r), jx, keep);
        }
        if (s >= p.lag && y < p.nitems) {
          const int ty = y / p.nchunk, jy = y - ty * p.nchunk;
          for (int r = 0; r < R; ++r) put(row_of<DT>(p, ty, r), jy, once);
        }
      }
      if (!ok) {
        // the copies already issued must land before the CTA's memory goes
        for (uint32_t j = n > uint32_t(kStages) ? n - kStages : 0; j < n; ++j) {
          const long long t0 = clock64();
          while (!mbar_test(saddr(&sh.full[j % kStages]), (j / kStages) & 1u) &&
                 clock64() - t0 < kTimeoutCycles) {
          }
        }
      }
    }
    __syncwarp();
  } else {
    consumer<DT>(p, sh, ring0, steps, err);
  }
}

// alpha[i, b, k] = the sum of tile (b,k)'s chunk partials in chunk order, and
// e_len[i, b] = 1 + sum_k prod_{j <= k} alpha_j over the first P-1 positions
// (Thm 3): one thread per (drafter, query).
__global__ void finish_kernel(const float* __restrict__ apart, int N, int B, int P, int nchunk,
                              float* __restrict__ alpha, float* __restrict__ e_len) {
  pdl_wait();
  const int64_t idx = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (idx >= int64_t(N) * B) return;
  const int64_t d = idx / B, b = idx - d * B, T = int64_t(B) * P;
  float e = 1.f, prod = 1.f;
  for (int k = 0; k < P; ++k) {
    const float* src = apart + (d * T + b * P + k) * nchunk;
    float a = 0.f;
    for (int j = 0; j < nchunk; ++j) a += src[j];
    alpha[d * T + b * P + k] = a;
    if (k < P - 1) {
      prod *= a;
      e += prod;
    }
  }
  if (e_len) e_len[idx] = e;
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

struct Layout {
  size_t stats, apart, cnt, total;
};

Layout layout(int N, int B, int P, int V) {
  const int64_t ntiles = int64_t(B) * P;
  const int64_t nchunk = (V + kChunk - 1) / kChunk;
  Layout L;
  L.stats = 0;
  L.apart = L.stats + align256(size_t(ntiles * (N + 1) * nchunk) * sizeof(float2));
  L.cnt = L.apart + align256(size_t(ntiles * N * nchunk) * sizeof(float));
  L.total = L.cnt + align256(size_t(ntiles) * sizeof(int));
  return L;
}

// SM count per device, queried on the first call (so that later calls can
// be captured into CUDA graphs); the kernel's shared-memory attribute is
// raised at the same time.  Keyed by device and guarded by a mutex, so host
// threads driving different GPUs may call concurrently.
template <int DT>
int sm_count() {
  static std::mutex mu;
  static int nsm_of[kMaxDevices] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
  std::lock_guard<std::mutex> lock(mu);
  if (!nsm_of[dev]) {
    int n = 0, per_sm = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaFuncSetAttribute(stream_kernel<DT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             int(shared_bytes())) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, stream_kernel<DT>, kThreads,
                                                      shared_bytes()) != cudaSuccess ||
        per_sm < 1)
      return 0;
    nsm_of[dev] = n;
  }
  return nsm_of[dev];
}

template <int DT>
hs_status launch_t(Params p, void* ws, float* alpha, float* e_len, cudaStream_t stream) {
  const int nsm = sm_count<DT>();
  if (nsm < 1) return HS_ERR_CUDA;
  const Layout L = layout(p.N, p.B, p.P, p.V);
  p.stats = reinterpret_cast<float2*>(static_cast<char*>(ws) + L.stats);
  p.apart = reinterpret_cast<float*>(static_cast<char*>(ws) + L.apart);
  p.cnt = reinterpret_cast<int*>(static_cast<char*>(ws) + L.cnt);
  if (cudaMemsetAsync(p.cnt, 0, size_t(p.ntiles) * sizeof(int), stream) != cudaSuccess)
    return HS_ERR_CUDA;
  // one CTA per SM, all resident (cooperative): every counter wait ends
  const int grid = p.nitems < nsm ? p.nitems : nsm;
  p.lag = 1 + (p.nchunk - 1) / grid;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.gridDim = dim3(unsigned(grid));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = shared_bytes();
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, stream_kernel<DT>, p) != cudaSuccess) return HS_ERR_CUDA;
  const int64_t nb = int64_t(p.N) * p.B;
  if (launch_pdl(finish_kernel, dim3(unsigned((nb + 127) / 128)), dim3(128), 0, stream,
                 static_cast<const float*>(p.apart), p.N, p.B, p.P, p.nchunk, alpha,
                 e_len) != cudaSuccess)
    return HS_ERR_CUDA;
  return HS_OK;
}

}  // namespace

bool eligible_sizes(int dtype, int N, int V, int greedy) {
  return !greedy && (dtype == HS_BF16 || dtype == HS_FP16) && N >= 1 && N <= kMaxN && V % 8 == 0;
}

bool eligible(const void* target, const void* drafter, int dtype, int N, int V, int greedy) {
  if (reinterpret_cast<uintptr_t>(target) % 16 || reinterpret_cast<uintptr_t>(drafter) % 16)
    return false;
  return eligible_sizes(dtype, N, V, greedy);
}

size_t workspace_bytes(int N, int B, int P, int V) { return layout(N, B, P, V).total; }

hs_status launch_impl(const void* target, const int32_t* path, int M, const void* drafter,
                      int dtype, int N, int B, int P, int V, float c, float* alpha, float* e_len,
                      void* ws, int* dev_status, cudaStream_t stream, int stall_tile,
                      long long wait_limit) {
  Params p = {};
  p.target = target;
  p.path = path;
  p.M = M;
  p.drafter = drafter;
  p.N = N;
  p.B = B;
  p.P = P;
  p.V = V;
  p.c = c;
  p.nchunk = (V + kChunk - 1) / kChunk;
  p.ntiles = B * P;
  p.nitems = p.ntiles * p.nchunk;
  p.dev_status = dev_status;
  p.stall_tile = stall_tile;
  p.wait_limit = wait_limit;
  return dtype == HS_BF16 ? launch_t<HS_BF16>(p, ws, alpha, e_len, stream)
                          : launch_t<HS_FP16>(p, ws, alpha, e_len, stream);
}

hs_status launch(const void* target, const int32_t* path, int M, const void* drafter, int dtype,
                 int N, int B, int P, int V, float c, float* alpha, float* e_len, void* ws,
                 int* dev_status, cudaStream_t stream) {
  return launch_impl(target, path, M, drafter, dtype, N, B, P, V, c, alpha, e_len, ws, dev_status,
                     stream, -1, kTimeoutCycles);
}

hs_status launch_wait_test(const void* target, const void* drafter, int dtype, int N, int B,
                           int P, int V, float c, long long wait_cycles, float* alpha,
                           float* e_len, void* ws, int* dev_status, cudaStream_t stream) {
  return launch_impl(target, nullptr, 0, drafter, dtype, N, B, P, V, c, alpha, e_len, ws,
                     dev_status, stream, 0, wait_cycles);
}

}  // namespace stream
}  // namespace hs
