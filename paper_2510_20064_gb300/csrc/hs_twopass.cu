// hs_twopass.cu -- stochastic feedback (Thm 1), two passes per row with the
// second served by L2, for shapes where the cluster kernel (hs_fused.cu)
// leaves SMs idle and the working set below fits in L2.
//
// One CTA per SM, no cluster; c = log2(e) / T throughout.
// The drafter rows of a call, ordered (tile, drafter), are split into even
// contiguous runs, one per CTA.  A CTA walks its run in groups of up to kG
// drafters of one tile:
//   pass 1: the tile's target offset o_t = c m + log2 sum_v 2^{c z_v - c m}
//           when the group starts a tile (or the run), so that
//           log2 p_v = c z_v - o_t, then each drafter row's offset o_i;
//   pass 2: the group's rows walked backwards (the most recently read part
//           first, while it is still in L2), each target chunk read once
//           for the group (from tensor memory, see below), summing
//           min(p_v, q_v) = 2^{min(c z_t - o_t, c z_d - o_i)}
//           (2^x is increasing, so the min moves inside: one exp2 per pair).
// One producer warp streams every chunk the consumers need, in their order,
// into a ring of 32 KB shared-memory stages with cp.async.bulk.  Pass 1 over
// the target parks its first kTmemChunks chunks (256 KB, a whole 128 256-logit
// bf16 row) in tensor memory, each thread its own words in its own lane, and
// pass 2 reads them from there; only the rest of a longer row comes back from
// L2, its loads asking L2 to keep the lines until the tile's last group.
// Pass 2's drafter loads mark theirs as last use.  Where a row's last chunk
// is at most half full, that chunk's arithmetic stops, warp by warp, after
// the last vector holding logits.  HBM reads each logit once
// as long as every SM's kG drafter rows and the target's tail stay in L2;
// the caller checks that (preferred()).
#include <math.h>
#include <stdint.h>

#include "hs_common.cuh"
#include "hs_twopass.h"

namespace hs {
namespace twopass {
namespace {

constexpr int kConsumerWarps = 16;
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kThreads = kConsumers + 32;       // + the producer warp
constexpr int kStages = 7;                      // ring stages (224 KB)
constexpr int kVecsPerThread = 4;               // 16-byte vectors of a stage per consumer
constexpr int kChunkVecs = kVecsPerThread * kConsumers;
constexpr int kChunkBytes = kChunkVecs * 16;    // 32 KB
constexpr int kG = 2;                           // drafters per group
constexpr int kWords = 4 * kVecsPerThread;      // 32-bit words of a chunk per thread
// Tensor memory: 128 lanes x 512 columns of 32 bits.  Consumer warp w owns
// lanes 32 (w % 4) .. +31 and columns 128 (w / 4) .. +127: kTmemChunks
// chunks of a row, kWords columns each.
static_assert(kConsumerWarps % 4 == 0, "warps share the four TMEM lane quadrants evenly");
constexpr int kTmemColsPerWarp = 512 / (kConsumerWarps / 4);
constexpr int kTmemChunks = kTmemColsPerWarp / kWords;
static_assert(kVecsPerThread == 4, "a chunk's words move to tensor memory 16 at a time");
constexpr long long kTimeoutCycles = 1LL << 31;  // about a second
constexpr float kFoldLimit = 64.f;  // |o| below which pass 2 folds R + L into one offset

template <int DT>
struct Pair;  // two logits of a 32-bit word as floats

template <>
struct Pair<HS_BF16> {
  __device__ static __forceinline__ float lo(uint32_t w) { return __uint_as_float(w << 16); }
  __device__ static __forceinline__ float hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
};
template <>
struct Pair<HS_FP16> {
  __device__ static __forceinline__ float lo(uint32_t w) {
    return __half2float(__ushort_as_half(static_cast<unsigned short>(w & 0xffffu)));
  }
  __device__ static __forceinline__ float hi(uint32_t w) {
    return __half2float(__ushort_as_half(static_cast<unsigned short>(w >> 16)));
  }
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
__device__ __forceinline__ uint64_t make_policy(int kind) {  // 0 normal, 1 keep, 2 last use
  uint64_t p;
  if (kind == 1)
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  else if (kind == 2)
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  else
    asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(p));
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
// ---- tensor memory (the target row between its two passes) ---------------------
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
// A chunk's 16 words of this thread into / out of 16 columns of its lane.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint4 (&v)[4]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, "
               "%9, %10, %11, %12, %13, %14, %15, %16};"
               :: "r"(taddr), "r"(v[0].x), "r"(v[0].y), "r"(v[0].z), "r"(v[0].w), "r"(v[1].x),
                  "r"(v[1].y), "r"(v[1].z), "r"(v[1].w), "r"(v[2].x), "r"(v[2].y), "r"(v[2].z),
                  "r"(v[2].w), "r"(v[3].x), "r"(v[3].y), "r"(v[3].z), "r"(v[3].w) : "memory");
}
// The load alone; tmem_wait_ld() below makes the registers valid.
__device__ __forceinline__ void tmem_ld16_async(uint32_t taddr, uint4 (&v)[4]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, "
               "%9, %10, %11, %12, %13, %14, %15}, [%16];"
               : "=r"(v[0].x), "=r"(v[0].y), "=r"(v[0].z), "=r"(v[0].w), "=r"(v[1].x),
                 "=r"(v[1].y), "=r"(v[1].z), "=r"(v[1].w), "=r"(v[2].x), "=r"(v[2].y),
                 "=r"(v[2].z), "=r"(v[2].w), "=r"(v[3].x), "=r"(v[3].y), "=r"(v[3].z),
                 "=r"(v[3].w) : "r"(taddr) : "memory");
}
// Waits for this thread's tensor-memory loads; the registers are passed
// through so that no use of them moves above the wait.
__device__ __forceinline__ void tmem_wait_ld(uint4 (&v)[4]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(v[0].x), "+r"(v[0].y), "+r"(v[0].z), "+r"(v[0].w), "+r"(v[1].x),
                 "+r"(v[1].y), "+r"(v[1].z), "+r"(v[1].w), "+r"(v[2].x), "+r"(v[2].y),
                 "+r"(v[2].z), "+r"(v[2].w), "+r"(v[3].x), "+r"(v[3].y), "+r"(v[3].z),
                 "+r"(v[3].w) :: "memory");
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint4 (&v)[4]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, "
               "%9, %10, %11, %12, %13, %14, %15}, [%16];"
               : "=r"(v[0].x), "=r"(v[0].y), "=r"(v[0].z), "=r"(v[0].w), "=r"(v[1].x),
                 "=r"(v[1].y), "=r"(v[1].z), "=r"(v[1].w), "=r"(v[2].x), "=r"(v[2].y),
                 "=r"(v[2].z), "=r"(v[2].w), "=r"(v[3].x), "=r"(v[3].y), "=r"(v[3].z),
                 "=r"(v[3].w) : "r"(taddr) : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Barrier of the consumer warps only (the producer warp never joins).
__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, %0;" :: "n"(kConsumers) : "memory");
}

// Per-warp posts of a group (the statistics of its rows, then its alpha
// partials), double-buffered by group parity: a buffer is rewritten two
// groups later, after barriers that every reader of its previous contents
// has passed.
struct Shared {
  uint64_t full[kStages], empty[kStages];
  float m[2][1 + kG][kConsumerWarps], s[2][1 + kG][kConsumerWarps];  // [group parity][row]
  int bad[2][1 + kG][kConsumerWarps];
  float acc[2][kG][kConsumerWarps];
  int error;
  uint32_t tmem_base;
};

struct Params {
  const void* target;
  const int32_t* path;
  const void* drafter;
  float* alpha;
  int* dev_status;
  int M, N, B, P, V;
  int t0;  // first tile of this kernel; it takes tiles t0 .. B*P-1 (0: all)
  float c;
};

// A CTA's group: drafters d0 .. d0+dn-1 of one tile, up to kG of them.
// with_t: the group starts the run's segment of its tile, so its pass 1
// reads the target; t_last: the segment's last group; shared: the tile has
// drafters in a neighbouring run too.
struct Group {
  int tile, d0, dn;
  bool with_t, t_last, shared;
};

// A CTA's walk over its run of drafter rows [rb, re) (tile-major), segment by
// segment -- a segment is the part of the run in one tile -- and in groups of
// up to kG drafters within a segment.  Even CTAs take the segments from the
// run's last tile back to its first, odd CTAs from the first on, so a tile
// split between two neighbouring runs is the first segment of both (read at
// the start of the call) or the last segment of both (read in both CTAs'
// final stretch): the second read of its target row can then come from L2.
struct Walk {
  int rb, re, N, tfirst, tlast, seg, tile, lo, hi, r;
  bool rev;
  __device__ void init(int rb_, int re_, int N_, bool rev_) {
    rb = rb_;
    re = re_;
    N = N_;
    rev = rev_;
    tfirst = rb / N;
    tlast = re > rb ? (re - 1) / N : tfirst - 1;
    seg = 0;
    if (!done()) start();
  }
  __device__ bool done() const { return seg > tlast - tfirst; }
  __device__ void start() {
    tile = rev ? tlast - seg : tfirst + seg;
    lo = rb > tile * N ? rb : tile * N;
    hi = re < (tile + 1) * N ? re : (tile + 1) * N;
    r = lo;
  }
  __device__ Group group() const {
    Group g;
    g.tile = tile;
    g.d0 = r - tile * N;
    g.dn = hi - r < kG ? hi - r : kG;
    g.with_t = r == lo;
    g.t_last = r + g.dn == hi;
    g.shared = lo > tile * N || hi < (tile + 1) * N;
    return g;
  }
  __device__ void advance(int dn) {
    r += dn;
    if (r >= hi) {
      ++seg;
      if (!done()) start();
    }
  }
};

// ---- consumer warps ---------------------------------------------------------------

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
// The two logits of a stored word as a packed pair.
template <int DT>
__device__ __forceinline__ uint64_t pair_of(uint32_t w) {
  return pack2(Pair<DT>::lo(w), Pair<DT>::hi(w));
}
// NaN-propagating packed max of two stored words, and the max of its pair.
template <int DT>
__device__ __forceinline__ uint32_t pmax(uint32_t a, uint32_t b) {
  uint32_t r;
  if (DT == HS_BF16)
    asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  else
    asm("max.NaN.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}


// Running statistics of a row in pass 1, in log2 units: an integer reference
// R (-inf until the row shows a finite logit) and two independent chains of
// packed partial sums of 2^{c z - R}; bad once a NaN or +inf logit was seen.
// R = ceil(c m) for m the max of the chunk that set it, so every offset and
// every rescale between references is exact and the sums are exactly
// relative to R (up to the rounding of each term).  Any reference gives the
// same normaliser R + log2 sum_v 2^{c z_v - R}; R only has to keep the terms
// finite, so it is set by the first chunk with a finite logit and raised only
// when a chunk's sum under it passes 2^100 (a term above 2^126 would
// overflow).  Terms far below R vanish as they would below the row max.
struct Stat {
  float R;
  uint64_t s2[2];
  bool bad;
};

template <int DT>
__device__ __forceinline__ Stat stat_init() {
  Stat st;
  st.R = -INFINITY;
  st.s2[0] = st.s2[1] = 0ull;
  st.bad = false;
  return st;
}

// The chunk's (the thread's 32 logits) sums of 2^{c z - R}, two packed pairs.
template <int DT>
__device__ __forceinline__ void chunk_sums(const uint4 (&v)[kVecsPerThread], uint64_t c2,
                                           float R, int nu, uint64_t& a, uint64_t& b) {
  const float off = R == -INFINITY ? 0.f : -R;  // all -inf so far: every term is 0
  const uint64_t off2 = pack2(off, off);
  a = b = 0ull;
#pragma unroll
  for (int u = 0; u < kVecsPerThread; ++u) {
    if (u < nu) {  // warp-uniform: only a row's last chunk has nu < kVecsPerThread
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
  }
}

// Fold one chunk into a row's statistics.  The chunk's max is only formed
// for the first chunk with a finite logit and when the sums under the
// current reference pass 2^100 or are not finite (NaN / +inf logits).
template <int DT>
__device__ __forceinline__ void stat_chunk(Stat& st, const uint4 (&v)[kVecsPerThread], float c,
                                           uint64_t c2, int nu) {
  uint64_t a, b;
  bool redo = st.R == -INFINITY;
  if (!redo) {
    chunk_sums<DT>(v, c2, st.R, nu, a, b);
    const uint64_t t2 = add2(a, b);
    redo = !(lo2(t2) + hi2(t2) <= 0x1p100f);
  }
  if (redo) {
    uint32_t mw = pmax<DT>(pmax<DT>(v[0].x, v[0].y), pmax<DT>(v[0].z, v[0].w));
#pragma unroll
    for (int u = 1; u < kVecsPerThread; ++u)
      mw = pmax<DT>(mw, pmax<DT>(pmax<DT>(v[u].x, v[u].y), pmax<DT>(v[u].z, v[u].w)));
    const float cm = max_nan(Pair<DT>::lo(mw), Pair<DT>::hi(mw));
    st.bad |= (cm != cm) || cm == INFINITY;
    const float Rn = ceilf(cm * c);  // -inf for an all -inf chunk, NaN stays out below
    if (Rn > st.R) {
      const float r = (st.R == -INFINITY) ? 0.f : ex2(st.R - Rn);  // an exact power of 2
      const uint64_t r2 = pack2(r, r), z2 = 0ull;
      st.s2[0] = fma2(st.s2[0], r2, z2);
      st.s2[1] = fma2(st.s2[1], r2, z2);
      st.R = Rn;
    }
    chunk_sums<DT>(v, c2, st.R, nu, a, b);
  }
  st.s2[0] = add2(st.s2[0], a);
  st.s2[1] = add2(st.s2[1], b);
}

// Every lane: the merge (R, S) of the warp's pairs (R, s), each s relative to
// its integer reference R: the largest reference first (one redux), then
// every sum rescaled to it once (by an exact power of 2) and added up.  (R is
// never NaN; a +inf R only comes with the row's bad flag.)
__device__ __forceinline__ void warp_merge(float& R, float& s) {
  float M;
  asm volatile("redux.sync.max.f32 %0, %1, 0xffffffff;" : "=f"(M) : "f"(R));  // warp-collective: kept in place
  s = (R == -INFINITY) ? 0.f : s * ex2(R - M);
  R = M;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
}

// Lane 0 of each warp posts the warp's merged (R, s, bad) of a row.
__device__ __forceinline__ void post_stat(const Stat& st, float* pm, float* ps, int* pb, int w,
                                          int l) {
  const uint64_t s2 = add2(st.s2[0], st.s2[1]);
  float R = st.R, s = lo2(s2) + hi2(s2);
  warp_merge(R, s);
  const bool bad = __any_sync(0xffffffffu, st.bad);
  if (l == 0) {
    pm[w] = R;
    ps[w] = s;
    pb[w] = bad;
  }
}

// A row's normaliser in log2 units, as its integer reference R and
// L = log2 sum_v 2^{c z_v - R}: log2 p_v = c z_v - R - L.  Both NaN for an
// unusable row (a NaN or +inf logit, or no finite logit).
struct Norm {
  float R, L;
};

// Every thread: the row's Norm from the warps' posts (lanes 0..15 read one
// each and the warp merges them).
__device__ __forceinline__ Norm row_norm(const float* pm, const float* ps, const int* pb, int l) {
  float R = l < kConsumerWarps ? pm[l] : -INFINITY;
  float s = l < kConsumerWarps ? ps[l] : 0.f;
  const bool bad = __any_sync(0xffffffffu, l < kConsumerWarps && pb[l] != 0);
  warp_merge(R, s);
  if (bad || R == -INFINITY || !(s > 0.f) || isinf(s)) {
    const float nan = __int_as_float(0x7fc00000);
    return Norm{nan, nan};
  }
  return Norm{R, __log2f(s)};
}

// The consumers' side of drafter rows rb .. re-1, group by group in the
// producer's order: pass 1 over the target row (when the group starts a
// tile or the run; its first kTmemChunks chunks also go to tensor memory)
// and over each drafter row, then pass 2 backwards, each target chunk (from
// tensor memory, or the ring past kTmemChunks) followed by the group's
// drafter chunks.  Every consumer
// thread runs the same control flow (also after a timeout, then on whatever
// the stages hold), so the consumer barriers always meet; a timed-out call
// reports HS_ERR_TIMEOUT and writes NaN.  A thread holds 4 vectors (32
// logits) of each stage; only a row's last chunk can end early, and only
// there are the vectors past the row's end replaced by -inf (kSkip: and a
// warp's arithmetic stops after the last of its vectors holding a logit).
template <int DT, bool kSkip>
__device__ __forceinline__ void consumer(const Params& p, Shared& sh, uint32_t ring0, int nvec,
                                         int nch, int rb, int re, float c, volatile int* err) {
  const int t = threadIdx.x, w = t >> 5, l = t & 31;
  const uint32_t tcol = sh.tmem_base + (uint32_t(32 * (w & 3)) << 16) +
                        uint32_t(kTmemColsPerWarp * (w >> 2));  // this thread's lane and columns
  const int T = p.B * p.P;
  uint32_t stage = 0, phase = 0;  // the next stage and its phase parity
  bool ok = true;
  const uint32_t ninf = DT == HS_BF16 ? 0xFF80FF80u : 0xFC00FC00u;
  const uint64_t c2 = pack2(c, c);
  // kSkip: the arithmetic of a row's last chunk stops at the vectors u that
  // hold logits for some lane of this warp (u * kConsumers + 32 w below the
  // chunk's vector count); the others are -inf for every lane
  const int tail_vecs = nvec - (nch - 1) * kChunkVecs - 32 * w;
  const int tail_nu = tail_vecs <= 0 ? 0
                      : (tail_vecs + kConsumers - 1) / kConsumers < kVecsPerThread
                          ? (tail_vecs + kConsumers - 1) / kConsumers
                          : kVecsPerThread;
  // the next stage into v; tail: the row's last chunk, whose vectors past
  // the row's end become -inf (callers pass a constant, ch == nch - 1)
  auto take = [&](int ch, bool tail, uint4 (&v)[kVecsPerThread]) {
    if (!mbar_wait(saddr(&sh.full[stage]), phase, err, p.dev_status)) ok = false;
    const uint32_t base = ring0 + stage * kChunkBytes + uint32_t(t) * 16u;
#pragma unroll
    for (int u = 0; u < kVecsPerThread; ++u) v[u] = lds128(base + uint32_t(u * kConsumers) * 16u);
    if (tail) {
#pragma unroll
      for (int u = 0; u < kVecsPerThread; ++u)
        if (ch * kChunkVecs + u * kConsumers + t >= nvec) v[u] = make_uint4(ninf, ninf, ninf, ninf);
    }
    // every consumer thread releases its own part of the stage (the stage's
    // barrier counts kConsumers arrivals): no warp-level hand-off needed
    mbar_arrive(saddr(&sh.empty[stage]));
    if (++stage == kStages) {
      stage = 0;
      phase ^= 1u;
    }
  };
  uint32_t rp = 0;  // buffers of the current group (group parity)
  // pass 1 over one row: each warp posts its merged statistics in slot
  // `slot` of the group (0: the target, 1 + i: drafter i of the group);
  // park: the row's first kTmemChunks chunks also go to tensor memory
  auto pass1 = [&](bool park, int slot) {
    Stat st = stat_init<DT>();
    auto step = [&](int ch, bool tail) {
      uint4 v[kVecsPerThread];
      take(ch, tail, v);
      if (park && ch < kTmemChunks) tmem_st16(tcol + uint32_t(kWords * ch), v);
      stat_chunk<DT>(st, v, c, c2, kSkip && tail ? tail_nu : kVecsPerThread);
    };
    for (int ch = 0; ch < nch - 1; ++ch) step(ch, false);
    step(nch - 1, true);
    if (park) asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    post_stat(st, sh.m[rp][slot], sh.s[rp][slot], sh.bad[rp][slot], w, l);
  };
  // after the group's consumer barrier: a row's normaliser in every thread
  // (NaN for an unusable row)
  auto norm_of = [&](int slot) {
    return row_norm(sh.m[rp][slot], sh.s[rp][slot], sh.bad[rp][slot], l);
  };
  Norm nt = {0.f, 0.f};   // normaliser of the current tile's target row
  bool bad_path = false;  // the current tile has an out-of-range path node
  Walk walk;
  walk.init(rb, re, p.N, (blockIdx.x & 1u) == 0u);
  for (; !walk.done(); ) {
    const Group g = walk.group();
    // pass 1 over the group's rows, each warp posting its statistics; one
    // consumer barrier, then every warp merges the posts of each row
    if (g.with_t) {
      bad_path = false;
      (void)target_row<DT>(p.target, p.path, p.M, p.P, g.tile, p.V, &bad_path);
      pass1(true, 0);
    }
#pragma unroll
    for (int gi = 0; gi < kG; ++gi)
      if (gi < g.dn) pass1(false, 1 + gi);
    consumer_sync();
    if (g.with_t) nt = norm_of(0);
    Norm nd[kG];
#pragma unroll
    for (int gi = 0; gi < kG; ++gi) nd[gi] = gi < g.dn ? norm_of(1 + gi) : Norm{0.f, 0.f};
    // The folded form takes each row's normaliser as one offset o = R + L,
    // held in fp32 to ulp(o)/2: alpha stays within 2.6e-6 relative while
    // |o| < kFoldLimit.  Otherwise (low temperatures, large logits) pass 2
    // keeps R and L apart: the target's terms use R_t alone, each drafter's
    // are shifted by L_t - L_d (a small number, full precision), and alpha
    // is scaled by 2^{-L_t} at the end.  NaN normalisers take the split form
    // and are flagged below.
    bool split = !(fabsf(nt.R + nt.L) < kFoldLimit);
#pragma unroll
    for (int gi = 0; gi < kG; ++gi)
      if (gi < g.dn) split |= !(fabsf(nd[gi].R + nd[gi].L) < kFoldLimit);
    const float tofs = split ? nt.R : nt.R + nt.L;
    const uint64_t ot2 = pack2(-tofs, -tofs);
    uint64_t od2[kG], sh2[kG];
#pragma unroll
    for (int gi = 0; gi < kG; ++gi) {
      const float dofs = split ? nd[gi].R : nd[gi].R + nd[gi].L;
      const float shift = split ? nt.L - nd[gi].L : 0.f;
      od2[gi] = pack2(-dofs, -dofs);
      sh2[gi] = pack2(shift, shift);
    }
    uint64_t acc[kG][2];  // two independent chains per drafter
#pragma unroll
    for (int gi = 0; gi < kG; ++gi) acc[gi][0] = acc[gi][1] = 0ull;
    // one chunk of pass 2: the target's words from tensor memory (tm) or the
    // ring, then each drafter's from the ring; full: the group has kG
    // drafters; sp: the split form (callers pass constants where they can, so
    // the loops below carry none of these tests)
    auto p2chunk = [&](int ch, bool tail, bool tm, bool full, bool sp) {
      uint4 v[kVecsPerThread], d[kVecsPerThread];
      // the target's words (tensor memory or ring) and the first drafter's:
      // the tensor-memory load is in flight while the drafter's chunk is taken
      if (tm) {
        tmem_ld16_async(tcol + uint32_t(kWords * ch), v);
        take(ch, tail, d);
        tmem_wait_ld(v);
      } else {
        take(ch, tail, v);
        take(ch, tail, d);
      }
      const int nu = kSkip && tail ? tail_nu : kVecsPerThread;
      float xt[8 * kVecsPerThread];  // log2 p of the thread's 32 logits
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
#pragma unroll
      for (int gi = 0; gi < kG; ++gi) {
        if (full || gi < g.dn) {
          if (gi > 0) take(ch, tail, d);
#pragma unroll
          for (int u = 0; u < kVecsPerThread; ++u) {
            if (u < nu) {
              const uint32_t wd[4] = {d[u].x, d[u].y, d[u].z, d[u].w};
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                uint64_t e = fma2(pair_of<DT>(wd[q]), c2, od2[gi]);
                if (sp) e = add2(e, sh2[gi]);
                acc[gi][q & 1] = add2(acc[gi][q & 1],
                                      pack2(ex2(fminf(xt[8 * u + 2 * q], lo2(e))),
                                            ex2(fminf(xt[8 * u + 2 * q + 1], hi2(e)))));
              }
            }
          }
        }
      }
    };
    auto pass2 = [&](bool full, bool sp) {
      p2chunk(nch - 1, true, nch - 1 < kTmemChunks, full, sp);
      int ch = nch - 2;
      for (; ch >= kTmemChunks; --ch) p2chunk(ch, false, false, full, sp);
      for (; ch >= 0; --ch) p2chunk(ch, false, true, full, sp);
    };
    if (!split)
      pass2(g.dn == kG, false);  // the usual case: one drafter pair form per group
    else
      pass2(g.dn == kG, true);
#pragma unroll
    for (int gi = 0; gi < kG; ++gi) {
      if (gi < g.dn) {
        const uint64_t a2 = add2(acc[gi][0], acc[gi][1]);
        const float a = warp_sum(lo2(a2) + hi2(a2));
        if (l == 0) sh.acc[rp][gi][w] = a;
      }
    }
    consumer_sync();
    if (w == 0) {
#pragma unroll
      for (int gi = 0; gi < kG; ++gi) {
        if (gi < g.dn) {
          float a = warp_sum(l < kConsumerWarps ? sh.acc[rp][gi][l] : 0.f);
          if (split) a *= ex2(-nt.L);
          if (l == 0) {
            const bool fine = ok && *err == 0;
            const bool good = fine && !bad_path && !(nt.L != nt.L) && !(nd[gi].L != nd[gi].L);
            if (!good && fine) report(p.dev_status, bad_path ? HS_ERR_INVALID_ARG : HS_ERR_NONFINITE);
            p.alpha[int64_t(g.d0 + gi) * T + g.tile] = good ? a : __int_as_float(0x7fc00000);
          }
        }
      }
    }
    rp ^= 1u;
    walk.advance(g.dn);
  }
  // every consumer warp is done with tensor memory before it is released
  tmem_fence_before();
  consumer_sync();
  tmem_fence_after();
  if (w == 0) tmem_dealloc512(sh.tmem_base);
}

size_t shared_bytes() {
  return ((sizeof(Shared) + 127) & ~size_t(127)) + size_t(kStages) * kChunkBytes;
}

template <int DT, bool kSkip>
__global__ void __launch_bounds__(kThreads, 1) twopass_kernel(const Params p) {
  extern __shared__ __align__(128) unsigned char smem[];
  Shared& sh = *reinterpret_cast<Shared*>(smem);
  const uint32_t ring0 = saddr(smem + ((sizeof(Shared) + 127) & ~size_t(127)));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(saddr(&sh.full[s]), 1);
      mbar_init(saddr(&sh.empty[s]), kConsumers);
    }
    sh.error = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // The shared memory keeps this kernel to one CTA per SM, so the allocation
  // can only wait for another kernel's CTA on the SM to finish.
  if (warp == 0) tmem_alloc512(saddr(&sh.tmem_base));
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();
  pdl_wait();  // the set-up above overlaps the previous kernel of the stream
  volatile int* err = &sh.error;
  const int nvec = p.V / 8;
  const int nch = (nvec + kChunkVecs - 1) / kChunkVecs;
  const int T = p.B * p.P;
  // this CTA's run of drafter rows (tile-major): an even split of rows
  // t0*N .. T*N-1
  const int64_t first = int64_t(p.t0) * p.N, total = int64_t(T - p.t0) * p.N;
  const int rb = int(first + total * blockIdx.x / gridDim.x);
  const int re = int(first + total * (blockIdx.x + 1) / gridDim.x);
  const float c = p.c;

  if (warp == kConsumerWarps) {
    // ------------------------------ producer ---------------------------------
    // Streams every chunk in the order the consumers take them (see consumer).
    if (lane == 0) {
      const uint64_t normal = make_policy(0), keep = make_policy(1), once = make_policy(2);
      uint32_t n = 0;  // chunks issued
      bool ok = true;
      auto put = [&](const char* row, int ch, uint64_t pol) {
        if (!ok) return;
        const uint32_t s = n % kStages;
        if (n >= kStages &&
            !mbar_wait(saddr(&sh.empty[s]), ((n / kStages) - 1) & 1u, err, p.dev_status)) {
          ok = false;
          return;
        }
        const int v0 = ch * kChunkVecs;
        const int nv = nvec - v0 < kChunkVecs ? nvec - v0 : kChunkVecs;
        bulk_fill(ring0 + s * kChunkBytes, saddr(&sh.full[s]), row + int64_t(v0) * 16,
                  uint32_t(nv) * 16u, pol);
        ++n;
      };
      auto drow = [&](int d, int tile) {
        return static_cast<const char*>(row_ptr<DT>(p.drafter, int64_t(d) * T + tile, p.V));
      };
      Walk walk;
      walk.init(rb, re, p.N, (blockIdx.x & 1u) == 0u);
      for (; !walk.done(); ) {
        const Group g = walk.group();
        bool bad_path = false;
        const char* tr = static_cast<const char*>(
            target_row<DT>(p.target, p.path, p.M, p.P, g.tile, p.V, &bad_path));
        if (g.with_t)  // chunks past kTmemChunks are read again in pass 2
          for (int ch = 0; ch < nch; ++ch) put(tr, ch, ch < kTmemChunks ? once : keep);
        for (int gi = 0; gi < g.dn; ++gi) {
          const char* dr = drow(g.d0 + gi, g.tile);
          for (int ch = 0; ch < nch; ++ch) put(dr, ch, normal);
        }
        for (int ch = nch - 1; ch >= 0; --ch) {
          if (ch >= kTmemChunks) put(tr, ch, g.t_last ? once : keep);
          for (int gi = 0; gi < g.dn; ++gi) put(drow(g.d0 + gi, g.tile), ch, once);
        }
        walk.advance(g.dn);
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
  } else {
    consumer<DT, kSkip>(p, sh, ring0, nvec, nch, rb, re, c, err);
  }
}

}  // namespace

bool preferred(int V, int elem_bytes, int tiles, int N, int sms, int cluster_sms,
               size_t l2_bytes) {
  if (cluster_sms >= sms || int64_t(tiles) * N < 2 * int64_t(sms)) return false;
  // per SM: kG drafter rows and the part of the target row past tensor memory
  const double row = double(V) * elem_bytes;
  const double tail = row - double(kTmemChunks) * kChunkBytes;
  const double working_set = (kG * row + (tail > 0 ? tail : 0.0)) * sms;
  return working_set <= 0.9 * double(l2_bytes);
}

int pair_grid(int V, int elem_bytes, int tiles, int N, int sms, size_t l2_bytes) {
  const int64_t rows = int64_t(tiles) * N;
  if (N % kG != 0 || rows >= 2 * int64_t(sms) || 10 * (rows / kG) < 7 * int64_t(sms)) return 0;
  const int64_t grid = rows / kG;
  const double row = double(V) * elem_bytes;
  const double tail = row - double(kTmemChunks) * kChunkBytes;
  const double working_set = (kG * row + (tail > 0 ? tail : 0.0)) * double(grid);
  return working_set <= 0.9 * double(l2_bytes) ? int(grid) : 0;
}

int long_row_grid(int V, int elem_bytes, int tiles, int N, int sms, size_t l2_bytes) {
  const int64_t rows = int64_t(tiles) * N;
  if (rows < 2 * int64_t(sms)) return pair_grid(V, elem_bytes, tiles, N, sms, l2_bytes);
  const double row = double(V) * elem_bytes;
  const double tail = row - double(kTmemChunks) * kChunkBytes;
  const double working_set = (kG * row + (tail > 0 ? tail : 0.0)) * sms;
  return working_set <= 2.0 * double(l2_bytes) ? sms : 0;
}

hs_status launch(const void* target, const int32_t* path, int M, const void* drafter, int dtype,
                 int N, int B, int P, int V, float c, int t0, int grid, float* alpha,
                 int* dev_status, cudaStream_t stream) {
  Params p;
  p.target = target;
  p.path = path;
  p.drafter = drafter;
  p.alpha = alpha;
  p.dev_status = dev_status;
  p.M = M;
  p.N = N;
  p.B = B;
  p.P = P;
  p.V = V;
  p.t0 = t0;
  p.c = c;
  const size_t smem = shared_bytes();
  // Rows whose last chunk is at most half full skip the arithmetic of its
  // empty part (V = 151 936: 1.5% faster); for fuller last chunks the guards
  // cost more than they save (V = 128 256: 1.5% slower), so that kernel has none.
  const int tail_vecs = V / 8 - (V / 8 - 1) / kChunkVecs * kChunkVecs;
  const bool skip = 2 * tail_vecs <= kChunkVecs;
  auto kern = dtype == HS_BF16
                  ? (skip ? twopass_kernel<HS_BF16, true> : twopass_kernel<HS_BF16, false>)
                  : (skip ? twopass_kernel<HS_FP16, true> : twopass_kernel<HS_FP16, false>);
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)) !=
      cudaSuccess)
    return HS_ERR_CUDA;
  return launch_pdl(kern, dim3(unsigned(grid)), dim3(kThreads), smem, stream, p) == cudaSuccess
             ? HS_OK
             : HS_ERR_CUDA;
}

}  // namespace twopass
}  // namespace hs

