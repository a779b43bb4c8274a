// hs_topl.cu -- feedback for an EAGLE draft tree with branching L (Thm 2):
// the target's token is accepted at a draft step iff it is among the L
// children the drafter proposes, its top-L tokens.  Stochastic target:
//   alpha[i,b,k] = sum_{v in Top_L(q_i)} p(v),   p = softmax(z_target / T);
// greedy target: alpha = 1[argmax p in Top_L(q_i)].  e_len by Thm 3.
//
//   topl_kernel   one warp per drafter row (i, b, k), or per 1/S of the row
//                 when rows are few.  The warp streams two segments:
//                   A  its 1/(N S) share of the target row of (b, k):
//                      NaN-propagating max, first argmax and
//                      sum_v 2^{(z_v - m) c}, c = log2(e) / T, per lane with
//                      rescaling, merged over the warp at the end;
//                   B  its drafter range: the warp keeps the range's L best
//                      (logit, -index) keys spread over its lanes (below).
//                 With 16-byte-aligned rows the segments pass through a
//                 per-warp ring of shared-memory stages that one lane fills
//                 with cp.async.bulk (mbarrier completion), so every warp has
//                 several steps in flight without holding them in registers.
//   alpha_kernel  one warp per drafter row: merges the N S target partials of
//                 its (b, k) and the S key lists of its row, and sums p over
//                 the row's top L, or over the first keep[row] of them when
//                 the tree was pruned (greedy target: compares with the first
//                 argmax); the last warp of each (i, b) to finish forms e_len.
// Every logit is read once.  The ranking is by the stored drafter logits
// (q's order does not depend on the temperature), ties toward the lower
// index, -inf last.
#include <math.h>
#include <stdint.h>

#include <climits>

#include "hs_common.cuh"
#include "hs_topl.h"

namespace hs {
namespace topl {
namespace {

// Small CTAs (4 independent warps): the SMs then get nearly equal shares of
// the warps (tree_path's 2048 rows are 512 CTAs, 3 or 4 per SM, where 256
// CTAs of 8 warps gave some SMs twice the work of others), and the register
// budget of 4 CTAs per SM (128) holds the warp's state without spilling.
constexpr int kThreads = 128;
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 4;                        // 16-byte vectors per lane per step
constexpr int kStages = 3;                        // ring stages per warp
constexpr int kStageBytes = 32 * kUnroll * 16;    // one warp step
constexpr int kPartSlots = 17;                    // L keys (<= 16) + flags
constexpr long long kTimeoutCycles = 2000000000;  // about 1 s

constexpr size_t ring_smem() { return size_t(kWarps) * kStages * (kStageBytes + 8); }

struct TStat {  // one share of a target row
  float m;      // max (stored logit) of the share
  float s;      // sum over the share of 2^{(z_v - m) c}
  int argmax;   // first index of the max (INT_MAX: none)
  int flags;    // bit 0: NaN or +inf in the share; bit 1: bad path node
};

struct Params {
  const void* target;
  const int32_t* path;
  const void* drafter;
  TStat* stats;      // [B*P][N*S]
  uint64_t* parts;   // [N*B*P][S][kPartSlots]
  int* counters;     // [N*B] warps done per (i, b), for e_len
  const int32_t* keep;  // [N*B*P] children kept by the tree's pruning, or null (all L)
  float* alpha;
  float* e_len;
  int* dev_status;
  int64_t nrows;     // N*B*P
  int M, N, B, P, V, L, S, greedy;
  float c;           // log2(e) / T
};

__host__ __device__ constexpr int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Order-preserving unsigned key of a non-NaN float (-inf lowest, +inf highest).
__device__ __forceinline__ uint32_t okey(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
// The float of an order key (the inverse of okey).
__device__ __forceinline__ float ofloat(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}
// The float of a key's value part, with the keys at or below okey(-inf) =
// 0x007fffff (the ones below it are NaN patterns) read as -inf.
__device__ __forceinline__ float key_float(uint64_t k) {
  const uint32_t h = uint32_t(k >> 32);
  return h <= 0x007fffffu ? -INFINITY : ofloat(h);
}

// (offset, sum) pairs over a warp: the larger offset and the rescaled sum.
__device__ __forceinline__ void merge_os(float& m, float& s, float c) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    const float M = max_nan(m, m2);
    const float a = (m == -INFINITY) ? 0.f : s * ex2((m - M) * c);
    const float b = (m2 == -INFINITY) ? 0.f : s2 * ex2((m2 - M) * c);
    m = M;
    s = a + b;
  }
}

// The warp's best key among the lanes' values (two 32-bit reductions: the
// value half, then the index half among the lanes holding that value).
__device__ __forceinline__ uint64_t warp_best(uint64_t k) {
  const uint32_t hi = uint32_t(k >> 32), lo = uint32_t(k);
  const uint32_t mh = __reduce_max_sync(0xffffffffu, hi);
  const uint32_t ml = __reduce_max_sync(0xffffffffu, hi == mh ? lo : 0u);
  return (uint64_t(mh) << 32) | ml;
}

__device__ __forceinline__ uint64_t shfl_u64(uint64_t k, int src) {
  const uint32_t hi = __shfl_sync(0xffffffffu, uint32_t(k >> 32), src);
  const uint32_t lo = __shfl_sync(0xffffffffu, uint32_t(k), src);
  return (uint64_t(hi) << 32) | lo;
}
__device__ __forceinline__ uint64_t shfl_up_u64(uint64_t k) {
  const uint32_t hi = __shfl_up_sync(0xffffffffu, uint32_t(k >> 32), 1);
  const uint32_t lo = __shfl_up_sync(0xffffffffu, uint32_t(k), 1);
  return (uint64_t(hi) << 32) | lo;
}

// (value, -index) key of a token: larger value first, then lower index.
__device__ __forceinline__ uint64_t token_key(float z, int v) {
  return (uint64_t(okey(z)) << 32) | (0xffffffffu - uint32_t(v));
}

// ---- per-warp ring: mbarriers and bulk copies --------------------------------

__device__ __forceinline__ uint32_t saddr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" :: "r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile("{\n\t.reg .pred p;\n\t"
               "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
               "selp.u32 %0, 1, 0, p;\n\t}"
               : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
  return ok != 0;
}
// Bounded wait for a stage (every lane); false after about a second.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  if (mbar_test(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_test(bar, parity))
    if (clock64() - t0 > kTimeoutCycles) return false;
  return true;
}
// One lane: stream `bytes` (a multiple of 16, 16-byte-aligned source) into a
// stage, completing its mbarrier's phase.  The fence orders the warp's
// earlier shared-memory reads of the stage before the copy's writes.
__device__ __forceinline__ void bulk_fill(uint32_t stage, uint32_t bar, const void* src,
                                          uint32_t bytes) {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
               :: "r"(bar), "r"(bytes) : "memory");
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes "
               "[%0], [%1], %2, [%3];"
               :: "r"(stage), "l"(src), "r"(bytes), "r"(bar) : "memory");
}
__device__ __forceinline__ uint4 lds128(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a) : "memory");
  return v;
}

// ---- 16-byte vectors of stored logits ---------------------------------------

template <int DT>
struct Vec;  // kN logits in one uint4, their maximum and their values

template <>
struct Vec<HS_BF16> {
  static constexpr int kN = 8;
  static constexpr uint32_t kNegInf = 0xFF80FF80u;
  __device__ static __forceinline__ uint32_t pmax(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
  }
  __device__ static __forceinline__ float at(uint4 w, int q) {
    const uint32_t x = q < 2 ? w.x : q < 4 ? w.y : q < 6 ? w.z : w.w;
    return __uint_as_float((q & 1) ? (x & 0xffff0000u) : (x << 16));
  }
  __device__ static __forceinline__ float at_dyn(uint4 w, int q) {  // q not a constant
    const uint32_t lo = (q & 2) ? w.y : w.x, hi = (q & 2) ? w.w : w.z;
    const uint32_t x = (q & 4) ? hi : lo;
    return __uint_as_float((x << (16 - 16 * (q & 1))) & 0xffff0000u);
  }
  __device__ static __forceinline__ float wfloat(uint32_t m) {  // max of a packed pair
    return max_nan(__uint_as_float(m << 16), __uint_as_float(m & 0xffff0000u));
  }
};

template <>
struct Vec<HS_FP16> {
  static constexpr int kN = 8;
  static constexpr uint32_t kNegInf = 0xFC00FC00u;
  __device__ static __forceinline__ uint32_t pmax(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("max.NaN.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
  }
  __device__ static __forceinline__ float half(uint32_t x, int hi) {
    return __half2float(__ushort_as_half(static_cast<unsigned short>(hi ? x >> 16 : x & 0xffffu)));
  }
  __device__ static __forceinline__ float at(uint4 w, int q) {
    const uint32_t x = q < 2 ? w.x : q < 4 ? w.y : q < 6 ? w.z : w.w;
    return half(x, q & 1);
  }
  __device__ static __forceinline__ float at_dyn(uint4 w, int q) {
    const uint32_t lo = (q & 2) ? w.y : w.x, hi = (q & 2) ? w.w : w.z;
    const uint32_t x = (q & 4) ? hi : lo;
    return __half2float(__ushort_as_half(static_cast<unsigned short>(x >> (16 * (q & 1)))));
  }
  __device__ static __forceinline__ float wfloat(uint32_t m) {
    return max_nan(half(m, 0), half(m, 1));
  }
};

template <>
struct Vec<HS_FP32> {
  static constexpr int kN = 4;
  static constexpr uint32_t kNegInf = 0xFF800000u;
  __device__ static __forceinline__ float at(uint4 w, int q) {
    return __uint_as_float(q == 0 ? w.x : q == 1 ? w.y : q == 2 ? w.z : w.w);
  }
  __device__ static __forceinline__ float at_dyn(uint4 w, int q) {
    const uint32_t lo = (q & 1) ? w.y : w.x, hi = (q & 1) ? w.w : w.z;
    return __uint_as_float((q & 2) ? hi : lo);
  }
  __device__ static __forceinline__ uint32_t pmax(uint32_t a, uint32_t b) {
    return __float_as_uint(max_nan(__uint_as_float(a), __uint_as_float(b)));
  }
  __device__ static __forceinline__ float wfloat(uint32_t m) { return __uint_as_float(m); }
};

// Vector of the row starting at logit v (-inf past the end of the row).
template <int DT, bool VEC>
__device__ __forceinline__ uint4 load_vec(const void* row, int64_t v, int V) {
  constexpr int kN = Vec<DT>::kN;
  if (VEC && v + kN <= V)
    return __ldg(reinterpret_cast<const uint4*>(static_cast<const char*>(row) +
                                                v * Elem<DT>::kBytes));
  uint32_t wd[4] = {Vec<DT>::kNegInf, Vec<DT>::kNegInf, Vec<DT>::kNegInf, Vec<DT>::kNegInf};
  if (DT == HS_FP32) {
#pragma unroll
    for (int q = 0; q < 4; ++q)
      if (v + q < V) wd[q] = __float_as_uint(Elem<DT>::one(row, v + q));
  } else {
    const uint16_t* h = static_cast<const uint16_t*>(row);
#pragma unroll
    for (int q = 0; q < 8; ++q)
      if (v + q < V) {
        const uint32_t bits = __ldg(h + v + q);
        wd[q / 2] = (q & 1) ? ((wd[q / 2] & 0xffffu) | (bits << 16))
                            : ((wd[q / 2] & 0xffff0000u) | bits);
      }
  }
  return make_uint4(wd[0], wd[1], wd[2], wd[3]);
}

// ---- segment B: the L best keys of a drafter range --------------------------
//
// The warp keeps the L best keys seen so far in lanes 0..L-1 (lane j holds the
// j-th best; 0: empty) and streams the range in steps of kUnroll vectors per
// lane.  Per step:
//   * packed NaN-propagating maxima give each vector's and the lane's
//     maximum; if no lane's maximum can beat the list's L-th key the step
//     costs nothing more;
//   * while the list is not full, the L-th largest lane maximum of the step
//     bounds the step's top L from below (at least L logits reach it);
//   * otherwise rounds: every lane proposes its best key above the floor and
//     below the last key it had inserted, and the proposals enter the list
//     largest first (a ballot finds the slot, a shuffle shifts the rest
//     down).  A lane whose proposal is rejected, or that had one candidate
//     only, is done with the step.
template <int DT>
__device__ __forceinline__ void topl_step(const uint4 (&cur)[kUnroll], const uint32_t (&pw)[kUnroll],
                                          float lm, int base, int lim, int L,
                                          uint64_t& key, uint64_t& tk) {
  constexpr int kN = Vec<DT>::kN;
  const int l = threadIdx.x & 31;
  uint64_t floor_key = tk;  // candidates must beat this key
  bool warm = false;
  if (tk == 0ull) {
    // list not full: the L-th largest lane maximum of this step, as a key
    // below every key of that value, bounds the step's top L from below
    uint32_t lk = (lm == lm) ? okey(lm) : 0u;
    uint32_t th = 0u;
    for (int q = 0; q < L; ++q) {
      const uint32_t mx = __reduce_max_sync(0xffffffffu, lk);
      th = mx;
      if (mx == 0u) break;
      const unsigned who = __ballot_sync(0xffffffffu, lk == mx);
      if (l == __ffs(who) - 1) lk = 0u;  // drop one lane holding it
    }
    floor_key = th == 0u ? 0ull : (uint64_t(th) << 32) - 1;
    warm = true;
  }
  // A key above the floor has a value >= the floor's value; NaN fails every
  // compare.  Below a warm-up floor a value equal to the bound enters; below
  // a key from an earlier step an equal value cannot (its index is larger),
  // so there the vector test is strict.
  const float fz0 = key_float(floor_key);
  if (!__any_sync(0xffffffffu, warm ? lm >= fz0 : lm > fz0)) return;
  uint32_t cmask = 0u;  // vectors that may hold a key above the floor
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) {
    const float vm = Vec<DT>::wfloat(pw[u]);
    if (warm ? vm >= fz0 : vm > fz0) cmask |= 1u << u;
  }
  uint64_t lub = ~0ull;  // keys this lane inserted in this step are >= lub
  while (__any_sync(0xffffffffu, cmask != 0u)) {
    const float fz = key_float(floor_key);
    uint64_t prop = 0ull;
    int cnt = 0;
    for (uint32_t m = cmask; m != 0u; m &= m - 1u) {
      const int u = __ffs(m) - 1;
      uint4 wv = cur[0];
#pragma unroll
      for (int j = 1; j < kUnroll; ++j)
        if (u == j) wv = cur[j];
      const int v0 = base + (u * 32 + l) * kN;
      uint32_t em = 0u;  // logits that pass the float prefilter
#pragma unroll
      for (int q = 0; q < kN; ++q) em |= (Vec<DT>::at(wv, q) >= fz ? 1u : 0u) << q;
      for (; em != 0u; em &= em - 1u) {
        const int q = __ffs(em) - 1;
        const uint64_t k = token_key(Vec<DT>::at_dyn(wv, q), v0 + q);
        if (v0 + q < lim && k > floor_key && k < lub) {
          ++cnt;
          if (k > prop) prop = k;
        }
      }
    }
    if (cnt <= 1) cmask = 0u;  // its only candidate is proposed now (or none)
    for (;;) {
      const uint64_t K = warp_best(prop);
      if (K <= floor_key) break;  // the rest are at or below the floor
      // insert K: lanes above its slot keep theirs, the rest shift down one
      const int slot = __popc(__ballot_sync(0xffffffffu, l < L && key > K));
      const uint64_t above = shfl_up_u64(key);
      if (l < L) key = l < slot ? key : (l == slot ? K : above);
      tk = shfl_u64(key, L - 1);
      if (tk > floor_key) floor_key = tk;
      if (prop == K) {
        lub = K;
        prop = 0ull;
      }
    }
    if (prop != 0ull) cmask = 0u;  // rejected: the lane's other keys are smaller
  }
}

// ---- segment A: a share of the target row -----------------------------------
// Packed fp32 pairs (two lanes of one 64-bit register pair): the same IEEE
// roundings as the scalar operations, two logits per instruction.
__device__ __forceinline__ uint64_t pack2(float lo, float hi) {
  uint64_t d;
  asm("mov.b64 %0, {%1, %2};" : "=l"(d) : "f"(lo), "f"(hi));
  return d;
}
__device__ __forceinline__ float lo2(uint64_t d) { return __uint_as_float(uint32_t(d)); }
__device__ __forceinline__ float hi2(uint64_t d) { return __uint_as_float(uint32_t(d >> 32)); }
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t mul2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// Per lane: running max tm (stored logit), first index of it, and the sum of
// 2^{(z - tm) c} over the lane's logits so far (rescaled when tm grows).
template <int DT>
__device__ __forceinline__ void stats_step(const uint4 (&cur)[kUnroll], float lm, int base,
                                           int greedy, float c, float& tm, float& ts,
                                           int& targ) {
  constexpr int kN = Vec<DT>::kN;
  const int l = threadIdx.x & 31;
  if (lm > tm) {  // a new running max (NaN compares false)
    ts = (tm == -INFINITY) ? 0.f : ts * ex2((tm - lm) * c);
    tm = lm;
    targ = INT_MAX;  // the lane visits its logits in increasing index order
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
#pragma unroll
      for (int q = 0; q < kN; ++q)
        if (targ == INT_MAX && Vec<DT>::at(cur[u], q) == lm)
          targ = base + (u * 32 + l) * kN + q;
  }
  if (!greedy && tm != -INFINITY) {
    // two logits at a time: (z - tm) then times c, then 2^x (-inf -> 0),
    // summed in two independent chains
    const uint64_t ntm2 = pack2(-tm, -tm), c2 = pack2(c, c);
    uint64_t sa = 0ull, sb = 0ull;
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
#pragma unroll
      for (int q = 0; q < kN; q += 2) {
        const uint64_t z2 = pack2(Vec<DT>::at(cur[u], q), Vec<DT>::at(cur[u], q + 1));
        const uint64_t e = mul2(add2(z2, ntm2), c2);
        const uint64_t x = pack2(ex2(lo2(e)), ex2(hi2(e)));
        if ((q >> 1) & 1)
          sb = add2(sb, x);
        else
          sa = add2(sa, x);
      }
    const uint64_t s2 = add2(sa, sb);
    ts += lo2(s2) + hi2(s2);
  }
}

// ---- the streaming kernel ---------------------------------------------------

template <int DT, bool TMA>
__global__ void __launch_bounds__(kThreads, 4) topl_kernel(const Params p) {
  extern __shared__ __align__(128) unsigned char smem[];
  constexpr int kN = Vec<DT>::kN;
  constexpr int kStep = 32 * kUnroll * kN;  // logits per warp step (positions fit in int: V < 2^30)
  constexpr int kEsz = Elem<DT>::kBytes;
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  pdl_wait();  // earlier kernels of the stream may still use the outputs and workspace
  if (blockIdx.x == 0 && p.e_len)
    for (int x = threadIdx.x; x < p.N * p.B; x += kThreads) p.counters[x] = 0;
  const int64_t gw = int64_t(blockIdx.x) * kWarps + w;
  const int64_t r = gw / p.S;  // drafter row (i, b, k)
  if (r >= p.nrows) return;    // whole warp
  const int part = int(gw - r * p.S);
  const int64_t BP = int64_t(p.B) * p.P;
  const int64_t tile = r % BP;
  const int i = int(r / BP);
  // segment A: share j of the N*S equal shares (whole steps) of the target row
  const int J = p.N * p.S, j = i * p.S + part;
  const int per_a = int(ceil_div(ceil_div(p.V, J), kStep) * kStep);
  const int a0 = int(int64_t(j) * per_a < p.V ? int64_t(j) * per_a : int64_t(p.V));
  const int a1 = a0 + per_a < p.V ? a0 + per_a : p.V;
  const int nA = int(ceil_div(a1 - a0, kStep));
  bool bad_path = false;
  const char* trow =
      static_cast<const char*>(target_row<DT>(p.target, p.path, p.M, p.P, tile, p.V, &bad_path));
  // segment B: part `part` of the S parts (whole steps) of the drafter row
  const int per_b = int(ceil_div(ceil_div(p.V, p.S), kStep) * kStep);
  const int e0 = int(int64_t(part) * per_b < p.V ? int64_t(part) * per_b : int64_t(p.V));
  const int lim = e0 + per_b < p.V ? e0 + per_b : p.V;
  const int nB = int(ceil_div(lim - e0, kStep));
  const char* drow = static_cast<const char*>(row_ptr<DT>(p.drafter, r, p.V));
  const int T = nA + nB;
  // step t covers logits [beg, end) of its segment's row
  auto range = [&](int t, const char*& row, int& beg, int& end) {
    if (t < nA) {
      row = trow;
      beg = a0 + t * kStep;
      end = a1;
    } else {
      row = drow;
      beg = e0 + (t - nA) * kStep;
      end = lim;
    }
  };
  const uint32_t ring = saddr(smem) + uint32_t(w) * kStages * kStageBytes;
  const uint32_t bars = saddr(smem) + uint32_t(kWarps * kStages * kStageBytes + w * kStages * 8);
  auto fill = [&](int t) {
    const char* row;
    int beg, end;
    range(t, row, beg, end);
    const int n = end - beg < kStep ? end - beg : kStep;
    bulk_fill(ring + uint32_t(t % kStages) * kStageBytes, bars + 8u * uint32_t(t % kStages),
              row + int64_t(beg) * kEsz, uint32_t(n * kEsz));
  };
  if (TMA) {
    if (l == 0) {
      for (int s = 0; s < kStages; ++s) mbar_init(bars + 8u * s);
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
      for (int t = 0; t < kStages && t < T; ++t) fill(t);
    }
    __syncwarp();
  }
  float tm = -INFINITY, ts = 0.f;  // segment A, per lane
  int targ = INT_MAX;
  bool tbad = false;
  uint64_t key = 0ull, tk = 0ull;  // segment B, see topl_step
  bool bad = false, any_finite = false;
  bool ok = true;
  int t = 0;
  for (; t < T; ++t) {
    const char* row;
    int beg, end;
    range(t, row, beg, end);
    uint4 cur[kUnroll];
    if (TMA) {
      const int s = t % kStages;
      ok = __all_sync(0xffffffffu, mbar_wait(bars + 8u * s, uint32_t(t / kStages) & 1u));
      if (!ok) break;
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int v = beg + (u * 32 + l) * kN;
        cur[u] = v < end ? lds128(ring + uint32_t(s) * kStageBytes + uint32_t(u * 32 + l) * 16u)
                         : make_uint4(Vec<DT>::kNegInf, Vec<DT>::kNegInf, Vec<DT>::kNegInf,
                                      Vec<DT>::kNegInf);
      }
    } else {
#pragma unroll
      for (int u = 0; u < kUnroll; ++u)
        cur[u] = load_vec<DT, false>(row, beg + (u * 32 + l) * kN, end);
    }
    // NaN-propagating maxima: one packed word per vector, then the lane's
    uint32_t pw[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
      pw[u] = Vec<DT>::pmax(Vec<DT>::pmax(cur[u].x, cur[u].y), Vec<DT>::pmax(cur[u].z, cur[u].w));
    uint32_t lw = pw[0];
#pragma unroll
    for (int u = 1; u < kUnroll; ++u) lw = Vec<DT>::pmax(lw, pw[u]);
    const float lm = Vec<DT>::wfloat(lw);
    if (TMA) {
      __syncwarp();  // every lane's reads of the stage are done: refill it
      if (l == 0 && t + kStages < T) fill(t + kStages);
    }
    if (t < nA) {
      tbad |= (lm != lm) || lm == INFINITY;
      stats_step<DT>(cur, lm, beg, p.greedy, p.c, tm, ts, targ);
    } else {
      bad |= (lm != lm) || lm == INFINITY;
      any_finite |= lm > -INFINITY;
      topl_step<DT>(cur, pw, lm, beg, lim, p.L, key, tk);
    }
  }
  if (TMA && !ok) {
    // a stage did not arrive in time: report, and let the copies already
    // issued (steps t .. t+kStages-1) land before the shared memory is freed
    if (l == 0) report(p.dev_status, HS_ERR_TIMEOUT);
    for (int u = t; u < t + kStages && u < T; ++u)
      (void)mbar_wait(bars + 8u * (u % kStages), uint32_t(u / kStages) & 1u);
  }
  // the share of the target row
  tbad = __any_sync(0xffffffffu, tbad);
  const float gm = warp_max_nan(tm);
  const int ga = warp_min_int(tm == gm ? targ : INT_MAX);
  float mm = tm, ss = ts;
  if (!p.greedy) merge_os(mm, ss, p.c);
  if (l == 0)
    p.stats[tile * J + j] = TStat{gm, ss, ga, (tbad || !ok ? 1 : 0) | (bad_path ? 2 : 0)};
  // the part's L best keys, and flags (bit 0: NaN, +inf or a timeout; bit 1:
  // a logit above -inf)
  bad = __any_sync(0xffffffffu, bad);
  any_finite = __any_sync(0xffffffffu, any_finite);
  uint64_t* out = p.parts + gw * kPartSlots;
  if (l < p.L) out[l] = key;
  if (l == 0) out[16] = (bad || !ok ? 1ull : 0ull) | (any_finite ? 2ull : 0ull);
}

// ---- alpha (and e_len) ------------------------------------------------------

template <int DT>
__global__ void __launch_bounds__(kThreads) alpha_kernel(const Params p) {
  pdl_wait();
  const int l = threadIdx.x & 31;
  const int64_t r = int64_t(blockIdx.x) * kWarps + (threadIdx.x >> 5);
  if (r >= p.nrows) return;  // whole warp
  const int64_t BP = int64_t(p.B) * p.P;
  const int64_t tile = r % BP;
  const int64_t ib = r / p.P;  // (i, b)
  // the target row of (b, k) from its J shares (lane q takes shares q, q+32,
  // ..., in index order): max, first argmax, and the sum relative to the max
  const int J = p.N * p.S;
  float m = -INFINITY, s = 0.f;
  int arg = INT_MAX, flags = 0;
  for (int q = l; q < J; q += 32) {
    const TStat t = p.stats[tile * J + q];
    flags |= t.flags;
    if (t.m > m) {
      s = (m == -INFINITY ? 0.f : s * ex2((m - t.m) * p.c)) + t.s;
      m = t.m;
      arg = t.argmax;
    } else if (t.m != -INFINITY) {
      s += t.s * ex2((t.m - m) * p.c);
    }
  }
  flags = int(__reduce_or_sync(0xffffffffu, unsigned(flags)));
  const float gm = warp_max_nan(m);
  const int ga = warp_min_int(m == gm ? arg : INT_MAX);
  if (!p.greedy) merge_os(m, s, p.c);  // s is now relative to gm
  // the row's L best keys: lane q holds the rank-q key
  const uint64_t* in = p.parts + r * p.S * kPartSlots;
  uint64_t key = 0ull, f = 0ull;
  if (p.S == 1) {
    key = l < p.L ? in[l] : 0ull;
    f = in[16];
  } else {
    // the parts' lists: at most 16 x 16 keys, 8 per lane
    uint64_t cand[8];
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
      const int slot = jj * 32 + l;  // (part, rank) = (slot / 16, slot % 16)
      cand[jj] = (slot / 16 < p.S && slot % 16 < p.L) ? in[(slot / 16) * kPartSlots + slot % 16]
                                                      : 0ull;
    }
    if (l < p.S) f = in[l * kPartSlots + 16];
    f = (__any_sync(0xffffffffu, f & 1ull) ? 1ull : 0ull) |
        (__any_sync(0xffffffffu, f & 2ull) ? 2ull : 0ull);
    for (int q = 0; q < p.L; ++q) {
      uint64_t lb = 0ull;
#pragma unroll
      for (int jj = 0; jj < 8; ++jj) lb = cand[jj] > lb ? cand[jj] : lb;
      const uint64_t best = warp_best(lb);
      if (best == 0ull) break;  // fewer than L tokens in the row
#pragma unroll
      for (int jj = 0; jj < 8; ++jj)
        if (cand[jj] == best) cand[jj] = 0ull;
      if (l == q) key = best;
    }
  }
  // the candidate set: the first `kept` of the row's L ranked keys (Thm 2's
  // remark on pruning: a pruned node keeps a prefix of its children)
  int kept = p.L;
  bool keep_bad = false;
  if (p.keep) {
    kept = __ldg(p.keep + r);
    keep_bad = kept < 0 || kept > p.L;
  }
  const bool target_ok =
      flags == 0 && gm != -INFINITY && (p.greedy || (isfinite(s) && s > 0.f));
  const bool ok = !(f & 1ull) && (f & 2ull) && target_ok && !keep_bad;
  const int mine = (l < kept && key != 0ull) ? int(0xffffffffu - uint32_t(key)) : -1;
  float a = 0.f;
  if (ok && mine >= 0) {
    if (p.greedy) {
      a = mine == ga ? 1.f : 0.f;
    } else {
      bool unused = false;
      const void* trow = target_row<DT>(p.target, p.path, p.M, p.P, tile, p.V, &unused);
      a = ex2((Elem<DT>::one(trow, mine) - gm) * p.c) / s;
    }
  }
  a = warp_sum(a);
  int last = 0;
  if (l == 0) {
    if (!ok) {
      a = __int_as_float(0x7fc00000);
      report(p.dev_status, (keep_bad || (flags & 2)) ? HS_ERR_INVALID_ARG : HS_ERR_NONFINITE);
    }
    p.alpha[r] = a;
    if (p.e_len) {
      __threadfence();  // alpha[r] before the count
      last = atomicAdd(&p.counters[ib], 1) == p.P - 1;
    }
  }
  // the last of the P warps of (i, b) forms e_len = 1 + sum_k prod_{j<=k} alpha_j
  // over k < P-1 (Thm 3)
  if (__shfl_sync(0xffffffffu, last, 0) && l == 0) {
    __threadfence();
    float e = 1.f, prod = 1.f;
    for (int k = 0; k < p.P - 1; ++k) {
      prod *= __ldcg(p.alpha + ib * p.P + k);
      e += prod;
    }
    p.e_len[ib] = e;
  }
}

// Warps per row: enough that the GPU holds about kWarpTarget warps when rows
// are few (at most 16, and never more parts than whole steps in the row).
constexpr int64_t kFewRows = 1216;     // below this many rows a row is split
constexpr int64_t kWarpTarget = 4864;  // 152 SMs x 32 warps
int split_of(int64_t rows, int V) {
  if (rows > kFewRows) return 1;  // splitting adds insertions; only for few rows
  int64_t S = (kWarpTarget + rows - 1) / rows;
  const int64_t steps = (int64_t(V) + 32 * kUnroll * 8 - 1) / (32 * kUnroll * 8);
  if (S > steps) S = steps;
  if (S > 16) S = 16;
  return S < 1 ? 1 : int(S);
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }
size_t stats_bytes(int N, int B, int P, int S) {
  return align256(size_t(B) * P * N * S * sizeof(TStat));
}
size_t parts_bytes(int N, int B, int P, int S) {
  return align256(size_t(N) * B * P * S * kPartSlots * sizeof(uint64_t));
}

template <int DT, bool TMA>
hs_status launch_t(const Params& p, cudaStream_t s) {
  const size_t smem = TMA ? ring_smem() : 0;
  if (TMA && cudaFuncSetAttribute(topl_kernel<DT, TMA>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  int(smem)) != cudaSuccess)
    return HS_ERR_CUDA;
  const int64_t warps = p.nrows * p.S;
  if (launch_pdl(topl_kernel<DT, TMA>, dim3(unsigned((warps + kWarps - 1) / kWarps)),
                 dim3(kThreads), smem, s, p) != cudaSuccess)
    return HS_ERR_CUDA;
  if (launch_pdl(alpha_kernel<DT>, dim3(unsigned((p.nrows + kWarps - 1) / kWarps)),
                 dim3(kThreads), 0, s, p) != cudaSuccess)
    return HS_ERR_CUDA;
  return HS_OK;
}

template <int DT>
hs_status launch_dt(bool vec, const Params& p, cudaStream_t s) {
  return vec ? launch_t<DT, true>(p, s) : launch_t<DT, false>(p, s);
}

}  // namespace

int kernel_count(int, int, int, int) { return 2; }

size_t workspace_bytes(int N, int B, int P, int V) {
  const int S = split_of(int64_t(N) * B * P, V);
  return stats_bytes(N, B, P, S) + parts_bytes(N, B, P, S) + size_t(N) * B * sizeof(int);
}

hs_status launch(const void* target, const int32_t* path, int M, const void* drafter, int dtype,
                 int N, int B, int P, int V, int L, const int32_t* keep, int greedy, float c,
                 float* alpha, float* e_len, void* ws, int* dev_status, cudaStream_t stream) {
  const int esz = dtype == HS_FP32 ? 4 : 2;
  const bool vec = (int64_t(V) * esz) % 16 == 0 && reinterpret_cast<uintptr_t>(target) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(drafter) % 16 == 0;
  Params p;
  p.target = target;
  p.path = path;
  p.drafter = drafter;
  p.nrows = int64_t(N) * B * P;
  p.M = M;
  p.N = N;
  p.B = B;
  p.P = P;
  p.V = V;
  p.L = L;
  p.keep = keep;
  p.S = split_of(p.nrows, V);
  p.greedy = greedy;
  p.c = c;
  char* w = static_cast<char*>(ws);
  p.stats = reinterpret_cast<TStat*>(w);
  p.parts = reinterpret_cast<uint64_t*>(w + stats_bytes(N, B, P, p.S));
  p.counters = reinterpret_cast<int*>(w + stats_bytes(N, B, P, p.S) + parts_bytes(N, B, P, p.S));
  p.alpha = alpha;
  p.e_len = e_len;
  p.dev_status = dev_status;
  switch (dtype) {
    case HS_BF16:
      return launch_dt<HS_BF16>(vec, p, stream);
    case HS_FP16:
      return launch_dt<HS_FP16>(vec, p, stream);
    default:
      return launch_dt<HS_FP32>(vec, p, stream);
  }
}

}  // namespace topl
}  // namespace hs
