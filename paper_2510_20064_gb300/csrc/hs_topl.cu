// hs_topl.cu -- feedback for an EAGLE draft tree with branching L (Thm 2):
// the target's token is accepted at a draft step iff it is among the L
// children the drafter proposes, its top-L tokens.  Stochastic target:
//   alpha[i,b,k] = sum_{v in Top_L(q_i)} p(v),   p = softmax(z_target / T);
// greedy target: alpha = 1[argmax p in Top_L(q_i)].  e_len by Thm 3.
//
//   target_stats_kernel  C CTAs per target row, each over a contiguous range:
//                        NaN-propagating max, first argmax, and
//                        sum_v 2^{z_v c - m c} in one pass (chunk-wise
//                        rescaling), c = log2(e) / T
//   topl_kernel          one warp per drafter row (or per part of a row, when
//                        rows are few): the warp keeps the row's L best
//                        (logit, -index) keys spread over its lanes, and a
//                        lane looks at its logits one by one only in vectors
//                        whose maximum can enter; then it combines the
//                        target row's C partials and sums p over those tokens
//   merge_kernel         rows split over S warps: the row's L best of the
//                        parts' lists, then the same sum
//   elen_kernel          prefix products of alpha_1..alpha_K
// The statistics kernel releases its dependent launch at once, so the top-L
// stream runs beside it; a warp waits for the statistics only once its row
// is done.
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

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 4;

struct TStat {  // one target row's range [part * per, (part + 1) * per)
  float m;      // max (stored logit) of the range
  float s;      // sum over the range of 2^{(z_v - m) c}
  int argmax;   // first index of the max (INT_MAX: none)
  int flags;    // bit 0: NaN or +inf in the range; bit 1: bad path node
};

template <int DT>
__host__ __device__ constexpr int64_t chunk_of() {
  return int64_t(kThreads) * kUnroll * Elem<DT>::kVec;
}

// Order-preserving unsigned key of a non-NaN float (-inf lowest, +inf highest).
__device__ __forceinline__ uint32_t okey(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
// The float of an order key (the inverse of okey).
__device__ __forceinline__ float ofloat(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
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

template <int DT, bool VEC>
__global__ void __launch_bounds__(kThreads) target_stats_kernel(
    const void* __restrict__ target, const int32_t* __restrict__ path, int M, int P, int V,
    int cpp, float c, TStat* __restrict__ stats) {
  pdl_wait();
  pdl_trigger();  // the top-L stream does not read these until its rows are done
  constexpr int kS = kUnroll * Elem<DT>::kVec;
  __shared__ float sm_m[kWarps], sm_s[kWarps];
  __shared__ int sm_a[kWarps];
  const int64_t tile = blockIdx.x;
  bool bad_path = false;
  const void* row = target_row<DT>(target, path, M, P, tile, V, &bad_path);
  float m = -INFINITY, s = 0.f;  // running max (stored logit) and sum relative to it
  int arg = INT_MAX;
  bool bad = false;
  const int64_t e0 = int64_t(blockIdx.y) * cpp * chunk_of<DT>();
  const int64_t e1 = e0 + int64_t(cpp) * chunk_of<DT>() < V ? e0 + int64_t(cpp) * chunk_of<DT>()
                                                            : int64_t(V);
  for (int64_t v0 = e0; v0 < e1; v0 += chunk_of<DT>()) {
    float x[kS];
    load_chunk<DT, VEC, kThreads, kUnroll>(row, v0, V, x);
    float cm = x[0];
#pragma unroll
    for (int q = 1; q < kS; ++q) cm = max_nan(cm, x[q]);
    bad |= (cm != cm) || cm == INFINITY;
    if (cm > m) {
      // a new running max: rescale the sum and take the first slot holding
      // it (slots visit increasing v, and an equal max in a later chunk
      // keeps the earlier index)
      s = (m == -INFINITY) ? 0.f : s * ex2((m - cm) * c);
      m = cm;
      arg = INT_MAX;
#pragma unroll
      for (int q = 0; q < kS; ++q) {
        const int64_t v = slot_pos<DT, VEC, kThreads>(v0, q, threadIdx.x);
        if (v < V && x[q] == cm && arg == INT_MAX) arg = int(v);
      }
    }
    if (m != -INFINITY) {
#pragma unroll
      for (int q = 0; q < kS; ++q) s += ex2((x[q] - m) * c);  // -inf past the row -> 0
    }
  }
  // the first index of the thread's max must be the first over all its chunks
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  const float wmax = warp_max_nan(m);
  const int warg = warp_min_int(m == wmax ? arg : INT_MAX);
  float mm = m, ss = s;
  merge_os(mm, ss, c);
  const bool any_bad = __syncthreads_or(bad);
  if (l == 0) {
    sm_m[w] = wmax;
    sm_s[w] = ss;
    sm_a[w] = warg;
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    float bm = l < kWarps ? sm_m[l] : -INFINITY;
    float bs = l < kWarps ? sm_s[l] : 0.f;
    int ba = l < kWarps ? sm_a[l] : INT_MAX;
    const float gm = warp_max_nan(bm);
    const int ga = warp_min_int(bm == gm ? ba : INT_MAX);
    merge_os(bm, bs, c);
    if (l == 0)
      stats[tile * gridDim.y + blockIdx.y] =
          TStat{gm, bs, ga, (any_bad ? 1 : 0) | (bad_path ? 2 : 0)};
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
__device__ __forceinline__ uint64_t token_key(float z, int64_t v) {
  return (uint64_t(okey(z)) << 32) | (0xffffffffu - uint32_t(v));
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

// One warp per drafter row (kWarps rows per CTA).  The warp keeps the L
// best keys of the row seen so far spread over lanes 0..L-1 (lane j holds
// the j-th best) and streams the row in steps of kUnroll vectors per lane,
// loading the next step before working on the current one.  A lane decodes
// a vector only when its maximum (packed max on the stored halves) can beat
// the warp's L-th key; those keys enter the list one at a time, largest
// first (warp-wide insertion: a ballot finds the slot, a shuffle shifts the
// rest down).  In the first step, while the list is not yet full, the L-th
// largest of the lanes' maxima bounds the candidates from below (at least L
// logits of the step reach it).  The warp then sums the target's p over
// the row's top L.
// The row's L best keys and its validity -> alpha (lanes q < L hold the
// rank-q key; 0 past the row's size).
// The target row's statistics from its C range partials (lanes 0..C-1, in
// range order): max, first argmax, and the sum relative to the max.
template <int DT>
__device__ __forceinline__ void alpha_of(uint64_t key, bool bad, bool any_finite, int L,
                                         const void* target, const int32_t* path, int M, int B,
                                         int P, int V, int greedy, float c, int C, int64_t r,
                                         const TStat* __restrict__ stats, float* alpha,
                                         int* dev_status) {
  const int l = threadIdx.x & 31;
  const int64_t tile = r % (int64_t(B) * P);
  const int mine = (l < L && key != 0ull) ? int(0xffffffffu - uint32_t(key)) : -1;
  const TStat ts = l < C ? stats[tile * C + l] : TStat{-INFINITY, 0.f, INT_MAX, 0};
  const int flags = int(__reduce_or_sync(0xffffffffu, unsigned(ts.flags)));
  const float gm = warp_max_nan(ts.m);
  const int ga = warp_min_int(ts.m == gm ? ts.argmax : INT_MAX);
  float mm = ts.m, ss = ts.s;
  if (!greedy) merge_os(mm, ss, c);
  const bool target_ok = flags == 0 && gm != -INFINITY && (greedy || (isfinite(ss) && ss > 0.f));
  const bool ok = !bad && any_finite && target_ok;
  float a = 0.f;
  if (ok && mine >= 0) {
    if (greedy) {
      a = mine == ga ? 1.f : 0.f;
    } else {
      bool unused = false;
      const void* trow = target_row<DT>(target, path, M, P, tile, V, &unused);
      a = ex2((Elem<DT>::one(trow, mine) - gm) * c) / ss;
    }
  }
  a = warp_sum(a);
  if (l == 0) {
    if (!ok) {
      a = __int_as_float(0x7fc00000);
      report(dev_status, (flags & 2) ? HS_ERR_INVALID_ARG : HS_ERR_NONFINITE);
    }
    alpha[r] = a;
  }
}

// Per-part output of a row split over S warps: the part's L best keys, and
// flags (bit 0: NaN or +inf seen, bit 1: a finite logit seen) in key slot 16.
constexpr int kPartSlots = 17;

template <int DT, bool VEC>
__global__ void __launch_bounds__(kThreads) topl_kernel(
    const void* __restrict__ target, const int32_t* __restrict__ path, int M,
    const void* __restrict__ drafter, int64_t nrows, int S, int B, int P, int V, int L,
    int greedy, float c, int C, const TStat* __restrict__ stats, uint64_t* __restrict__ parts,
    float* __restrict__ alpha, int* dev_status) {
  // no wait here: the drafter rows are inputs, and the statistics are read
  // only after the wait below
  constexpr int kN = Vec<DT>::kN;
  constexpr int64_t kWarpStep = int64_t(32) * kUnroll * kN;
  const int l = threadIdx.x & 31;
  const int64_t gw = int64_t(blockIdx.x) * kWarps + (threadIdx.x >> 5);
  const int64_t r = gw / S;  // drafter row (i, b, k)
  const int part = int(gw - r * S);
  if (r >= nrows) return;  // whole warp
  const void* row = row_ptr<DT>(drafter, r, V);
  // this warp's part of the row: [e0, lim), whole warp steps except the last
  const int64_t per = ((int64_t(V) + S - 1) / S + kWarpStep - 1) / kWarpStep * kWarpStep;
  const int64_t e0 = int64_t(part) * per;
  const int lim = int(e0 + per < V ? e0 + per : V);
  uint64_t key = 0ull;  // lane j < L: the j-th best key so far (0: empty)
  uint64_t tk = 0ull;   // the L-th best key (0 until L keys are in)
  bool bad = false, any_finite = false;
  uint4 cur[kUnroll], nxt[kUnroll];
#pragma unroll
  for (int u = 0; u < kUnroll; ++u)
    cur[u] = load_vec<DT, VEC>(row, e0 + int64_t(u * 32 + l) * kN, lim);
  for (int64_t base = e0; base < lim; base += kWarpStep) {
    if (base + kWarpStep < lim) {
#pragma unroll
      for (int u = 0; u < kUnroll; ++u)
        nxt[u] = load_vec<DT, VEC>(row, base + kWarpStep + int64_t(u * 32 + l) * kN, lim);
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
    bad |= (lm != lm) || lm == INFINITY;
    any_finite |= lm > -INFINITY;
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
    // The floor's value as a float (order keys up to okey(-inf) = 0x007fffff
    // stand for -inf; the ones below it are NaN patterns).  A key above the
    // floor has a value >= it; NaN fails every compare.  Below a warm-up
    // floor a value equal to the bound enters; below a key from an earlier
    // step an equal value cannot (its index is larger), so there the
    // vector test is strict.
    const uint32_t fh0 = uint32_t(floor_key >> 32);
    const float fz0 = fh0 <= 0x007fffffu ? -INFINITY : ofloat(fh0);
    if (__any_sync(0xffffffffu, warm ? lm >= fz0 : lm > fz0)) {
      uint32_t cmask = 0u;  // vectors that may hold a key above the floor
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const float vm = Vec<DT>::wfloat(pw[u]);
        if (warm ? vm >= fz0 : vm > fz0) cmask |= 1u << u;
      }
      // Each round, every lane proposes its best key above the floor and
      // below the last key it had inserted (lub); the proposals enter the
      // list largest first.  A lane whose proposal is rejected, or that had
      // no second candidate, is done with this step.
      uint64_t lub = ~0ull;
      while (__any_sync(0xffffffffu, cmask != 0u)) {
        const uint32_t fh = uint32_t(floor_key >> 32);
        const float fz = fh <= 0x007fffffu ? -INFINITY : ofloat(fh);
        uint64_t prop = 0ull;
        int cnt = 0;
        for (uint32_t m = cmask; m != 0u; m &= m - 1u) {
          const int u = __ffs(m) - 1;
          uint4 wv = cur[0];
#pragma unroll
          for (int j = 1; j < kUnroll; ++j)
            if (u == j) wv = cur[j];
          const int64_t v0 = base + int64_t(u * 32 + l) * kN;
          uint32_t em = 0u;
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
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) cur[u] = nxt[u];
  }
  bad = __any_sync(0xffffffffu, bad);
  any_finite = __any_sync(0xffffffffu, any_finite);
  pdl_wait();  // the statistics kernel (and with it every earlier one) is done
  if (S == 1) {
    alpha_of<DT>(key, bad, any_finite, L, target, path, M, B, P, V, greedy, c, C, r, stats,
                 alpha, dev_status);
    return;
  }
  uint64_t* out = parts + gw * kPartSlots;
  if (l < L) out[l] = key;
  if (l == 0) out[16] = (bad ? 1ull : 0ull) | (any_finite ? 2ull : 0ull);
}

// Rows split over S warps: one warp per row merges the parts' L best keys
// (at most 16 x 16, up to 8 per lane) into the row's L best, then alpha.
template <int DT>
__global__ void __launch_bounds__(kThreads) merge_kernel(
    const void* __restrict__ target, const int32_t* __restrict__ path, int M, int64_t nrows,
    int S, int B, int P, int V, int L, int greedy, float c, int C,
    const TStat* __restrict__ stats, const uint64_t* __restrict__ parts,
    float* __restrict__ alpha, int* dev_status) {
  pdl_wait();
  const int l = threadIdx.x & 31;
  const int64_t r = int64_t(blockIdx.x) * kWarps + (threadIdx.x >> 5);
  if (r >= nrows) return;  // whole warp
  const uint64_t* in = parts + r * S * kPartSlots;
  uint64_t cand[8];
  bool bad = false, any_finite = false;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int slot = j * 32 + l;  // (part, rank) = (slot / 16, slot % 16)
    cand[j] = (slot / 16 < S && slot % 16 < L) ? in[(slot / 16) * kPartSlots + slot % 16] : 0ull;
  }
  if (l < S) {
    const uint64_t f = in[l * kPartSlots + 16];
    bad = f & 1ull;
    any_finite = (f & 2ull) != 0ull;
  }
  bad = __any_sync(0xffffffffu, bad);
  any_finite = __any_sync(0xffffffffu, any_finite);
  uint64_t key = 0ull;  // lane q: the row's rank-q key
  for (int q = 0; q < L; ++q) {
    uint64_t lb = 0ull;
#pragma unroll
    for (int j = 0; j < 8; ++j) lb = cand[j] > lb ? cand[j] : lb;
    const uint64_t best = warp_best(lb);
    if (best == 0ull) break;  // fewer than L tokens in the row
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (cand[j] == best) cand[j] = 0ull;
    if (l == q) key = best;
  }
  alpha_of<DT>(key, bad, any_finite, L, target, path, M, B, P, V, greedy, c, C, r, stats, alpha,
               dev_status);
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

// Warps per row: enough that the GPU holds about kWarpTarget rows-in-flight
// of streaming warps when rows are few (at most 16, and never more parts
// than whole warp steps in the row).
constexpr int64_t kWarpTarget = 2432;  // 152 SMs x 16 warps
int split_of(int64_t rows, int V) {
  if (2 * rows > kWarpTarget) return 1;  // splitting adds insertions; only for few rows
  int64_t S = (kWarpTarget + rows - 1) / rows;
  const int64_t steps = (int64_t(V) + 32 * kUnroll * 8 - 1) / (32 * kUnroll * 8);
  if (S > steps) S = steps;
  if (S > 16) S = 16;
  return S < 1 ? 1 : int(S);
}
// Target statistics: C ranges of cpp chunks per row, about 4 chunks each.
int stat_cpp(int V) {
  const int64_t nchunk = (int64_t(V) + chunk_of<HS_FP32>() - 1) / chunk_of<HS_FP32>();
  const int64_t C = (nchunk + 3) / 4 < 16 ? (nchunk + 3) / 4 : 16;
  return int((nchunk + C - 1) / C);
}
template <int DT>
int stat_parts(int V) {
  const int64_t span = int64_t(stat_cpp(V)) * chunk_of<DT>();
  return int((V + span - 1) / span);
}
int stat_parts_max(int V) { return stat_parts<HS_FP32>(V); }  // the most ranges of any dtype
size_t parts_offset(int B, int P, int V) {
  return (size_t(B) * P * stat_parts_max(V) * sizeof(TStat) + 255) & ~size_t(255);
}

template <int DT, bool VEC>
hs_status launch_t(const void* target, const int32_t* path, int M, const void* drafter, int N,
                   int B, int P, int V, int L, int greedy, float c, float* alpha, float* e_len,
                   void* ws, int* dev_status, cudaStream_t s) {
  TStat* stats = static_cast<TStat*>(ws);
  const unsigned tiles = unsigned(int64_t(B) * P);
  const int C = stat_parts<DT>(V);
  if (launch_pdl(target_stats_kernel<DT, VEC>, dim3(tiles, unsigned(C)), dim3(kThreads), 0, s,
                 target, path, M, P, V, stat_cpp(V), c, stats) != cudaSuccess)
    return HS_ERR_CUDA;
  const int64_t rows = int64_t(N) * B * P;
  const int S = split_of(rows, V);
  uint64_t* parts = reinterpret_cast<uint64_t*>(static_cast<char*>(ws) + parts_offset(B, P, V));
  const int64_t warps = rows * S;
  if (launch_pdl(topl_kernel<DT, VEC>, dim3(unsigned((warps + kWarps - 1) / kWarps)),
                 dim3(kThreads), 0, s, target, path, M, drafter, rows, S, B, P, V, L, greedy, c,
                 C, stats, parts, alpha, dev_status) != cudaSuccess)
    return HS_ERR_CUDA;
  if (S > 1 &&
      launch_pdl(merge_kernel<DT>, dim3(unsigned((rows + kWarps - 1) / kWarps)), dim3(kThreads),
                 0, s, target, path, M, rows, S, B, P, V, L, greedy, c, C, stats, parts, alpha,
                 dev_status) != cudaSuccess)
    return HS_ERR_CUDA;
  if (e_len) {
    const int64_t nb = int64_t(N) * B;
    if (launch_pdl(elen_kernel, dim3(unsigned((nb + 255) / 256)), dim3(256), 0, s, alpha, nb, P,
                   e_len) != cudaSuccess)
      return HS_ERR_CUDA;
  }
  return HS_OK;
}

template <int DT>
hs_status launch_dt(bool vec, const void* target, const int32_t* path, int M,
                    const void* drafter, int N, int B, int P, int V, int L, int greedy, float c,
                    float* alpha, float* e_len, void* ws, int* dev_status, cudaStream_t s) {
  if (vec)
    return launch_t<DT, true>(target, path, M, drafter, N, B, P, V, L, greedy, c, alpha, e_len,
                              ws, dev_status, s);
  return launch_t<DT, false>(target, path, M, drafter, N, B, P, V, L, greedy, c, alpha, e_len,
                             ws, dev_status, s);
}

}  // namespace

int kernel_count(int N, int B, int P, int V) {
  return split_of(int64_t(N) * B * P, V) > 1 ? 4 : 3;
}

size_t workspace_bytes(int N, int B, int P, int V) {
  const int64_t rows = int64_t(N) * B * P;
  const int S = split_of(rows, V);
  return parts_offset(B, P, V) +
         (S > 1 ? size_t(rows) * S * kPartSlots * sizeof(uint64_t) : 0);
}

hs_status launch(const void* target, const int32_t* path, int M, const void* drafter, int dtype,
                 int N, int B, int P, int V, int L, int greedy, float c, float* alpha,
                 float* e_len, void* ws, int* dev_status, cudaStream_t stream) {
  const int esz = dtype == HS_FP32 ? 4 : 2;
  const bool vec = (int64_t(V) * esz) % 16 == 0 && reinterpret_cast<uintptr_t>(target) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(drafter) % 16 == 0;
  switch (dtype) {
    case HS_BF16:
      return launch_dt<HS_BF16>(vec, target, path, M, drafter, N, B, P, V, L, greedy, c, alpha,
                                e_len, ws, dev_status, stream);
    case HS_FP16:
      return launch_dt<HS_FP16>(vec, target, path, M, drafter, N, B, P, V, L, greedy, c, alpha,
                                e_len, ws, dev_status, stream);
    default:
      return launch_dt<HS_FP32>(vec, target, path, M, drafter, N, B, P, V, L, greedy, c, alpha,
                                e_len, ws, dev_status, stream);
  }
}

}  // namespace topl
}  // namespace hs
