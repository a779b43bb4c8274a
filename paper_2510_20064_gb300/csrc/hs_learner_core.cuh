// hs_learner_core.cuh -- one learner round for one query, by one warp (lane
// i = drafter i, N <= 32): Hedge (App. B.1 remark) or NormalHedge (App. D.6
// figure, steps 2-5).  Shared by the learner kernels (hs_learner.cu) and the
// delayed-feedback kernels (hs_delayed.cu).
//
// NormalHedge's scale is found by a warp-parallel bisection: with x_i =
// [R_i]_+ / max R and kappa = (max R)^2 / (2c), the scale equation becomes
// g(kappa) = (1/N) sum_i exp(kappa x_i^2) - e = 0 with g increasing and the
// root in [1, 1 + ln N] (g(1) <= 0 since every term is <= e; g(1 + ln N) >= 0
// since the x = 1 term alone is N e).  Each round the 32 lanes evaluate g at
// 32 interior points of the bracket and keep the sub-interval where g changes
// sign, shrinking it 33-fold; 6 rounds take it below fp32 resolution.  The
// terms exp(kappa x_j^2) of g are formed as 2^{kappa y_j}, y_j = x_j^2 log2(e),
// with the hardware exp2 (about 2^-22 relative), and the drafters beyond N
// carry y = -inf, so they add exact zeros and the sums run over whole groups
// of 8 lanes.  Then p_i is proportional to x_i exp(kappa x_i^2), which equals
// ([R_i]_+/c) exp([R_i]_+^2 / 2c) up to the common factor.
#pragma once

#include <math.h>
#include <stdint.h>

#include "hs_common.cuh"

namespace hs {
namespace learner {

constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(kFull, v, o));
  return v;
}

__device__ __forceinline__ float warp_min(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(kFull, v, o));
  return v;
}

// One round for the calling warp's query.  Lane i < N holds drafter i:
//   f      its loss this round (ignored by Hedge when add_loss is false);
//   state  Hedge: cumulative loss L (L += f when add_loss);
//          NormalHedge: regret R (R += sum_j p_j (f_j - f_i));
//   p      NormalHedge: p_t in; both: the normalised weights out;
// returns the choice: Hedge the first argmin of L; NormalHedge the first
// argmax of R when max R > 0, else 0 (uniform weights).
__device__ __forceinline__ int round(int learner, int N, float eta, float f, bool add_loss,
                                     float& state, float& p) {
  const int lane = threadIdx.x & 31;
  const bool act = lane < N;
  float w;
  int sel;
  if (learner == HS_HEDGE) {
    // ---- Hedge: w = exp(-eta (L - min L)) / Z, choice = first argmin L ----
    float L = act ? state : 0.f;
    if (add_loss) L += f;
    state = L;
    const float Lmin = warp_min(act ? L : INFINITY);
    const unsigned tie = __ballot_sync(kFull, act && L == Lmin);
    sel = tie ? __ffs(tie) - 1 : 0;
    w = act ? expf(-eta * (L - Lmin)) : 0.f;
  } else {
    // ---- NormalHedge steps 2-3: R_i += sum_j p_j (l_j - l_i) ----
    // (lanes >= N hold p = 0 and f = 0, so their terms are exact zeros)
    const float pi = act ? p : 0.f;
    const float fi = act ? f : 0.f;
    float inc = 0.f;
    for (int j0 = 0; j0 < N; j0 += 8) {
#pragma unroll
      for (int jj = 0; jj < 8; ++jj) {
        const float pj = __shfl_sync(kFull, pi, j0 + jj);
        const float fj = __shfl_sync(kFull, fi, j0 + jj);
        inc = fmaf(pj, fj - fi, inc);
      }
    }
    const float R = act ? state + inc : -INFINITY;
    state = R;
    const float Rmax = warp_max(R);
    if (!(Rmax > 0.f)) {
      // no positive regret: the scale equation has no root, p is uniform
      w = act ? 1.f : 0.f;
      sel = 0;
    } else {
      // ---- step 4 by warp-parallel bisection on kappa (see file header) ----
      const float x = act ? fmaxf(R, 0.f) / Rmax : 0.f;
      const float x2 = x * x;
      const float y = act ? x2 * kLog2e : -INFINITY;
      float lo = 1.f, hi = 1.f + logf(float(N));
      const float e1 = 2.71828182845904523536f;
      for (int r = 0; r < 6; ++r) {
        const float kap = lo + (hi - lo) * float(lane + 1) * (1.f / 33.f);
        float g = 0.f;
        for (int j0 = 0; j0 < N; j0 += 8) {
#pragma unroll
          for (int jj = 0; jj < 8; ++jj) g += ex2(kap * __shfl_sync(kFull, y, j0 + jj));
        }
        const unsigned up = __ballot_sync(kFull, g >= e1 * float(N));
        const int first = up ? __ffs(up) - 1 : 32;  // first point with g >= 0
        const float klo = __shfl_sync(kFull, kap, first > 0 ? first - 1 : 0);
        const float khi = __shfl_sync(kFull, kap, first < 32 ? first : 31);
        if (first > 0) lo = klo;
        if (first < 32) hi = khi;
      }
      const float kap = 0.5f * (lo + hi);
      // ---- step 5: p_i proportional to x_i exp(kappa x_i^2) ----
      w = act ? x * expf(kap * x2) : 0.f;
      const unsigned top = __ballot_sync(kFull, act && R == Rmax);
      sel = top ? __ffs(top) - 1 : 0;
    }
  }
  float z = w;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(kFull, z, o);
  p = w / z;
  return sel;
}

}  // namespace learner
}  // namespace hs
