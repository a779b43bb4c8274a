// hs_learner.cu -- loss (Sec. 3.3), Hedge (App. B.1 remark) and NormalHedge
// (App. D.6 figure) for B independent queries: one warp per query, lane i =
// drafter i (N <= 32); the round itself is hs_learner_core.cuh.
#include <math.h>
#include <stdint.h>

#include "hs_common.cuh"
#include "hs_learner_core.cuh"

namespace hs {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kWarpsPerBlock = 4;

enum LossSrc { kLossGiven = 0, kLossLength = 1, kLossAccept = 2, kLossNone = 3 };

struct LearnerArgs {
  const float* alpha;    // [N,B,P]
  const float* e_len;    // [N,B]
  const float* loss_in;  // [N,B]
  int loss_src;
  int N, B, P;
  int learner;  // HS_HEDGE / HS_NORMALHEDGE
  float eta;
  const float* state_in;  // Hedge: L, NormalHedge: R
  float* state_out;       // may alias state_in, or NULL
  int hedge_add_loss;     // Hedge: L += f before the weights
  const float* p_in;      // NormalHedge: p_t
  float* weights_out;     // [N,B]
  float* loss_out;        // [N,B] or NULL
  const int32_t* sel_in;  // [B] or NULL: drafter played this round
  int32_t* sel_out;       // [B]
  float* played;          // [B] or NULL: += f[sel_in]
};

__global__ void __launch_bounds__(kWarpsPerBlock * 32) learner_kernel(LearnerArgs a) {
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int64_t b = int64_t(blockIdx.x) * kWarpsPerBlock + (threadIdx.x >> 5);
  if (b >= a.B) return;  // whole warp leaves together
  const int N = a.N;
  const bool act = lane < N;
  const int64_t ib = int64_t(lane) * a.B + b;

  // ---- loss of this round (Sec. 3.3; chunk form of App. B.3) ----
  float f = 0.f;
  if (act) {
    if (a.loss_src == kLossGiven) {
      f = a.loss_in[ib];
    } else if (a.loss_src == kLossLength) {
      f = 1.f - a.e_len[ib] / float(a.P);  // 1 - E / (K+1)
    } else if (a.loss_src == kLossAccept) {
      const int K = a.P - 1;
      const float* al = a.alpha + ib * a.P;
      float s = 0.f;
      for (int k = 0; k < K; ++k) s += 1.f - al[k];
      f = s / float(K);
    }
    if (a.loss_out) a.loss_out[ib] = f;
  }
  if (a.played) {
    const int s = a.sel_in ? a.sel_in[b] : 0;
    const bool ok = s >= 0 && s < N;
    const float fs = __shfl_sync(kFull, f, ok ? s : 0);
    if (lane == 0) a.played[b] += ok ? fs : __int_as_float(0x7fc00000);
  }

  float state = act ? a.state_in[ib] : 0.f;
  float p = (act && a.learner == HS_NORMALHEDGE) ? a.p_in[ib] : 0.f;
  const int sel = learner::round(a.learner, N, a.eta, f, a.hedge_add_loss != 0, state, p);
  if (act && a.state_out) a.state_out[ib] = state;
  if (act) a.weights_out[ib] = p;
  if (lane == 0) a.sel_out[b] = sel;
}

bool aligned4(const void* p) { return reinterpret_cast<uintptr_t>(p) % 4 == 0; }

hs_status launch(const LearnerArgs& a, void* stream) {
  const unsigned blocks = unsigned((int64_t(a.B) + kWarpsPerBlock - 1) / kWarpsPerBlock);
  if (launch_pdl(learner_kernel, dim3(blocks), dim3(kWarpsPerBlock * 32), 0,
                 static_cast<cudaStream_t>(stream), a) != cudaSuccess)
    return HS_ERR_CUDA;
  return cudaGetLastError() == cudaSuccess ? HS_OK : HS_ERR_CUDA;
}

hs_status check_nb(int N, int B) {
  if (N < 1 || B < 1) return HS_ERR_INVALID_ARG;
  if (N > HS_MAX_LEARNER_N) return HS_ERR_UNSUPPORTED;
  if (int64_t(N) * B >= (int64_t(1) << 31)) return HS_ERR_INVALID_ARG;
  return HS_OK;
}

}  // namespace
}  // namespace hs

extern "C" hs_status hs_hedge_update(const float* cum_loss, int N, int B, float eta,
                                     float* weights, int32_t* selected, void* stream) {
  hs_status st = hs::check_nb(N, B);
  if (st != HS_OK) return st;
  if (!cum_loss || !weights || !selected || !(isfinite(eta) && eta >= 0.f))
    return HS_ERR_INVALID_ARG;
  if (!hs::aligned4(cum_loss) || !hs::aligned4(weights) || !hs::aligned4(selected))
    return HS_ERR_MISALIGNED;
  hs::LearnerArgs a = {};
  a.loss_src = hs::kLossNone;
  a.N = N; a.B = B; a.P = 1;
  a.learner = HS_HEDGE;
  a.eta = eta;
  a.state_in = cum_loss;
  a.weights_out = weights;
  a.sel_out = selected;
  return hs::launch(a, stream);
}

extern "C" hs_status hs_normalhedge_update(float* regret, const float* loss, float* weights, int N,
                                           int B, int32_t* selected, void* stream) {
  hs_status st = hs::check_nb(N, B);
  if (st != HS_OK) return st;
  if (!regret || !loss || !weights || !selected) return HS_ERR_INVALID_ARG;
  if (!hs::aligned4(regret) || !hs::aligned4(loss) || !hs::aligned4(weights) ||
      !hs::aligned4(selected))
    return HS_ERR_MISALIGNED;
  hs::LearnerArgs a = {};
  a.loss_src = hs::kLossGiven;
  a.loss_in = loss;
  a.N = N; a.B = B; a.P = 1;
  a.learner = HS_NORMALHEDGE;
  a.state_in = regret;
  a.state_out = regret;
  a.p_in = weights;
  a.weights_out = weights;
  a.sel_out = selected;
  return hs::launch(a, stream);
}

extern "C" hs_status hs_learner_step(const float* alpha, const float* e_len, int N, int B, int P,
                                     int loss_kind, int learner, float eta, float* state,
                                     float* weights, float* loss_out, int32_t* selected,
                                     float* played_loss, void* stream) {
  hs_status st = hs::check_nb(N, B);
  if (st != HS_OK) return st;
  if (P < 1 || int64_t(N) * B * P >= (int64_t(1) << 40)) return HS_ERR_INVALID_ARG;
  if (loss_kind != HS_LOSS_LENGTH && loss_kind != HS_LOSS_ACCEPT) return HS_ERR_INVALID_ARG;
  if (learner != HS_HEDGE && learner != HS_NORMALHEDGE) return HS_ERR_INVALID_ARG;
  if (loss_kind == HS_LOSS_LENGTH && !e_len) return HS_ERR_INVALID_ARG;
  if (loss_kind == HS_LOSS_ACCEPT && (!alpha || P < 2)) return HS_ERR_INVALID_ARG;
  if (!state || !weights || !selected) return HS_ERR_INVALID_ARG;
  if (learner == HS_HEDGE && !(isfinite(eta) && eta >= 0.f)) return HS_ERR_INVALID_ARG;
  if (!hs::aligned4(alpha) || !hs::aligned4(e_len) || !hs::aligned4(state) ||
      !hs::aligned4(weights) || !hs::aligned4(loss_out) || !hs::aligned4(selected) ||
      !hs::aligned4(played_loss))
    return HS_ERR_MISALIGNED;
  hs::LearnerArgs a = {};
  a.alpha = alpha;
  a.e_len = e_len;
  a.loss_src = loss_kind == HS_LOSS_LENGTH ? hs::kLossLength : hs::kLossAccept;
  a.N = N; a.B = B; a.P = P;
  a.learner = learner;
  a.eta = eta;
  a.state_in = state;
  a.state_out = state;
  a.hedge_add_loss = 1;
  a.p_in = weights;
  a.weights_out = weights;
  a.loss_out = loss_out;
  a.sel_in = selected;
  a.sel_out = selected;
  a.played = played_loss;
  return hs::launch(a, stream);
}
