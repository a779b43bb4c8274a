// hs_delayed.cu -- the learner under delayed and censored feedback, and
// sampled play, for B independent queries:
//   sample_kernel         QFI-D's "play a_t according to p" (App. B.1): an
//                         inverse-CDF draw with a caller-supplied uniform,
//                         one thread per query, fp32 sums in index order
//   chunk_learner_kernel  chunk-level game with the chunk horizon k_h (App.
//                         B.3): the losses use positions 1..k_h only; or the
//                         losses alone, for a queue of delayed vectors
//   apply_kernel          QFI-D catch-up over a queue of chunk-level loss
//                         vectors (App. B.1; the batched feedback of B.5)
//   token_append_kernel   the verified tokens of a chunk join each query's
//                         token stream (a ring of gamma values)
//   token_learner_kernel  QFI-D catch-up (App. B.1): every revealed token loss
//                         not yet consumed (Sec. 3.2, Fig. "Token-Level Game
//                         with Delay") is fed to the base learner in token
//                         order, one round each, then the choice stands
// The learner kernels run one warp per query, lane i = drafter i (N <= 32).
#include <math.h>
#include <stdint.h>

#include "hs_common.cuh"
#include "hs_learner_core.cuh"

namespace hs {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kWarpsPerBlock = 4;

bool aligned(const void* p, uintptr_t a) { return reinterpret_cast<uintptr_t>(p) % a == 0; }

hs_status check_nb(int N, int B) {
  if (N < 1 || B < 1) return HS_ERR_INVALID_ARG;
  if (N > HS_MAX_LEARNER_N) return HS_ERR_UNSUPPORTED;
  if (int64_t(N) * B >= (int64_t(1) << 31)) return HS_ERR_INVALID_ARG;
  return HS_OK;
}

unsigned warp_blocks(int B) { return unsigned((int64_t(B) + kWarpsPerBlock - 1) / kWarpsPerBlock); }

// ---- sampled play ---------------------------------------------------------------

__global__ void sample_kernel(const float* __restrict__ w, int N, int B,
                              const float* __restrict__ uniforms, int32_t* __restrict__ selected,
                              int* dev_status) {
  pdl_wait();
  const int64_t b = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const float u = uniforms[b];
  bool ok = u >= 0.f && u < 1.f;
  float total = 0.f;
  for (int i = 0; i < N; ++i) {
    const float x = w[int64_t(i) * B + b];
    ok = ok && x >= 0.f && !isinf(x);
    total += x;
  }
  ok = ok && total > 0.f && !isinf(total);
  int pick = -1;
  if (ok) {
    // the first running sum above u * total (it grows only at a positive
    // weight); the last positive weight if rounding leaves none above it
    const float thr = u * total;
    float run = 0.f;
    for (int i = 0; i < N; ++i) {
      const float x = w[int64_t(i) * B + b];
      run += x;
      if (x > 0.f) pick = i;
      if (run > thr) break;
    }
  } else {
    report(dev_status, HS_ERR_NONFINITE);
  }
  selected[b] = pick;
}

// ---- chunk-level round with a chunk horizon ------------------------------------

struct ChunkArgs {
  const float* alpha;    // [N,B,P]
  const int32_t* k_h;    // [B]
  int N, B, P, loss_kind, learner;
  float eta;
  float* state;          // [N,B]
  float* weights;        // [N,B]
  float* loss_out;       // [N,B] or NULL
  int32_t* selected;     // [B]
  float* played;         // [B] or NULL
  int* dev_status;
  int update;            // 0: write the losses only
};

__global__ void __launch_bounds__(kWarpsPerBlock * 32) chunk_learner_kernel(ChunkArgs a) {
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int64_t b = int64_t(blockIdx.x) * kWarpsPerBlock + (threadIdx.x >> 5);
  if (b >= a.B) return;  // whole warp
  const int k = a.k_h[b];
  if (k < 0 || k > a.P - 1) {  // this query's round is skipped
    if (lane == 0) report(a.dev_status, HS_ERR_INVALID_ARG);
    return;
  }
  const bool act = lane < a.N;
  const int64_t ib = int64_t(lane) * a.B + b;
  // losses over the verified positions 1..k (Thm 3 with K = k; the
  // acceptance rate over k tokens); k = 0 carries no information: 0
  float f = 0.f;
  if (act && k > 0) {
    const float* al = a.alpha + ib * a.P;
    if (a.loss_kind == HS_LOSS_LENGTH) {
      float e = 1.f, prod = 1.f;
      for (int j = 0; j < k; ++j) {
        prod *= al[j];
        e += prod;
      }
      f = 1.f - e / float(k + 1);
    } else {
      float s = 0.f;
      for (int j = 0; j < k; ++j) s += 1.f - al[j];
      f = s / float(k);
    }
  }
  if (act && a.loss_out) a.loss_out[ib] = f;
  if (!a.update) return;
  if (a.played) {
    const int s = a.selected[b];
    const bool ok = s >= 0 && s < a.N;
    const float fs = __shfl_sync(kFull, f, ok ? s : 0);
    if (lane == 0) a.played[b] += ok ? fs : __int_as_float(0x7fc00000);
  }
  float state = act ? a.state[ib] : 0.f;
  float p = (act && a.learner == HS_NORMALHEDGE) ? a.weights[ib] : 0.f;
  const int sel = learner::round(a.learner, a.N, a.eta, f, true, state, p);
  if (act) {
    a.state[ib] = state;
    a.weights[ib] = p;
  }
  if (lane == 0) a.selected[b] = sel;
}

// ---- a queue of chunk-level loss vectors -----------------------------------------

struct ApplyArgs {
  const float* queue;    // [Q,N,B]: vector c sits in slot (first + c) mod Q
  int Q, first, count, N, B, learner;
  float eta;
  float* state;          // [N,B]
  float* weights;        // [N,B]
  int32_t* selected;     // [B]
};

__global__ void __launch_bounds__(kWarpsPerBlock * 32) apply_kernel(ApplyArgs a) {
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int64_t b = int64_t(blockIdx.x) * kWarpsPerBlock + (threadIdx.x >> 5);
  if (b >= a.B) return;  // whole warp
  const bool act = lane < a.N;
  const int64_t ib = int64_t(lane) * a.B + b;
  float state = act ? a.state[ib] : 0.f;
  float p = (act && a.learner == HS_NORMALHEDGE) ? a.weights[ib] : 0.f;
  int sel = 0;
  for (int c = 0; c < a.count; ++c) {  // FIFO
    const int64_t slot = (int64_t(a.first) + c) % a.Q;
    const float f = act ? a.queue[(slot * a.N + lane) * a.B + b] : 0.f;
    sel = learner::round(a.learner, a.N, a.eta, f, true, state, p);
  }
  if (act) {
    a.state[ib] = state;
    a.weights[ib] = p;
  }
  if (lane == 0) a.selected[b] = sel;
}

// ---- token stream and the QFI-D catch-up ----------------------------------------

struct TokenArgs {
  float* gamma;          // [B,H,N]: gamma of drafter i at token s is [b, s mod H, i]
  int32_t* who;          // [B,H]: drafter that played token s
  int64_t* n_tok;        // [B] tokens in the stream
  int64_t* n_done;       // [B] tokens whose loss has been consumed
  int N, B, H;
  // append
  const float* alpha;    // [N,B,P]
  const int32_t* k_h;    // [B]
  int P;
  // catch-up
  int K, loss_kind, learner;
  int64_t accept_first;
  float eta;
  float* state;          // [N,B]
  float* weights;        // [N,B]
  int32_t* selected;     // [B]
  float* played;         // [B] or NULL
  int* dev_status;
};

__global__ void __launch_bounds__(kWarpsPerBlock * 32) token_append_kernel(TokenArgs a) {
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int64_t b = int64_t(blockIdx.x) * kWarpsPerBlock + (threadIdx.x >> 5);
  if (b >= a.B) return;  // whole warp
  const int k = a.k_h[b];
  if (k < 0 || k > a.P - 1) {
    if (lane == 0) report(a.dev_status, HS_ERR_INVALID_ARG);
    return;
  }
  const int64_t n = a.n_tok[b];
  if (n + k + 1 - a.n_done[b] > a.H) {  // the ring would overwrite unconsumed tokens
    if (lane == 0) report(a.dev_status, HS_ERR_UNSUPPORTED);
    return;
  }
  // the chunk's verified tokens: its k accepted drafts and the target's token
  for (int j = 0; j <= k; ++j) {
    const int64_t slot = int64_t(b) * a.H + (n + j) % a.H;
    if (lane < a.N) a.gamma[slot * a.N + lane] = a.alpha[(int64_t(lane) * a.B + b) * a.P + j];
    if (lane == 0) a.who[slot] = a.selected[b];
  }
  if (lane == 0) a.n_tok[b] = n + k + 1;
}

// Tokens of a stream of n whose loss is revealed (Fig. "Token-Level Game with
// Delay"): f_{<=n} for the acceptance-rate loss, f_{<=n-K} for the length
// loss; with hybrid losses the first accept_first use the acceptance rate.
__device__ __forceinline__ int64_t revealed(int64_t n, int K, int loss_kind,
                                            int64_t accept_first) {
  int64_t late = loss_kind == HS_LOSS_LENGTH ? n - K : n;
  if (late < 0) late = 0;
  const int64_t early = n < accept_first ? n : accept_first;
  return late > early ? late : early;
}

__global__ void __launch_bounds__(kWarpsPerBlock * 32) token_learner_kernel(TokenArgs a) {
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int64_t b = int64_t(blockIdx.x) * kWarpsPerBlock + (threadIdx.x >> 5);
  if (b >= a.B) return;  // whole warp
  const bool act = lane < a.N;
  const int64_t ib = int64_t(lane) * a.B + b;
  const int64_t n = a.n_tok[b];
  int64_t d = a.n_done[b];
  const int64_t ready = revealed(n, a.K, a.loss_kind, a.accept_first);
  if (d >= ready) return;  // nothing new: the choice stands
  float state = act ? a.state[ib] : 0.f;
  float p = (act && a.learner == HS_NORMALHEDGE) ? a.weights[ib] : 0.f;
  const float* g = a.gamma + int64_t(b) * a.H * a.N + lane;
  float own = 0.f;
  int sel = 0;
  int slot = int(d % a.H);  // ring slot of token d
  for (; d < ready; ++d, slot = slot + 1 == a.H ? 0 : slot + 1) {  // FIFO: token order
    float f = 0.f;
    if (act) {
      if (d < a.accept_first || a.loss_kind == HS_LOSS_ACCEPT) {
        f = 1.f - g[int64_t(slot) * a.N];
      } else {
        // Thm 3 for a K-token draft starting at token d; the window's loads
        // are issued 8 at a time (slots wrap once at most: K <= H)
        float e = 1.f, prod = 1.f;
        for (int j0 = 0; j0 < a.K; j0 += 8) {
          float v[8];
#pragma unroll
          for (int jj = 0; jj < 8; ++jj) {
            int sj = slot + j0 + jj;
            sj -= sj >= a.H ? a.H : 0;
            v[jj] = j0 + jj < a.K ? g[int64_t(sj) * a.N] : 1.f;
          }
#pragma unroll
          for (int jj = 0; jj < 8; ++jj)
            if (j0 + jj < a.K) {
              prod *= v[jj];
              e += prod;
            }
        }
        f = 1.f - e / float(a.K + 1);
      }
    }
    const int pl = a.who[int64_t(b) * a.H + slot];
    own += __shfl_sync(kFull, f, pl >= 0 && pl < a.N ? pl : 0);
    sel = learner::round(a.learner, a.N, a.eta, f, true, state, p);
  }
  if (act) {
    a.state[ib] = state;
    a.weights[ib] = p;
  }
  if (lane == 0) {
    a.selected[b] = sel;
    a.n_done[b] = d;
    if (a.played) a.played[b] += own;
  }
}

}  // namespace
}  // namespace hs

extern "C" hs_status hs_sample_select(const float* weights, int N, int B, const float* uniforms,
                                      int32_t* selected, int* dev_status, void* stream) {
  hs_status st = hs::check_nb(N, B);
  if (st != HS_OK) return st;
  if (!weights || !uniforms || !selected) return HS_ERR_INVALID_ARG;
  if (!hs::aligned(weights, 4) || !hs::aligned(uniforms, 4) || !hs::aligned(selected, 4) ||
      !hs::aligned(dev_status, 4))
    return HS_ERR_MISALIGNED;
  if (hs::launch_pdl(hs::sample_kernel, dim3(unsigned((int64_t(B) + 127) / 128)), dim3(128), 0,
                     static_cast<cudaStream_t>(stream), weights, N, B, uniforms, selected,
                     dev_status) != cudaSuccess)
    return HS_ERR_CUDA;
  return HS_OK;
}

extern "C" hs_status hs_chunk_learner_step(const float* alpha, const int32_t* k_h, int N, int B,
                                           int P, int loss_kind, int learner, float eta,
                                           float* state, float* weights, float* loss_out,
                                           int32_t* selected, float* played_loss,
                                           int* dev_status, void* stream) {
  hs_status st = hs::check_nb(N, B);
  if (st != HS_OK) return st;
  if (P < 1 || int64_t(N) * B * P >= (int64_t(1) << 40)) return HS_ERR_INVALID_ARG;
  if (loss_kind != HS_LOSS_LENGTH && loss_kind != HS_LOSS_ACCEPT) return HS_ERR_INVALID_ARG;
  if (learner != HS_HEDGE && learner != HS_NORMALHEDGE) return HS_ERR_INVALID_ARG;
  if (!alpha || !k_h || !state || !weights || !selected) return HS_ERR_INVALID_ARG;
  if (learner == HS_HEDGE && !(isfinite(eta) && eta >= 0.f)) return HS_ERR_INVALID_ARG;
  if (!hs::aligned(alpha, 4) || !hs::aligned(k_h, 4) || !hs::aligned(state, 4) ||
      !hs::aligned(weights, 4) || !hs::aligned(loss_out, 4) || !hs::aligned(selected, 4) ||
      !hs::aligned(played_loss, 4) || !hs::aligned(dev_status, 4))
    return HS_ERR_MISALIGNED;
  hs::ChunkArgs a = {alpha, k_h, N, B, P, loss_kind, learner, eta, state, weights, loss_out,
                     selected, played_loss, dev_status, 1};
  if (hs::launch_pdl(hs::chunk_learner_kernel, dim3(hs::warp_blocks(B)),
                     dim3(hs::kWarpsPerBlock * 32), 0, static_cast<cudaStream_t>(stream),
                     a) != cudaSuccess)
    return HS_ERR_CUDA;
  return HS_OK;
}

namespace {
hs_status check_ring(const float* gamma, const int32_t* who, int N, int B, int H,
                     const int64_t* n_tok, const int64_t* n_done, const int* dev_status) {
  hs_status st = hs::check_nb(N, B);
  if (st != HS_OK) return st;
  if (H < 1 || double(B) * double(H) * double(N) >= 9.0e18) return HS_ERR_INVALID_ARG;
  if (!gamma || !who || !n_tok || !n_done) return HS_ERR_INVALID_ARG;
  if (!hs::aligned(gamma, 4) || !hs::aligned(who, 4) || !hs::aligned(n_tok, 8) ||
      !hs::aligned(n_done, 8) || !hs::aligned(dev_status, 4))
    return HS_ERR_MISALIGNED;
  return HS_OK;
}
}  // namespace

extern "C" hs_status hs_token_append(const float* alpha, const int32_t* k_h, int N, int B, int P,
                                     const int32_t* selected, float* gamma_ring,
                                     int32_t* who_ring, int H, int64_t* n_tok,
                                     const int64_t* n_done, int* dev_status, void* stream) {
  hs_status st = check_ring(gamma_ring, who_ring, N, B, H, n_tok, n_done, dev_status);
  if (st != HS_OK) return st;
  if (P < 1 || !alpha || !k_h || !selected) return HS_ERR_INVALID_ARG;
  if (!hs::aligned(alpha, 4) || !hs::aligned(k_h, 4) || !hs::aligned(selected, 4))
    return HS_ERR_MISALIGNED;
  hs::TokenArgs a = {};
  a.gamma = gamma_ring;
  a.who = who_ring;
  a.n_tok = n_tok;
  a.n_done = const_cast<int64_t*>(n_done);  // read only by this kernel
  a.N = N;
  a.B = B;
  a.H = H;
  a.alpha = alpha;
  a.k_h = k_h;
  a.P = P;
  a.selected = const_cast<int32_t*>(selected);  // read only by this kernel
  a.dev_status = dev_status;
  if (hs::launch_pdl(hs::token_append_kernel, dim3(hs::warp_blocks(B)),
                     dim3(hs::kWarpsPerBlock * 32), 0, static_cast<cudaStream_t>(stream),
                     a) != cudaSuccess)
    return HS_ERR_CUDA;
  return HS_OK;
}

extern "C" hs_status hs_token_learner_step(const float* gamma_ring, const int32_t* who_ring,
                                           int N, int B, int H, const int64_t* n_tok,
                                           int64_t* n_done, int K, int loss_kind,
                                           int64_t accept_first, int learner, float eta,
                                           float* state, float* weights, int32_t* selected,
                                           float* played_loss, int* dev_status, void* stream) {
  hs_status st = check_ring(gamma_ring, who_ring, N, B, H, n_tok, n_done, dev_status);
  if (st != HS_OK) return st;
  if (K < 1 || K > H || accept_first < 0) return HS_ERR_INVALID_ARG;
  if (loss_kind != HS_LOSS_LENGTH && loss_kind != HS_LOSS_ACCEPT) return HS_ERR_INVALID_ARG;
  if (learner != HS_HEDGE && learner != HS_NORMALHEDGE) return HS_ERR_INVALID_ARG;
  if (!state || !weights || !selected) return HS_ERR_INVALID_ARG;
  if (learner == HS_HEDGE && !(isfinite(eta) && eta >= 0.f)) return HS_ERR_INVALID_ARG;
  if (!hs::aligned(state, 4) || !hs::aligned(weights, 4) || !hs::aligned(selected, 4) ||
      !hs::aligned(played_loss, 4))
    return HS_ERR_MISALIGNED;
  hs::TokenArgs a = {};
  a.gamma = const_cast<float*>(gamma_ring);  // read only by this kernel
  a.who = const_cast<int32_t*>(who_ring);
  a.n_tok = const_cast<int64_t*>(n_tok);
  a.n_done = n_done;
  a.N = N;
  a.B = B;
  a.H = H;
  a.K = K;
  a.loss_kind = loss_kind;
  a.learner = learner;
  a.accept_first = accept_first;
  a.eta = eta;
  a.state = state;
  a.weights = weights;
  a.selected = selected;
  a.played = played_loss;
  a.dev_status = dev_status;
  if (hs::launch_pdl(hs::token_learner_kernel, dim3(hs::warp_blocks(B)),
                     dim3(hs::kWarpsPerBlock * 32), 0, static_cast<cudaStream_t>(stream),
                     a) != cudaSuccess)
    return HS_ERR_CUDA;
  return HS_OK;
}

extern "C" hs_status hs_chunk_losses(const float* alpha, const int32_t* k_h, int N, int B, int P,
                                     int loss_kind, float* loss_out, int* dev_status,
                                     void* stream) {
  if (N < 1 || B < 1 || P < 1 || int64_t(N) * B * P >= (int64_t(1) << 40))
    return HS_ERR_INVALID_ARG;
  if (N > HS_MAX_LEARNER_N) return HS_ERR_UNSUPPORTED;
  if (loss_kind != HS_LOSS_LENGTH && loss_kind != HS_LOSS_ACCEPT) return HS_ERR_INVALID_ARG;
  if (!alpha || !k_h || !loss_out) return HS_ERR_INVALID_ARG;
  if (!hs::aligned(alpha, 4) || !hs::aligned(k_h, 4) || !hs::aligned(loss_out, 4) ||
      !hs::aligned(dev_status, 4))
    return HS_ERR_MISALIGNED;
  hs::ChunkArgs a = {alpha, k_h, N, B, P, loss_kind, HS_HEDGE, 0.f, nullptr, nullptr, loss_out,
                     nullptr, nullptr, dev_status, 0};
  if (hs::launch_pdl(hs::chunk_learner_kernel, dim3(hs::warp_blocks(B)),
                     dim3(hs::kWarpsPerBlock * 32), 0, static_cast<cudaStream_t>(stream),
                     a) != cudaSuccess)
    return HS_ERR_CUDA;
  return HS_OK;
}

extern "C" hs_status hs_learner_apply(const float* queue, int Q, int first, int count, int N,
                                      int B, int learner, float eta, float* state,
                                      float* weights, int32_t* selected, void* stream) {
  hs_status st = hs::check_nb(N, B);
  if (st != HS_OK) return st;
  if (Q < 1 || first < 0 || first >= Q || count < 0 || count > Q) return HS_ERR_INVALID_ARG;
  if (learner != HS_HEDGE && learner != HS_NORMALHEDGE) return HS_ERR_INVALID_ARG;
  if (!queue || !state || !weights || !selected) return HS_ERR_INVALID_ARG;
  if (learner == HS_HEDGE && !(isfinite(eta) && eta >= 0.f)) return HS_ERR_INVALID_ARG;
  if (!hs::aligned(queue, 4) || !hs::aligned(state, 4) || !hs::aligned(weights, 4) ||
      !hs::aligned(selected, 4))
    return HS_ERR_MISALIGNED;
  if (count == 0) return HS_OK;  // QFI-D with an empty queue: nothing to do
  hs::ApplyArgs a = {queue, Q, first, count, N, B, learner, eta, state, weights, selected};
  if (hs::launch_pdl(hs::apply_kernel, dim3(hs::warp_blocks(B)), dim3(hs::kWarpsPerBlock * 32),
                     0, static_cast<cudaStream_t>(stream), a) != cudaSuccess)
    return HS_ERR_CUDA;
  return HS_OK;
}

// App. B.5's schedule (host only; see the header for the reading).
extern "C" hs_status hs_schedule_next(const hs_schedule_config* cfg, hs_schedule_state* st,
                                      int tokens, hs_schedule_action* act) {
  if (!cfg || !st || !act) return HS_ERR_INVALID_ARG;
  if (cfg->warmup_rounds < 0 || cfg->batch_rounds < 1 || cfg->skip_tokens < 0 ||
      cfg->hybrid_vectors < 0 || tokens < 0)
    return HS_ERR_INVALID_ARG;
  const int64_t r = st->rounds;
  bool evaluate, apply;
  if (r < cfg->warmup_rounds) {  // full information every round
    evaluate = apply = true;
    st->tokens_since_eval = 0;
  } else {
    st->tokens_since_eval += tokens;
    evaluate = st->tokens_since_eval >= cfg->skip_tokens;
    if (evaluate) st->tokens_since_eval = 0;
    apply = (r - cfg->warmup_rounds + 1) % cfg->batch_rounds == 0;
  }
  act->evaluate = evaluate ? 1 : 0;
  act->loss_kind =
      (evaluate && st->vectors_made < cfg->hybrid_vectors) ? HS_LOSS_ACCEPT : HS_LOSS_LENGTH;
  if (evaluate) {
    ++st->vectors_made;
    ++st->vectors_queued;
  }
  act->apply = (apply && st->vectors_queued > 0) ? 1 : 0;
  if (act->apply) st->vectors_queued = 0;
  st->rounds = r + 1;
  return HS_OK;
}
