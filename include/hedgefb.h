/*
 * hedgefb.h -- C ABI of libhedgefb, the GB300 (sm_103a) implementation of
 * HedgeSpec's panoramic-feedback path ("Not-a-Bandit: Provably No-Regret
 * Drafter Selection in Speculative Decoding for LLMs", arXiv 2510.20064).
 *
 * After a verification step the verified tokens have been prefilled into
 * every drafter (Sec. 3.2), so each drafter i has logits at the same P = K+1
 * positions as the target.  From those logits this library computes
 *   alpha[i,b,k] -- the token acceptance probability gamma (Sec. 3.2):
 *                   sum_v min(p(v), q_i(v)) (Thm 1), or, in greedy mode, the
 *                   indicator that argmax q_i == argmax p (Thm 2, L = 1);
 *   e_len[i,b]   -- the acceptance-length estimate of Thm 3,
 *                   1 + sum_{k=1..K} prod_{j<=k} alpha_j, with gamma_{K+1} = 0;
 * and then runs the learner: the Sec. 3.3 loss, Hedge (App. B.1 remark) or
 * NormalHedge (App. D.6 figure), and the choice of the next drafter.
 *
 * Conventions shared by every call
 *  - Shapes are row-major and contiguous.  Index names: N drafters, B
 *    queries, P = K+1 positions, V vocabulary entries.  [N,B] arrays hold
 *    element (i,b) at i*B + b.
 *  - Every pointer marked "device" is device memory owned by the caller; the
 *    library allocates nothing and keeps no state between calls.
 *  - Logits are bf16, fp16 or fp32 (hs_dtype); probabilities, losses, state
 *    and weights are fp32; indices are int32.
 *  - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *    default stream).  Argument errors are detected on the host, before any
 *    launch, and returned; nothing is launched then.  HS_ERR_CUDA reports a
 *    failed launch (cudaGetLastError).
 *  - Data errors are found on the device.  A logit row holding NaN or +inf,
 *    or holding only -inf, makes every alpha that uses the row NaN (and the
 *    e_len that uses it); then, if dev_status is not NULL, HS_ERR_NONFINITE
 *    is stored to *dev_status.  An out-of-range path index stores
 *    HS_ERR_INVALID_ARG the same way.  The library never clears *dev_status:
 *    set it to HS_OK before the call and read it after synchronising.
 *    -inf logits are legal (masked vocabulary).
 *  - Nothing traps; no kernel waits without a bound.
 */
#ifndef HEDGEFB_H
#define HEDGEFB_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  HS_OK = 0,
  HS_ERR_INVALID_ARG = 1,  /* bad size, null pointer, T <= 0, short workspace */
  HS_ERR_UNSUPPORTED = 2,  /* well-formed but outside what is built (e.g. N > 32 for a learner) */
  HS_ERR_MISALIGNED = 3,   /* a pointer not aligned to its element type */
  HS_ERR_NONFINITE = 4,    /* device-side: NaN / +inf / all -inf logit row */
  HS_ERR_CUDA = 5,         /* a CUDA launch failed */
  HS_ERR_TIMEOUT = 6       /* device-side: a bounded wait ran out */
} hs_status;

typedef enum { HS_BF16 = 0, HS_FP16 = 1, HS_FP32 = 2 } hs_dtype;
typedef enum { HS_LOSS_LENGTH = 0, HS_LOSS_ACCEPT = 1 } hs_loss;
typedef enum { HS_HEDGE = 0, HS_NORMALHEDGE = 1 } hs_learner;

/* Largest N the learner calls accept (one warp lane per drafter). */
#define HS_MAX_LEARNER_N 32

/* Human-readable name of a status code; never NULL. */
const char* hs_status_string(int status);

/* Library version, 10000*major + 100*minor + patch. */
int hs_version(void);

/* Bytes of device workspace hs_feedback / hs_feedback_path need for these
 * sizes (0 is a valid answer).  Returns 0 for invalid sizes as well; those
 * calls then fail with HS_ERR_INVALID_ARG. */
size_t hs_feedback_workspace_size(int N, int B, int P, int V, int dtype, int greedy);

/* Number of kernels one hs_feedback / hs_feedback_path call with these
 * arguments launches (for launch accounting); 0 for invalid sizes. */
int hs_feedback_kernel_count(int N, int B, int P, int V, int dtype, int greedy);

/* Panoramic feedback along a verified chain (Sec. 3.2; Thm 1, Thm 2 with
 * L = 1, Thm 3).
 *   target     device, [B,P,V] logits of the target at the P = K+1 verified
 *              positions (Sec. 2.2 step 2: p(x_{t+k} | x_{<t+k}), k = 1..K+1).
 *   drafter    device, [N,B,P,V] logits of every drafter prefilled with the
 *              same verified tokens (Sec. 3.2).
 *   dtype      hs_dtype of both logit tensors.
 *   temperature  T > 0, finite: p = softmax(z_target / T), q_i =
 *              softmax(z_i / T).  Ignored when greedy != 0.
 *   greedy     0: alpha = sum_v min(p(v), q_i(v)), fp32 accumulation.
 *              1: alpha = 1 if argmax q_i == argmax p else 0, argmax over the
 *                 stored logits, lowest index on ties (exact).
 *   alpha      device, out, [N,B,P] fp32 -- all P positions.  The last one
 *              (k = K+1) is the first position of the next chunk; it is not
 *              used by e_len (gamma_{K+1} := 0 in Thm 3).
 *   e_len      device, out, [N,B] fp32 -- 1 + sum_{k=1..K} prod_{j<=k} alpha_j,
 *              in [1, K+1].  May be NULL.
 *   workspace  device, hs_feedback_workspace_size(...) bytes, 256-byte
 *              aligned; may be NULL when that size is 0.  Its contents need
 *              no initialisation and are garbage afterwards.
 *   dev_status device, one int, or NULL (see conventions).
 * Limits: N, B, P, V >= 1; N*B*P*V < 2^62.  Misaligned logit pointers (not
 * a multiple of the element size) give HS_ERR_MISALIGNED. */
hs_status hs_feedback(const void* target, const void* drafter, int dtype, int N,
                      int B, int P, int V, float temperature, int greedy,
                      float* alpha, float* e_len, void* workspace,
                      size_t workspace_bytes, int* dev_status, void* stream);

/* Bytes of the fixed device scratch behind hs_feedback_static. */
#define HS_STATIC_SCRATCH_BYTES (16u << 20)

/* hs_feedback without a workspace argument, for callers that cannot
 * allocate device memory at call time: a serving loop whose memory is
 * reserved up front by another allocator, or code that must not pay for (or
 * synchronise on) cudaMalloc while requests are in flight.  Same arguments
 * and results as hs_feedback, minus `workspace` / `workspace_bytes`.  The
 * paper has no counterpart; this is a deployment convenience.
 *  - The kernels that need scratch (greedy argmax partials, the streaming
 *    and two-pass stochastic paths) use a fixed array of
 *    HS_STATIC_SCRATCH_BYTES bytes compiled into the library; every GPU that
 *    loads the library keeps it until the process exits.  The call makes no
 *    cudaMalloc, cudaFree or other allocating call.
 *  - Sizes whose hs_feedback_workspace_size exceeds HS_STATIC_SCRATCH_BYTES
 *    return HS_ERR_UNSUPPORTED before any launch.
 *  - The first call on a device looks up the array's device address
 *    (cudaGetSymbolAddress, with that device current); make that first call
 *    before capturing a stream into a CUDA graph.  The address belongs to
 *    the device's current context: every call compares that context's id
 *    with the one the address was found in, and a device reset (which
 *    replaces the context) makes the next call look it up again, so that
 *    call, too, belongs before any capture.
 *  - Every call on a device shares the one array, which keeps the last
 *    call's contents; whatever must start at zero is cleared by the call
 *    itself.  Calls whose executions overlap on the GPU (different streams,
 *    or graphs replayed concurrently) race on it: order them. */
hs_status hs_feedback_static(const void* target, const void* drafter, int dtype, int N,
                             int B, int P, int V, float temperature, int greedy,
                             float* alpha, float* e_len, int* dev_status, void* stream);

/* As hs_feedback, but the target rows come from a draft tree (Sec. 2.3,
 * Fig. "illus_gamma"): row k of query b is tree_target[b, path_idx[b,k], :].
 *   tree_target  device, [B,M,V] logits at the M tree nodes of each query.
 *   path_idx     device, [B,P] int32 node indices of the verified
 *                root-to-leaf path, each in [0, M).  An index outside that
 *                range makes the alphas of that (b,k) NaN and stores
 *                HS_ERR_INVALID_ARG to *dev_status.
 * Only the P path rows of each query are read. */
hs_status hs_feedback_path(const void* tree_target, const int32_t* path_idx,
                           int M, const void* drafter, int dtype, int N, int B,
                           int P, int V, float temperature, int greedy,
                           float* alpha, float* e_len, void* workspace,
                           size_t workspace_bytes, int* dev_status,
                           void* stream);

/* Largest branching L the draft-tree entries accept. */
#define HS_MAX_TREE_L 16

/* Bytes of device workspace hs_feedback_topl / hs_feedback_topl_path need
 * (the target rows' share statistics, each drafter row's candidate list and
 * one counter per (drafter, query)); 0 for invalid sizes. */
size_t hs_feedback_topl_workspace_size(int N, int B, int P, int V);

/* Number of kernels one hs_feedback_topl / hs_feedback_topl_path call with
 * these sizes launches (for launch accounting); 0 for invalid sizes. */
int hs_feedback_topl_kernel_count(int N, int B, int P, int V);

/* Panoramic feedback for an EAGLE draft tree with branching L (Sec. 2.3,
 * Thm 2): the drafter proposes its L most likely tokens as the children of
 * a node, and the target's token is accepted iff it is one of them.  Same
 * arguments and layouts as hs_feedback, plus
 *   L          1 <= L <= HS_MAX_TREE_L: the drafter's candidate set is
 *              Top_L(q_i), its L tokens with the largest stored logits
 *              (the ranking of q does not depend on T), ties toward the
 *              lower index, -inf logits last; L >= V takes every token.
 *   greedy     0: alpha = sum_{v in Top_L(q_i)} p(v), p = softmax(z_target/T),
 *                 fp32.  1: alpha = 1 if argmax p (stored logits, lowest
 *                 index on ties) is in Top_L(q_i), else 0 -- exact.  With
 *                 L = 1 this is hs_feedback's greedy rule.
 *   workspace  device, hs_feedback_topl_workspace_size(...) bytes, 256-byte
 *              aligned (required).
 * The candidate set is the plain top L; hs_feedback_topl_pruned below takes
 * the pruned sets of EAGLE-2's dynamic pruning.  Errors as in hs_feedback; a
 * drafter row with NaN, +inf or no finite logit gives NaN and
 * HS_ERR_NONFINITE. */
hs_status hs_feedback_topl(const void* target, const void* drafter, int dtype, int N,
                           int B, int P, int V, float temperature, int greedy, int L,
                           float* alpha, float* e_len, void* workspace,
                           size_t workspace_bytes, int* dev_status, void* stream);

/* hs_feedback_topl with the target rows taken from a draft tree, as in
 * hs_feedback_path (tree_target [B,M,V], path_idx [B,P] int32). */
hs_status hs_feedback_topl_path(const void* tree_target, const int32_t* path_idx,
                                int M, const void* drafter, int dtype, int N, int B,
                                int P, int V, float temperature, int greedy, int L,
                                float* alpha, float* e_len, void* workspace,
                                size_t workspace_bytes, int* dev_status,
                                void* stream);

/* Tree-mode feedback with EAGLE-2's dynamic pruning (Sec. 2.3, the remark
 * closing Thm 2: with pruning, the candidate set of a node is its pruned set
 * of children).  A node's children are the drafter's L highest-ranked tokens
 * and each is scored by the node's score times q(child), so pruning by score
 * keeps a prefix of that ranking.  Same arguments as hs_feedback_topl, plus
 *   keep  device, [N,B,P] int32, caller-owned: keep[i,b,k] in [0, L] is the
 *         number of children drafter i's tree kept at the node of position k
 *         of query b; the candidate set is the first keep[i,b,k] tokens of
 *         Top_L(q_i) (0: every child was pruned, alpha = 0).  keep = L
 *         everywhere gives hs_feedback_topl's result.  Must be non-null and
 *         4-byte aligned (HS_ERR_INVALID_ARG / HS_ERR_MISALIGNED before any
 *         launch).  A value outside [0, L] makes that alpha NaN and stores
 *         HS_ERR_INVALID_ARG to *dev_status.
 * Workspace: hs_feedback_topl_workspace_size(N, B, P, V); launches:
 * hs_feedback_topl_kernel_count(N, B, P, V). */
hs_status hs_feedback_topl_pruned(const void* target, const void* drafter, int dtype, int N,
                                  int B, int P, int V, float temperature, int greedy, int L,
                                  const int32_t* keep, float* alpha, float* e_len,
                                  void* workspace, size_t workspace_bytes, int* dev_status,
                                  void* stream);

/* hs_feedback_topl_pruned with the target rows taken from a draft tree, as
 * in hs_feedback_path (tree_target [B,M,V], path_idx [B,P] int32). */
hs_status hs_feedback_topl_pruned_path(const void* tree_target, const int32_t* path_idx,
                                       int M, const void* drafter, int dtype, int N, int B,
                                       int P, int V, float temperature, int greedy, int L,
                                       const int32_t* keep, float* alpha, float* e_len,
                                       void* workspace, size_t workspace_bytes,
                                       int* dev_status, void* stream);

/* Hedge weights from cumulative losses (App. B.1 remark: w_i <- w_i
 * exp(-eta l_i) from w = 1, normalised, i.e. w = exp(-eta L) / Z).
 *   cum_loss  device, [N,B] fp32 cumulative loss L per (drafter, query).
 *   eta       learning rate, finite and >= 0.
 *   weights   device, out, [N,B] fp32, each column sums to 1.
 *   selected  device, out, [B] int32: first argmin_i L[i,b] (= argmax of w).
 * Limits: 1 <= N <= HS_MAX_LEARNER_N, B >= 1. */
hs_status hs_hedge_update(const float* cum_loss, int N, int B, float eta,
                          float* weights, int32_t* selected, void* stream);

/* One NormalHedge round (App. D.6 figure, steps 2-5) for B queries.
 *   regret    device, in/out, [N,B] fp32: R_{t-1} in, R_t out, where
 *             R_t = R_{t-1} + l_A - l evaluated as sum_j p_j (l_j - l_i).
 *   loss      device, [N,B] fp32 losses l_t of this round.
 *   weights   device, in/out, [N,B] fp32: p_t in (initially 1/N), p_{t+1}
 *             out: p_i proportional to ([R_i]_+/c) exp([R_i]_+^2 / 2c) with
 *             c solving (1/N) sum_i exp([R_i]_+^2 / 2c) = e; uniform when no
 *             R_i is positive.
 *   selected  device, out, [B] int32: argmax of p_{t+1} -- the first argmax
 *             of R when max R > 0, else 0.
 * Limits: 1 <= N <= HS_MAX_LEARNER_N, B >= 1. */
hs_status hs_normalhedge_update(float* regret, const float* loss,
                                float* weights, int N, int B,
                                int32_t* selected, void* stream);

/* Fused learner round: loss from the feedback (Sec. 3.3), learner update and
 * next choice, for B independent queries.
 *   alpha, e_len  device, [N,B,P] and [N,B] fp32 from hs_feedback.
 *   loss_kind     HS_LOSS_LENGTH: f = 1 - e_len / (K+1)      (needs e_len)
 *                 HS_LOSS_ACCEPT: f = (1/K) sum_{k<=K} (1 - alpha_k)
 *                                 (needs alpha and P >= 2)
 *   learner       HS_HEDGE:       state = cumulative loss L, L += f, then
 *                                 hs_hedge_update's weights and choice
 *                 HS_NORMALHEDGE: state = cumulative regret R, then
 *                                 hs_normalhedge_update's round
 *   eta           Hedge learning rate (ignored by NormalHedge).
 *   state, weights  device, in/out, [N,B] fp32.
 *   loss_out      device, out, [N,B] fp32 losses f, or NULL.
 *   selected      device, in/out, [B] int32: the drafter played this round
 *                 in, the next round's choice out.
 *   played_loss   device, in/out, [B] fp32, or NULL: += f[selected_in],
 *                 the learner's own loss term of the Sec. 3.1 regret.
 * Limits: 1 <= N <= HS_MAX_LEARNER_N, B >= 1, P >= 1. */
hs_status hs_learner_step(const float* alpha, const float* e_len, int N, int B,
                          int P, int loss_kind, int learner, float eta,
                          float* state, float* weights, float* loss_out,
                          int32_t* selected, float* played_loss, void* stream);

/* Sampled play (App. B.1, QFI-D: "play a_t according to p", here by
 * sampling from p): for query b, the first drafter i whose running sum
 * weights[0,b] + ... + weights[i,b] exceeds uniforms[b] times the column's
 * total, both sums in fp32 in index order and the threshold rounded once; a
 * zero weight is never drawn, and if rounding leaves no running sum above the
 * threshold the last positive weight is drawn.
 *   weights   device, [N,B] fp32: finite, >= 0, some positive per column
 *             (e.g. the weights a learner call wrote).
 *   uniforms  device, [B] fp32 in [0, 1), from the caller's generator.
 *   selected  device, out, [B] int32; -1 for a column or uniform outside
 *             those rules, which also sets *dev_status = HS_ERR_NONFINITE.
 * Limits: 1 <= N <= HS_MAX_LEARNER_N, B >= 1. */
hs_status hs_sample_select(const float* weights, int N, int B, const float* uniforms,
                           int32_t* selected, int* dev_status, void* stream);

/* Chunk-level learner round with a chunk horizon (App. B.3, game "Chunk-
 * Level Game"; Sec. 3.2 on censoring): as hs_learner_step, but query b's
 * chosen drafter had k_h[b] accepted draft tokens, so only positions
 * 1..k_h[b] were verified and the losses use those alone (Thm 3 with
 * K = k_h[b]):
 *   HS_LOSS_LENGTH  f = 1 - (1 + sum_{k<=k_h} prod_{j<=k} alpha_j)/(k_h+1)
 *   HS_LOSS_ACCEPT  f = (1/k_h) sum_{k<=k_h} (1 - alpha_k)
 * and k_h[b] = 0 gives f = 0 (no information).  e_len is not an input: it is
 * formed from alpha.
 *   k_h       device, [B] int32, 0 <= k_h[b] <= P-1; a query outside that
 *             range keeps its state and sets *dev_status =
 *             HS_ERR_INVALID_ARG.
 * Other arguments as hs_learner_step (loss_out and played_loss may be NULL).
 */
hs_status hs_chunk_learner_step(const float* alpha, const int32_t* k_h, int N, int B,
                                int P, int loss_kind, int learner, float eta,
                                float* state, float* weights, float* loss_out,
                                int32_t* selected, float* played_loss, int* dev_status,
                                void* stream);

/* Token-level game with delay (Sec. 3.2, Fig. "Token-Level Game with Delay")
 * run through QFI-D (App. B.1).  Each query keeps a stream of its verified
 * tokens' acceptance probabilities in a caller-owned ring:
 *   gamma_ring  device, [B,H,N] fp32: gamma of drafter i at token s (0-based)
 *               of query b sits at [b, s mod H, i];
 *   who_ring    device, [B,H] int32: the drafter that played token s;
 *   n_tok       device, [B] int64: tokens in the stream (start at 0);
 *   n_done      device, [B] int64: tokens whose loss the learner consumed
 *               (start at 0).
 * hs_token_append, after a chunk's feedback: the chunk's k_h[b] accepted
 * draft tokens and the target's token that ends it join the stream with
 * gamma_i = alpha[i,b,0..k_h[b]], played by selected[b].  k_h as in
 * hs_chunk_learner_step.  A query whose ring would overwrite unconsumed
 * tokens (n_tok + k_h + 1 - n_done > H) is not appended and sets *dev_status
 * = HS_ERR_UNSUPPORTED.  Size the ring H >= K + 2P to never meet this with
 * one learner call per chunk. */
hs_status hs_token_append(const float* alpha, const int32_t* k_h, int N, int B, int P,
                          const int32_t* selected, float* gamma_ring, int32_t* who_ring,
                          int H, int64_t* n_tok, const int64_t* n_done, int* dev_status,
                          void* stream);

/* hs_token_learner_step, before a chunk's choice: QFI-D's catch-up.  Every
 * token loss that is revealed and not yet consumed is fed to the base
 * learner (HS_HEDGE or HS_NORMALHEDGE, state and weights as in
 * hs_learner_step) in token order, one round each; selected[b] becomes the
 * last round's choice (unchanged when nothing was revealed).  Token s's loss
 * is 1 - gamma_s (HS_LOSS_ACCEPT), or 1 - E/(K+1) with E = 1 +
 * sum_{k=1..K} prod_{j<k} gamma_{s+j} (HS_LOSS_LENGTH, Thm 3 for a K-token
 * draft starting at s).  With n tokens in the stream, f_s is revealed for
 * s < n (acceptance) or s < n - K (length), as in the figure; hybrid losses
 * (App. B.5): tokens s < accept_first use the acceptance loss and are
 * revealed at once.  played_loss (or NULL) [B] += f_s[the drafter that
 * played s] for each consumed token.  1 <= K <= H. */
hs_status hs_token_learner_step(const float* gamma_ring, const int32_t* who_ring, int N,
                                int B, int H, const int64_t* n_tok, int64_t* n_done,
                                int K, int loss_kind, int64_t accept_first, int learner,
                                float eta, float* state, float* weights,
                                int32_t* selected, float* played_loss, int* dev_status,
                                void* stream);

/* The chunk-level losses of hs_chunk_learner_step alone, without a learner
 * update: loss_out [N,B] (device, fp32), e.g. one slot of a queue of delayed
 * loss vectors for hs_learner_apply.  k_h as there (a query outside the range
 * keeps its loss_out entries and sets *dev_status = HS_ERR_INVALID_ARG). */
hs_status hs_chunk_losses(const float* alpha, const int32_t* k_h, int N, int B, int P,
                          int loss_kind, float* loss_out, int* dev_status, void* stream);

/* QFI-D's catch-up over a queue of chunk-level loss vectors (App. B.1; the
 * batched feedback of App. B.5): vectors c = 0..count-1, in slots
 * (first + c) mod Q of queue [Q,N,B] (device, fp32), are fed to the base
 * learner in that order, one round each, for every query; state, weights
 * and the choice as in hs_learner_step (selected[b] = the last round's
 * choice).  0 <= first < Q, 0 <= count <= Q; count = 0 launches nothing. */
hs_status hs_learner_apply(const float* queue, int Q, int first, int count, int N, int B,
                           int learner, float eta, float* state, float* weights,
                           int32_t* selected, void* stream);

/* The practical schedule of App. B.5 ("skipping updates", batched delayed
 * feedback, warm-up, "hybrid losses"), host only.  A round is one
 * speculative chunk; after it hs_schedule_next decides, from the chunk's
 * token count:
 *   - in the first warmup_rounds rounds: evaluate every drafter on the
 *     chunk and apply the vector at once (full information each round);
 *   - afterwards: evaluate only when at least skip_tokens tokens were
 *     generated since the last evaluation (this chunk's included); queue the
 *     vectors, and apply the queue once every batch_rounds rounds counted
 *     from the end of the warm-up (only when something is queued);
 *   - the first hybrid_vectors vectors use HS_LOSS_ACCEPT, later ones
 *     HS_LOSS_LENGTH.
 * The paper's example setting is warmup 6, batch 12, skip 6. */
typedef struct {
  int warmup_rounds;
  int batch_rounds;   /* >= 1 */
  int skip_tokens;
  int hybrid_vectors;
} hs_schedule_config;

typedef struct {      /* zero-initialise before the first round */
  int64_t rounds;
  int64_t tokens_since_eval;
  int64_t vectors_made;
  int64_t vectors_queued;
} hs_schedule_state;

typedef struct {
  int evaluate;   /* 1: run the feedback on this chunk and queue its loss vector */
  int loss_kind;  /* HS_LOSS_ACCEPT / HS_LOSS_LENGTH: that vector's loss */
  int apply;      /* 1: feed the whole queue to the learner before the next choice */
} hs_schedule_action;

hs_status hs_schedule_next(const hs_schedule_config* cfg, hs_schedule_state* state,
                           int tokens, hs_schedule_action* action);

/* ---- test hook (the paper has no counterpart) ----------------------------
 * Exercises the bounded-wait error path of the library's kernels on a GPU
 * without faulting or hanging it.  It runs the streaming stochastic kernel
 * (the one hs_feedback uses for V > 153 600) with one change: the wait of
 * tile (b,k) = (0,0) for its statistics asks for one count more than exist,
 * so it can only run out, and every wait on a tile's statistics count is
 * limited to `wait_cycles` SM clock cycles instead of about a second.  Tile (0,0)'s waits then report
 * HS_ERR_TIMEOUT to *dev_status and its alphas (and the e_len of query 0)
 * come out NaN; every other alpha is the one hs_feedback computes, and the
 * CUDA context stays usable.  Same arguments as hs_feedback (stochastic,
 * chain target), plus wait_cycles >= 1; dev_status is required.  Takes only
 * shapes the streaming kernel takes (bf16/fp16, V % 8 == 0, N <= 32,
 * 16-byte-aligned logits), else HS_ERR_UNSUPPORTED; workspace as
 * hs_feedback_workspace_size reports for the same sizes. */
hs_status hs_test_stream_wait_timeout(const void* target, const void* drafter, int dtype,
                                      int N, int B, int P, int V, float temperature,
                                      long long wait_cycles, float* alpha, float* e_len,
                                      void* workspace, size_t workspace_bytes,
                                      int* dev_status, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* HEDGEFB_H */
