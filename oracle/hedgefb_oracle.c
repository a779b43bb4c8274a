/*
 * hedgefb_oracle.c -- plain, slow, fp64 CPU restatement of the HedgeSpec
 * panoramic-feedback path ("Not-a-Bandit", arXiv 2510.20064).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the oracle that the CUDA library is
 * checked against.  Only the test-suite, the smoke check and the CPU-baseline
 * leg of the benchmark may load it.  It shares no code, header, table or
 * constant with the CUDA library and never calls into it.
 *
 * Every function evaluates the paper's definition directly, in fp64, with
 * plain loops in index order:
 *   - Thm 1 (Sec. 2.2):      alpha = sum_x min(p(x), q(x)) = 1 - TV(p, q)
 *   - Thm 2 with L = 1 and a greedy target (Sec. 2.3): greedy alpha is the
 *                            indicator that the two argmaxes agree
 *   - Thm 2 (Sec. 2.3), EAGLE tree with branching L: alpha is the target's
 *                            mass on the drafter's top-L tokens
 *   - Thm 3 (Sec. 3.2):      counterfactual acceptance-length estimator
 *   - Sec. 3.3 / App. B.3:   length loss and acceptance-rate loss
 *   - App. B.1 remark:       Hedge, w_i <- w_i exp(-eta l_i), normalised
 *   - App. D.6 (Fig. "NormalHedge"): NormalHedge regret update, scale c and
 *                            weights
 *   - App. B.1 (QFI-D):      a draw "according to p" by the inverse CDF, and
 *                            the FIFO catch-up of delayed loss vectors
 *   - App. B.3:              chunk-level losses with the chunk horizon k_h
 *   - Sec. 3.2 (Fig. "Token-Level Game with Delay"): per-token losses and
 *                            the rule of when each is revealed
 *   - App. B.5:              warm-up, skipped and batched updates, hybrid
 *                            losses (a schedule), and a batch fed FIFO
 * Input logits are read as the very bytes the GPU reads: bf16 is widened by
 * a 16-bit shift, fp16 by its IEEE-754 binary16 definition, fp32 as is; all
 * three conversions to double are exact.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum { ORC_BF16 = 0, ORC_FP16 = 1, ORC_FP32 = 2 };
enum { ORC_OK = 0, ORC_BADARG = 1, ORC_NONFINITE = 4 };
enum { ORC_LOSS_LENGTH = 0, ORC_LOSS_ACCEPT = 1 };
enum { ORC_HEDGE = 0, ORC_NORMALHEDGE = 1 };

/* ---- exact decode of one stored logit -------------------------------- */

static double decode_bf16(uint16_t h) {
  uint32_t bits = ((uint32_t)h) << 16;  /* bf16 is the top half of binary32 */
  float f;
  memcpy(&f, &bits, sizeof f);
  return (double)f;
}

static double decode_fp16(uint16_t h) {
  int sign = (h >> 15) & 1;
  int expo = (h >> 10) & 0x1f;
  int mant = h & 0x3ff;
  double v;
  if (expo == 0)
    v = ldexp((double)mant, -24);                  /* subnormal: mant * 2^-24 */
  else if (expo == 31)
    v = mant ? NAN : INFINITY;
  else
    v = ldexp((double)(mant + 1024), expo - 25);   /* (1 + mant/1024) 2^(e-15) */
  return sign ? -v : v;
}

double orc_decode(const void* base, int dtype, int64_t idx) {
  if (dtype == ORC_BF16) return decode_bf16(((const uint16_t*)base)[idx]);
  if (dtype == ORC_FP16) return decode_fp16(((const uint16_t*)base)[idx]);
  return (double)((const float*)base)[idx];
}

/* ---- one row: softmax at temperature T (the p(.) / q(.) of Thm 1) ---- */

/* A row is usable when it holds no NaN, no +inf and at least one finite
 * value; -inf entries are masked vocabulary and have probability 0. */
static int row_ok(const void* row, int dtype, int V) {
  int any_finite = 0;
  for (int v = 0; v < V; ++v) {
    double z = orc_decode(row, dtype, v);
    if (isnan(z) || z == INFINITY) return 0;
    if (z != -INFINITY) any_finite = 1;
  }
  return any_finite;
}

/* P[v] = exp(z_v/T - lse),  lse = m + log sum_v exp(z_v/T - m),  m = max z/T. */
int orc_row_probs(const void* row, int dtype, int V, double T, double* P) {
  if (!row_ok(row, dtype, V)) {
    for (int v = 0; v < V; ++v) P[v] = NAN;
    return ORC_NONFINITE;
  }
  double m = -INFINITY;
  for (int v = 0; v < V; ++v) {
    double s = orc_decode(row, dtype, v) / T;
    if (s > m) m = s;
  }
  double sum = 0.0;
  for (int v = 0; v < V; ++v) sum += exp(orc_decode(row, dtype, v) / T - m);
  double lse = m + log(sum);
  for (int v = 0; v < V; ++v) P[v] = exp(orc_decode(row, dtype, v) / T - lse);
  return ORC_OK;
}

/* First index of the largest stored logit (ties -> lowest index; -0 == +0).
 * Returns -1 for an unusable row. */
int orc_row_argmax(const void* row, int dtype, int V) {
  if (!row_ok(row, dtype, V)) return -1;
  int best = 0;
  double bz = orc_decode(row, dtype, 0);
  for (int v = 1; v < V; ++v) {
    double z = orc_decode(row, dtype, v);
    if (z > bz) { bz = z; best = v; }
  }
  return best;
}

/* Thm 1: acceptance probability of one draft position = sum_x min(p, q). */
double orc_overlap(const double* P, const double* Q, int V) {
  double a = 0.0;
  for (int v = 0; v < V; ++v) a += (P[v] < Q[v]) ? P[v] : Q[v];
  return a;
}

/* Thm 1, right-hand side: TV(p, q) = 1/2 sum_x |p(x) - q(x)|. */
double orc_tv(const double* P, const double* Q, int V) {
  double t = 0.0;
  for (int v = 0; v < V; ++v) t += fabs(P[v] - Q[v]);
  return 0.5 * t;
}

/* alpha for one (target row, drafter row) pair.
 * Stochastic: Thm 1.  Greedy: Thm 2 with branching L = 1 under a greedy
 * (argmax) target -- the drafted token is accepted iff both argmaxes agree. */
int orc_alpha_pair(const void* zt, const void* zd, int dtype, int V, double T,
                   int greedy, double* alpha) {
  if (greedy) {
    int jt = orc_row_argmax(zt, dtype, V), jd = orc_row_argmax(zd, dtype, V);
    if (jt < 0 || jd < 0) { *alpha = NAN; return ORC_NONFINITE; }
    *alpha = (jt == jd) ? 1.0 : 0.0;
    return ORC_OK;
  }
  double* P = (double*)malloc(sizeof(double) * (size_t)V);
  double* Q = (double*)malloc(sizeof(double) * (size_t)V);
  int st = orc_row_probs(zt, dtype, V, T, P);
  st |= orc_row_probs(zd, dtype, V, T, Q);
  *alpha = st ? NAN : orc_overlap(P, Q, V);
  free(P);
  free(Q);
  return st ? ORC_NONFINITE : ORC_OK;
}

/* ---- Thm 3: counterfactual acceptance length ------------------------- */

/* Sum of prefix products: 1 + sum_{k=1..K} prod_{j<=k} gamma_j.
 * gamma[0..K-1] are gamma_1..gamma_K; gamma_{K+1} := 0 is implicit. */
double orc_elen_prefix(const double* gamma, int K) {
  double e = 1.0, prod = 1.0;
  for (int k = 0; k < K; ++k) {
    prod *= gamma[k];
    e += prod;
  }
  return e;
}

/* The estimator exactly as Thm 3 prints it:
 * sum_{k=1..K+1} k (1 - gamma_k) prod_{j=1..k-1} gamma_j,  gamma_{K+1} = 0. */
double orc_elen_thm3(const double* gamma, int K) {
  double e = 0.0;
  for (int k = 1; k <= K + 1; ++k) {
    double gk = (k <= K) ? gamma[k - 1] : 0.0;
    double prod = 1.0;
    for (int j = 1; j <= k - 1; ++j) prod *= gamma[j - 1];
    e += (double)k * (1.0 - gk) * prod;
  }
  return e;
}

/* Sec. 3.3 (chunk form, App. B.3): f = 1 - E_len / (K+1). */
double orc_loss_length(double e_len, int K) { return 1.0 - e_len / (double)(K + 1); }

/* App. B.3 acceptance-rate loss over a chunk of K drafted tokens:
 * f = (1/K) sum_{j=1..K} (1 - gamma_j). */
double orc_loss_accept(const double* gamma, int K) {
  double s = 0.0;
  for (int k = 0; k < K; ++k) s += 1.0 - gamma[k];
  return s / (double)K;
}

/* ---- whole feedback call ---------------------------------------------- */

/* target [B,P,V] (or, with path != NULL, a tree [B,M,V] whose rows
 * path[b*P+k] lie on the verified path), drafter [N,B,P,V].
 * Writes alpha [N,B,P] for every position and e_len [N,B] from
 * alpha_1..alpha_K, K = P-1 (gamma_{K+1} := 0 in Thm 3). */
static int feedback_impl(const void* target, const int32_t* path, int M,
                         const void* drafter, int dtype, int N, int B, int P,
                         int V, double T, int greedy, double* alpha,
                         double* e_len) {
  if (N < 1 || B < 1 || P < 1 || V < 1 || (!greedy && !(T > 0.0)))
    return ORC_BADARG;
  size_t esz = (dtype == ORC_FP32) ? 4 : 2;
  int status = ORC_OK;
  double* Pt = (double*)malloc(sizeof(double) * (size_t)V);
  double* Q = (double*)malloc(sizeof(double) * (size_t)V);
  for (int b = 0; b < B; ++b) {
    for (int k = 0; k < P; ++k) {
      int64_t trow = path ? ((int64_t)b * M + path[b * P + k]) : ((int64_t)b * P + k);
      if (path && (path[b * P + k] < 0 || path[b * P + k] >= M)) {
        free(Pt);
        free(Q);
        return ORC_BADARG;
      }
      const char* zt = (const char*)target + (size_t)trow * V * esz;
      int jt = -1, st_t = ORC_OK;
      if (greedy)
        jt = orc_row_argmax(zt, dtype, V);
      else
        st_t = orc_row_probs(zt, dtype, V, T, Pt);
      for (int i = 0; i < N; ++i) {
        int64_t drow = ((int64_t)i * B + b) * P + k;
        const char* zd = (const char*)drafter + (size_t)drow * V * esz;
        double a;
        if (greedy) {
          int jd = orc_row_argmax(zd, dtype, V);
          a = (jt < 0 || jd < 0) ? NAN : (jt == jd ? 1.0 : 0.0);
        } else {
          int st_d = orc_row_probs(zd, dtype, V, T, Q);
          a = (st_t || st_d) ? NAN : orc_overlap(Pt, Q, V);
        }
        if (isnan(a)) status = ORC_NONFINITE;
        alpha[drow] = a;
      }
    }
  }
  for (int i = 0; i < N; ++i)
    for (int b = 0; b < B; ++b)
      e_len[i * B + b] = orc_elen_prefix(alpha + ((size_t)i * B + b) * P, P - 1);
  free(Pt);
  free(Q);
  return status;
}

int orc_feedback(const void* target, const void* drafter, int dtype, int N,
                 int B, int P, int V, double T, int greedy, double* alpha,
                 double* e_len) {
  return feedback_impl(target, NULL, 0, drafter, dtype, N, B, P, V, T, greedy,
                       alpha, e_len);
}

int orc_feedback_path(const void* tree, const int32_t* path, int M,
                      const void* drafter, int dtype, int N, int B, int P,
                      int V, double T, int greedy, double* alpha,
                      double* e_len) {
  if (M < 1 || !path) return ORC_BADARG;
  return feedback_impl(tree, path, M, drafter, dtype, N, B, P, V, T, greedy,
                       alpha, e_len);
}

/* ---- Thm 2: EAGLE draft tree with branching L -------------------------- */

/* Top_L(q) of one drafter row: the L tokens the drafter ranks first.  The
 * ranking is by the stored logit (softmax at any temperature keeps the
 * order), larger first, ties toward the lower index; -inf logits rank last
 * (their q is 0) and NaN never occurs here (unusable rows are rejected).
 * Selection sort over the row, one pass per rank: plain and slow.  Writes
 * idx[0..L-1] in rank order; L is at most V. */
void orc_topl_set(const void* zd, int dtype, int V, int L, int* idx) {
  for (int r = 0; r < L; ++r) {
    int best = -1;
    double bz = 0.0;
    for (int v = 0; v < V; ++v) {
      int taken = 0;
      for (int q = 0; q < r; ++q)
        if (idx[q] == v) { taken = 1; break; }
      if (taken) continue;
      double z = orc_decode(zd, dtype, v);
      if (best < 0 || z > bz) { best = v; bz = z; }
    }
    idx[r] = best;
  }
}

/* alpha for one (target row, drafter row) pair under Thm 2: the target's
 * token is accepted iff it lies in the drafter's candidate set Top_L(q).
 * Stochastic target: alpha = sum_{v in Top_L(q)} p(v).  Greedy target:
 * alpha = 1[argmax p in Top_L(q)].  With L = 1 and a greedy target this is
 * the argmax-agreement rule of the greedy mode. */
int orc_alpha_topl(const void* zt, const void* zd, int dtype, int V, double T,
                   int greedy, int L, double* alpha) {
  if (L < 1) return ORC_BADARG;
  if (L > V) L = V;
  if (!row_ok(zd, dtype, V)) { *alpha = NAN; return ORC_NONFINITE; }
  int* idx = (int*)malloc(sizeof(int) * (size_t)L);
  orc_topl_set(zd, dtype, V, L, idx);
  int st = ORC_OK;
  if (greedy) {
    int jt = orc_row_argmax(zt, dtype, V);
    if (jt < 0) {
      *alpha = NAN;
      st = ORC_NONFINITE;
    } else {
      double a = 0.0;
      for (int r = 0; r < L; ++r)
        if (idx[r] == jt) a = 1.0;
      *alpha = a;
    }
  } else {
    double* Pt = (double*)malloc(sizeof(double) * (size_t)V);
    st = orc_row_probs(zt, dtype, V, T, Pt);
    double a = 0.0;
    for (int r = 0; r < L; ++r) a += Pt[idx[r]];
    *alpha = st ? NAN : a;
    free(Pt);
  }
  free(idx);
  return st;
}

/* A whole feedback call under Thm 2 (same layouts as orc_feedback /
 * orc_feedback_path; path == NULL for a chain target). */
int orc_feedback_topl(const void* target, const int32_t* path, int M,
                      const void* drafter, int dtype, int N, int B, int P,
                      int V, double T, int greedy, int L, double* alpha,
                      double* e_len) {
  if (N < 1 || B < 1 || P < 1 || V < 1 || L < 1 || (!greedy && !(T > 0.0)))
    return ORC_BADARG;
  if (path && M < 1) return ORC_BADARG;
  size_t esz = (dtype == ORC_FP32) ? 4 : 2;
  int status = ORC_OK;
  for (int b = 0; b < B; ++b) {
    for (int k = 0; k < P; ++k) {
      if (path && (path[b * P + k] < 0 || path[b * P + k] >= M)) return ORC_BADARG;
      int64_t row_t = (int64_t)b * P + k;               /* chain: target[b, k] */
      if (path) row_t = (int64_t)b * M + path[b * P + k];  /* tree: its path row */
      const char* zt = (const char*)target + (size_t)row_t * V * esz;
      for (int i = 0; i < N; ++i) {
        const int64_t row_d = ((int64_t)i * B + b) * P + k;  /* drafter[i, b, k] */
        const char* zd = (const char*)drafter + (size_t)row_d * V * esz;
        double a;
        if (orc_alpha_topl(zt, zd, dtype, V, T, greedy, L, &a) != ORC_OK) status = ORC_NONFINITE;
        alpha[row_d] = a;
      }
    }
  }
  for (int i = 0; i < N; ++i)
    for (int b = 0; b < B; ++b) {
      const double* gam = alpha + ((size_t)i * B + b) * P;  /* alpha_1..alpha_K */
      e_len[i * B + b] = orc_elen_prefix(gam, P - 1);
    }
  return status;
}

/* ---- Thm 2 with EAGLE-2's dynamic pruning ------------------------------ */

/* The remark closing Thm 2: when the draft tree is pruned, the candidate set
 * of a node is its pruned set of children instead of Top_L(q).  A node's
 * children are the drafter's L highest-ranked tokens and each is scored by
 * the node's own score times q(child), so pruning by score keeps a prefix of
 * that ranking: the first `keep` tokens of Top_L(q), 0 <= keep <= L (keep =
 * 0: every child was pruned and the target's token cannot be accepted).
 * alpha = sum over that prefix of p(v) (stochastic target) or 1[argmax p in
 * the prefix] (greedy target).  keep outside [0, L] is an argument error
 * (alpha NaN, ORC_BADARG); an unusable drafter or target row gives NaN and
 * ORC_NONFINITE. */
int orc_alpha_topl_pruned(const void* zt, const void* zd, int dtype, int V, double T,
                          int greedy, int L, int keep, double* alpha) {
  if (L < 1 || keep < 0 || keep > L) { *alpha = NAN; return ORC_BADARG; }
  if (!row_ok(zd, dtype, V)) { *alpha = NAN; return ORC_NONFINITE; }
  int n = L < V ? L : V;
  int* idx = (int*)malloc(sizeof(int) * (size_t)n);
  orc_topl_set(zd, dtype, V, n, idx);          /* Top_L(q), in rank order */
  int kept = keep < n ? keep : n;             /* the pruned set: idx[0..kept-1] */
  int st = ORC_OK;
  if (greedy) {
    int jt = orc_row_argmax(zt, dtype, V);
    if (jt < 0) {
      *alpha = NAN;
      st = ORC_NONFINITE;
    } else {
      double a = 0.0;
      for (int r = 0; r < kept; ++r)
        if (idx[r] == jt) a = 1.0;
      *alpha = a;
    }
  } else {
    double* Pt = (double*)malloc(sizeof(double) * (size_t)V);
    st = orc_row_probs(zt, dtype, V, T, Pt);
    double a = 0.0;
    for (int r = 0; r < kept; ++r) a += Pt[idx[r]];
    *alpha = st ? NAN : a;
    free(Pt);
  }
  free(idx);
  return st;
}

/* A whole pruned-tree feedback call: as orc_feedback_topl, with keep[N,B,P]
 * (element (i*B + b)*P + k) the number of children drafter i's tree kept at
 * the node of position k of query b.  Returns ORC_BADARG if any keep is out
 * of range (those alphas NaN), else ORC_NONFINITE if any row was unusable. */
int orc_feedback_topl_pruned(const void* target, const int32_t* path, int M,
                             const void* drafter, int dtype, int N, int B, int P,
                             int V, double T, int greedy, int L, const int32_t* keep,
                             double* alpha, double* e_len) {
  if (N < 1 || B < 1 || P < 1 || V < 1 || L < 1 || (!greedy && !(T > 0.0)))
    return ORC_BADARG;
  if (path && M < 1) return ORC_BADARG;
  size_t esz = (dtype == ORC_FP32) ? 4 : 2;
  int bad_keep = 0, bad_row = 0;
  for (int b = 0; b < B; ++b) {
    for (int k = 0; k < P; ++k) {
      if (path && (path[b * P + k] < 0 || path[b * P + k] >= M)) return ORC_BADARG;
      const int64_t row_tgt = path ? (int64_t)b * M + path[b * P + k]  /* tree: path row */
                                   : (int64_t)b * P + k;               /* chain: target[b, k] */
      const char* zt = (const char*)target + (size_t)row_tgt * V * esz;
      for (int i = 0; i < N; ++i) {
        const int64_t row_drf = ((int64_t)i * B + b) * P + k;  /* drafter[i, b, k] */
        const char* zd = (const char*)drafter + (size_t)row_drf * V * esz;
        double a;
        int st = orc_alpha_topl_pruned(zt, zd, dtype, V, T, greedy, L, keep[row_drf], &a);
        if (st == ORC_BADARG) bad_keep = 1;
        else if (st != ORC_OK) bad_row = 1;
        alpha[row_drf] = a;
      }
    }
  }
  for (int i = 0; i < N; ++i)
    for (int b = 0; b < B; ++b) {
      const double* gam = alpha + ((size_t)i * B + b) * P;  /* alpha_1..alpha_K */
      e_len[(size_t)i * B + b] = orc_elen_prefix(gam, P - 1);  /* Thm 3 */
    }
  return bad_keep ? ORC_BADARG : (bad_row ? ORC_NONFINITE : ORC_OK);
}

/* ---- learners ---------------------------------------------------------- */

/* Hedge (App. B.1 remark): starting from w = 1, w_i <- w_i exp(-eta l_i)
 * after every loss vector, so w_i = exp(-eta L_i) with L the cumulative loss;
 * Predict normalises.  exp(-eta (L_i - min L)) is the same vector up to the
 * common factor exp(eta min L).  The played drafter is the argmax of the
 * weights, i.e. the first argmin of L. */
void orc_hedge(const double* L, int N, double eta, double* w, int* sel) {
  int best = 0;
  for (int i = 1; i < N; ++i)
    if (L[i] < L[best]) best = i;
  double z = 0.0;
  for (int i = 0; i < N; ++i) {
    w[i] = exp(-eta * (L[i] - L[best]));
    z += w[i];
  }
  for (int i = 0; i < N; ++i) w[i] /= z;
  *sel = best;
}

/* (1/N) sum_i exp(([R_i]_+)^2 / (2c)) - e : the NormalHedge scale equation. */
static double nh_phi(const double* R, int N, double c) {
  double s = 0.0;
  for (int i = 0; i < N; ++i) {
    double r = R[i] > 0.0 ? R[i] : 0.0;
    s += exp(r * r / (2.0 * c));
  }
  return s / (double)N - exp(1.0);
}

/* NormalHedge, one round (App. D.6, Fig. "NormalHedge", steps 2-5).
 * p holds p_t on entry and p_{t+1} on exit; R holds R_{t-1} / R_t.
 * Steps 2-3 add l_A - l_i with l_A = sum_j p_j l_j.  Because sum_j p_j = 1
 * this increment is sum_j p_j (l_j - l_i), which is how it is evaluated: the
 * two agree to rounding, and this form is exactly 0 for a drafter whose loss
 * ties every other's (frequent with greedy feedback, whose losses are
 * quantised), where l_A - l_i would leave rounding noise that the scale
 * equation then amplifies.
 * If no regret is positive the scale equation has no root; p_{t+1} is then
 * uniform.  The played drafter is the argmax of p_{t+1}: the first argmax of
 * R when max R > 0 (p is strictly increasing in [R]_+ there and zero for
 * R <= 0), else drafter 0 (uniform weights, ties to the lowest index). */
int orc_normalhedge(double* R, const double* loss, double* p, int N, int* sel,
                    double* c_out) {
  for (int i = 0; i < N; ++i) {                      /* steps 2-3 */
    double inc = 0.0;
    for (int j = 0; j < N; ++j) inc += p[j] * (loss[j] - loss[i]);
    R[i] += inc;
  }
  int best = 0;
  for (int i = 1; i < N; ++i)
    if (R[i] > R[best]) best = i;
  double rmax = R[best];
  if (!(rmax > 0.0)) {
    for (int i = 0; i < N; ++i) p[i] = 1.0 / (double)N;
    *sel = 0;
    if (c_out) *c_out = NAN;
    return ORC_OK;
  }
  /* step 4: phi is strictly decreasing in c; phi(lo) >= 0 because the largest
   * term alone is N e there, phi(hi) <= 0 because every term is <= e there. */
  double lo = rmax * rmax / (2.0 * (1.0 + log((double)N)));
  double hi = rmax * rmax / 2.0;
  for (int it = 0; it < 400 && (hi - lo) > 1e-15 * hi; ++it) {
    double mid = 0.5 * (lo + hi);
    if (nh_phi(R, N, mid) > 0.0)
      lo = mid;
    else
      hi = mid;
  }
  double c = 0.5 * (lo + hi);
  double z = 0.0;                                    /* step 5 */
  for (int i = 0; i < N; ++i) {
    double r = R[i] > 0.0 ? R[i] : 0.0;
    p[i] = (r / c) * exp(r * r / (2.0 * c));
    z += p[i];
  }
  for (int i = 0; i < N; ++i) p[i] /= z;
  *sel = best;
  if (c_out) *c_out = c;
  return ORC_OK;
}

/* One learner round for B independent queries, arrays [N,B] (element i*B+b),
 * alpha [N,B,P], e_len [N,B].  loss_kind selects the Sec. 3.3 length loss or
 * the acceptance-rate loss; learner_kind selects Hedge (state = cumulative
 * loss L) or NormalHedge (state = cumulative regret R, weights = p_t in,
 * p_{t+1} out).  selected[b] holds the drafter played this round on entry
 * and the next round's choice on exit; when played != NULL, played[b]
 * accumulates f_t[i_t], the learner's own loss in the Sec. 3.1 regret. */
int orc_learner_step(const double* alpha, const double* e_len, int N, int B,
                     int P, int loss_kind, int learner_kind, double eta,
                     double* state, double* weights, double* loss_out,
                     int* selected, double* played) {
  int K = P - 1;
  if (N < 1 || B < 1 || P < 1) return ORC_BADARG;
  if (loss_kind == ORC_LOSS_ACCEPT && K < 1) return ORC_BADARG;
  double* f = (double*)malloc(sizeof(double) * (size_t)N);
  double* col = (double*)malloc(sizeof(double) * (size_t)N);
  double* w = (double*)malloc(sizeof(double) * (size_t)N);
  double* g = (double*)malloc(sizeof(double) * (size_t)(P > 0 ? P : 1));
  for (int b = 0; b < B; ++b) {
    for (int i = 0; i < N; ++i) {
      if (loss_kind == ORC_LOSS_LENGTH) {
        f[i] = orc_loss_length(e_len[i * B + b], K);
      } else {
        for (int k = 0; k < P; ++k) g[k] = alpha[((size_t)i * B + b) * P + k];
        f[i] = orc_loss_accept(g, K);
      }
      if (loss_out) loss_out[i * B + b] = f[i];
    }
    if (played) played[b] += f[selected[b]];
    for (int i = 0; i < N; ++i) col[i] = state[i * B + b];
    int sel = 0;
    if (learner_kind == ORC_HEDGE) {
      for (int i = 0; i < N; ++i) col[i] += f[i];
      orc_hedge(col, N, eta, w, &sel);
    } else {
      for (int i = 0; i < N; ++i) w[i] = weights[i * B + b];
      orc_normalhedge(col, f, w, N, &sel, NULL);
    }
    for (int i = 0; i < N; ++i) {
      state[i * B + b] = col[i];
      weights[i * B + b] = w[i];
    }
    selected[b] = sel;
  }
  free(f);
  free(col);
  free(w);
  free(g);
  return ORC_OK;
}

/* ---- App. B.1 (QFI-D): playing an action "according to p" -------------- */

/* A draw from the weights by the inverse CDF, with a uniform u in [0, 1)
 * supplied by the caller: the first i whose running sum w_0 + ... + w_i
 * exceeds u times the total.  This is an integer decided by floating-point
 * sums, so it is decided in the kernels' precision: fp32, both sums in index
 * order, the threshold u * total rounded once.  The running sum can first
 * exceed the threshold only where it grows, i.e. at a positive weight, so a
 * zero weight is never drawn; if rounding leaves every running sum at or
 * below the threshold (u next to 1), the last positive weight is drawn.
 * Returns -1 for unusable input: u outside [0, 1), a negative, NaN or
 * infinite weight, or no positive weight. */
int orc_sample_select(const float* w, int N, float u) {
  if (!(u >= 0.0f && u < 1.0f)) return -1;
  float total = 0.0f;
  for (int i = 0; i < N; ++i) {
    if (!(w[i] >= 0.0f) || isinf(w[i])) return -1;
    total += w[i];
  }
  if (!(total > 0.0f) || isinf(total)) return -1;
  const float thr = u * total;
  float run = 0.0f;
  int last_pos = -1;
  for (int i = 0; i < N; ++i) {
    run += w[i];
    if (w[i] > 0.0f) last_pos = i;
    if (run > thr) return i;
  }
  return last_pos;
}

/* ---- App. B.3 chunk-level game with a chunk horizon k_h ----------------- */

/* The losses of one chunk whose chosen drafter had k accepted draft tokens:
 * Thm 3 with K = k (gamma_1..gamma_k, gamma_{k+1} := 0), and the acceptance
 * rate over the k tokens.  The positions after k were not verified (the
 * censoring of Sec. 3.2) and are not read.  k = 0 carries no information:
 * both losses are 0 (E_len = 1 = K+1, and an empty average is taken as 0). */
double orc_chunk_loss(const double* gamma, int k, int loss_kind) {
  if (k <= 0) return 0.0;
  if (loss_kind == ORC_LOSS_LENGTH) return orc_loss_length(orc_elen_prefix(gamma, k), k);
  return orc_loss_accept(gamma, k);
}

/* Base.Update with one loss vector for one query, then Base.Predict (App.
 * B.1, QFI-D): Hedge keeps the cumulative loss in st and forms w from it;
 * NormalHedge keeps the regret in st and w = p_t in, p_{t+1} out. */
static void base_update(int learner_kind, double eta, const double* lv, double* st, double* wt,
                        int N, int* choice) {
  if (learner_kind == ORC_HEDGE) {
    for (int i = 0; i < N; ++i) st[i] = st[i] + lv[i];
    orc_hedge(st, N, eta, wt, choice);
  } else {
    orc_normalhedge(st, lv, wt, N, choice, NULL);
  }
}

/* One chunk-level round for B queries (arrays [N,B], alpha [N,B,P]) when
 * query b's chosen drafter had k_h[b] accepted draft tokens, 0 <= k_h[b] <=
 * P-1; otherwise as orc_learner_step (loss_out, selected and played alike). */
int orc_chunk_learner_step(const double* alpha, int N, int B, int P, const int* k_h,
                           int loss_kind, int learner_kind, double eta, double* state,
                           double* weights, double* loss_out, int* selected, double* played) {
  if (N < 1 || B < 1 || P < 1) return ORC_BADARG;
  for (int b = 0; b < B; ++b)
    if (k_h[b] < 0 || k_h[b] > P - 1) return ORC_BADARG;
  double* lv = (double*)malloc(sizeof(double) * (size_t)N);
  double* st = (double*)malloc(sizeof(double) * (size_t)N);
  double* wt = (double*)malloc(sizeof(double) * (size_t)N);
  double* gm = (double*)malloc(sizeof(double) * (size_t)P);
  for (int b = 0; b < B; ++b) {
    for (int i = 0; i < N; ++i) {
      for (int k = 0; k < P; ++k) gm[k] = alpha[((size_t)i * B + b) * P + k];
      lv[i] = orc_chunk_loss(gm, k_h[b], loss_kind);
      if (loss_out) loss_out[i * B + b] = lv[i];
      st[i] = state[i * B + b];
      wt[i] = weights[i * B + b];
    }
    if (played) played[b] = played[b] + lv[selected[b]];
    int choice = 0;
    base_update(learner_kind, eta, lv, st, wt, N, &choice);
    for (int i = 0; i < N; ++i) {
      state[i * B + b] = st[i];
      weights[i * B + b] = wt[i];
    }
    selected[b] = choice;
  }
  free(lv);
  free(st);
  free(wt);
  free(gm);
  return ORC_OK;
}

/* ---- Sec. 3.2 token-level game with delay, through QFI-D (App. B.1) ----- */

/* The loss of choosing drafter i at token s (0-based) of a query's token
 * stream g_i[0..]: the acceptance-rate loss 1 - g_i[s], or the length loss
 * of a K-token draft starting at s, 1 - E/(K+1) with E from g_i[s..s+K-1]
 * (Thm 3). */
double orc_token_loss(const double* g, int64_t s, int K, int loss_kind) {
  if (loss_kind == ORC_LOSS_ACCEPT) return 1.0 - g[s];
  return orc_loss_length(orc_elen_prefix(g + s, K), K);
}

/* How many of a stream's first n tokens have a revealed loss (Fig. "Token-
 * Level Game with Delay"): at the end of a chunk that ends at token n (1-
 * based), f_{<=n} is revealed for the acceptance-rate loss and f_{<=n-K} for
 * the length loss.  With hybrid losses (App. B.5) the first `accept_first`
 * tokens use the acceptance-rate loss, the rest loss_kind. */
int64_t orc_token_revealed(int64_t n, int K, int loss_kind, int64_t accept_first) {
  int64_t late = (loss_kind == ORC_LOSS_LENGTH) ? n - K : n;
  if (late < 0) late = 0;
  int64_t early = n < accept_first ? n : accept_first;
  return late > early ? late : early;
}

/* A whole token-level session for B queries through QFI-D.  For chunk h =
 * 0..H-1 and every query b:
 *   1. catch up: pop every revealed, unprocessed token loss in token order
 *      (FIFO) and feed it to Base (Update, then Predict);
 *   2. play: sel[h*B+b] = Base's choice (the last Update's Predict; with no
 *      Update yet, the caller's initial choice sel0[b]);
 *   3. the chunk's k_h[h*B+b]+1 verified tokens join the stream, with
 *      gamma = alpha[h] at positions 0..k_h of (i, b), each recorded as
 *      played by sel[h*B+b].
 * alpha [H,N,B,P] (gamma of drafter i at position k of chunk h, b),
 * k_h [H,B] in 0..P-1; state/weights [N,B] as in orc_learner_step (initial
 * values in, final out); played [B] (or NULL) += f_s[drafter that played s]
 * for every processed token s; processed [B] (or NULL) = tokens processed. */
int orc_token_session(const double* alpha, const int* k_h, int H, int N, int B, int P, int K,
                      int loss_kind, int64_t accept_first, int learner_kind, double eta,
                      double* state, double* weights, const int* sel0, int* sel, double* played,
                      int64_t* processed) {
  if (N < 1 || B < 1 || P < 1 || H < 0 || K < 1) return ORC_BADARG;
  for (int64_t x = 0; x < (int64_t)H * B; ++x)
    if (k_h[x] < 0 || k_h[x] > P - 1) return ORC_BADARG;
  const int64_t cap = (int64_t)H * P + 1;
  double* stream = (double*)malloc(sizeof(double) * (size_t)(N * cap));
  int* who = (int*)malloc(sizeof(int) * (size_t)cap);
  double* lv = (double*)malloc(sizeof(double) * (size_t)N);
  double* st = (double*)malloc(sizeof(double) * (size_t)N);
  double* wt = (double*)malloc(sizeof(double) * (size_t)N);
  for (int b = 0; b < B; ++b) {
    int64_t n = 0, done = 0;
    int choice = sel0[b];
    for (int i = 0; i < N; ++i) {
      st[i] = state[i * B + b];
      wt[i] = weights[i * B + b];
    }
    double own = 0.0;
    for (int h = 0; h < H; ++h) {
      const int64_t ready = orc_token_revealed(n, K, loss_kind, accept_first);
      for (; done < ready; ++done) {
        const int kind = done < accept_first ? ORC_LOSS_ACCEPT : loss_kind;
        for (int i = 0; i < N; ++i) lv[i] = orc_token_loss(stream + (size_t)i * cap, done, K, kind);
        own += lv[who[done]];
        base_update(learner_kind, eta, lv, st, wt, N, &choice);
      }
      sel[(size_t)h * B + b] = choice;
      const int kk = k_h[(size_t)h * B + b];
      for (int k = 0; k <= kk; ++k) {
        for (int i = 0; i < N; ++i)
          stream[(size_t)i * cap + n] = alpha[(((size_t)h * N + i) * B + b) * P + k];
        who[n] = choice;
        ++n;
      }
    }
    for (int i = 0; i < N; ++i) {
      state[i * B + b] = st[i];
      weights[i * B + b] = wt[i];
    }
    if (played) played[b] += own;
    if (processed) processed[b] = done;
  }
  free(stream);
  free(who);
  free(lv);
  free(st);
  free(wt);
  return ORC_OK;
}

/* ---- App. B.5 practical heuristics: warm-up, batched and skipped updates,
 * hybrid losses -------------------------------------------------------------- */

/* QFI-D's catch-up over a batch of chunk-level loss vectors: the `count`
 * vectors lv[c][N][B] are fed to Base in order (c = 0 first), one round each,
 * for every query; state/weights/selected as in orc_learner_step. */
int orc_learner_apply(const double* lv, int count, int N, int B, int learner_kind, double eta,
                      double* state, double* weights, int* selected) {
  if (N < 1 || B < 1 || count < 0) return ORC_BADARG;
  double* one = (double*)malloc(sizeof(double) * (size_t)N);
  double* st = (double*)malloc(sizeof(double) * (size_t)N);
  double* wt = (double*)malloc(sizeof(double) * (size_t)N);
  for (int b = 0; b < B; ++b) {
    for (int i = 0; i < N; ++i) {
      st[i] = state[i * B + b];
      wt[i] = weights[i * B + b];
    }
    int choice = selected[b];
    for (int c = 0; c < count; ++c) {
      for (int i = 0; i < N; ++i) one[i] = lv[((size_t)c * N + i) * B + b];
      base_update(learner_kind, eta, one, st, wt, N, &choice);
    }
    for (int i = 0; i < N; ++i) {
      state[i * B + b] = st[i];
      weights[i * B + b] = wt[i];
    }
    selected[b] = choice;
  }
  free(one);
  free(st);
  free(wt);
  return ORC_OK;
}

/* The schedule of App. B.5, read as follows.  A round is one speculative
 * chunk, after which the schedule decides:
 *   - during the first warmup rounds: evaluate every drafter on the chunk
 *     (panoramic feedback, one loss vector) and apply it at once (full
 *     information every round);
 *   - afterwards, "skipping updates by a fixed number of tokens": evaluate
 *     only when at least skip_tokens tokens were generated since the last
 *     evaluation (counting this chunk's), and "delayed batched feedback":
 *     queue the vectors and apply the queue (FIFO, QFI-D) once every
 *     batch_rounds rounds after the warm-up;
 *   - "hybrid losses": the first hybrid_vectors loss vectors use the
 *     acceptance-rate loss, later ones the length loss.
 * State: s[0] rounds so far, s[1] tokens since the last evaluation, s[2]
 * vectors made, s[3] vectors queued and not applied.  Outputs: act[0]
 * evaluate, act[1] the loss kind of that vector, act[2] apply the queue
 * (including this round's vector) before the next choice. */
int orc_schedule_next(int warmup, int batch_rounds, int skip_tokens, int hybrid_vectors,
                      int64_t* s, int tokens, int* act) {
  if (warmup < 0 || batch_rounds < 1 || skip_tokens < 0 || hybrid_vectors < 0 || tokens < 0)
    return ORC_BADARG;
  const int64_t r = s[0];
  int evaluate, apply;
  if (r < warmup) {
    evaluate = 1;
    apply = 1;
    s[1] = 0;
  } else {
    s[1] += tokens;
    evaluate = s[1] >= skip_tokens;
    if (evaluate) s[1] = 0;
    apply = ((r - warmup + 1) % batch_rounds) == 0;
  }
  act[0] = evaluate;
  act[1] = (evaluate && s[2] < hybrid_vectors) ? ORC_LOSS_ACCEPT : ORC_LOSS_LENGTH;
  if (evaluate) {
    s[2] += 1;
    s[3] += 1;
  }
  act[2] = apply && s[3] > 0;
  if (act[2]) s[3] = 0;
  s[0] = r + 1;
  return ORC_OK;
}
