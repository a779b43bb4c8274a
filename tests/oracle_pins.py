"""Pins for the fp64 oracle: facts the paper and the mathematics fix.

Every ``check_*`` takes an ``oracle.Oracle`` and raises AssertionError when
the oracle disagrees with the fact it checks.  ``test_oracle_pins.py`` runs
them against the oracle as built; ``test_oracle_mutants.py`` runs them
against copies of the oracle with one planted mistake each and expects at
least one check to fail for every mistake.

Nothing here re-types an oracle formula: probabilities come from
``scipy.special.softmax``, bf16/fp16 decoding from numpy bit operations and
numpy's float16, and the remaining checks use closed forms, invariants,
the paper's worked example and Monte-Carlo runs of the speculative-decoding
rule (Sec. 2.2).
"""
from __future__ import annotations

import json
import math
import os

import numpy as np
from scipy.special import softmax
from scipy.stats import chi2

import oracle as orc

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


# ---- helpers (independent of the oracle) ---------------------------------

def bf16_bits(x) -> np.ndarray:
    """fp32 -> bf16 bit pattern, round to nearest even (finite inputs)."""
    u = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


def bf16_value(bits) -> np.ndarray:
    with np.errstate(invalid="ignore"):  # signalling-NaN patterns widen to NaN
        return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def stored(z, kind: str) -> np.ndarray:
    z = np.asarray(z, np.float32)
    if kind == "bf16":
        return bf16_bits(z)
    if kind == "fp16":
        return z.astype(np.float16)
    return z


def value(s: np.ndarray) -> np.ndarray:
    if s.dtype == np.uint16:
        return bf16_value(s)
    return s.astype(np.float64)


def probs(s: np.ndarray, T: float) -> np.ndarray:
    return softmax(value(s) / T)


KINDS = ("bf16", "fp16", "fp32")


# ---- decoding --------------------------------------------------------------

def check_decode_all_16bit(o):
    """Every bf16 and fp16 bit pattern decodes to its exact value."""
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    want_bf = bf16_value(bits)
    want_h = bits.view(np.float16).astype(np.float64)
    for arr, want in ((bits, want_bf), (bits.view(np.float16), want_h)):
        got = o.decode(arr)
        fin = ~np.isnan(want)
        assert np.array_equal(got[fin], want[fin])
        assert np.all(np.isnan(got[~fin]))


# ---- Thm 1: alpha = sum min(p, q) = 1 - TV ----------------------------------

def check_identical_rows(o):
    rng = np.random.default_rng(1)
    for kind in KINDS:
        z = stored(rng.normal(0, 3, 257), kind)
        for T in (0.5, 1.0, 2.0):
            a, st = o.alpha_pair(z, z, T, False)
            assert st == orc.OK and abs(a - 1.0) < 1e-12


def check_disjoint_supports(o):
    """Complementary -inf masks: p and q share no support, so alpha = 0 exactly."""
    rng = np.random.default_rng(2)
    V = 64
    zt = rng.normal(0, 2, V).astype(np.float32)
    zd = rng.normal(0, 2, V).astype(np.float32)
    zt[1::2] = -np.inf
    zd[0::2] = -np.inf
    for kind in KINDS:
        a, st = o.alpha_pair(stored(zt, kind), stored(zd, kind), 1.0, False)
        assert st == orc.OK and a == 0.0


def check_one_minus_tv(o):
    """alpha equals 1 - TV(p, q) with p, q from scipy's softmax at z/T."""
    rng = np.random.default_rng(3)
    for kind in KINDS:
        for V in (1, 2, 7, 100, 1000):
            for T in (0.3, 0.7, 1.0, 2.5):
                zt = stored(rng.normal(0, 3, V), kind)
                zd = stored(value(zt) + rng.normal(0, 1.5, V), kind)
                p, q = probs(zt, T), probs(zd, T)
                want = 1.0 - 0.5 * np.abs(p - q).sum()
                a, st = o.alpha_pair(zt, zd, T, False)
                assert st == orc.OK and abs(a - want) < 1e-12, (kind, V, T, a, want)


def check_row_probs(o):
    rng = np.random.default_rng(4)
    for kind in KINDS:
        z = stored(rng.normal(0, 4, 300), kind)
        P, st = o.row_probs(z, 0.7)
        assert st == orc.OK
        assert np.allclose(P, probs(z, 0.7), rtol=1e-12, atol=1e-300)


def check_tv_function(o):
    rng = np.random.default_rng(5)
    p = softmax(rng.normal(size=50))
    q = softmax(rng.normal(size=50))
    assert abs(o.tv(p, q) - (1.0 - np.minimum(p, q).sum())) < 1e-13
    assert abs(o.overlap(p, q) + o.tv(p, q) - 1.0) < 1e-13


def check_symmetry_and_shift(o):
    rng = np.random.default_rng(6)
    zt = (rng.integers(-64, 64, 200) / 16.0).astype(np.float32)
    zd = (rng.integers(-64, 64, 200) / 16.0).astype(np.float32)
    a, _ = o.alpha_pair(zt, zd, 0.9, False)
    b, _ = o.alpha_pair(zd, zt, 0.9, False)
    c, _ = o.alpha_pair(zt + np.float32(8.0), zd - np.float32(3.0), 0.9, False)
    assert abs(a - b) < 1e-13 and abs(a - c) < 1e-13


def check_mc_accept_reject(o):
    """Monte Carlo of the Sec. 2.2 rule on V = 6: the empirical acceptance rate
    matches alpha (Thm 1) within 5 sigma and the emitted token follows p."""
    rng = np.random.default_rng(7)
    V, n = 6, 400_000
    zt = rng.normal(0, 1.5, V).astype(np.float32)
    zd = rng.normal(0, 1.5, V).astype(np.float32)
    T = 0.8
    p, q = probs(zt, T), probs(zd, T)
    a, st = o.alpha_pair(zt, zd, T, False)
    assert st == orc.OK
    draft = rng.choice(V, size=n, p=q)
    acc = rng.random(n) < p[draft] / q[draft]
    rate = acc.mean()
    sigma = math.sqrt(a * (1 - a) / n)
    assert abs(rate - a) < 5 * sigma + 1e-12, (rate, a, sigma)
    resid = np.maximum(p - q, 0.0)
    resid /= resid.sum()
    out = np.where(acc, draft, rng.choice(V, size=n, p=resid))
    counts = np.bincount(out, minlength=V)
    stat = ((counts - n * p) ** 2 / (n * p)).sum()
    assert stat < chi2.ppf(1 - 1e-6, V - 1), stat


# ---- greedy: Thm 2 with L = 1 under a greedy target --------------------------

def check_greedy_matches_argmax(o):
    rng = np.random.default_rng(8)
    for kind in KINDS:
        for _ in range(50):
            V = int(rng.integers(1, 40))
            zt = stored(rng.integers(-4, 4, V).astype(np.float32), kind)  # many ties
            zd = stored(rng.integers(-4, 4, V).astype(np.float32), kind)
            want = 1.0 if np.argmax(value(zt)) == np.argmax(value(zd)) else 0.0
            a, st = o.alpha_pair(zt, zd, 1.0, True)
            assert st == orc.OK and a == want


def check_greedy_ties_lowest_index(o):
    row = np.array([1.0, 3.0, 3.0, 2.0], np.float32)
    assert o.row_argmax(row) == 1
    assert o.row_argmax(np.array([-0.0, 0.0, -1.0], np.float32)) == 0
    assert o.row_argmax(np.array([-np.inf, -5.0, -5.0], np.float32)) == 1
    a, _ = o.alpha_pair(row, np.array([0, 5, 5, 0], np.float32), 1.0, True)
    assert a == 1.0
    a, _ = o.alpha_pair(row, np.array([0, 4, 5, 0], np.float32), 1.0, True)
    assert a == 0.0


def check_small_temperature_limit(o):
    """With a clear top-1 gap, stochastic alpha at T -> 0 tends to greedy alpha."""
    rng = np.random.default_rng(9)
    seen = set()
    for trial in range(20):
        V = 50
        zt = rng.normal(0, 1, V).astype(np.float32)
        zd = rng.normal(0, 1, V).astype(np.float32)
        top = int(rng.integers(V))
        zt[top] += 20.0
        zd[top if trial % 2 == 0 else (top + 1 + int(rng.integers(V - 1))) % V] += 20.0
        g, _ = o.alpha_pair(zt, zd, 1.0, True)
        s, _ = o.alpha_pair(zt, zd, 0.02, False)
        assert abs(g - s) < 1e-6
        seen.add(g)
    assert seen == {0.0, 1.0}


def check_nonfinite_rows(o):
    good = np.array([0.0, 1.0, 2.0], np.float32)
    for bad in ([np.nan, 0.0, 1.0], [np.inf, 0.0, 1.0], [-np.inf] * 3):
        bad = np.array(bad, np.float32)
        for greedy in (False, True):
            a, st = o.alpha_pair(good, bad, 1.0, greedy)
            assert st == orc.NONFINITE and math.isnan(a)
    a, st = o.alpha_pair(good, np.array([-np.inf, 0.0, 1.0], np.float32), 1.0, False)
    assert st == orc.OK and 0.0 < a < 1.0


# ---- Thm 3: acceptance-length estimator --------------------------------------

def check_elen_constant_alpha(o):
    """Constant gamma = a: 1 + a + ... + a^K = (1 - a^{K+1}) / (1 - a)."""
    for K in (0, 1, 2, 5, 8):
        for a in (0.0, 0.25, 0.6, 0.95, 1.0):
            want = K + 1.0 if a == 1.0 else (1 - a ** (K + 1)) / (1 - a)
            g = [a] * K
            assert abs(o.elen_prefix(g) - want) < 1e-12
            assert abs(o.elen_thm3(g) - want) < 1e-12


def check_elen_forms_and_range(o):
    rng = np.random.default_rng(10)
    for K in range(0, 10):
        for _ in range(20):
            g = rng.random(K)
            e1, e2 = o.elen_prefix(g), o.elen_thm3(g)
            assert abs(e1 - e2) < 1e-12
            assert 1.0 - 1e-15 <= e1 <= K + 1 + 1e-12


def check_worked_example(o):
    with open(os.path.join(GOLDEN, "censoring_example.json")) as f:
        ex = json.load(f)
    for case in ex["cases"]:
        assert len(case["gamma"]) == case["K"]
        assert abs(o.elen_thm3(case["gamma"]) - case["expected_accept_length"]) < 1e-12
        assert abs(o.elen_prefix(case["gamma"]) - case["expected_accept_length"]) < 1e-12


def check_mc_chunk_length(o):
    """Monte Carlo of one speculative-decoding chunk (Sec. 2.2) with fixed
    per-position (p_k, q_k): the mean number of tokens a chunk emits (accepted
    drafts + the resampled or bonus token) matches e_len within 5 sigma.
    Position-wise distributions that do not depend on the realised prefix are
    the case in which the product form of Thm 3 is exact."""
    rng = np.random.default_rng(11)
    K, V, n, T = 4, 5, 300_000, 1.0
    tgt = rng.normal(0, 1.2, (1, K + 1, V)).astype(np.float32)
    drf = (tgt[None] + rng.normal(0, 0.8, (1, 1, K + 1, V))).astype(np.float32)
    alpha, e_len, st = o.feedback(tgt, drf, T, False)
    assert st == orc.OK
    emitted = np.ones(n)
    alive = np.ones(n, bool)
    for k in range(K):
        p, q = probs(tgt[0, k], T), probs(drf[0, 0, k], T)
        draft = rng.choice(V, size=n, p=q)
        alive &= rng.random(n) < p[draft] / q[draft]
        emitted += alive
    sd = emitted.std() / math.sqrt(n)
    assert abs(emitted.mean() - e_len[0, 0]) < 5 * sd, (emitted.mean(), e_len[0, 0], sd)


def check_losses(o):
    """Sec. 3.3: the length loss is 0 for a drafter that always reaches K+1
    and 1 - 1/(K+1) for one that never passes a draft; the accept-rate loss
    is 0 / 1 at gamma = 1 / 0 and lies in [0, 1]."""
    for K in (1, 3, 8):
        assert abs(o.loss_length(o.elen_prefix([1.0] * K), K)) < 1e-15
        assert abs(o.loss_length(o.elen_prefix([0.0] * K), K) - (1 - 1 / (K + 1))) < 1e-15
        assert abs(o.loss_accept([1.0] * K)) < 1e-15
        assert abs(o.loss_accept([0.0] * K) - 1.0) < 1e-15
        g = np.linspace(0.1, 0.9, K)
        assert abs(o.loss_accept(g) - (1 - g.mean())) < 1e-15


# ---- feedback call layout ------------------------------------------------------

def check_feedback_layout(o):
    """alpha[i,b,k] pairs target row (b,k) with drafter row (i,b,k)."""
    rng = np.random.default_rng(12)
    N, B, P, V, T = 3, 2, 4, 16, 0.9
    for kind in KINDS:
        tgt = stored(rng.normal(0, 2, (B, P, V)), kind)
        drf = stored(value(tgt)[None] + rng.normal(0, 1 + np.arange(N)[:, None, None, None],
                                                    (N, B, P, V)), kind)
        alpha, e_len, st = o.feedback(tgt, drf, T, False)
        assert st == orc.OK
        for i in range(N):
            for b in range(B):
                for k in range(P):
                    p, q = probs(tgt[b, k], T), probs(drf[i, b, k], T)
                    assert abs(alpha[i, b, k] - (1 - 0.5 * np.abs(p - q).sum())) < 1e-12
                assert abs(e_len[i, b] - o.elen_thm3(alpha[i, b, :P - 1])) < 1e-12
        ga, ge, st = o.feedback(tgt, drf, T, True)
        for i in range(N):
            for b in range(B):
                for k in range(P):
                    want = float(np.argmax(value(tgt[b, k])) == np.argmax(value(drf[i, b, k])))
                    assert ga[i, b, k] == want


def check_feedback_path(o):
    """The tree form reads target rows path[b,k] of a [B,M,V] tensor."""
    rng = np.random.default_rng(13)
    N, B, P, M, V = 2, 3, 4, 11, 24
    tree = rng.normal(0, 2, (B, M, V)).astype(np.float32)
    path = np.stack([rng.choice(M, P, replace=False) for _ in range(B)]).astype(np.int32)
    gathered = np.stack([tree[b, path[b]] for b in range(B)])
    drf = (gathered[None] + rng.normal(0, 1, (N, B, P, V))).astype(np.float32)
    a1, e1, _ = o.feedback(tree, drf, 1.0, False, path=path)
    for i in range(N):
        for b in range(B):
            for k in range(P):
                p, q = probs(gathered[b, k], 1.0), probs(drf[i, b, k], 1.0)
                assert abs(a1[i, b, k] - (1 - 0.5 * np.abs(p - q).sum())) < 1e-12


# ---- Hedge (App. B.1 remark) ----------------------------------------------------

def check_hedge_multiplicative(o):
    """Sequential w <- w exp(-eta l), normalised, equals the oracle's weights
    from the cumulative loss; the choice is the first argmax of the weights."""
    rng = np.random.default_rng(14)
    N, eta = 6, 0.37
    w = np.ones(N) / N
    L = np.zeros(N)
    for t in range(60):
        f = rng.random(N)
        w = w * np.exp(-eta * f)
        w /= w.sum()
        L += f
        got, sel = o.hedge(L, eta)
        assert np.allclose(got, w, rtol=1e-10, atol=0)
        assert sel == int(np.argmax(w))
    got, sel = o.hedge(np.zeros(N), eta)
    assert np.allclose(got, 1.0 / N) and sel == 0
    # the same run through the batched learner round (state = cumulative loss)
    w = np.ones(N) / N
    state, weights, sel = np.zeros((N, 1)), np.full((N, 1), 1.0 / N), np.zeros(1, np.int32)
    for t in range(40):
        f = rng.random(N)
        w = w * np.exp(-eta * f)
        w /= w.sum()
        state, weights, _, sel, _ = o.learner_step(np.zeros((N, 1, 2)), 2.0 * (1.0 - f[:, None]),
                                                   orc.LOSS_LENGTH, orc.HEDGE, eta, state,
                                                   weights, sel)
        assert np.allclose(weights[:, 0], w, rtol=1e-10, atol=0)
        assert sel[0] == int(np.argmax(w))


def _hedge_regret(o, losses, eta):
    T, N = losses.shape
    state = np.zeros((N, 1))
    weights = np.full((N, 1), 1.0 / N)
    sel = np.zeros(1, np.int32)
    exp_loss = 0.0
    for t in range(T):
        f = losses[t][:, None]
        exp_loss += float((weights[:, 0] * f[:, 0]).sum())
        # length loss with P = 1 is identically 0, so feed the loss through
        # e_len: f = 1 - e_len / (K+1) with K = 1  =>  e_len = 2 (1 - f)
        alpha = np.zeros((N, 1, 2))
        state, weights, loss, sel, _ = o.learner_step(alpha, 2.0 * (1.0 - f), orc.LOSS_LENGTH,
                                                      orc.HEDGE, eta, state, weights, sel)
        assert np.allclose(loss, f, atol=1e-15)
    return exp_loss - losses.sum(axis=0).min()


def check_hedge_regret_bound(o):
    """Hedge's expected regret obeys ln N / eta + eta T / 8 (here 45.6 for
    N = 8, T = 2000, eta = sqrt(8 ln N / T)) on a switching-expert sequence."""
    rng = np.random.default_rng(15)
    N, T = 8, 2000
    eta = math.sqrt(8 * math.log(N) / T)
    losses = rng.random((T, N)) * 0.6 + 0.2
    for t in range(T):
        losses[t, (t // 250) % N] = rng.random() * 0.2
    reg = _hedge_regret(o, losses, eta)
    assert reg <= math.log(N) / eta + eta * T / 8


# ---- NormalHedge (App. D.6 figure) --------------------------------------------

def check_normalhedge_closed_form(o):
    """k experts share regret r > 0, the rest are negative: the scale is
    c = r^2 / (2 ln((N (e-1) + k) / k)) and those k weights are 1/k each."""
    for N, k, r in ((8, 1, 3.0), (8, 3, 0.7), (16, 5, 12.0), (2, 2, 0.01)):
        R = np.full(N, -1.0)
        R[:k] = r
        Rn, p, sel, c = o.normalhedge(R, np.zeros(N), np.full(N, 1.0 / N))
        want = r * r / (2 * math.log((N * (math.e - 1) + k) / k))
        assert abs(c - want) < 1e-12 * want
        assert np.allclose(p[:k], 1.0 / k, rtol=1e-12) and np.all(p[k:] == 0.0)
        assert sel == 0


def check_normalhedge_equation(o):
    """For random regrets the returned c solves (1/N) sum exp([R]_+^2/2c) = e,
    and p is proportional to the gradient of that potential in R."""
    rng = np.random.default_rng(16)
    for _ in range(30):
        N = int(rng.integers(2, 33))
        R0 = rng.normal(0, 3, N)
        loss = rng.random(N)
        p0 = rng.dirichlet(np.ones(N))
        R, p, sel, c = o.normalhedge(R0, loss, p0)
        if R.max() <= 0:
            continue
        Rp = np.maximum(R, 0)
        assert abs(np.exp(Rp ** 2 / (2 * c)).mean() - math.e) < 1e-12
        phi = lambda x: np.exp(np.maximum(x, 0) ** 2 / (2 * c)).sum()
        h = 1e-6
        grad = np.array([(phi(R + h * np.eye(N)[i]) - phi(R - h * np.eye(N)[i])) / (2 * h)
                         for i in range(N)])
        assert np.allclose(p, grad / grad.sum(), rtol=1e-5, atol=1e-9)
        assert sel == int(np.argmax(R))


def check_normalhedge_regret_update(o):
    """Step 3: R_i += l_A - l_i with l_A = sum p_i l_i, so the p-weighted
    increments vanish and increments differ by the loss differences."""
    rng = np.random.default_rng(17)
    N = 7
    R0 = rng.normal(0, 1, N)
    loss = rng.random(N)
    p0 = rng.dirichlet(np.ones(N))
    R, _, _, _ = o.normalhedge(R0, loss, p0)
    d = R - R0
    assert abs((p0 * d).sum()) < 1e-14
    assert np.allclose(d[:, None] - d[None, :], loss[None, :] - loss[:, None], atol=1e-14)


def check_normalhedge_uniform(o):
    """No positive regret: the scale equation has no root and p is uniform;
    the initial state (R = 0, p = 1/N) stays there under equal losses."""
    N = 5
    R, p, sel, c = o.normalhedge(np.zeros(N), np.full(N, 0.4), np.full(N, 1.0 / N))
    assert np.allclose(p, 1.0 / N) and sel == 0 and np.all(R == 0)
    R, p, sel, c = o.normalhedge(np.array([-3.0, -1.0, -2.0, -0.5, -4.0]), np.zeros(N),
                                 np.full(N, 1.0 / N))
    assert np.allclose(p, 1.0 / N) and sel == 0
    R, p, sel, c = o.normalhedge(np.zeros(1), np.array([0.3]), np.ones(1))
    assert p[0] == 1.0 and sel == 0


def check_learner_step_played_loss(o):
    """played[b] accumulates f_t[i_t] for the drafter chosen before round t."""
    rng = np.random.default_rng(18)
    N, B, P = 4, 3, 3
    state = np.zeros((N, B))
    weights = np.full((N, B), 1.0 / N)
    sel = np.array([2, 0, 3], np.int32)
    played = np.zeros(B)
    alpha = rng.random((N, B, P))
    e_len = np.array([[o.elen_prefix(alpha[i, b, :P - 1]) for b in range(B)] for i in range(N)])
    for learner in (orc.HEDGE, orc.NORMALHEDGE):
        for loss_kind in (orc.LOSS_LENGTH, orc.LOSS_ACCEPT):
            s2, w2, loss, sel2, pl = o.learner_step(alpha, e_len, loss_kind, learner, 0.5,
                                                     state, weights, sel, played)
            assert np.allclose(pl, loss[sel, np.arange(B)], atol=1e-15)
            if loss_kind == orc.LOSS_ACCEPT:
                assert np.allclose(loss, 1 - alpha[:, :, :P - 1].mean(axis=2), atol=1e-15)
            else:
                assert np.allclose(loss, 1 - e_len / P, atol=1e-15)
            if learner == orc.HEDGE:
                assert np.allclose(s2, loss, atol=1e-15)
                assert np.array_equal(sel2, np.argmin(loss, axis=0))
            assert np.allclose(w2.sum(axis=0), 1.0)


# ---- Thm 2: EAGLE tree with branching L ----------------------------------------

def topl_numpy(stored_row: np.ndarray, L: int) -> np.ndarray:
    """The L tokens ranked first by stored logit, ties toward the lower index
    (numpy lexsort: primary key -value, secondary key the index)."""
    z = value(stored_row)
    order = np.lexsort((np.arange(z.size), -z))
    return order[:min(L, z.size)]


def check_topl_set_lexsort(o):
    """Top_L on tie-heavy rows (logits on a 1/4 grid, some -inf) equals the
    lexsort ranking, for every L."""
    rng = np.random.default_rng(41)
    for kind in KINDS:
        for V in (1, 5, 64, 300):
            z = (rng.integers(-12, 12, V) / 4.0).astype(np.float32)
            z[rng.random(V) < 0.1] = -np.inf
            s = stored(z, kind)
            for L in sorted({1, 2, 3, 7, 16, V}):
                assert np.array_equal(o.topl_set(s, L), topl_numpy(s, L)), (kind, V, L)


def check_topl_alpha_scipy(o):
    """alpha = sum of scipy's softmax(z_t / T) over the drafter's top-L tokens."""
    rng = np.random.default_rng(42)
    for kind in KINDS:
        for V in (2, 9, 100, 1000):
            zt = stored(rng.normal(0, 3, V), kind)
            zd = stored(value(zt) + rng.normal(0, 1.5, V), kind)
            for T in (0.5, 1.0, 2.0):
                p = probs(zt, T)
                for L in (1, 3, 10):
                    want = p[topl_numpy(zd, L)].sum()
                    a, st = o.alpha_topl(zt, zd, T, False, L)
                    assert st == orc.OK and abs(a - want) < 1e-12, (kind, V, T, L, a, want)


def check_topl_special_cases(o):
    """L = 1 under a greedy target is the argmax-agreement rule; L >= V puts
    every token in the candidate set, so alpha = 1."""
    rng = np.random.default_rng(43)
    for kind in KINDS:
        for trial in range(20):
            V = int(rng.integers(2, 40))
            zt = stored(rng.integers(-4, 4, V).astype(np.float32), kind)
            zd = stored(rng.integers(-4, 4, V).astype(np.float32), kind)
            a, st = o.alpha_topl(zt, zd, 1.0, True, 1)
            want = 1.0 if np.argmax(value(zt)) == np.argmax(value(zd)) else 0.0
            assert st == orc.OK and a == want
            for greedy in (False, True):
                a, st = o.alpha_topl(zt, zd, 0.8, greedy, V + int(rng.integers(0, 3)))
                assert st == orc.OK and abs(a - 1.0) < 1e-12


def check_topl_greedy_target_membership(o):
    """Greedy target: alpha = 1 exactly when the target's argmax is among the
    drafter's top-L tokens."""
    rng = np.random.default_rng(44)
    for trial in range(200):
        V = int(rng.integers(3, 30))
        L = int(rng.integers(1, V))
        zt = rng.integers(-5, 5, V).astype(np.float32)
        zd = rng.integers(-5, 5, V).astype(np.float32)
        a, st = o.alpha_topl(zt, zd, 1.0, True, L)
        want = 1.0 if np.argmax(zt) in set(topl_numpy(zd, L).tolist()) else 0.0
        assert st == orc.OK and a == want, (V, L)


def check_topl_mc_eagle(o):
    """Monte Carlo of Thm 2 on V = 8: the target's sampled token is accepted
    iff the drafter put it among its L children; the empirical rate matches
    alpha within 5 sigma."""
    rng = np.random.default_rng(45)
    V, n = 8, 400_000
    zt = rng.normal(0, 1.5, V).astype(np.float32)
    zd = rng.normal(0, 1.5, V).astype(np.float32)
    T = 0.9
    p = probs(zt, T)
    children = np.argsort(-zd, kind="stable")[:3]   # the drafter's 3 most likely tokens
    x = rng.choice(V, size=n, p=p)
    rate = np.isin(x, children).mean()
    a, st = o.alpha_topl(zt, zd, T, False, 3)
    sigma = math.sqrt(a * (1 - a) / n)
    assert st == orc.OK and abs(rate - a) < 5 * sigma + 1e-12, (rate, a, sigma)


def check_topl_nonfinite(o):
    rng = np.random.default_rng(46)
    zt = rng.normal(0, 1, 50).astype(np.float32)
    zd = rng.normal(0, 1, 50).astype(np.float32)
    bad = zd.copy()
    bad[7] = np.nan
    a, st = o.alpha_topl(zt, bad, 1.0, False, 4)
    assert st == orc.NONFINITE and np.isnan(a)
    badt = zt.copy()
    badt[3] = np.inf
    for greedy in (False, True):
        a, st = o.alpha_topl(badt, zd, 1.0, greedy, 4)
        assert st == orc.NONFINITE and np.isnan(a)


def check_feedback_topl_layout(o):
    """The whole-call layout: alpha[i,b,k] pairs target row (b,k) (or its path
    row) with drafter row (i,b,k); e_len is 1 + sum of cumulative products of
    alpha_1..alpha_K."""
    rng = np.random.default_rng(47)
    N, B, P, V, L, T = 3, 2, 4, 40, 5, 0.9
    tgt = stored(rng.normal(0, 2, (B, P, V)), "bf16")
    drf = stored(value(tgt)[None] + rng.normal(0, 1, (N, B, P, V)), "bf16")
    M = 6
    tree = stored(rng.normal(0, 2, (B, M, V)), "bf16")
    path = rng.integers(0, M, (B, P)).astype(np.int32)
    for use_path in (False, True):
        a, e, st = o.feedback_topl(tree if use_path else tgt, drf, T, False, L,
                                   path if use_path else None)
        assert st == orc.OK
        for i in range(N):
            for b in range(B):
                for k in range(P):
                    zt = tree[b, path[b, k]] if use_path else tgt[b, k]
                    want = probs(zt, T)[topl_numpy(drf[i, b, k], L)].sum()
                    assert abs(a[i, b, k] - want) < 1e-12
                want_e = 1.0 + np.cumprod(a[i, b, :P - 1]).sum()
                assert abs(e[i, b] - want_e) < 1e-12


ALL_CHECKS = [v for k, v in sorted(globals().items()) if k.startswith("check_")]
