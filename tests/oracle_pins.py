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


# ---- Thm 2 with EAGLE-2's dynamic pruning --------------------------------------

def check_topl_pruned_prefix_scipy(o):
    """Pruned candidate set = the first `keep` of the lexsort ranking: alpha
    is scipy's softmax(z_t / T) summed over them (stochastic target), or
    whether numpy's argmax of the target is among them (greedy target), for
    every keep from 0 to L on tie-heavy rows with -inf masks."""
    rng = np.random.default_rng(48)
    for kind in KINDS:
        for V in (3, 20, 300):
            zt = stored(rng.normal(0, 2.5, V), kind)
            zd = (rng.integers(-10, 10, V) / 4.0).astype(np.float32)
            zd[rng.random(V) < 0.15] = -np.inf
            zd = stored(zd, kind)
            for L in (1, 4, 16):
                rank = topl_numpy(zd, L)
                for keep in range(L + 1):
                    prefix = rank[:keep]
                    for T in (0.6, 1.7):
                        a, st = o.alpha_topl_pruned(zt, zd, T, False, L, keep)
                        want = probs(zt, T)[prefix].sum()
                        assert st == orc.OK and abs(a - want) < 1e-12, (kind, V, L, keep, T)
                    a, st = o.alpha_topl_pruned(zt, zd, 1.0, True, L, keep)
                    want = 1.0 if int(np.argmax(value(zt))) in set(prefix.tolist()) else 0.0
                    assert st == orc.OK and a == want, (kind, V, L, keep)


def check_topl_pruned_reductions(o):
    """keep = L is the unpruned rule of Thm 2; keep = 1 under a greedy target
    is the argmax-agreement rule; keep = 0 accepts nothing; alpha never
    decreases as the pruning keeps more children."""
    rng = np.random.default_rng(49)
    for trial in range(60):
        V = int(rng.integers(2, 60))
        L = int(rng.integers(1, 17))
        zt = stored(rng.normal(0, 2, V), "bf16")
        zd = stored(value(zt) + rng.normal(0, 1.5, V), "bf16")
        for greedy in (False, True):
            a_full, st = o.alpha_topl(zt, zd, 0.9, greedy, L)
            a, st2 = o.alpha_topl_pruned(zt, zd, 0.9, greedy, L, L)
            assert st == st2 == orc.OK and a == a_full
            a0, st = o.alpha_topl_pruned(zt, zd, 0.9, greedy, L, 0)
            assert st == orc.OK and a0 == 0.0
            prev = -1.0
            for keep in range(L + 1):
                a, st = o.alpha_topl_pruned(zt, zd, 0.9, greedy, L, keep)
                assert st == orc.OK and a >= prev
                prev = a
        a, st = o.alpha_topl_pruned(zt, zd, 1.0, True, L, 1)
        want = 1.0 if np.argmax(value(zt)) == np.argmax(value(zd)) else 0.0
        assert st == orc.OK and a == want


def check_topl_pruned_mc_eagle2(o):
    """Monte Carlo of a pruned EAGLE-2 node on V = 8: the drafter expands its
    L = 5 most likely tokens, scores each child by the node's score times
    q(child), and drops the children scoring below a threshold; the target's
    sampled token is accepted iff a surviving child matches it.  The
    survivors are a prefix of the ranking, and the empirical acceptance rate
    matches alpha with keep = their number, within 5 sigma."""
    rng = np.random.default_rng(50)
    V, n, L, T = 8, 400_000, 5, 0.8
    zt = rng.normal(0, 1.5, V).astype(np.float32)
    zd = rng.normal(0, 1.5, V).astype(np.float32)
    q = softmax(zd.astype(np.float64))
    children = np.argsort(-zd, kind="stable")[:L]
    node_score = 0.6
    scores = node_score * q[children]
    threshold = np.sort(scores)[-3] * (1 - 1e-9)   # three children survive
    survivors = children[scores >= threshold]
    assert np.array_equal(survivors, children[:len(survivors)]), "pruning keeps a prefix"
    x = rng.choice(V, size=n, p=probs(zt, T))
    rate = np.isin(x, survivors).mean()
    a, st = o.alpha_topl_pruned(zt, zd, T, False, L, len(survivors))
    sigma = math.sqrt(a * (1 - a) / n)
    assert st == orc.OK and len(survivors) == 3
    assert abs(rate - a) < 5 * sigma + 1e-12, (rate, a, sigma)


def check_topl_pruned_invalid(o):
    """keep outside [0, L] is an argument error (NaN); unusable rows give
    NaN and the non-finite status; a whole call reports the argument error
    first and still fills every other alpha."""
    rng = np.random.default_rng(51)
    zt = rng.normal(0, 1, 30).astype(np.float32)
    zd = rng.normal(0, 1, 30).astype(np.float32)
    for keep in (-1, 5):
        a, st = o.alpha_topl_pruned(zt, zd, 1.0, False, 4, keep)
        assert st == orc.BADARG and np.isnan(a)
    bad = zd.copy()
    bad[2] = np.nan
    a, st = o.alpha_topl_pruned(zt, bad, 1.0, False, 4, 2)
    assert st == orc.NONFINITE and np.isnan(a)
    N, B, P, V = 2, 2, 3, 30
    tgt = stored(rng.normal(0, 2, (B, P, V)), "fp32")
    drf = stored(rng.normal(0, 2, (N, B, P, V)), "fp32")
    keep = rng.integers(0, 5, (N, B, P)).astype(np.int32)
    keep[1, 0, 2] = 6
    a, e, st = o.feedback_topl_pruned(tgt, drf, 1.0, False, 4, keep)
    assert st == orc.BADARG and np.isnan(a[1, 0, 2]) and np.isnan(a).sum() == 1


def check_feedback_topl_pruned_layout(o):
    """The whole-call layout with per-row keep: alpha[i,b,k] pairs target row
    (b,k) (or its path row) with drafter row (i,b,k) and that row's keep;
    e_len is 1 + the sum of cumulative products of alpha_1..alpha_K."""
    rng = np.random.default_rng(52)
    N, B, P, V, L, T = 3, 2, 4, 40, 6, 0.9
    tgt = stored(rng.normal(0, 2, (B, P, V)), "bf16")
    drf = stored(value(tgt)[None] + rng.normal(0, 1, (N, B, P, V)), "bf16")
    keep = rng.integers(0, L + 1, (N, B, P)).astype(np.int32)
    M = 6
    tree = stored(rng.normal(0, 2, (B, M, V)), "bf16")
    path = rng.integers(0, M, (B, P)).astype(np.int32)
    for use_path in (False, True):
        a, e, st = o.feedback_topl_pruned(tree if use_path else tgt, drf, T, False, L, keep,
                                          path if use_path else None)
        assert st == orc.OK
        for i in range(N):
            for b in range(B):
                for k in range(P):
                    zt = tree[b, path[b, k]] if use_path else tgt[b, k]
                    want = probs(zt, T)[topl_numpy(drf[i, b, k], L)[:keep[i, b, k]]].sum()
                    assert abs(a[i, b, k] - want) < 1e-12
                want_e = 1.0 + np.cumprod(a[i, b, :P - 1]).sum()
                assert abs(e[i, b] - want_e) < 1e-12


# ---- App. B.1 (QFI-D): sampled play --------------------------------------------

def check_sample_select_searchsorted(o):
    """The draw is numpy's searchsorted (side='right') of u * total into the
    fp32 running sums (np.cumsum accumulates in index order), so the first
    running sum above the threshold; the last positive weight when none is."""
    rng = np.random.default_rng(60)
    for _ in range(400):
        N = int(rng.integers(1, 33))
        w = rng.random(N).astype(np.float32)
        w[rng.random(N) < 0.3] = 0.0
        if not w.any():
            w[int(rng.integers(N))] = np.float32(0.5)
        csum = np.cumsum(w, dtype=np.float32)
        for u in list(rng.random(6).astype(np.float32)) + [np.float32(0.0)]:
            thr = np.float32(u) * csum[-1]
            want = int(np.searchsorted(csum, thr, side="right"))
            if want == N:
                want = int(np.flatnonzero(w > 0)[-1])
            got = o.sample_select(w, float(u))
            assert got == want, (w, u, got, want)
            assert w[got] > 0


def check_sample_select_frequencies(o):
    """Over many uniforms each drafter is drawn with frequency w_i / sum w
    (within 5 sigma), including exact zeros for zero weights."""
    w = np.array([0.05, 0.0, 0.4, 0.15, 0.3, 0.1], np.float32)
    rng = np.random.default_rng(61)
    n = 100_000
    counts = np.zeros(len(w), np.int64)
    for u in rng.random(n).astype(np.float32):
        counts[o.sample_select(w, float(u))] += 1
    p = w / w.sum()
    sd = np.sqrt(n * p * (1 - p))
    assert counts[1] == 0
    assert np.all(np.abs(counts - n * p) <= 5 * sd + 1e-9), counts


def check_sample_select_invalid(o):
    w = np.array([0.3, 0.7], np.float32)
    for u in (1.0, -0.25, float("nan")):
        assert o.sample_select(w, u) == -1
    for bad in ([0.0, 0.0], [0.5, -0.1], [np.inf, 1.0], [np.nan, 1.0]):
        assert o.sample_select(np.array(bad, np.float32), 0.5) == -1
    assert o.sample_select(np.array([0.0, 0.0, 1.0], np.float32), 0.0) == 2
    u_top = float(np.nextafter(np.float32(1.0), np.float32(0.0)))
    assert o.sample_select(np.array([0.0, 1.0, 0.0], np.float32), u_top) == 1


# ---- App. B.3: chunk-level game with a chunk horizon -------------------------------

def check_chunk_loss_reduces_to_fixed_K(o):
    """k = K is the fixed-horizon loss; k = 1 is 1 - (1 + g1)/2 and 1 - g1;
    constant gamma a gives E = (1 - a^{k+1})/(1 - a); positions after k are
    never read; k = 0 gives 0."""
    rng = np.random.default_rng(62)
    for _ in range(50):
        P = int(rng.integers(2, 12))
        g = rng.random(P)
        K = P - 1
        assert o.chunk_loss(g, K, orc.LOSS_LENGTH) == o.loss_length(o.elen_prefix(g[:K]), K)
        assert o.chunk_loss(g, K, orc.LOSS_ACCEPT) == o.loss_accept(g[:K])
        assert abs(o.chunk_loss(g, 1, orc.LOSS_LENGTH) - (1 - (1 + g[0]) / 2)) < 1e-15
        assert abs(o.chunk_loss(g, 1, orc.LOSS_ACCEPT) - (1 - g[0])) < 1e-15
        k = int(rng.integers(1, P))
        h = g.copy()
        h[k:] = rng.random(P - k)
        for kind in (orc.LOSS_LENGTH, orc.LOSS_ACCEPT):
            assert o.chunk_loss(g, k, kind) == o.chunk_loss(h, k, kind)
            assert o.chunk_loss(g, 0, kind) == 0.0
        a = float(rng.random())
        e = (1 - a ** (k + 1)) / (1 - a)
        assert abs(o.chunk_loss(np.full(P, a), k, orc.LOSS_LENGTH) - (1 - e / (k + 1))) < 1e-13


def check_chunk_learner_step_matches_fixed_horizon(o):
    """Query b of a chunk-level round with horizon k_h[b] is the fixed-horizon
    round on that query's first k_h[b]+1 positions."""
    rng = np.random.default_rng(63)
    N, B, P = 5, 6, 7
    for learner in (orc.HEDGE, orc.NORMALHEDGE):
        for kind in (orc.LOSS_LENGTH, orc.LOSS_ACCEPT):
            alpha = rng.random((N, B, P))
            k_h = rng.integers(1, P, B)
            state = rng.random((N, B)) * (0.5 if learner == orc.HEDGE else 0.2)
            weights = rng.dirichlet(np.ones(N), B).T.copy()
            sel = rng.integers(0, N, B).astype(np.int32)
            played = rng.random(B)
            st, w, loss, s2, pl = o.chunk_learner_step(alpha, k_h, kind, learner, 0.3, state,
                                                        weights, sel, played)
            for b in range(B):
                k = int(k_h[b])
                a_b = alpha[:, b:b + 1, :k + 1]
                e_b = np.array([[o.elen_prefix(a_b[i, 0, :k])] for i in range(N)])
                st1, w1, l1, s1, p1 = o.learner_step(a_b, e_b, kind, learner, 0.3,
                                                     state[:, b:b + 1], weights[:, b:b + 1],
                                                     sel[b:b + 1], played[b:b + 1])
                assert np.array_equal(st[:, b], st1[:, 0]) and np.array_equal(w[:, b], w1[:, 0])
                assert np.array_equal(loss[:, b], l1[:, 0]) and s2[b] == s1[0]
                assert pl[b] == p1[0]


# ---- Sec. 3.2 token-level game with delay, QFI-D (App. B.1) ---------------------------

def check_token_loss_window(o):
    """The length loss of token s is the chunk loss of a K-token chunk that
    starts at s; the acceptance loss is 1 - g[s]."""
    rng = np.random.default_rng(64)
    g = rng.random(40)
    for K in (1, 3, 8):
        for s in range(0, 40 - K):
            assert o.token_loss(g, s, K, orc.LOSS_LENGTH) == o.chunk_loss(g[s:s + K], K,
                                                                         orc.LOSS_LENGTH)
            assert abs(o.token_loss(g, s, K, orc.LOSS_ACCEPT) - (1 - g[s])) < 1e-15


def check_token_revealed_paper_rule(o):
    """Fig. "Token-Level Game with Delay": at the end of a chunk ending at
    token t the player knows f_{<=t} (acceptance) or f_{<=t-K} (length);
    hybrid losses reveal the first accept_first tokens early."""
    assert o.token_revealed(10, 4, orc.LOSS_LENGTH) == 6
    assert o.token_revealed(3, 4, orc.LOSS_LENGTH) == 0
    assert o.token_revealed(10, 4, orc.LOSS_ACCEPT) == 10
    assert o.token_revealed(5, 8, orc.LOSS_LENGTH, accept_first=3) == 3
    assert o.token_revealed(2, 8, orc.LOSS_LENGTH, accept_first=3) == 2
    assert o.token_revealed(20, 8, orc.LOSS_LENGTH, accept_first=3) == 12


def _session_inputs(rng, H, N, B, P):
    alpha = rng.random((H, N, B, P))
    k_h = rng.integers(0, P, (H, B))
    return alpha, k_h


def _stream(alpha, k_h, b):
    H, N, _, P = alpha.shape
    return np.concatenate([alpha[h, :, b, :k_h[h, b] + 1] for h in range(H)], axis=1)


def check_token_session_hedge_sum(o):
    """Hedge through QFI-D: the final cumulative loss is the initial one plus
    the plain sum of the revealed token losses (order does not matter), the
    weights are Hedge's closed form of it, and the processed count is the
    revealed count of the stream before the last chunk's tokens."""
    rng = np.random.default_rng(65)
    H, N, B, P, K = 9, 4, 3, 5, 4
    alpha, k_h = _session_inputs(rng, H, N, B, P)
    for kind, first in ((orc.LOSS_ACCEPT, 0), (orc.LOSS_LENGTH, 0), (orc.LOSS_LENGTH, 5)):
        state0 = rng.random((N, B))
        st, w, sel, played, done = o.token_session(alpha, k_h, K, kind, orc.HEDGE, 0.4, state0,
                                                   np.full((N, B), 1.0 / N), np.zeros(B),
                                                   accept_first=first)
        for b in range(B):
            g = _stream(alpha, k_h, b)
            n_before_last = g.shape[1] - (k_h[H - 1, b] + 1)
            ready = o.token_revealed(n_before_last, K, kind, first)
            assert done[b] == ready
            tot = np.zeros(N)
            for s_ in range(ready):
                if s_ < first or kind == orc.LOSS_ACCEPT:
                    tot += 1.0 - g[:, s_]
                else:
                    csum = np.cumprod(g[:, s_:s_ + K], axis=1).sum(axis=1)
                    tot += 1.0 - (1.0 + csum) / (K + 1)
            assert np.allclose(st[:, b], state0[:, b] + tot, rtol=0, atol=1e-12)
            ww, ss = o.hedge(st[:, b], 0.4)
            assert np.array_equal(w[:, b], ww) and sel[H - 1, b] == (ss if ready else 0)


def check_token_session_normalhedge_fifo(o):
    """NormalHedge through QFI-D: the revealed losses are fed in token order
    (FIFO), one NormalHedge round each, before every chunk's choice."""
    rng = np.random.default_rng(66)
    H, N, B, P, K = 8, 5, 2, 4, 3
    alpha, k_h = _session_inputs(rng, H, N, B, P)
    for kind in (orc.LOSS_ACCEPT, orc.LOSS_LENGTH):
        st, w, sel, played, done = o.token_session(alpha, k_h, K, kind, orc.NORMALHEDGE, 0.0,
                                                   np.zeros((N, B)), np.full((N, B), 1.0 / N),
                                                   np.zeros(B))
        for b in range(B):
            g = _stream(alpha, k_h, b)
            R, p, choice, n, d, own = np.zeros(N), np.full(N, 1.0 / N), 0, 0, 0, 0.0
            who = []
            for h in range(H):
                ready = o.token_revealed(n, K, kind)
                while d < ready:
                    f = np.array([o.token_loss(g[i], d, K, kind) for i in range(N)])
                    own += f[who[d]]
                    R, p, choice, _ = o.normalhedge(R, f, p)
                    d += 1
                assert sel[h, b] == choice
                who += [choice] * (k_h[h, b] + 1)
                n += k_h[h, b] + 1
            assert np.array_equal(st[:, b], R) and np.array_equal(w[:, b], p)
            assert done[b] == d and abs(played[b] - own) < 1e-12


def check_token_session_unrevealed_is_unseen(o):
    """The choice for chunk h depends only on revealed losses: changing the
    gamma of tokens whose loss is not yet revealed leaves sel[h] alone."""
    rng = np.random.default_rng(67)
    H, N, B, P, K = 6, 4, 1, 5, 4
    alpha, k_h = _session_inputs(rng, H, N, B, P)
    k_h[:] = P - 1
    args = (K, orc.LOSS_LENGTH, orc.HEDGE, 0.5, np.zeros((N, B)), np.full((N, B), 0.25),
            np.zeros(B))
    _, _, sel, _, _ = o.token_session(alpha, k_h, *args)
    # at chunk 3 the stream holds 3*P tokens, of which the first 3*P-K are
    # revealed; perturb the later ones (they sit in chunk 2)
    alt = alpha.copy()
    n3 = 3 * P
    for t in range(n3 - K + 1, n3):
        h, k = divmod(t, P)
        alt[h, :, 0, k] = rng.random(N)
    _, _, sel2, _, _ = o.token_session(alt, k_h, *args)
    assert sel2[3, 0] == sel[3, 0]


# ---- App. B.5 practical heuristics ----------------------------------------------

def check_schedule_hand_trace(o):
    """warm-up 2, batch 3, skip 6 tokens, hybrid 2 vectors, worked by hand:
    rounds 0-1 warm-up (evaluate, apply; the two acceptance-rate vectors);
    then the token count since the last evaluation runs 7 (eval), 3, 6 (eval),
    9 (eval), 1, 2, 10 (eval), 6 (eval), and the queue is applied at rounds
    4 and 7 (every 3rd round after the warm-up; round 10 would be next)."""
    got = o.schedule(2, 3, 6, 2, [5, 4, 7, 3, 3, 9, 1, 1, 8, 6])
    A, Ln = orc.LOSS_ACCEPT, orc.LOSS_LENGTH
    want = [(1, A, 1), (1, A, 1), (1, Ln, 0), (0, Ln, 0), (1, Ln, 1), (1, Ln, 0), (0, Ln, 0),
            (0, Ln, 1), (1, Ln, 0), (1, Ln, 0)]
    assert got == want, got


def check_schedule_invariants(o):
    """On random token counts: warm-up rounds evaluate and apply; later an
    evaluation happens exactly when the tokens since the last one reach the
    skip count; applies fall every batch_rounds rounds after the warm-up and
    only with something queued; the first hybrid vectors are acceptance-rate
    ones, all later ones length ones."""
    rng = np.random.default_rng(68)
    for _ in range(40):
        W, Bt, S, Hy = (int(rng.integers(0, 8)), int(rng.integers(1, 14)),
                        int(rng.integers(0, 15)), int(rng.integers(0, 10)))
        toks = rng.integers(1, 10, 120)
        dec = o.schedule(W, Bt, S, Hy, toks)
        since, made, queued = 0, 0, 0
        for r, (ev, kind, ap) in enumerate(dec):
            if r < W:
                assert ev == 1 and ap == 1
                since = 0
            else:
                since += int(toks[r])
                assert ev == (since >= S)
                if ev:
                    since = 0
                assert ap == ((((r - W + 1) % Bt) == 0) and (queued + ev) > 0)
            if ev:
                assert kind == (orc.LOSS_ACCEPT if made < Hy else orc.LOSS_LENGTH)
                made += 1
                queued += 1
            if ap:
                queued = 0


def check_learner_apply_batches(o):
    """A batch fed through QFI-D: Hedge ends at the plain sum of the vectors
    (and Hedge's closed form of it); NormalHedge equals one NormalHedge round
    per vector in queue order; an empty batch changes nothing."""
    rng = np.random.default_rng(69)
    C, N, B = 7, 5, 4
    lv = rng.random((C, N, B))
    st0 = rng.random((N, B))
    w0 = np.full((N, B), 1.0 / N)
    s0 = rng.integers(0, N, B)
    st, w, sel = o.learner_apply(lv, orc.HEDGE, 0.7, st0, w0, s0)
    assert np.allclose(st, st0 + lv.sum(axis=0), rtol=0, atol=1e-12)
    for b in range(B):
        ww, ss = o.hedge(st[:, b], 0.7)
        assert np.array_equal(w[:, b], ww) and sel[b] == ss
    st, w, sel = o.learner_apply(lv, orc.NORMALHEDGE, 0.0, np.zeros((N, B)), w0, s0)
    for b in range(B):
        R, p = np.zeros(N), np.full(N, 1.0 / N)
        for c in range(C):
            R, p, ch, _ = o.normalhedge(R, lv[c, :, b], p)
        assert np.array_equal(st[:, b], R) and np.array_equal(w[:, b], p) and sel[b] == ch
    st, w, sel = o.learner_apply(lv[:0], orc.NORMALHEDGE, 0.0, st0, w0, s0)
    assert np.array_equal(st, st0) and np.array_equal(w, w0) and np.array_equal(sel, s0)


ALL_CHECKS = [v for k, v in sorted(globals().items()) if k.startswith("check_")]
