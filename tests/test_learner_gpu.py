"""hs_hedge_update / hs_normalhedge_update / hs_learner_step against the fp64
oracle, through the C ABI.

Per-round cases give both sides the same fp32 inputs and compare element by
element.  The selected drafter is an argmax decided in fp32 on the GPU and
in fp64 in the oracle; it must match exactly unless the oracle's own top two
are within the fp32 error of the state, in which case the GPU's pick must be
one of those near-tied drafters (both are then correct).  The number of such
rounds is reported and is 0 in every case below.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import paper_2510_20064_gb300 as hf
from paper_2510_20064_gb300 import synth
from parity_util import ATOL_WEIGHTS, RTOL_ALPHA, RTOL_WEIGHTS, assert_rel, oracle_feedback, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def cuda(x, dtype=torch.float32):
    return torch.tensor(np.asarray(x), dtype=dtype, device=DEV).contiguous()


def check_sel(gpu_sel, ref_sel, key, lower_is_better, tol):
    """Exact match, except where the oracle's key has a near-tie at the top."""
    ties = 0
    for b in range(len(ref_sel)):
        g, r = int(gpu_sel[b]), int(ref_sel[b])
        if g == r:
            continue
        kg, kr = key[g, b], key[r, b]
        scale = max(1.0, abs(kr))
        assert abs(kg - kr) <= tol * scale, (
            f"query {b}: gpu chose {g} (key {kg}), oracle {r} (key {kr})")
        ties += 1
    return ties


@pytest.mark.parametrize("N", [1, 2, 8, 16, 32])
@pytest.mark.parametrize("eta", [0.0, 0.0912, 0.5, 3.0])
def test_hedge_update(N, eta):
    rng = np.random.default_rng(N * 100 + int(eta * 10))
    B = 37
    L = (rng.random((N, B)) * 20).astype(np.float32)
    if N > 2:
        L[1, :5] = L[0, :5]  # exact ties -> lowest index
    w, sel = hf.hs_hedge_update(cuda(L), eta)
    torch.cuda.synchronize()
    o = oracle.get()
    for b in range(B):
        rw, rs = o.hedge(L[:, b], eta)
        assert_rel(to_np(w)[:, b], rw, RTOL_WEIGHTS, "hedge weights", ATOL_WEIGHTS)
        assert int(sel[b]) == rs


@pytest.mark.parametrize("N", [1, 2, 7, 8, 16, 32])
def test_normalhedge_update(N):
    rng = np.random.default_rng(N)
    B = 64
    R = rng.normal(0, 3, (N, B)).astype(np.float32)
    R[:, :4] = -np.abs(R[:, :4]) - 1.5       # stays <= 0 after a round (|increment| <= 1)
    if N >= 3:
        R[:3, 4:8] = 2.5                       # tied top regrets
    loss = rng.random((N, B)).astype(np.float32)
    loss[:, 4:8] = 0.25                        # equal losses keep the ties exact
    p = rng.dirichlet(np.ones(N), size=B).T.astype(np.float32)
    Rg, pg, sg = cuda(R), cuda(p), torch.empty(B, dtype=torch.int32, device=DEV)
    hf.hs_normalhedge_update(Rg, cuda(loss), pg, sg)
    torch.cuda.synchronize()
    o = oracle.get()
    ref_R = np.empty((N, B)); ref_p = np.empty((N, B)); ref_s = np.empty(B, int)
    for b in range(B):
        ref_R[:, b], ref_p[:, b], ref_s[b], _ = o.normalhedge(R[:, b], loss[:, b], p[:, b])
    assert_rel(to_np(Rg), ref_R, 1e-5, "regret", atol=1e-6)
    assert_rel(to_np(pg), ref_p, RTOL_WEIGHTS, "normalhedge weights", ATOL_WEIGHTS)
    ties = check_sel(sg.cpu().numpy(), ref_s, ref_R, False, 1e-5)
    assert ties == 0
    assert np.allclose(to_np(pg)[:, :4], 1.0 / N)


@pytest.mark.parametrize("learner", [hf.HS_HEDGE, hf.HS_NORMALHEDGE])
@pytest.mark.parametrize("loss_kind", [hf.HS_LOSS_LENGTH, hf.HS_LOSS_ACCEPT])
def test_learner_step(learner, loss_kind):
    rng = np.random.default_rng(10 * learner + loss_kind)
    N, B, P = 8, 50, 6
    alpha = rng.random((N, B, P)).astype(np.float32)
    e_len = (1 + rng.random((N, B)) * (P - 1)).astype(np.float32)
    state = (rng.normal(0, 2, (N, B)) if learner else rng.random((N, B)) * 10).astype(np.float32)
    weights = rng.dirichlet(np.ones(N), size=B).T.astype(np.float32)
    sel = rng.integers(0, N, B).astype(np.int32)
    played = rng.random(B).astype(np.float32)
    g = [cuda(state), cuda(weights), cuda(sel, torch.int32), cuda(played)]
    loss_out = torch.empty(N, B, device=DEV)
    hf.hs_learner_step(cuda(alpha), cuda(e_len), loss_kind, learner, 0.3, g[0], g[1], g[2],
                       loss_out=loss_out, played_loss=g[3])
    torch.cuda.synchronize()
    rs, rw, rl, rsel, rp = oracle.get().learner_step(alpha, e_len, loss_kind, learner, 0.3,
                                                     state, weights, sel, played)
    assert_rel(to_np(loss_out), rl, 1e-6, "loss", atol=1e-7)
    assert_rel(to_np(g[0]), rs, 1e-5, "state", atol=1e-6)
    assert_rel(to_np(g[1]), rw, RTOL_WEIGHTS, "weights", ATOL_WEIGHTS)
    assert_rel(to_np(g[3]), rp, 1e-6, "played loss")
    assert check_sel(g[2].cpu().numpy(), rsel, rs, learner == hf.HS_HEDGE, 1e-5) == 0


def test_tiny_chain_trajectory():
    """50 rounds of the tiny chain (fresh logits each round, Hedge eta = 0.5),
    GPU feedback + learner against oracle feedback + oracle learner."""
    w = synth.WORKLOADS["tiny_chain"]
    o = oracle.get()
    for greedy in (False, True):
        N, B = w.N, w.B
        state = torch.zeros(N, B, device=DEV)
        weights = torch.full((N, B), 1.0 / N, device=DEV)
        sel = torch.zeros(B, dtype=torch.int32, device=DEV)
        played = torch.zeros(B, device=DEV)
        r_state, r_w = np.zeros((N, B)), np.full((N, B), 1.0 / N)
        r_sel, r_played = np.zeros(B, np.int32), np.zeros(B)
        ties = 0
        for rnd in range(w.rounds):
            d = synth.make_inputs(w, rnd=rnd, device=DEV)
            alpha, e_len = hf.hs_feedback(d["target"], d["drafter"], w.temperature, greedy)
            hf.hs_learner_step(alpha, e_len, hf.HS_LOSS_LENGTH, hf.HS_HEDGE, w.eta, state,
                               weights, sel, played_loss=played)
            ra, re, _ = oracle_feedback(d, w.temperature, greedy)
            r_state, r_w, _, r_sel, r_played = o.learner_step(ra, re, oracle.LOSS_LENGTH,
                                                              oracle.HEDGE, w.eta, r_state, r_w,
                                                              r_sel, r_played)
            torch.cuda.synchronize()
            if greedy:
                assert np.array_equal(to_np(alpha), ra)
            else:
                assert_rel(to_np(alpha), ra, RTOL_ALPHA, f"alpha round {rnd}")
            assert_rel(to_np(state), r_state, 1e-5, f"cum loss round {rnd}", atol=1e-6)
            assert_rel(to_np(weights), r_w, RTOL_WEIGHTS, f"weights round {rnd}", ATOL_WEIGHTS)
            ties += check_sel(sel.cpu().numpy(), r_sel, r_state, True, 1e-5)
        assert ties == 0
        assert_rel(to_np(played), r_played, 1e-5, "played loss")


@pytest.mark.parametrize("learner", [hf.HS_HEDGE, hf.HS_NORMALHEDGE])
def test_switching_session_learner(learner):
    """2000 rounds of the long session's expert schedule, fed as seeded
    synthetic acceptance rates (expert (b + t//250) mod 8 accepts ~0.9, the
    others ~0.45) to both learners.

    Every 50th round is compared with the oracle's learner given identical
    inputs (the same fp32 alpha and the GPU's state, weights and choice from
    before the round): state within the rounding of one fp32 round, weights
    within 1e-4 relative, the choice exact.  Separately the oracle runs the
    whole trajectory in fp64 from the start; the GPU's fp32 state may then
    differ by the rounding it accumulates, at most t rounds of (half an ulp
    of the state + (N + 2) 2^-23), and the choices may differ only where the
    oracle's top two are within that drift."""
    N, B, P, T = 8, 16, 6, 2000
    eta = math.sqrt(8 * math.log(N) / T)
    rng = np.random.default_rng(77)
    state = torch.zeros(N, B, device=DEV)
    weights = torch.full((N, B), 1.0 / N, device=DEV)
    sel = torch.zeros(B, dtype=torch.int32, device=DEV)
    played = torch.zeros(B, device=DEV)
    r_state, r_w = np.zeros((N, B)), np.full((N, B), 1.0 / N)
    r_sel, r_played = np.zeros(B, np.int32), np.zeros(B)
    cum = np.zeros((N, B))
    ties = 0
    round_err = (N + 2) * 2.0 ** -23
    for t in range(T):
        expert = (np.arange(B) + t // 250) % N
        alpha = (0.3 + 0.3 * rng.random((N, B, P))).astype(np.float32)
        alpha[expert, np.arange(B)] = (0.85 + 0.1 * rng.random((B, P))).astype(np.float32)
        ga = cuda(alpha)
        dummy_e = torch.ones(N, B, device=DEV)
        check = t % 50 == 49 or t == T - 1
        if check:
            before = [to_np(state), to_np(weights), sel.cpu().numpy(), to_np(played)]
        hf.hs_learner_step(ga, dummy_e, hf.HS_LOSS_ACCEPT, learner, eta, state, weights, sel,
                           played_loss=played)
        r_state, r_w, loss, r_sel_new, r_played = o_step(alpha, learner, eta, r_state, r_w,
                                                         r_sel, r_played)
        cum += loss
        if check:
            torch.cuda.synchronize()
            g_state, g_w, g_sel = to_np(state), to_np(weights), sel.cpu().numpy()
            # one round from identical inputs
            i_state, i_w, _, i_sel, _ = o_step(alpha, learner, eta, *before)
            assert_rel(g_state, i_state, 1e-6, f"state round {t}", atol=round_err)
            assert_rel(g_w, i_w, RTOL_WEIGHTS, f"weights round {t}", ATOL_WEIGHTS)
            assert check_sel(g_sel, i_sel, i_state, learner == hf.HS_HEDGE, 1e-5) == 0, t
            # the fp64 trajectory: accumulated fp32 rounding only
            drift = (t + 1) * (2.0 ** -24 * np.abs(r_state).max() + round_err)
            assert np.all(np.abs(g_state - r_state) <= drift), (t, float(
                np.abs(g_state - r_state).max()), drift)
            ties += check_sel(g_sel, r_sel_new, r_state, learner == hf.HS_HEDGE, 2 * drift)
        r_sel = r_sel_new
    assert ties == 0
    regret = (r_played - cum.min(axis=0)).mean()
    drift = T * (2.0 ** -24 * np.abs(r_played).max() + 2.0 ** -23)
    assert np.all(np.abs(to_np(played) - r_played) <= drift)
    print(f"learner {learner}: mean cumulative regret over {B} queries = {regret:.3f}")


def o_step(alpha, learner, eta, state, weights, sel, played):
    N, B, P = alpha.shape
    return oracle.get().learner_step(alpha, np.ones((N, B)), oracle.LOSS_ACCEPT, learner, eta,
                                     state, weights, sel, played)
