"""Sampled play (App. B.1), the chunk-level game with a chunk horizon (App.
B.3) and the token-level game with delay through QFI-D (Sec. 3.2, App. B.1,
hybrid losses of App. B.5) against the oracle, through the C ABI."""
import numpy as np
import pytest
import torch

import oracle
import paper_2510_20064_gb300 as hf
from parity_util import RTOL_WEIGHTS, assert_rel, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    hf.lib()
    assert torch.cuda.is_available()


def test_sample_select_bit_exact():
    """The draw is an integer from fp32 sums in index order on both sides."""
    rng = np.random.default_rng(1)
    o = oracle.get()
    for N in (1, 2, 7, 32):
        B = 512
        w = rng.random((N, B)).astype(np.float32)
        w[rng.random((N, B)) < 0.3] = 0.0
        w[0, (w > 0).sum(axis=0) == 0] = 0.25
        u = rng.random(B).astype(np.float32)
        u[:4] = [0.0, np.nextafter(np.float32(1), np.float32(0)), 0.5, 0.999]
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        sel = hf.hs_sample_select(torch.from_numpy(w).to(DEV), torch.from_numpy(u).to(DEV),
                                  dev_status=status)
        want = np.array([o.sample_select(w[:, b], float(u[b])) for b in range(B)])
        assert np.array_equal(sel.cpu().numpy(), want)
        assert int(status.item()) == hf.HS_OK


def test_sample_select_invalid_columns():
    w = torch.tensor([[0.5, 0.0, -0.1, 0.3], [0.5, 0.0, 0.6, float("nan")]], device=DEV)
    u = torch.tensor([1.0, 0.5, 0.5, 0.5], device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    sel = hf.hs_sample_select(w, u, dev_status=status)
    assert sel.cpu().tolist() == [-1, -1, -1, -1]
    assert int(status.item()) == hf.HS_ERR_NONFINITE


def test_sample_select_frequencies():
    """Drawn over many uniforms, each drafter's frequency is its weight."""
    N, B = 6, 200_000
    w1 = torch.tensor([0.05, 0.0, 0.4, 0.15, 0.3, 0.1], device=DEV)
    w = w1[:, None].expand(N, B).contiguous()
    g = torch.Generator(device=DEV).manual_seed(7)
    u = torch.rand(B, generator=g, device=DEV)
    sel = hf.hs_sample_select(w, u).cpu().numpy()
    counts = np.bincount(sel, minlength=N)
    p = w1.cpu().numpy() / w1.sum().item()
    assert counts[1] == 0
    assert np.all(np.abs(counts - B * p) <= 5 * np.sqrt(B * p * (1 - p)) + 1e-9)


def _near_tie(state, weights, learner, sel_a, sel_b, b):
    if learner == hf.HS_HEDGE:
        L = state[:, b]
        return abs(L[sel_a] - L[sel_b]) <= 1e-4 * max(1.0, abs(L).max())
    return abs(weights[sel_a, b] - weights[sel_b, b]) <= 1e-4 * weights[:, b].max()


@pytest.mark.parametrize("learner", [hf.HS_HEDGE, hf.HS_NORMALHEDGE])
@pytest.mark.parametrize("loss_kind", [hf.HS_LOSS_LENGTH, hf.HS_LOSS_ACCEPT])
def test_chunk_learner_matches_oracle(learner, loss_kind):
    rng = np.random.default_rng(2)
    o = oracle.get()
    N, B, P, eta = 8, 64, 9, 0.3
    state = np.zeros((N, B))
    weights = np.full((N, B), 1.0 / N)
    sel = np.zeros(B, np.int32)
    played = np.zeros(B)
    g_state = torch.zeros(N, B, device=DEV)
    g_w = torch.full((N, B), 1.0 / N, device=DEV)
    g_sel = torch.zeros(B, dtype=torch.int32, device=DEV)
    g_pl = torch.zeros(B, device=DEV)
    g_loss = torch.empty(N, B, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    for rnd in range(20):
        alpha = rng.random((N, B, P)).astype(np.float32)
        k_h = rng.integers(0, P, B).astype(np.int32)
        state, weights, loss, sel_o, played = o.chunk_learner_step(
            alpha, k_h, loss_kind, learner, eta, state, weights, sel, played)
        hf.hs_chunk_learner_step(torch.from_numpy(alpha).to(DEV), torch.from_numpy(k_h).to(DEV),
                                 loss_kind, learner, eta, g_state, g_w, g_sel, loss_out=g_loss,
                                 played_loss=g_pl, dev_status=status)
        assert_rel(to_np(g_loss), loss, 1e-5, f"loss round {rnd}", atol=1e-6)
        assert_rel(to_np(g_w), weights, RTOL_WEIGHTS, f"weights round {rnd}", atol=1e-6)
        gs = g_sel.cpu().numpy()
        for b in np.flatnonzero(gs != sel_o):
            assert _near_tie(state, weights, learner, gs[b], sel_o[b], b), (rnd, b)
        sel = gs.copy()  # both sides continue from the GPU's choice
    assert_rel(to_np(g_pl), played, 1e-4, "played loss")
    assert int(status.item()) == hf.HS_OK


def test_chunk_learner_rejects_bad_horizon():
    N, B, P = 4, 3, 5
    alpha = torch.rand(N, B, P, device=DEV)
    k_h = torch.tensor([1, 5, -1], dtype=torch.int32, device=DEV)
    state = torch.zeros(N, B, device=DEV)
    w = torch.full((N, B), 0.25, device=DEV)
    sel = torch.zeros(B, dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    hf.hs_chunk_learner_step(alpha, k_h, hf.HS_LOSS_LENGTH, hf.HS_HEDGE, 0.5, state, w, sel,
                             dev_status=status)
    assert int(status.item()) == hf.HS_ERR_INVALID_ARG
    s = state.cpu().numpy()
    assert np.all(s[:, 1:] == 0) and np.any(s[:, 0] != 0)


def run_token_session(alpha, k_h, K, loss_kind, learner, eta, accept_first, H_ring):
    """The GPU session: before each chunk the QFI-D catch-up, after it the
    chunk's verified tokens join the stream."""
    Hc, N, B, P = alpha.shape
    ts = hf.TokenStream(N, B, H_ring, DEV)
    state = torch.zeros(N, B, device=DEV)
    w = torch.full((N, B), 1.0 / N, device=DEV)
    sel = torch.zeros(B, dtype=torch.int32, device=DEV)
    played = torch.zeros(B, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    sels = []
    a_dev = torch.from_numpy(alpha.astype(np.float32)).to(DEV)
    k_dev = torch.from_numpy(k_h.astype(np.int32)).to(DEV)
    for h in range(Hc):
        hf.hs_token_learner_step(ts, K, loss_kind, learner, eta, state, w, sel,
                                 accept_first=accept_first, played_loss=played,
                                 dev_status=status)
        sels.append(sel.cpu().numpy().copy())
        hf.hs_token_append(ts, a_dev[h].contiguous(), k_dev[h].contiguous(), sel,
                           dev_status=status)
    torch.cuda.synchronize()
    return (to_np(state), to_np(w), np.array(sels), to_np(played),
            ts.n_done.cpu().numpy(), int(status.item()))


@pytest.mark.parametrize("learner", [hf.HS_HEDGE, hf.HS_NORMALHEDGE])
@pytest.mark.parametrize("loss_kind,accept_first", [(hf.HS_LOSS_ACCEPT, 0),
                                                    (hf.HS_LOSS_LENGTH, 0),
                                                    (hf.HS_LOSS_LENGTH, 12)])
def test_token_session_matches_oracle(learner, loss_kind, accept_first):
    """QFI-D over a 40-chunk session with variable chunk lengths: the choice
    before every chunk, the final state and weights, the learner's own loss
    and the count of consumed tokens."""
    rng = np.random.default_rng(3)
    Hc, N, B, P, K, eta = 40, 8, 32, 9, 8, 0.2
    alpha = rng.random((Hc, N, B, P)).astype(np.float32).astype(np.float64)
    k_h = rng.integers(0, P, (Hc, B))
    st, w, sels, played, done, status = run_token_session(alpha, k_h, K, loss_kind, learner,
                                                          eta, accept_first, H_ring=K + 2 * P)
    assert status == hf.HS_OK
    o_st, o_w, o_sel, o_pl, o_done = oracle.get().token_session(
        alpha, k_h, K, loss_kind, learner, eta, np.zeros((N, B)), np.full((N, B), 1.0 / N),
        np.zeros(B), accept_first=accept_first)
    assert np.array_equal(done, o_done)
    assert_rel(w, o_w, RTOL_WEIGHTS, "weights", atol=1e-6)
    assert_rel(st, o_st, 1e-4, "state", atol=1e-4)
    mism = np.argwhere(sels != o_sel)
    if len(mism):
        # a choice that differs sends a different drafter's tokens into the
        # played loss; only a near tie may cause it
        pytest.fail(f"{len(mism)} choices differ, first at chunk/query {mism[0]}")
    assert_rel(played, o_pl, 1e-4, "played loss")


def test_token_ring_overflow_is_refused():
    N, B, P, K = 4, 2, 5, 4
    ts = hf.TokenStream(N, B, 6, DEV)  # room for one chunk of 5 tokens only
    alpha = torch.rand(N, B, P, device=DEV)
    k_h = torch.full((B,), P - 1, dtype=torch.int32, device=DEV)
    sel = torch.zeros(B, dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    hf.hs_token_append(ts, alpha, k_h, sel, dev_status=status)
    assert int(status.item()) == hf.HS_OK
    hf.hs_token_append(ts, alpha, k_h, sel, dev_status=status)
    assert int(status.item()) == hf.HS_ERR_UNSUPPORTED
    assert ts.n_tok.cpu().tolist() == [5, 5]


@pytest.mark.parametrize("learner", [hf.HS_HEDGE, hf.HS_NORMALHEDGE])
def test_scheduled_session_matches_oracle(learner):
    """App. B.5: the paper's example schedule (warm-up 6, batch 12, skip 6
    tokens) with 3 hybrid vectors drives the losses-only kernel into a device
    queue and the FIFO catch-up kernel; decisions, weights and choices after
    every applied batch match the oracle's schedule and learner."""
    rng = np.random.default_rng(4)
    o = oracle.get()
    R, N, B, P, Q, eta = 80, 8, 32, 9, 64, 0.25
    cfg = (6, 12, 6, 3)
    sch = hf.Schedule(*cfg)
    ks = rng.integers(0, P, R)
    dec = o.schedule(*cfg, ks + 1)
    queue = torch.zeros(Q, N, B, device=DEV)
    state = torch.zeros(N, B, device=DEV)
    w = torch.full((N, B), 1.0 / N, device=DEV)
    sel = torch.zeros(B, dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    o_state, o_w, o_sel = np.zeros((N, B)), np.full((N, B), 1.0 / N), np.zeros(B, np.int32)
    pending, head, tail, applies = [], 0, 0, 0
    for r in range(R):
        ev, kind, ap = sch.next(int(ks[r]) + 1)
        assert (ev, kind, ap) == dec[r], r
        alpha = rng.random((N, B, P)).astype(np.float32)
        if ev:
            k_h = torch.full((B,), int(ks[r]), dtype=torch.int32, device=DEV)
            hf.hs_chunk_losses(torch.from_numpy(alpha).to(DEV), k_h, kind,
                               loss_out=queue[tail % Q], dev_status=status)
            lv = np.array([[o.chunk_loss(alpha[i, b], int(ks[r]), kind) for b in range(B)]
                           for i in range(N)])
            assert_rel(to_np(queue[tail % Q]), lv, 1e-5, f"losses round {r}", atol=1e-6)
            pending.append(lv)
            tail += 1
        if ap:
            hf.hs_learner_apply(queue, head % Q, tail - head, learner, eta, state, w, sel)
            o_state, o_w, o_sel = o.learner_apply(np.stack(pending), learner, eta, o_state, o_w,
                                                  o_sel)
            pending, head = [], tail
            applies += 1
            assert_rel(to_np(w), o_w, RTOL_WEIGHTS, f"weights after round {r}", atol=1e-6)
            gs = sel.cpu().numpy()
            for b in np.flatnonzero(gs != o_sel):
                assert _near_tie(o_state, o_w, learner, gs[b], o_sel[b], b), (r, b)
            o_sel = gs.copy()
    assert applies >= 8 and int(status.item()) == hf.HS_OK
