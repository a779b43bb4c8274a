"""The long session (N = 8 drafters, B = 128 queries, K = 5, V = 151936 bf16,
2000 verification rounds, the expert drafter of query b switching to
(b + t // 250) mod 8 every 250 rounds) run through the C ABI exactly as a
server would run it: hs_feedback on fresh logits every round, then
hs_learner_step with the length loss (Sec. 3.3) for Hedge and NormalHedge
side by side.

On rounds 0, 1, 249, 250, 251, 1000 and 1999 (the first rounds, both sides
of the first expert switch, the middle and the end):
  * every alpha and e_len of the call against the oracle on the same stored
    bytes, at 1e-5 relative (Thm 1, Thm 3);
  * each learner's round against the oracle's learner given identical
    inputs: the GPU's fp32 alpha and e_len and the GPU's state, weights and
    choice from before the round.  Weights within 1e-4 relative, the state
    within fp32 rounding, the choice exact (App. B.1 remark: Hedge; App. D.6:
    NormalHedge).
Over the whole session, a property the paper's analysis fixes at any size:
Hedge's weight-averaged loss has regret at most ln N / eta + eta T / 8
against the best fixed drafter in hindsight (Sec. 3.1).
"""
import math

import numpy as np
import pytest
import torch

import oracle
import paper_2510_20064_gb300 as hf
from paper_2510_20064_gb300 import synth
from parity_util import (ATOL_WEIGHTS, RTOL_ALPHA, RTOL_WEIGHTS, assert_rel,
                         oracle_feedback_parallel, to_np)
from test_learner_gpu import check_sel

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
CHECKED = (0, 1, 249, 250, 251, 1000, 1999)


def test_long_session_rounds_match_oracle():
    w = synth.WORKLOADS["long_session"]
    N, B, P, T = w.N, w.B, w.P, w.rounds
    eta = w.eta
    o = oracle.get()
    ws = torch.empty(max(1, hf.hs_feedback_workspace_size(N, B, P, w.V, hf.HS_BF16, False)),
                     dtype=torch.uint8, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    alpha = torch.empty(N, B, P, device=DEV)
    e_len = torch.empty(N, B, device=DEV)
    learners = {}
    for name, kind, okind in (("hedge", hf.HS_HEDGE, oracle.HEDGE),
                              ("normalhedge", hf.HS_NORMALHEDGE, oracle.NORMALHEDGE)):
        learners[name] = dict(kind=kind, okind=okind, state=torch.zeros(N, B, device=DEV),
                              weights=torch.full((N, B), 1.0 / N, device=DEV),
                              sel=torch.zeros(B, dtype=torch.int32, device=DEV),
                              played=torch.zeros(B, device=DEV),
                              loss=torch.empty(N, B, device=DEV))
    cum_loss = torch.zeros(N, B, dtype=torch.float64, device=DEV)
    hedge_avg = torch.zeros(B, dtype=torch.float64, device=DEV)  # sum_t <w_t, f_t>
    ties = 0
    for t in range(T):
        d = synth.make_inputs(w, rnd=t, device=DEV)
        hf.hs_feedback(d["target"], d["drafter"], w.temperature, False, alpha=alpha, e_len=e_len,
                       workspace=ws, dev_status=status)
        check = t in CHECKED
        if check:
            torch.cuda.synchronize()
            ra, re, rst = oracle_feedback_parallel(d, w.temperature, False)
            assert rst == 0
            assert_rel(to_np(alpha), ra, RTOL_ALPHA, f"alpha, round {t}")
            assert_rel(to_np(e_len), re, RTOL_ALPHA, f"e_len, round {t}")
            g_alpha = alpha.cpu().numpy()
            g_elen = e_len.cpu().numpy()
        for name, L in learners.items():
            if check:
                before = [L[k].cpu().numpy().copy() for k in ("state", "weights", "sel", "played")]
            w_t = L["weights"].double() if name == "hedge" else None
            hf.hs_learner_step(alpha, e_len, hf.HS_LOSS_LENGTH, L["kind"], eta, L["state"],
                               L["weights"], L["sel"], loss_out=L["loss"],
                               played_loss=L["played"])
            if name == "hedge":
                hedge_avg += (w_t * L["loss"].double()).sum(dim=0)
                cum_loss += L["loss"].double()
            if check:
                rs, rw, rl, rsel, rp = o.learner_step(g_alpha, g_elen, oracle.LOSS_LENGTH,
                                                      L["okind"], eta, *before)
                torch.cuda.synchronize()
                what = f"{name}, round {t}"
                assert_rel(to_np(L["loss"]), rl, 1e-6, f"loss {what}", atol=1e-7)
                # one fp32 round on fp32 state: half an ulp of the state, plus
                # the fp32 loss (2^-24) and, for NormalHedge, the increment
                # sum_j p_j (f_j - f_i) over N products (N 2^-23)
                assert_rel(to_np(L["state"]), rs, 1e-6, f"state {what}",
                           atol=(N + 2) * 2.0 ** -23)
                assert_rel(to_np(L["played"]), rp, 1e-6, f"played loss {what}", atol=1e-6)
                assert_rel(to_np(L["weights"]), rw, RTOL_WEIGHTS, f"weights {what}",
                           ATOL_WEIGHTS)
                ties += check_sel(L["sel"].cpu().numpy(), rsel, rs, name == "hedge", 1e-5)
        del d
    torch.cuda.synchronize()
    assert int(status.item()) == hf.HS_OK
    assert ties == 0, f"{ties} near-tied choices"
    # Hedge's regret bound on the weight-averaged loss (Sec. 3.1)
    best = cum_loss.min(dim=0).values
    regret = (hedge_avg - best).cpu().numpy()
    bound = math.log(N) / eta + eta * T / 8
    assert np.all(regret <= bound), (float(regret.max()), bound)
    played = {k: (L["played"].double() - best).mean().item() for k, L in learners.items()}
    print(f"long session: mean regret of the played drafter, hedge {played['hedge']:.3f}, "
          f"normalhedge {played['normalhedge']:.3f}; weight-averaged Hedge regret max "
          f"{regret.max():.3f} <= {bound:.1f}")
