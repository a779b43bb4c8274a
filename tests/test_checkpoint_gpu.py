"""Checkpoint and resume of a learner session, through the C ABI.

All learner state lives in caller-owned device arrays (the library keeps
none), so a checkpoint is a copy of those arrays and a resume is a copy
back.  A session of 1000 rounds is run twice: once straight through, and
once stopped after round 500, its arrays written to a file, read back into
freshly allocated tensors and continued.  The two runs must agree bit for
bit, for the chunk-level learners (Hedge, NormalHedge; Sec. 3.3 losses) and
for the token-level game with delay (QFI-D over the token stream, App. B.1
and Sec. 3.2) with sampled play.
"""
import numpy as np
import pytest
import torch

import paper_2510_20064_gb300 as hf

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
N, B, P = 8, 64, 6
K = P - 1
ROUNDS, STOP = 1000, 500
ETA = 0.0912


def round_inputs(t):
    """Seeded per-round alpha [N,B,P], accepted counts k_h [B] and uniforms [B]."""
    rng = np.random.default_rng(1000 + t)
    expert = (np.arange(B) + t // 250) % N
    alpha = 0.3 + 0.3 * rng.random((N, B, P))
    alpha[expert, np.arange(B)] = 0.85 + 0.1 * rng.random((B, P))
    a = torch.tensor(alpha, dtype=torch.float32, device=DEV)
    k_h = torch.tensor(rng.integers(0, K + 1, B), dtype=torch.int32, device=DEV)
    u = torch.tensor(rng.random(B), dtype=torch.float32, device=DEV)
    return a, k_h, u


def e_len_of(a):
    prod = torch.cumprod(a[..., :-1], dim=-1)
    return 1.0 + prod.sum(dim=-1)


STREAM_FIELDS = ("gamma", "who", "n_tok", "n_done")  # the token stream's device arrays


def fresh(kind):
    st = {"state": torch.zeros(N, B, device=DEV),
          "weights": torch.full((N, B), 1.0 / N, device=DEV),
          "sel": torch.zeros(B, dtype=torch.int32, device=DEV),
          "played": torch.zeros(B, device=DEV)}
    if kind == "token":
        ts = hf.TokenStream(N, B, K + 2 * P, DEV)
        st.update({f: getattr(ts, f) for f in STREAM_FIELDS})
    return st


def stream_of(st):
    """A TokenStream over the arrays in st (a fresh one, or one read back
    from a checkpoint)."""
    ts = hf.TokenStream(N, B, st["gamma"].shape[1], DEV)
    for f in STREAM_FIELDS:
        getattr(ts, f).copy_(st[f])
    return ts


def play(kind, learner, st, t0, t1, status):
    ts = stream_of(st) if kind == "token" else None
    for t in range(t0, t1):
        a, k_h, u = round_inputs(t)
        if kind == "chunk":
            hf.hs_learner_step(a, e_len_of(a), hf.HS_LOSS_LENGTH, learner, ETA, st["state"],
                               st["weights"], st["sel"], played_loss=st["played"])
        else:
            hf.hs_token_append(ts, a, k_h, st["sel"], dev_status=status)
            arg = torch.empty(B, dtype=torch.int32, device=DEV)
            hf.hs_token_learner_step(ts, K, hf.HS_LOSS_LENGTH, learner, ETA, st["state"],
                                     st["weights"], arg, played_loss=st["played"],
                                     dev_status=status)
            hf.hs_sample_select(st["weights"], u, selected=st["sel"], dev_status=status)
    if ts is not None:  # the stream's arrays back into st
        for f in STREAM_FIELDS:
            st[f].copy_(getattr(ts, f))


@pytest.mark.parametrize("kind", ["chunk", "token"])
@pytest.mark.parametrize("learner", [hf.HS_HEDGE, hf.HS_NORMALHEDGE])
def test_resume_is_bit_exact(kind, learner, tmp_path):
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    straight = fresh(kind)
    play(kind, learner, straight, 0, ROUNDS, status)

    first = fresh(kind)
    play(kind, learner, first, 0, STOP, status)
    torch.cuda.synchronize()
    path = tmp_path / "session.npz"
    np.savez(path, **{k: v.cpu().numpy() for k, v in first.items()})
    del first
    saved = np.load(path)
    resumed = {k: torch.tensor(saved[k], device=DEV) for k in saved.files}
    play(kind, learner, resumed, STOP, ROUNDS, status)
    torch.cuda.synchronize()
    assert int(status.item()) == hf.HS_OK, hf.hs_status_string(int(status.item()))
    for k in straight:
        a, b = straight[k].cpu().numpy(), resumed[k].cpu().numpy()
        assert a.dtype == b.dtype and np.array_equal(a, b), f"{k} differs after the resume"
    assert int(straight["sel"].max()) < N
