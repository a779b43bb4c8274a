"""libhedgefb loads without a GPU, exports every symbol its header declares,
and rejects bad arguments on the host before any CUDA call.  CPU only: no
call here reaches a kernel launch."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "hedgefb.h")


@pytest.fixture(scope="module")
def hf():
    import paper_2510_20064_gb300 as hf
    from paper_2510_20064_gb300 import build
    if not os.path.exists(hf.LIB_PATH) or any(
            os.path.getmtime(os.path.join(build.CSRC, f)) > os.path.getmtime(hf.LIB_PATH)
            for f in os.listdir(build.CSRC)):
        build.build()
    return hf


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(hs_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for want in ("hs_feedback", "hs_feedback_path", "hs_hedge_update", "hs_normalhedge_update",
                 "hs_learner_step", "hs_feedback_workspace_size", "hs_status_string"):
        assert want in names


def test_every_declared_symbol_is_exported(hf):
    lib = hf.lib()
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert name in hf.SIGNATURES, f"binding lacks {name}"


def test_status_strings(hf):
    for code in range(7):
        assert hf.hs_status_string(code).startswith("HS_")
    assert "UNKNOWN" in hf.hs_status_string(99)
    assert hf.hs_version() >= 100


def test_workspace_sizes(hf):
    ws = hf.hs_feedback_workspace_size
    assert ws(0, 1, 1, 1, hf.HS_BF16, 0) == 0
    assert ws(1, 1, 1, 1, 7, 0) == 0
    for N, B, P, V in ((2, 1, 5, 1000), (4, 8, 7, 151936), (8, 64, 9, 128256), (8, 128, 6, 151936)):
        for g in (0, 1):
            n = ws(N, B, P, V, hf.HS_BF16, g)
            assert n % 256 == 0 and 0 < n < (1 << 31)


FAKE = 0x10000  # never dereferenced: every call below fails validation first


def call_feedback(hf, target=FAKE, drafter=FAKE, dtype=0, N=2, B=1, P=3, V=64, T=1.0, greedy=0,
                  alpha=FAKE, e_len=FAKE, ws=FAKE, ws_bytes=1 << 20, status=None):
    return hf.lib().hs_feedback(target, drafter, dtype, N, B, P, V, T, greedy, alpha, e_len, ws,
                                ws_bytes, status, None)


def test_feedback_rejects_bad_arguments(hf):
    E = hf
    assert call_feedback(hf, N=0) == E.HS_ERR_INVALID_ARG
    assert call_feedback(hf, V=0) == E.HS_ERR_INVALID_ARG
    assert call_feedback(hf, P=-1) == E.HS_ERR_INVALID_ARG
    assert call_feedback(hf, dtype=5) == E.HS_ERR_INVALID_ARG
    assert call_feedback(hf, target=None) == E.HS_ERR_INVALID_ARG
    assert call_feedback(hf, alpha=None) == E.HS_ERR_INVALID_ARG
    assert call_feedback(hf, T=0.0) == E.HS_ERR_INVALID_ARG
    assert call_feedback(hf, T=-1.0) == E.HS_ERR_INVALID_ARG
    assert call_feedback(hf, T=float("nan")) == E.HS_ERR_INVALID_ARG
    assert call_feedback(hf, T=float("inf")) == E.HS_ERR_INVALID_ARG
    assert call_feedback(hf, target=FAKE + 1) == E.HS_ERR_MISALIGNED
    assert call_feedback(hf, dtype=2, drafter=FAKE + 2) == E.HS_ERR_MISALIGNED
    assert call_feedback(hf, alpha=FAKE + 2) == E.HS_ERR_MISALIGNED
    assert call_feedback(hf, ws_bytes=16) == E.HS_ERR_INVALID_ARG
    assert call_feedback(hf, ws=None) == E.HS_ERR_INVALID_ARG
    assert call_feedback(hf, ws=FAKE + 16) == E.HS_ERR_MISALIGNED
    assert call_feedback(hf, N=1 << 20) == E.HS_ERR_UNSUPPORTED
    assert call_feedback(hf, N=1 << 20, B=1 << 20, P=1 << 10) == E.HS_ERR_INVALID_ARG


def test_feedback_path_rejects_bad_arguments(hf):
    f = hf.lib().hs_feedback_path
    args = [FAKE, FAKE, 85, FAKE, 0, 2, 1, 4, 64, 1.0, 0, FAKE, FAKE, FAKE, 1 << 20, None, None]
    bad = list(args); bad[1] = None
    assert f(*bad) == hf.HS_ERR_INVALID_ARG
    bad = list(args); bad[2] = 0
    assert f(*bad) == hf.HS_ERR_INVALID_ARG
    bad = list(args); bad[1] = FAKE + 2
    assert f(*bad) == hf.HS_ERR_MISALIGNED
    bad = list(args); bad[9] = 0.0
    assert f(*bad) == hf.HS_ERR_INVALID_ARG


def test_learner_rejects_bad_arguments(hf):
    lib = hf.lib()
    assert lib.hs_hedge_update(FAKE, 0, 4, 0.5, FAKE, FAKE, None) == hf.HS_ERR_INVALID_ARG
    assert lib.hs_hedge_update(FAKE, 33, 4, 0.5, FAKE, FAKE, None) == hf.HS_ERR_UNSUPPORTED
    assert lib.hs_hedge_update(FAKE, 8, 4, -0.5, FAKE, FAKE, None) == hf.HS_ERR_INVALID_ARG
    assert lib.hs_hedge_update(FAKE, 8, 4, float("nan"), FAKE, FAKE, None) == hf.HS_ERR_INVALID_ARG
    assert lib.hs_hedge_update(FAKE + 1, 8, 4, 0.5, FAKE, FAKE, None) == hf.HS_ERR_MISALIGNED
    assert lib.hs_normalhedge_update(FAKE, None, FAKE, 8, 4, FAKE, None) == hf.HS_ERR_INVALID_ARG
    assert lib.hs_normalhedge_update(FAKE, FAKE, FAKE, 40, 4, FAKE, None) == hf.HS_ERR_UNSUPPORTED
    step = lib.hs_learner_step
    base = [FAKE, FAKE, 8, 4, 6, hf.HS_LOSS_LENGTH, hf.HS_NORMALHEDGE, 0.0, FAKE, FAKE, None,
            FAKE, None, None]
    for idx, val, want in ((5, 9, hf.HS_ERR_INVALID_ARG), (6, 5, hf.HS_ERR_INVALID_ARG),
                           (4, 0, hf.HS_ERR_INVALID_ARG), (1, None, hf.HS_ERR_INVALID_ARG),
                           (8, None, hf.HS_ERR_INVALID_ARG), (11, FAKE + 3, hf.HS_ERR_MISALIGNED),
                           (2, 33, hf.HS_ERR_UNSUPPORTED)):
        bad = list(base); bad[idx] = val
        assert step(*bad) == want, (idx, val)
    bad = list(base); bad[5] = hf.HS_LOSS_ACCEPT; bad[4] = 1
    assert step(*bad) == hf.HS_ERR_INVALID_ARG
    bad = list(base); bad[6] = hf.HS_HEDGE; bad[7] = float("inf")
    assert step(*bad) == hf.HS_ERR_INVALID_ARG


def test_delayed_entries_reject_bad_arguments(hf):
    lib = hf.lib()
    E = hf
    sample = [FAKE, 8, 4, FAKE, FAKE, None, None]
    for idx, val, want in ((1, 0, E.HS_ERR_INVALID_ARG), (1, 33, E.HS_ERR_UNSUPPORTED),
                           (3, None, E.HS_ERR_INVALID_ARG), (4, FAKE + 2, E.HS_ERR_MISALIGNED)):
        bad = list(sample); bad[idx] = val
        assert lib.hs_sample_select(*bad) == want, (idx, val)
    chunk = [FAKE, FAKE, 8, 4, 6, E.HS_LOSS_LENGTH, E.HS_HEDGE, 0.5, FAKE, FAKE, None, FAKE, None,
             None, None]
    for idx, val, want in ((1, None, E.HS_ERR_INVALID_ARG), (4, 0, E.HS_ERR_INVALID_ARG),
                           (5, 4, E.HS_ERR_INVALID_ARG), (7, -1.0, E.HS_ERR_INVALID_ARG),
                           (1, FAKE + 1, E.HS_ERR_MISALIGNED), (2, 40, E.HS_ERR_UNSUPPORTED)):
        bad = list(chunk); bad[idx] = val
        assert lib.hs_chunk_learner_step(*bad) == want, (idx, val)
    app = [FAKE, FAKE, 8, 4, 6, FAKE, FAKE, FAKE, 32, FAKE, FAKE, None, None]
    for idx, val, want in ((8, 0, E.HS_ERR_INVALID_ARG), (9, None, E.HS_ERR_INVALID_ARG),
                           (9, FAKE + 4, E.HS_ERR_MISALIGNED), (5, None, E.HS_ERR_INVALID_ARG),
                           (2, 33, E.HS_ERR_UNSUPPORTED)):
        bad = list(app); bad[idx] = val
        assert lib.hs_token_append(*bad) == want, (idx, val)
    tok = [FAKE, FAKE, 8, 4, 32, FAKE, FAKE, 8, E.HS_LOSS_LENGTH, 0, E.HS_NORMALHEDGE, 0.0, FAKE,
           FAKE, FAKE, None, None, None]
    for idx, val, want in ((7, 0, E.HS_ERR_INVALID_ARG), (7, 33, E.HS_ERR_INVALID_ARG),
                           (9, -1, E.HS_ERR_INVALID_ARG), (8, 2, E.HS_ERR_INVALID_ARG),
                           (10, 2, E.HS_ERR_INVALID_ARG), (6, FAKE + 4, E.HS_ERR_MISALIGNED),
                           (12, None, E.HS_ERR_INVALID_ARG)):
        bad = list(tok); bad[idx] = val
        assert lib.hs_token_learner_step(*bad) == want, (idx, val)


def test_schedule_matches_oracle(hf):
    """hs_schedule_next is host code: its decisions equal the oracle's on
    random token counts and settings, including the paper's example."""
    import numpy as np

    import oracle
    o = oracle.get()
    rng = np.random.default_rng(5)
    settings = [(6, 12, 6, 3)] + [(int(rng.integers(0, 9)), int(rng.integers(1, 15)),
                                   int(rng.integers(0, 16)), int(rng.integers(0, 12)))
                                  for _ in range(30)]
    for cfg in settings:
        toks = rng.integers(0, 10, 200)
        sch = hf.Schedule(*cfg)
        assert [sch.next(int(t)) for t in toks] == o.schedule(*cfg, toks), cfg


def test_schedule_rejects_bad_settings(hf):
    for cfg in ((6, 0, 6, 0), (-1, 12, 6, 0), (6, 12, -2, 0), (6, 12, 6, -1)):
        with pytest.raises(hf.HedgeFBError):
            hf.Schedule(*cfg).next(5)
    with pytest.raises(hf.HedgeFBError):
        hf.Schedule().next(-1)


def test_binding_refuses_cpu_tensors(hf):
    import torch
    t = torch.zeros(1, 3, 8)
    with pytest.raises(ValueError):
        hf.hs_feedback(t, torch.zeros(2, 1, 3, 8))


def test_pruned_tree_entries_reject_bad_keep(hf):
    """The pruned tree-mode entries refuse a null or misaligned kept-count
    array before anything reaches the GPU."""
    lib = hf.lib()
    P = ctypes.c_void_p
    for keep, want in ((None, hf.HS_ERR_INVALID_ARG), (P(FAKE + 2), hf.HS_ERR_MISALIGNED)):
        st = lib.hs_feedback_topl_pruned(P(FAKE), P(FAKE), hf.HS_BF16, 2, 2, 3, 64, 1.0, 0, 4,
                                         keep, P(FAKE), P(FAKE), P(FAKE), 1 << 20, None, None)
        assert st == want
        st = lib.hs_feedback_topl_pruned_path(P(FAKE), P(FAKE), 5, P(FAKE), hf.HS_BF16, 2, 2, 3,
                                              64, 1.0, 0, 4, keep, P(FAKE), P(FAKE), P(FAKE),
                                              1 << 20, None, None)
        assert st == want


def test_wait_timeout_hook_refuses_other_shapes(hf):
    """The bounded-wait test hook takes only the streaming kernel's shapes
    and a positive limit, and needs the status word; anything else is
    refused before anything reaches the GPU."""
    lib = hf.lib()
    fake = ctypes.c_void_p(FAKE)
    lim = ctypes.c_longlong
    assert lib.hs_test_stream_wait_timeout(fake, fake, hf.HS_FP32, 2, 1, 2, 200000, 1.0,
                                           lim(1000), fake, fake, fake, 1 << 30, fake,
                                           None) == hf.HS_ERR_UNSUPPORTED
    assert lib.hs_test_stream_wait_timeout(fake, fake, hf.HS_BF16, 2, 1, 2, 200000, 1.0,
                                           lim(0), fake, fake, fake, 1 << 30, fake,
                                           None) == hf.HS_ERR_INVALID_ARG
    assert lib.hs_test_stream_wait_timeout(fake, fake, hf.HS_BF16, 2, 1, 2, 200000, 1.0,
                                           lim(1000), fake, fake, fake, 1 << 30, None,
                                           None) == hf.HS_ERR_INVALID_ARG
