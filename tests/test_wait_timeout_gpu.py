"""The bounded-wait error path on a GPU, without faulting or hanging it.

hs_test_stream_wait_timeout runs the streaming stochastic kernel with tile
(0,0)'s wait for its statistics made unsatisfiable and every wait limited to
a short number of clock cycles: the wait runs out, HS_ERR_TIMEOUT reaches
the status word, tile (0,0)'s alphas come out NaN and every other alpha is
the one hs_feedback computes.  The next ordinary call on the same GPU then
runs normally and matches the oracle.
"""
import ctypes

import numpy as np
import pytest
import torch

import paper_2510_20064_gb300 as hf
from paper_2510_20064_gb300 import synth
from parity_util import RTOL_ALPHA, assert_rel, oracle_feedback, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def test_wait_runs_out_and_the_context_stays_usable():
    # V above the cluster kernel's range: the streaming kernel's shapes
    w = synth.Workload("timeout", N=3, B=2, P=3, V=200000, dtype="bf16", temperature=0.9,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=61)
    N, B, P, V = w.N, w.B, w.P, w.V
    ws_bytes = hf.hs_feedback_workspace_size(N, B, P, V, hf.HS_BF16, False)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=DEV)
    alpha = torch.full((N, B, P), 7.0, device=DEV)
    e_len = torch.full((N, B), 7.0, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    st = hf.lib().hs_test_stream_wait_timeout(
        hf._ptr(d["target"]), hf._ptr(d["drafter"]), hf.HS_BF16, N, B, P, V, 0.9,
        ctypes.c_longlong(200_000), hf._ptr(alpha), hf._ptr(e_len), hf._ptr(ws), ws_bytes,
        hf._ptr(status), stream)
    assert st == hf.HS_OK
    torch.cuda.synchronize()
    assert int(status.item()) == hf.HS_ERR_TIMEOUT
    a, e = to_np(alpha), to_np(e_len)
    assert np.isnan(a[:, 0, 0]).all(), "the timed-out tile's alphas must be NaN"
    assert np.isnan(e[:, 0]).all() and not np.isnan(e[:, 1:]).any()
    ra, re, rst = oracle_feedback(d, 0.9, False)
    assert rst == 0
    mask = np.ones_like(ra, dtype=bool)
    mask[:, 0, 0] = False
    assert_rel(a[mask], ra[mask], RTOL_ALPHA, "alpha of the tiles that completed")
    # the same GPU, the same buffers: an ordinary call is unaffected
    status.zero_()
    a2, e2 = hf.hs_feedback(d["target"], d["drafter"], 0.9, False, alpha=alpha, e_len=e_len,
                            workspace=ws, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == hf.HS_OK
    assert_rel(to_np(a2), ra, RTOL_ALPHA, "alpha after the timeout")
    assert_rel(to_np(e2), re, RTOL_ALPHA, "e_len after the timeout")
