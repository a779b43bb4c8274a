"""hs_feedback_static -- the entry point for callers that cannot allocate
device memory when they call (their memory is reserved up front by another
allocator, or allocation latency is not acceptable mid-request) -- gives the
same results as hs_feedback, through the C ABI, on two calls in a row.

The cases below exercise every kernel family that needs scratch: greedy
(per-chunk argmax partials), the streaming stochastic kernel (row
statistics, alpha partials and tile counters that must restart at zero on
each call) and the two-pass stochastic kernels (fp32 logits), plus the
cluster kernel, which needs none.  The file's name makes pytest collect it
last.
"""
import ctypes

import numpy as np
import pytest
import torch

import paper_2510_20064_gb300 as hf
from paper_2510_20064_gb300 import synth
from parity_util import to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"

CASES = [
    ("greedy", dict(N=4, B=3, P=5, V=151936, dtype="bf16"), True),
    ("streaming", dict(N=3, B=8, P=4, V=200000, dtype="bf16"), False),
    ("two_pass_fp32", dict(N=3, B=2, P=4, V=5000, dtype="fp32"), False),
    ("cluster", dict(N=4, B=2, P=7, V=151936, dtype="bf16"), False),
]


def _static_call(d, T, greedy, alpha, e_len, status):
    N, B, P, V = d["drafter"].shape
    code = {torch.bfloat16: hf.HS_BF16, torch.float16: hf.HS_FP16,
            torch.float32: hf.HS_FP32}[d["drafter"].dtype]
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return hf.lib().hs_feedback_static(
        ctypes.c_void_p(d["target"].data_ptr()), ctypes.c_void_p(d["drafter"].data_ptr()), code,
        N, B, P, V, float(T), int(greedy), ctypes.c_void_p(alpha.data_ptr()),
        ctypes.c_void_p(e_len.data_ptr()), ctypes.c_void_p(status.data_ptr()), stream)


@pytest.mark.parametrize("name,sizes,greedy", CASES, ids=[c[0] for c in CASES])
def test_static_matches_hs_feedback(name, sizes, greedy):
    w = synth.Workload(name, target="zipf", sigma="qwen", temperature=0.8, **sizes)
    N, B, P = w.N, w.B, w.P
    ref_a, ref_e = [], []
    for call in range(2):
        d = synth.make_inputs(w, device=DEV, seed=300 + 17 * call)
        a, e = hf.hs_feedback(d["target"], d["drafter"], w.temperature, greedy)
        torch.cuda.synchronize()
        ref_a.append(to_np(a))
        ref_e.append(to_np(e))
        alpha = torch.full((N, B, P), float("nan"), device=DEV)
        e_len = torch.full((N, B), float("nan"), device=DEV)
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        st = _static_call(d, w.temperature, greedy, alpha, e_len, status)
        torch.cuda.synchronize()
        assert st == hf.HS_OK, hf.hs_status_string(st)
        assert int(status.item()) == hf.HS_OK
        # the same kernels on the same bytes: results are identical, so any
        # leftover of the previous call in the shared scratch would show
        assert np.array_equal(to_np(alpha), ref_a[-1], equal_nan=True), f"{name} alpha, call {call}"
        assert np.array_equal(to_np(e_len), ref_e[-1], equal_nan=True), f"{name} e_len, call {call}"
    assert not np.array_equal(ref_a[0], ref_a[1]), "the two calls must see different inputs"


def test_static_rejects_sizes_beyond_its_scratch():
    need = hf.hs_feedback_workspace_size(32, 4096, 9, 151936, hf.HS_BF16, True)
    assert need > 16 << 20
    st = hf.lib().hs_feedback_static(ctypes.c_void_p(16), ctypes.c_void_p(16), hf.HS_BF16, 32,
                                     4096, 9, 151936, 1.0, 1, ctypes.c_void_p(16),
                                     ctypes.c_void_p(16), None, None)
    assert st == hf.HS_ERR_UNSUPPORTED
