"""hs_feedback_topl / hs_feedback_topl_path (Thm 2, EAGLE tree with branching
L) against the fp64 oracle, through the C ABI.

alpha is the target's probability mass on the drafter's top-L tokens; the
candidate set depends only on the stored drafter logits, so the greedy
results (and the sets behind the stochastic ones) must match exactly.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2510_20064_gb300 as hf
from paper_2510_20064_gb300 import synth
from parity_util import RTOL_ALPHA, assert_rel, per_query_parallel, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
W = synth.WORKLOADS


@pytest.fixture(scope="module", autouse=True)
def _lib():
    hf.lib()
    assert torch.cuda.is_available()


def run(d, T, greedy, L):
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    if "path" in d:
        a, e = hf.hs_feedback_topl_path(d["target"], d["path"], d["drafter"], L, T, greedy,
                                        dev_status=status)
    else:
        a, e = hf.hs_feedback_topl(d["target"], d["drafter"], L, T, greedy, dev_status=status)
    torch.cuda.synchronize()
    return to_np(a), to_np(e), int(status.item())


def oracle_topl(d, T, greedy, L):
    path = d.get("path")
    return oracle.get().feedback_topl(synth.storage_numpy(d["target"]),
                                      synth.storage_numpy(d["drafter"]), T, greedy, L,
                                      path=None if path is None else path.cpu().numpy())


def compare(d, T, greedy, L):
    a, e, st = run(d, T, greedy, L)
    ra, re, rst = oracle_topl(d, T, greedy, L)
    assert rst == 0 and st == hf.HS_OK, (rst, st)
    if greedy:
        assert np.array_equal(a, ra), "greedy alpha must be bit-exact"
        assert np.array_equal(e, re), "greedy e_len must be bit-exact"
    else:
        assert_rel(a, ra, RTOL_ALPHA, f"alpha L={L}")
        assert_rel(e, re, RTOL_ALPHA, f"e_len L={L}")
    return a


CASES = [
    # workload, size overrides (the paper's vocabularies: many chunks, ragged tail)
    ("qwen3_8b_chain", dict(B=2, N=3, P=3)),
    ("llama3_batch", dict(B=2, N=4, P=3)),
    ("tree_path", dict(B=2, N=3)),
    ("tiny_chain", {}),
]


@pytest.mark.parametrize("name,sizes", CASES, ids=[c[0] for c in CASES])
@pytest.mark.parametrize("L", [1, 3, 10, 16])
def test_topl_matches_oracle(name, sizes, L):
    w = W[name]
    d = synth.make_inputs(w, device=DEV, seed=700 + L, **sizes)
    for greedy in (False, True):
        compare(d, w.temperature, greedy, L)


@pytest.mark.parametrize("dtype", ["bf16", "fp16", "fp32"])
def test_topl_dtypes_and_ragged_vocab(dtype):
    w = synth.Workload("rag", N=2, B=2, P=3, V=20001, dtype=dtype, temperature=0.8,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=11)
    for L in (2, 16):
        for greedy in (False, True):
            compare(d, 0.8, greedy, L)


def test_topl_ties_and_masks():
    """Integer logits (many ties at the L boundary) and -inf masked tokens:
    the lower index must win, exactly as the oracle ranks."""
    g = torch.Generator(device=DEV).manual_seed(3)
    N, B, P, V = 3, 2, 3, 9000
    tgt = torch.randint(-6, 6, (B, P, V), generator=g, device=DEV).float()
    drf = torch.randint(-6, 6, (N, B, P, V), generator=g, device=DEV).float()
    drf[torch.rand(N, B, P, V, generator=g, device=DEV) < 0.2] = float("-inf")
    for dt in (torch.bfloat16, torch.float32):
        d = {"target": tgt.to(dt).contiguous(), "drafter": drf.to(dt).contiguous()}
        for L in (1, 5, 16):
            compare(d, 1.0, True, L)
            compare(d, 1.0, False, L)


def test_topl_adversarial_order():
    """Ascending drafter logits make every token displace a kept one (the
    slow path of the per-thread lists); descending ones reject nearly all."""
    N, B, P, V = 2, 1, 2, 30000
    ramp = torch.linspace(-8, 8, V, device=DEV)
    tgt = torch.randn(B, P, V, generator=torch.Generator(device=DEV).manual_seed(4), device=DEV)
    drf = torch.stack([ramp, ramp.flip(0)]).reshape(N, 1, 1, V).expand(N, B, P, V)
    d = {"target": tgt.to(torch.bfloat16).contiguous(),
         "drafter": drf.to(torch.bfloat16).contiguous()}
    for L in (1, 7, 16):
        for greedy in (False, True):
            compare(d, 1.0, greedy, L)


def test_topl_special_cases():
    w = synth.Workload("small", N=2, B=2, P=4, V=10, dtype="bf16", temperature=1.0,
                       target="gauss", sigma="tiny")
    d = synth.make_inputs(w, device=DEV, seed=5)
    a, e, st = run(d, 1.0, False, 16)          # L >= V: every token is a child
    assert st == hf.HS_OK and np.all(np.abs(a - 1.0) < 1e-6)
    a1, _, _ = run(d, 1.0, True, 1)            # L = 1, greedy: hs_feedback's greedy rule
    ag, _ = hf.hs_feedback(d["target"], d["drafter"], 1.0, True)
    assert np.array_equal(a1, to_np(ag))


def test_topl_nonfinite_and_bad_path():
    w = W["qwen3_8b_chain"]
    d = synth.make_inputs(w, device=DEV, B=2, N=3, P=3, V=5000)
    d["drafter"][1, 0, 2, 17] = float("nan")
    d["drafter"][2, 1, 0, :] = float("-inf")
    d["target"][1, 1, 4999] = float("inf")
    for greedy in (False, True):
        a, e, st = run(d, 1.0, greedy, 4)
        ra, re, rst = oracle_topl(d, 1.0, greedy, 4)
        assert st == hf.HS_ERR_NONFINITE and rst == oracle.NONFINITE
        assert np.array_equal(np.isnan(a), np.isnan(ra))
    t = W["tree_path"]
    dt = synth.make_inputs(t, device=DEV, B=2, N=2)
    dt["path"][1, 2] = 999
    a, e, st = run(dt, 1.0, False, 4)
    assert st == hf.HS_ERR_INVALID_ARG and np.all(np.isnan(a[:, 1, 2]))


def test_topl_argument_errors():
    d = synth.make_inputs(W["tiny_chain"], device=DEV)
    for L in (0, 17):
        with pytest.raises(hf.HedgeFBError):
            hf.hs_feedback_topl(d["target"], d["drafter"], L, 1.0, False)


@pytest.mark.parametrize("name", ["llama3_batch", "tree_path"])
def test_topl_full_size_sampled(name):
    """The benchmark's sizes, sampled (i, b, k) against the oracle pair by pair."""
    w = W[name]
    d = synth.make_inputs(w, device=DEV, seed=9)
    L = 10
    o = oracle.get()
    path = d.get("path")
    rng = np.random.default_rng(0)
    samples = [(int(rng.integers(w.N)), int(rng.integers(w.B)), int(rng.integers(w.P)))
               for _ in range(6)]
    for greedy in (False, True):
        a, e, st = run(d, w.temperature, greedy, L)
        assert st == hf.HS_OK
        for (i, b, k) in samples:
            trow = d["target"][b, int(path[b, k])] if path is not None else d["target"][b, k]
            ra, _ = o.alpha_topl(synth.storage_numpy(trow),
                                 synth.storage_numpy(d["drafter"][i, b, k]), w.temperature,
                                 greedy, L)
            if greedy:
                assert a[i, b, k] == ra
            else:
                assert abs(a[i, b, k] - ra) <= RTOL_ALPHA * abs(ra), (i, b, k, a[i, b, k], ra)


# ---- EAGLE-2's dynamic pruning (the remark closing Thm 2) ----------------------

def run_pruned(d, T, greedy, L, keep):
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    kt = torch.tensor(keep, dtype=torch.int32, device=DEV)
    if "path" in d:
        a, e = hf.hs_feedback_topl_pruned_path(d["target"], d["path"], d["drafter"], L, kt, T,
                                               greedy, dev_status=status)
    else:
        a, e = hf.hs_feedback_topl_pruned(d["target"], d["drafter"], L, kt, T, greedy,
                                          dev_status=status)
    torch.cuda.synchronize()
    return to_np(a), to_np(e), int(status.item())


def oracle_pruned(d, T, greedy, L, keep):
    o = oracle.get()
    return per_query_parallel(
        lambda t, dr, pa, kp: o.feedback_topl_pruned(t, dr, T, greedy, L, kp, path=pa), d, keep)


PRUNED = [
    ("qwen3_8b_chain", dict(B=2, N=3, P=3), (1, 4, 10, 16)),
    ("tree_path", dict(B=2, N=3), (1, 4, 10, 16)),
    ("tree_path", {}, (10,)),  # the full tree_path call: 2048 rows, one warp each
]


@pytest.mark.parametrize("name,sizes,L", [(n, s, L) for n, s, Ls in PRUNED for L in Ls],
                         ids=[f"{n}{'_full' if not s else ''}_L{L}" for n, s, Ls in PRUNED
                              for L in Ls])
def test_pruned_matches_oracle(name, sizes, L):
    """Per-row kept-children counts drawn from 0..L (every value occurs):
    every alpha and e_len against the oracle; the candidate sets are exact."""
    w = W[name]
    d = synth.make_inputs(w, device=DEV, seed=800 + L, **sizes)
    N, B, P = d["drafter"].shape[:3]
    rng = np.random.default_rng(900 + L)
    keep = rng.integers(0, L + 1, (N, B, P)).astype(np.int32)
    keep.reshape(-1)[:L + 1] = np.arange(L + 1)
    for greedy in (False, True):
        a, e, st = run_pruned(d, w.temperature, greedy, L, keep)
        ra, re, rst = oracle_pruned(d, w.temperature, greedy, L, keep)
        assert st == hf.HS_OK and rst == 0, (st, rst)
        if greedy:
            assert np.array_equal(a, ra) and np.array_equal(e, re)
        else:
            assert_rel(a, ra, RTOL_ALPHA, f"pruned alpha L={L}")
            assert_rel(e, re, RTOL_ALPHA, f"pruned e_len L={L}")
        assert np.all(a[keep == 0] == 0.0)


def test_pruned_keep_all_is_unpruned():
    """keep = L everywhere gives hs_feedback_topl's alphas bit for bit."""
    w = W["llama3_batch"]
    d = synth.make_inputs(w, device=DEV, seed=811, B=2, N=4, P=3)
    keep = np.full(d["drafter"].shape[:3], 10, np.int32)
    for greedy in (False, True):
        a, e, st = run_pruned(d, w.temperature, greedy, 10, keep)
        a0, e0, st0 = run(d, w.temperature, greedy, 10)
        assert st == st0 == hf.HS_OK
        assert np.array_equal(a, a0) and np.array_equal(e, e0)


def test_pruned_keep_out_of_range():
    """A kept count outside [0, L] makes only that alpha NaN and reports
    HS_ERR_INVALID_ARG; a null keep pointer is refused before any launch."""
    w = W["qwen3_8b_chain"]
    d = synth.make_inputs(w, device=DEV, seed=812, B=2, N=2, P=3, V=5000)
    keep = np.full((2, 2, 3), 2, np.int32)
    keep[1, 0, 2] = 5
    keep[0, 1, 1] = -1
    a, e, st = run_pruned(d, 0.7, False, 4, keep)
    assert st == hf.HS_ERR_INVALID_ARG
    assert np.isnan(a[1, 0, 2]) and np.isnan(a[0, 1, 1]) and np.isnan(a).sum() == 2
    ra, re, rst = oracle_pruned(d, 0.7, False, 4, keep)
    assert rst == oracle.BADARG
    assert_rel(a, ra, RTOL_ALPHA, "alpha next to a bad keep")
    alpha = torch.empty(2, 2, 3, device=DEV)
    st = hf.lib().hs_feedback_topl_pruned(
        hf._ptr(d["target"]), hf._ptr(d["drafter"]), hf.HS_BF16, 2, 2, 3, 5000, 0.7, 0, 4, None,
        hf._ptr(alpha), None, None, 0, None, None)
    assert st == hf.HS_ERR_INVALID_ARG


@pytest.mark.parametrize("dtype", ["bf16", "fp16", "fp32"])
def test_pruned_dtypes_masks_and_extremes(dtype):
    """Pruned candidate sets on every storage dtype, a ragged vocabulary with
    masked (-inf) tokens, and the extreme counts: every child pruned (alpha
    exactly 0) and none pruned, in one call."""
    w = synth.Workload("pruned", N=3, B=2, P=4, V=20001, dtype=dtype, temperature=0.8,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=820)
    mask = torch.rand(w.V, device=DEV) < 0.2
    d["drafter"][..., mask] = float("-inf")
    d["target"][..., mask.roll(3)] = float("-inf")
    L = 7
    rng = np.random.default_rng(821)
    keep = rng.integers(0, L + 1, (w.N, w.B, w.P)).astype(np.int32)
    keep[0] = 0
    keep[1] = L
    for greedy in (False, True):
        a, e, st = run_pruned(d, w.temperature, greedy, L, keep)
        ra, re, rst = oracle_pruned(d, w.temperature, greedy, L, keep)
        assert st == hf.HS_OK and rst == 0, (st, rst)
        if greedy:
            assert np.array_equal(a, ra) and np.array_equal(e, re)
        else:
            assert_rel(a, ra, RTOL_ALPHA, f"pruned alpha {dtype}")
            assert_rel(e, re, RTOL_ALPHA, f"pruned e_len {dtype}")
        assert np.all(a[0] == 0.0) and np.all(e[0] == 1.0)
