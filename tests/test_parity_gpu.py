"""hs_feedback / hs_feedback_path against the fp64 oracle, through the C ABI.

Reduced cases keep the paper-shaped vocabularies (V = 128256 / 151936, so
every row spans many vocab chunks and ends in a ragged one) with fewer
drafters, queries or positions, and are compared element by element.
Full-size cases run the benchmark's exact sizes and compare every output of
a call in both modes (the oracle spread over the host cores by query).
"""
import numpy as np
import pytest
import torch

import paper_2510_20064_gb300 as hf
from paper_2510_20064_gb300 import synth
from parity_util import (RTOL_ALPHA, assert_rel, oracle_alpha_rows, oracle_feedback,
                         oracle_feedback_parallel, to_np)

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
W = synth.WORKLOADS


@pytest.fixture(scope="module", autouse=True)
def _lib():
    hf.lib()
    assert torch.cuda.is_available()


def run(d, T, greedy, **kw):
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    if "path" in d:
        a, e = hf.hs_feedback_path(d["target"], d["path"], d["drafter"], T, greedy,
                                   dev_status=status, **kw)
    else:
        a, e = hf.hs_feedback(d["target"], d["drafter"], T, greedy, dev_status=status, **kw)
    torch.cuda.synchronize()
    return to_np(a), to_np(e), int(status.item())


def compare_full(d, T, greedy):
    a, e, st = run(d, T, greedy)
    ra, re, rst = oracle_feedback(d, T, greedy)
    assert st == hf.HS_OK and rst == 0
    if greedy:
        assert np.array_equal(a, ra), "greedy alpha must be bit-exact"
        assert np.array_equal(e, re), "greedy e_len must be bit-exact"
    else:
        assert_rel(a, ra, RTOL_ALPHA, "alpha")
        assert_rel(e, re, RTOL_ALPHA, "e_len")
    return a, e


REDUCED = [
    ("tiny_chain", {}, (False, True)),
    ("qwen3_8b_chain", dict(B=2), (False, True)),
    ("llama3_batch", dict(B=3, N=8), (False, True)),
    ("tree_path", dict(B=2), (False, True)),
    ("long_session", dict(B=2), (False, True)),
]


@pytest.mark.parametrize("name,sizes,modes", REDUCED, ids=[r[0] for r in REDUCED])
def test_reduced_workloads(name, sizes, modes):
    w = W[name]
    d = synth.make_inputs(w, device=DEV, **sizes)
    for greedy in modes:
        compare_full(d, w.temperature, greedy)


@pytest.mark.parametrize("V", [1, 2, 7, 8, 9, 1000, 8191, 8193, 20001, 151937])
@pytest.mark.parametrize("dtype", ["bf16", "fp16", "fp32"])
def test_ragged_vocab(V, dtype):
    w = synth.Workload("ragged", N=3, B=2, P=3, V=V, dtype=dtype, temperature=0.9,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=100 + V)
    compare_full(d, 0.9, False)
    compare_full(d, 0.9, True)


@pytest.mark.parametrize("T", [0.05, 0.3, 1.0, 5.0])
def test_temperatures(T):
    w = W["llama3_batch"]
    d = synth.make_inputs(w, device=DEV, B=1, N=4, P=3)
    compare_full(d, T, False)


def test_identical_and_disjoint_rows():
    g = torch.Generator(device=DEV).manual_seed(5)
    B, P, V, N = 2, 4, 40000, 3
    tgt = torch.randn(B, P, V, generator=g, device=DEV).to(torch.bfloat16)
    drf = tgt[None].repeat(N, 1, 1, 1).contiguous()
    a, e, st = run({"target": tgt, "drafter": drf}, 0.8, False)
    assert st == 0 and np.all(np.abs(a - 1) < 1e-5) and np.all(np.abs(e - P) < 1e-4)
    a, e, st = run({"target": tgt, "drafter": drf}, 0.8, True)
    assert np.all(a == 1) and np.all(e == P)
    neg = torch.tensor(float("-inf"), device=DEV, dtype=torch.bfloat16)
    even = torch.arange(V, device=DEV) % 2 == 0
    t2 = torch.where(even, tgt, neg).contiguous()
    d2 = torch.where(~even, drf, neg).contiguous()
    a, e, st = run({"target": t2, "drafter": d2}, 0.8, False)
    assert st == 0 and np.all(a == 0.0) and np.all(e == 1.0)


def test_nonfinite_rows_flagged():
    w = W["qwen3_8b_chain"]
    d = synth.make_inputs(w, device=DEV, B=2, N=3, P=3, V=5000)
    d["drafter"][1, 0, 2, 17] = float("nan")
    d["drafter"][2, 1, 0, :] = float("-inf")
    d["target"][1, 1, 4999] = float("inf")
    for greedy in (False, True):
        a, e, st = run(d, 1.0, greedy)
        assert st == hf.HS_ERR_NONFINITE
        ra, re, rst = oracle_feedback(d, 1.0, greedy)
        assert rst == hf.HS_ERR_NONFINITE
        assert np.isnan(a[1, 0, 2]) and np.isnan(a[2, 1, 0]) and np.all(np.isnan(a[:, 1, 1]))
        if greedy:
            assert np.array_equal(np.isnan(a), np.isnan(ra))
            ok = ~np.isnan(ra)
            assert np.array_equal(a[ok], ra[ok])
        else:
            assert_rel(a, ra, RTOL_ALPHA, "alpha with NaN rows")
            assert_rel(e, re, RTOL_ALPHA, "e_len with NaN rows")


def test_masked_vocabulary():
    """-inf entries are legal: masked tokens carry probability 0."""
    w = W["llama3_batch"]
    d = synth.make_inputs(w, device=DEV, B=2, N=2, P=3, V=10000)
    mask = torch.rand(d["target"].shape[-1], device=DEV) < 0.3
    d["target"][..., mask] = float("-inf")
    d["drafter"][..., mask.roll(7)] = float("-inf")
    compare_full(d, 1.0, False)
    compare_full(d, 1.0, True)


def test_degenerate_sizes():
    w = W["qwen3_8b_chain"]
    for N, B, P, V in ((1, 1, 1, 1), (1, 1, 1, 5), (1, 3, 1, 300), (5, 1, 2, 1)):
        d = synth.make_inputs(w, device=DEV, N=N, B=B, P=P, V=V)
        a, e = compare_full(d, 0.7, False)
        if P == 1:
            assert np.all(e == 1.0)
        if V == 1:
            assert np.allclose(a, 1.0)
        compare_full(d, 0.7, True)


def test_greedy_ties_lowest_index():
    B, P, V = 1, 2, 64
    tgt = torch.zeros(B, P, V, device=DEV, dtype=torch.bfloat16)
    drf = torch.zeros(2, B, P, V, device=DEV, dtype=torch.bfloat16)
    tgt[0, 0, [5, 9]] = 3.0       # target argmax = 5 (first of the tie)
    drf[0, 0, 0, [9, 5]] = 3.0    # same tie: argmax 5 -> accepted
    drf[1, 0, 0, 9] = 3.0         # argmax 9 -> rejected
    tgt[0, 1, 60] = -0.0          # all zeros: first index 0 wins
    a, _, _ = run({"target": tgt, "drafter": drf}, 1.0, True)
    assert a[0, 0, 0] == 1.0 and a[1, 0, 0] == 0.0 and a[0, 0, 1] == 1.0 and a[1, 0, 1] == 1.0


def test_unaligned_views_take_the_scalar_path():
    """Logit tensors starting one element past a 16-byte boundary."""
    w = W["qwen3_8b_chain"]
    d = synth.make_inputs(w, device=DEV, B=2, N=2, P=3, V=4096)
    buf_t = torch.empty(d["target"].numel() + 1, dtype=torch.bfloat16, device=DEV)
    buf_d = torch.empty(d["drafter"].numel() + 1, dtype=torch.bfloat16, device=DEV)
    t = buf_t[1:].view(d["target"].shape)
    dr = buf_d[1:].view(d["drafter"].shape)
    t.copy_(d["target"])
    dr.copy_(d["drafter"])
    assert t.data_ptr() % 16 != 0
    compare_full({"target": t, "drafter": dr}, 0.7, False)


def test_path_index_out_of_range():
    w = W["tree_path"]
    d = synth.make_inputs(w, device=DEV, B=2, N=2)
    d["path"][1, 2] = w.M  # one past the last node
    a, e, st = run(d, 1.0, False)
    assert st == hf.HS_ERR_INVALID_ARG
    assert np.all(np.isnan(a[:, 1, 2])) and not np.any(np.isnan(a[:, 0, :]))


def test_workspace_and_outputs_reused():
    """Two calls in a row on the same buffers give identical results."""
    w = W["qwen3_8b_chain"]
    d = synth.make_inputs(w, device=DEV, B=2, N=4, P=3)
    a1, e1, _ = run(d, 0.7, False)
    a2, e2, _ = run(d, 0.7, False)
    assert np.array_equal(a1, a2) and np.array_equal(e1, e2)


# ---- full benchmark sizes ---------------------------------------------------

FULL = ["qwen3_8b_chain", "llama3_batch", "tree_path", "long_session"]


@pytest.mark.parametrize("name", FULL)
def test_full_size_every_output(name):
    """The benchmark's exact sizes, in the launch configuration bench.py
    times: every alpha and e_len of a whole call against the oracle (run on
    every host core), stochastic at 1e-5 relative and greedy bit-exact."""
    w = W[name]
    d = synth.make_inputs(w, device=DEV)
    for greedy in (False, True):
        a, e, st = run(d, w.temperature, greedy)
        ra, re, rst = oracle_feedback_parallel(d, w.temperature, greedy)
        assert st == hf.HS_OK and rst == 0
        if greedy:
            assert np.array_equal(a, ra), f"{name}: greedy alpha must be bit-exact"
            assert np.array_equal(e, re), f"{name}: greedy e_len must be bit-exact"
        else:
            assert_rel(a, ra, RTOL_ALPHA, f"{name} alpha")
            assert_rel(e, re, RTOL_ALPHA, f"{name} e_len")
        # properties that hold at any size
        assert not np.isnan(a).any()
        assert np.all(a >= 0) and np.all(a <= 1 + 1e-5)
        assert np.all(e >= 1 - 1e-6) and np.all(e <= w.P + 1e-4)


# ---- both feedback paths ------------------------------------------------------
# bf16/fp16 rows with V % 8 == 0, 16-byte-aligned logits and N <= 32 take the
# single-read cluster kernel (the cluster size, up to 16, that keeps the most
# SMs busy) up to V = 153600 -- or the two-pass-per-SM kernel when there are at
# least two drafter rows per SM and its L2 working set fits -- and the
# persistent streaming kernel above; everything else takes the fallback
# two-pass kernels.  These cases cross each boundary.

@pytest.mark.parametrize("V", [8, 4096, 19200, 19208, 38400, 38408, 76800, 76808, 128256,
                               151936, 153600, 153608, 262144])
def test_cluster_sizes(V):
    w = synth.Workload("vsweep", N=3, B=2, P=3, V=V, dtype="bf16", temperature=0.8,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=7 + V)
    compare_full(d, 0.8, False)


@pytest.mark.parametrize("N", [1, 31, 32, 33])
def test_drafter_counts(N):
    w = W["llama3_batch"]
    d = synth.make_inputs(w, device=DEV, N=N, B=1, P=2, V=20000)
    compare_full(d, 1.0, False)


@pytest.mark.parametrize("greedy", [False, True])
def test_long_chain(greedy):
    """P = 40 scored positions (more than a warp's 32 lanes): the greedy
    finalize carries its prefix product of alpha from one group of 32
    positions to the next; drafter 0 copies the target, so its alphas are 1
    at every position and e_len reaches P.  Every alpha and e_len compared."""
    w = synth.Workload("long_chain", N=3, B=2, P=40, V=4096, dtype="bf16", temperature=0.9,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=12)
    d["drafter"][0] = d["target"]
    a, e = compare_full(d, 0.9, greedy)
    if greedy:
        assert np.all(a[0] == 1.0) and np.all(e[0] == 40.0)


def test_more_tiles_than_resident_clusters():
    """B*P = 1200 tiles: every resident cluster loops over many tiles."""
    w = W["qwen3_8b_chain"]
    d = synth.make_inputs(w, device=DEV, N=2, B=200, P=6, V=38400)
    a, e, st = run(d, 0.7, False)
    assert st == 0
    rng = np.random.default_rng(3)
    samples = [(int(rng.integers(2)), int(rng.integers(200)), int(rng.integers(6)))
               for _ in range(40)]
    ref = oracle_alpha_rows(d, samples, 0.7, False)
    assert_rel(np.array([a[s] for s in samples]), ref, RTOL_ALPHA, "many-tile alpha")


def test_fp16_full_vocab():
    w = synth.Workload("fp16", N=4, B=2, P=3, V=151936, dtype="fp16", temperature=0.7,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=11)
    compare_full(d, 0.7, False)
    compare_full(d, 0.7, True)


def test_streaming_kernel_many_tiles():
    """V above the cluster kernel's range with many tiles per CTA and 240
    drafter rows of an odd N (fewer than two per SM, no drafter pairs), so the
    streaming kernel takes the call."""
    w = synth.Workload("big_vocab", N=5, B=24, P=2, V=200000, dtype="bf16", temperature=0.9,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=21)
    a, e, st = run(d, 0.9, False)
    assert st == 0
    rng = np.random.default_rng(4)
    samples = [(int(rng.integers(5)), int(rng.integers(24)), int(rng.integers(2)))
               for _ in range(30)]
    ref = oracle_alpha_rows(d, samples, 0.9, False)
    assert_rel(np.array([a[s] for s in samples]), ref, RTOL_ALPHA, "streaming alpha")
    col = oracle_alpha_rows(d, [(2, 7, k) for k in range(2)], 0.9, False)
    assert_rel(np.array([e[2, 7]]), np.array([1.0 + np.cumprod(col[:-1]).sum()]), RTOL_ALPHA,
               "streaming e_len")


@pytest.mark.parametrize("N,B,P", [(2, 80, 2), (4, 8, 7)])
def test_two_pass_kernel_long_rows(N, B, P):
    """Rows of 200 000 logits, longer than the cluster kernel holds: with 320
    drafter rows the two-pass kernel takes the call on every SM (its L2 working
    set above L2, so some second passes come from HBM), with 224 rows of
    N = 4 one CTA per drafter pair; every alpha and e_len is compared."""
    w = synth.Workload("long_rows", N=N, B=B, P=P, V=200000, dtype="bf16", temperature=0.9,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=22 + N)
    compare_full(d, 0.9, False)


def test_streaming_kernel_lagged_steps():
    """Rows of 2 600 000 logits: 159 chunks per row, more than there are SMs,
    so a tile's items span steps and each overlap comes two steps after its
    statistics; every alpha and e_len is compared."""
    w = synth.Workload("huge_vocab", N=2, B=1, P=2, V=2_600_000, dtype="bf16", temperature=0.9,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=23)
    compare_full(d, 0.9, False)


@pytest.mark.parametrize("T", [0.05, 5.0])
def test_streaming_kernel_fp16_max_drafters(T):
    """fp16, N = 32 (the most the kernel takes) and V = 160 000 at extreme
    temperatures, with the first 100 000 logits of one query's rows masked to
    -inf (its chunks' references come from the rest); every alpha and e_len
    is compared.  At T = 0.05 the noisiest drafters barely overlap the target
    (alpha ~1e-43), so alpha also gets the V * 2^-126 absolute floor of the
    flush to zero below fp32's normal range."""
    w = synth.Workload("big_vocab", N=32, B=2, P=2, V=160000, dtype="fp16", temperature=T,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=24)
    d["target"][1, :, :100000] = float("-inf")
    d["drafter"][:, 1, :, :100000] = float("-inf")
    a, e, st = run(d, T, False)
    ra, re, rst = oracle_feedback(d, T, False)
    assert st == hf.HS_OK and rst == 0
    assert_rel(a, ra, RTOL_ALPHA, "alpha", atol=w.V * 2.0 ** -126)
    assert_rel(e, re, RTOL_ALPHA, "e_len")
    assert np.nanmax(ra) > 0.1, "some pairs must overlap well above the flush floor"


def test_streaming_kernel_flags_bad_rows():
    """V above the cluster kernel's range: a NaN drafter logit in a row's last
    chunk, a +inf one in its first and a drafter row with no finite logit only
    make their own alphas NaN (HS_ERR_NONFINITE); an out-of-range path node
    makes its tile's alphas NaN (HS_ERR_INVALID_ARG)."""
    w = synth.Workload("big_vocab", N=3, B=4, P=3, V=200000, dtype="bf16", temperature=1.0,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=25)
    d["drafter"][2, 3, 1, 199999] = float("nan")
    d["drafter"][0, 1, 0, 7] = float("inf")
    d["drafter"][1, 2, 2, :] = float("-inf")
    a, e, st = run(d, 1.0, False)
    ra, re, rst = oracle_feedback(d, 1.0, False)
    assert st == hf.HS_ERR_NONFINITE
    assert np.array_equal(np.isnan(a), np.isnan(ra)) and np.isnan(a).sum() == 3
    assert np.isnan(a[2, 3, 1]) and np.isnan(a[0, 1, 0]) and np.isnan(a[1, 2, 2])
    assert_rel(a, ra, RTOL_ALPHA, "alpha next to a NaN row")
    t = synth.make_inputs(W["tree_path"], device=DEV, B=3, N=2, V=200000, seed=26)
    t["path"][2, 1] = -1
    a, e, st = run(t, 1.0, False)
    assert st == hf.HS_ERR_INVALID_ARG
    assert np.isnan(a[:, 2, 1]).all() and np.isnan(a).sum() == 2
    t["path"][2, 1] = 3
    compare_full(t, 1.0, False)


@pytest.mark.parametrize("dtype", ["bf16", "fp16"])
def test_two_pass_kernel_every_alpha(dtype):
    """320 tiles of 76808-logit rows: the cluster kernel would hold them on 144
    of the SMs and the rows of every SM fit in L2, so the two-pass kernel
    takes the call (one CTA per SM, the second pass from L2); every alpha and
    e_len is compared."""
    w = synth.Workload("two_pass", N=2, B=80, P=4, V=76808, dtype=dtype, temperature=0.8,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=41)
    compare_full(d, 0.8, False)


def test_two_pass_kernel_flags_bad_rows():
    """A NaN drafter row, and an out-of-range path node: only their alphas
    are NaN, with the status the other kernels report."""
    w = synth.Workload("two_pass", N=2, B=80, P=4, V=76808, dtype="bf16", temperature=1.0,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=42)
    d["drafter"][1, 77, 3, 5] = float("nan")      # in a row's first chunk
    d["drafter"][0, 12, 1, 70000] = float("inf")  # in a late chunk
    a, e, st = run(d, 1.0, False)
    ra, re, rst = oracle_feedback(d, 1.0, False)
    assert st == hf.HS_ERR_NONFINITE
    assert np.array_equal(np.isnan(a), np.isnan(ra)) and np.isnan(a).sum() == 2
    assert np.isnan(a[1, 77, 3]) and np.isnan(a[0, 12, 1])
    assert_rel(a, ra, RTOL_ALPHA, "alpha next to a NaN row")
    t = synth.make_inputs(W["tree_path"], device=DEV, B=80, N=2, V=76808, seed=43)
    t["path"][79, 2] = 999
    a, e, st = run(t, 1.0, False)
    assert st == hf.HS_ERR_INVALID_ARG
    assert np.isnan(a[:, 79, 2]).all() and np.isnan(a).sum() == 2


@pytest.mark.parametrize("dtype", ["bf16", "fp16"])
def test_two_pass_kernel_one_pair_per_cta(dtype):
    """224 drafter rows (N = 4, 56 tiles): fewer than two per SM, so the
    two-pass kernel runs one CTA per pair of drafters of a tile (112 CTAs),
    each reading its tile's target row; every alpha and e_len is compared."""
    w = synth.Workload("pairs", N=4, B=8, P=7, V=76808, dtype=dtype, temperature=0.7,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=49)
    compare_full(d, 0.7, False)


@pytest.mark.parametrize("V,dtype", [(32776, "bf16"), (36872, "fp16"), (200000, "fp16")])
def test_two_pass_kernel_short_last_chunk(V, dtype):
    """Rows whose last 16 384-logit chunk is at most half full, where each
    warp stops that chunk's arithmetic after its last vector holding logits:
    one 8-logit vector in the last chunk (V = 32776, so warps 1-15 have none),
    513 vectors (V = 36872, one lane of warp 0 holds a second vector), and
    424 vectors (V = 200000, warps 14 and 15 have none).  One CTA per drafter
    pair; every alpha and e_len is compared."""
    w = synth.Workload("pairs", N=4, B=8, P=7, V=V, dtype=dtype, temperature=0.8,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=53 + V)
    compare_full(d, 0.8, False)


def test_two_pass_kernel_groups_cross_tiles():
    """N = 5 drafters: the 1600 drafter rows are split evenly over the SMs in
    runs that start and end inside tiles (such a run reads the tile's target
    row again), walked in groups of two, of one at a tile's end and at the
    start of an odd CTA's run; every alpha and e_len is compared."""
    w = synth.Workload("two_pass", N=5, B=64, P=5, V=76808, dtype="bf16", temperature=0.9,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=44)
    compare_full(d, 0.9, False)


@pytest.mark.parametrize("dtype", ["bf16", "fp16"])
def test_two_pass_kernel_qwen_vocab(dtype):
    """Qwen-vocabulary rows (V = 151936) and 960 drafter rows: the target row
    is longer than the 256 KB tensor memory holds, so pass 2 reads its first
    eight chunks from tensor memory and the last two from the ring."""
    w = synth.Workload("two_pass", N=3, B=40, P=8, V=151936, dtype=dtype, temperature=0.7,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=45)
    compare_full(d, 0.7, False)


@pytest.mark.parametrize("T", [0.05, 5.0])
def test_two_pass_kernel_row_extremes(T):
    """The two-pass kernel at extreme temperatures on rows whose largest
    logits sit at the end of the vocabulary (so the first chunk's max is a
    low reference that later chunks must raise), with the first 40000 logits
    of one query's rows masked to -inf; every alpha and e_len is compared."""
    w = synth.Workload("two_pass", N=2, B=80, P=4, V=76808, dtype="bf16", temperature=T,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=46)
    d["target"] = torch.flip(d["target"], dims=[-1]).contiguous()
    d["drafter"] = torch.flip(d["drafter"], dims=[-1]).contiguous()
    d["target"][3, :, :40000] = float("-inf")
    d["drafter"][:, 3, :, :40000] = float("-inf")
    compare_full(d, T, False)


@pytest.mark.parametrize("V", [38408, 65536])
def test_two_pass_kernel_short_rows(V):
    """The shortest rows the two-pass kernel takes (the cluster kernel needs 3
    or 4 CTAs per row there, leaving SMs idle): three chunks with a ragged
    tail (V = 38408), and four full chunks (V = 65536)."""
    w = synth.Workload("two_pass", N=3, B=64, P=5, V=V, dtype="bf16", temperature=0.9,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=47 + V)
    compare_full(d, 0.9, False)


@pytest.mark.parametrize("T", [0.05, 0.5])
def test_two_pass_kernel_large_logits(T):
    """Logits three times the synthetic scale (max around 30): at these
    temperatures a row's log2 normaliser reaches the hundreds, where one fp32
    offset would hold it only to ~3e-5; the kernel keeps its integer reference
    and log2-sum apart there, and every alpha stays within 1e-5 relative.
    Some pairs are nearly disjoint (alpha ~1e-41): terms below the fp32 normal
    range, 2^-126, flush to zero (ex2.approx.ftz), so the comparison also
    allows V * 2^-126 ~ 1e-33 absolute."""
    w = synth.Workload("two_pass", N=2, B=80, P=4, V=76808, dtype="bf16", temperature=T,
                       target="zipf", sigma="qwen")
    d = synth.make_inputs(w, device=DEV, seed=48)
    d["target"] = (d["target"].float() * 3).to(torch.bfloat16)
    d["drafter"] = (d["drafter"].float() * 3).to(torch.bfloat16)
    a, e, st = run(d, T, False)
    ra, re, rst = oracle_feedback(d, T, False)
    assert st == hf.HS_OK and rst == 0
    floor = w.V * 2.0 ** -126
    assert_rel(a, ra, RTOL_ALPHA, "alpha", atol=floor)
    assert_rel(e, re, RTOL_ALPHA, "e_len")
    assert np.nanmax(ra) > 0.1, "some pairs must overlap well above the flush floor"
