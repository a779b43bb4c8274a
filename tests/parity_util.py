"""Helpers for the GPU-vs-oracle parity tests."""
from __future__ import annotations

import concurrent.futures as cf
import os

import numpy as np
import torch

import oracle
from paper_2510_20064_gb300 import synth

# Spec tolerances: alpha and e_len within 1e-5 relative (fp32
# accumulation against the fp64 oracle), weights within 1e-4 relative.
RTOL_ALPHA = 1e-5
RTOL_WEIGHTS = 1e-4
ATOL_WEIGHTS = 1e-7   # fp32 weights far below the largest one carry no relative meaning


def assert_rel(gpu, ref, rtol, what, atol=0.0):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    assert gpu.shape == ref.shape, (what, gpu.shape, ref.shape)
    nan_g, nan_r = np.isnan(gpu), np.isnan(ref)
    assert np.array_equal(nan_g, nan_r), f"{what}: NaN pattern differs"
    g, r = gpu[~nan_r], ref[~nan_r]
    err = np.abs(g - r)
    bound = rtol * np.abs(r) + atol
    bad = err > bound
    if bad.any():
        j = int(np.argmax(err / np.maximum(bound, 1e-300)))
        raise AssertionError(f"{what}: {int(bad.sum())}/{bad.size} outside rtol={rtol} "
                             f"atol={atol}; worst gpu={g[j]!r} ref={r[j]!r}")


def to_np(t: torch.Tensor) -> np.ndarray:
    return t.detach().double().cpu().numpy()


def oracle_feedback(d: dict, T: float, greedy: bool):
    path = d.get("path")
    return oracle.get().feedback(synth.storage_numpy(d["target"]), synth.storage_numpy(d["drafter"]),
                                 T, greedy, path=None if path is None else path.cpu().numpy())


def oracle_alpha_rows(d: dict, samples, T: float, greedy: bool) -> np.ndarray:
    """Oracle alpha for sampled (i, b, k), reading only those rows."""
    o = oracle.get()
    out = np.empty(len(samples))
    path = d.get("path")
    for n, (i, b, k) in enumerate(samples):
        trow = d["target"][b, int(path[b, k])] if path is not None else d["target"][b, k]
        a, _ = o.alpha_pair(synth.storage_numpy(trow), synth.storage_numpy(d["drafter"][i, b, k]),
                            T, greedy)
        out[n] = a
    return out


def host_threads() -> int:
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:
        return os.cpu_count() or 1


def per_query_parallel(call, d: dict, keep: np.ndarray | None = None):
    """Run a whole-call oracle function on every host core: the queries are
    independent, so each thread calls `call(target, drafter, path[, keep])`
    on one query's rows (contiguous copies) and the results are stacked in
    query order -- the same arithmetic and outputs as one call over all
    queries.  Returns (alpha, e_len, first non-zero status or 0)."""
    t_np = synth.storage_numpy(d["target"])
    d_np = synth.storage_numpy(d["drafter"])
    path = d.get("path")
    path_np = None if path is None else path.cpu().numpy().astype(np.int32)
    B = d_np.shape[1]

    def one(b):
        args = [np.ascontiguousarray(t_np[b:b + 1]), np.ascontiguousarray(d_np[:, b:b + 1]),
                None if path_np is None else np.ascontiguousarray(path_np[b:b + 1])]
        if keep is not None:
            args.append(np.ascontiguousarray(keep[:, b:b + 1]))
        return call(*args)

    with cf.ThreadPoolExecutor(max_workers=host_threads()) as ex:
        parts = list(ex.map(one, range(B)))
    alpha = np.concatenate([a for a, _, _ in parts], axis=1)
    e_len = np.concatenate([e for _, e, _ in parts], axis=1)
    status = next((st for _, _, st in parts if st != 0), 0)
    return alpha, e_len, status


def oracle_feedback_parallel(d: dict, T: float, greedy: bool):
    """oracle_feedback on every host core (per_query_parallel)."""
    o = oracle.get()
    return per_query_parallel(lambda t, dr, pa: o.feedback(t, dr, T, greedy, path=pa), d)
