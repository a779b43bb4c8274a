"""fp64 CPU oracle for the HedgeSpec panoramic-feedback path.

TEST INFRASTRUCTURE ONLY: this package is imported by ``tests/``, by
``__graft_entry__.smoke()`` and by the CPU-baseline leg of ``bench.py``, and
by nothing else.  It wraps ``hedgefb_oracle.c`` (plain C, fp64) through
ctypes and takes numpy arrays only; it never touches the CUDA library.

Logit arrays are passed as their stored bytes: ``np.uint16`` for bf16,
``np.float16`` for fp16, ``np.float32`` for fp32.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "hedgefb_oracle.c")
_LIB = os.path.join(_HERE, "libhedgefb_oracle.so")

BF16, FP16, FP32 = 0, 1, 2
LOSS_LENGTH, LOSS_ACCEPT = 0, 1
HEDGE, NORMALHEDGE = 0, 1
OK, BADARG, NONFINITE = 0, 1, 4


def build(src: str = _SRC, out: str = _LIB) -> str:
    """Compile the oracle with gcc (IEEE fp64, no contraction, no fast-math)."""
    cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fPIC", "-shared",
           "-o", out, src, "-lm"]
    subprocess.run(cmd, check=True)
    return out


def _bind(lib):
    P, I, D, L = ctypes.c_void_p, ctypes.c_int, ctypes.c_double, ctypes.c_int64
    sig = {
        "orc_decode": ([P, I, L], D),
        "orc_row_probs": ([P, I, I, D, P], I),
        "orc_row_argmax": ([P, I, I], I),
        "orc_overlap": ([P, P, I], D),
        "orc_tv": ([P, P, I], D),
        "orc_alpha_pair": ([P, P, I, I, D, I, P], I),
        "orc_elen_prefix": ([P, I], D),
        "orc_elen_thm3": ([P, I], D),
        "orc_loss_length": ([D, I], D),
        "orc_loss_accept": ([P, I], D),
        "orc_feedback": ([P, P, I, I, I, I, I, D, I, P, P], I),
        "orc_feedback_path": ([P, P, I, P, I, I, I, I, I, D, I, P, P], I),
        "orc_topl_set": ([P, I, I, I, P], None),
        "orc_alpha_topl": ([P, P, I, I, D, I, I, P], I),
        "orc_feedback_topl": ([P, P, I, P, I, I, I, I, I, D, I, I, P, P], I),
        "orc_alpha_topl_pruned": ([P, P, I, I, D, I, I, I, P], I),
        "orc_feedback_topl_pruned": ([P, P, I, P, I, I, I, I, I, D, I, I, P, P, P], I),
        "orc_hedge": ([P, I, D, P, P], None),
        "orc_normalhedge": ([P, P, P, I, P, P], I),
        "orc_learner_step": ([P, P, I, I, I, I, I, D, P, P, P, P, P], I),
        "orc_sample_select": ([P, I, ctypes.c_float], I),
        "orc_chunk_loss": ([P, I, I], D),
        "orc_chunk_learner_step": ([P, I, I, I, P, I, I, D, P, P, P, P, P], I),
        "orc_token_loss": ([P, L, I, I], D),
        "orc_token_revealed": ([L, I, I, L], L),
        "orc_token_session": ([P, P, I, I, I, I, I, I, L, I, D, P, P, P, P, P, P], I),
        "orc_learner_apply": ([P, I, I, I, I, D, P, P, P], I),
        "orc_schedule_next": ([I, I, I, I, P, I, P], I),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    return lib


def _ptr(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def dtype_code(arr: np.ndarray) -> int:
    if arr.dtype == np.uint16:
        return BF16
    if arr.dtype == np.float16:
        return FP16
    if arr.dtype == np.float32:
        return FP32
    raise TypeError(f"logits must be uint16 (bf16 bits), float16 or float32, got {arr.dtype}")


class Oracle:
    """ctypes binding of one build of ``hedgefb_oracle.c``."""

    def __init__(self, path: str | None = None):
        if path is None:
            path = _LIB
            if (not os.path.exists(path)
                    or os.path.getmtime(path) < os.path.getmtime(_SRC)):
                build()
        self.lib = _bind(ctypes.CDLL(path))

    # ---- per-row pieces ----------------------------------------------------

    def row_probs(self, row: np.ndarray, T: float):
        row = np.ascontiguousarray(row)
        out = np.empty(row.shape[-1], np.float64)
        st = self.lib.orc_row_probs(_ptr(row), dtype_code(row), row.shape[-1], float(T),
                                    _ptr(out))
        return out, st

    def row_argmax(self, row: np.ndarray) -> int:
        row = np.ascontiguousarray(row)
        return self.lib.orc_row_argmax(_ptr(row), dtype_code(row), row.shape[-1])

    def decode(self, row: np.ndarray) -> np.ndarray:
        row = np.ascontiguousarray(row).reshape(-1)
        return np.array([self.lib.orc_decode(_ptr(row), dtype_code(row), i)
                         for i in range(row.shape[0])])

    def overlap(self, p, q) -> float:
        p, q = _f64(p), _f64(q)
        return self.lib.orc_overlap(_ptr(p), _ptr(q), p.shape[0])

    def tv(self, p, q) -> float:
        p, q = _f64(p), _f64(q)
        return self.lib.orc_tv(_ptr(p), _ptr(q), p.shape[0])

    def alpha_pair(self, zt: np.ndarray, zd: np.ndarray, T: float, greedy: bool):
        zt, zd = np.ascontiguousarray(zt), np.ascontiguousarray(zd)
        assert zt.dtype == zd.dtype and zt.shape == zd.shape
        out = ctypes.c_double()
        st = self.lib.orc_alpha_pair(_ptr(zt), _ptr(zd), dtype_code(zt), zt.shape[-1],
                                     float(T), int(bool(greedy)), ctypes.byref(out))
        return out.value, st

    # ---- Thm 3 and losses --------------------------------------------------

    def elen_prefix(self, gamma) -> float:
        g = _f64(gamma)
        return self.lib.orc_elen_prefix(_ptr(g), g.shape[0])

    def elen_thm3(self, gamma) -> float:
        g = _f64(gamma)
        return self.lib.orc_elen_thm3(_ptr(g), g.shape[0])

    def loss_length(self, e_len: float, K: int) -> float:
        return self.lib.orc_loss_length(float(e_len), int(K))

    def loss_accept(self, gamma) -> float:
        g = _f64(gamma)
        return self.lib.orc_loss_accept(_ptr(g), g.shape[0])

    # ---- whole feedback call -----------------------------------------------

    def feedback(self, target: np.ndarray, drafter: np.ndarray, T: float, greedy: bool,
                 path: np.ndarray | None = None):
        """alpha [N,B,P] and e_len [N,B] in fp64; returns (alpha, e_len, status).

        target is [B,P,V] (chain) or [B,M,V] with ``path`` [B,P] int32 (tree
        rows on the verified path); drafter is [N,B,P,V]."""
        target = np.ascontiguousarray(target)
        drafter = np.ascontiguousarray(drafter)
        assert target.dtype == drafter.dtype
        N, B, P, V = drafter.shape
        alpha = np.empty((N, B, P), np.float64)
        e_len = np.empty((N, B), np.float64)
        if path is None:
            assert target.shape == (B, P, V)
            st = self.lib.orc_feedback(_ptr(target), _ptr(drafter), dtype_code(target),
                                       N, B, P, V, float(T), int(bool(greedy)),
                                       _ptr(alpha), _ptr(e_len))
        else:
            path = np.ascontiguousarray(path, dtype=np.int32)
            M = target.shape[1]
            assert target.shape == (B, M, V) and path.shape == (B, P)
            st = self.lib.orc_feedback_path(_ptr(target), _ptr(path), M, _ptr(drafter),
                                            dtype_code(target), N, B, P, V, float(T),
                                            int(bool(greedy)), _ptr(alpha), _ptr(e_len))
        return alpha, e_len, st

    # ---- Thm 2: EAGLE tree with branching L ---------------------------------

    def topl_set(self, row: np.ndarray, L: int) -> np.ndarray:
        """Top_L(q) of one drafter row, in rank order (ties -> lower index)."""
        row = np.ascontiguousarray(row)
        L = min(int(L), row.shape[-1])
        idx = np.empty(L, np.int32)
        self.lib.orc_topl_set(_ptr(row), dtype_code(row), row.shape[-1], L, _ptr(idx))
        return idx

    def alpha_topl(self, zt: np.ndarray, zd: np.ndarray, T: float, greedy: bool, L: int):
        zt = np.ascontiguousarray(zt)
        zd = np.ascontiguousarray(zd)
        a = ctypes.c_double()
        st = self.lib.orc_alpha_topl(_ptr(zt), _ptr(zd), dtype_code(zt), zt.shape[-1], float(T),
                                     int(bool(greedy)), int(L), ctypes.byref(a))
        return a.value, st

    def feedback_topl(self, target: np.ndarray, drafter: np.ndarray, T: float, greedy: bool,
                      L: int, path: np.ndarray | None = None):
        """As feedback() with Thm 2's acceptance: alpha = the target's mass
        on the drafter's top-L tokens (greedy target: whether its argmax is
        among them)."""
        target = np.ascontiguousarray(target)
        drafter = np.ascontiguousarray(drafter)
        assert target.dtype == drafter.dtype
        N, B, P, V = drafter.shape
        alpha = np.empty((N, B, P), np.float64)
        e_len = np.empty((N, B), np.float64)
        if path is None:
            assert target.shape == (B, P, V)
            pp, M = None, 0
        else:
            pp = np.ascontiguousarray(path, dtype=np.int32)
            M = target.shape[1]
            assert target.shape == (B, M, V) and pp.shape == (B, P)
        st = self.lib.orc_feedback_topl(_ptr(target), None if pp is None else _ptr(pp), M,
                                        _ptr(drafter), dtype_code(target), N, B, P, V, float(T),
                                        int(bool(greedy)), int(L), _ptr(alpha), _ptr(e_len))
        return alpha, e_len, st

    def alpha_topl_pruned(self, zt: np.ndarray, zd: np.ndarray, T: float, greedy: bool, L: int,
                          keep: int):
        zt = np.ascontiguousarray(zt)
        zd = np.ascontiguousarray(zd)
        a = ctypes.c_double()
        st = self.lib.orc_alpha_topl_pruned(_ptr(zt), _ptr(zd), dtype_code(zt), zt.shape[-1],
                                            float(T), int(bool(greedy)), int(L), int(keep),
                                            ctypes.byref(a))
        return a.value, st

    def feedback_topl_pruned(self, target: np.ndarray, drafter: np.ndarray, T: float,
                             greedy: bool, L: int, keep: np.ndarray,
                             path: np.ndarray | None = None):
        """feedback_topl() with the dynamically pruned candidate sets: the
        first keep[i,b,k] of drafter row (i,b,k)'s top-L tokens."""
        target = np.ascontiguousarray(target)
        drafter = np.ascontiguousarray(drafter)
        assert target.dtype == drafter.dtype
        N, B, P, V = drafter.shape
        keep = np.ascontiguousarray(keep, dtype=np.int32)
        assert keep.shape == (N, B, P)
        alpha = np.empty((N, B, P), np.float64)
        e_len = np.empty((N, B), np.float64)
        if path is None:
            assert target.shape == (B, P, V)
            pp, M = None, 0
        else:
            pp = np.ascontiguousarray(path, dtype=np.int32)
            M = target.shape[1]
            assert target.shape == (B, M, V) and pp.shape == (B, P)
        st = self.lib.orc_feedback_topl_pruned(_ptr(target), None if pp is None else _ptr(pp), M,
                                               _ptr(drafter), dtype_code(target), N, B, P, V,
                                               float(T), int(bool(greedy)), int(L), _ptr(keep),
                                               _ptr(alpha), _ptr(e_len))
        return alpha, e_len, st

    # ---- learners ----------------------------------------------------------

    def hedge(self, L, eta: float):
        L = _f64(L)
        w = np.empty_like(L)
        sel = ctypes.c_int()
        self.lib.orc_hedge(_ptr(L), L.shape[0], float(eta), _ptr(w), ctypes.byref(sel))
        return w, sel.value

    def normalhedge(self, R, loss, p):
        """One NormalHedge round; returns (R_t, p_{t+1}, selected, c_t)."""
        R, loss, p = _f64(R).copy(), _f64(loss), _f64(p).copy()
        sel, c = ctypes.c_int(), ctypes.c_double()
        self.lib.orc_normalhedge(_ptr(R), _ptr(loss), _ptr(p), R.shape[0],
                                 ctypes.byref(sel), ctypes.byref(c))
        return R, p, sel.value, c.value

    def learner_step(self, alpha, e_len, loss_kind: int, learner_kind: int, eta: float,
                     state, weights, selected, played=None):
        """One batched learner round; arrays [N,B] (alpha [N,B,P]).

        Returns (state, weights, loss, selected, played) as new arrays."""
        alpha, e_len = _f64(alpha), _f64(e_len)
        N, B, P = alpha.shape
        state, weights = _f64(state).copy(), _f64(weights).copy()
        sel = np.ascontiguousarray(selected, dtype=np.int32).copy()
        loss = np.empty((N, B), np.float64)
        pl = None if played is None else _f64(played).copy()
        st = self.lib.orc_learner_step(_ptr(alpha), _ptr(e_len), N, B, P, int(loss_kind),
                                       int(learner_kind), float(eta), _ptr(state),
                                       _ptr(weights), _ptr(loss), _ptr(sel),
                                       None if pl is None else _ptr(pl))
        if st != OK:
            raise ValueError(f"oracle learner_step rejected its arguments (status {st})")
        return state, weights, loss, sel, pl


    # ---- App. B.1 (QFI-D): sampled play; App. B.3 / Sec. 3.2 delayed games ----

    def sample_select(self, w, u: float) -> int:
        """Inverse-CDF draw from fp32 weights w[N] with uniform u (fp32)."""
        w = np.ascontiguousarray(w, dtype=np.float32)
        return int(self.lib.orc_sample_select(_ptr(w), w.shape[0], float(np.float32(u))))

    def chunk_loss(self, gamma, k: int, loss_kind: int) -> float:
        g = _f64(gamma)
        return float(self.lib.orc_chunk_loss(_ptr(g), int(k), int(loss_kind)))

    def chunk_learner_step(self, alpha, k_h, loss_kind: int, learner_kind: int, eta: float,
                           state, weights, selected, played=None):
        """Chunk-level round with per-query chunk horizon k_h[B]; returns
        (state, weights, loss, selected, played) as new arrays."""
        alpha = _f64(alpha)
        N, B, P = alpha.shape
        kh = np.ascontiguousarray(k_h, dtype=np.int32)
        state, weights = _f64(state).copy(), _f64(weights).copy()
        sel = np.ascontiguousarray(selected, dtype=np.int32).copy()
        loss = np.empty((N, B), np.float64)
        pl = None if played is None else _f64(played).copy()
        st = self.lib.orc_chunk_learner_step(_ptr(alpha), N, B, P, _ptr(kh), int(loss_kind),
                                             int(learner_kind), float(eta), _ptr(state),
                                             _ptr(weights), _ptr(loss), _ptr(sel),
                                             None if pl is None else _ptr(pl))
        if st != OK:
            raise ValueError(f"oracle chunk_learner_step rejected its arguments (status {st})")
        return state, weights, loss, sel, pl

    def token_loss(self, g, s: int, K: int, loss_kind: int) -> float:
        g = _f64(g)
        return float(self.lib.orc_token_loss(_ptr(g), int(s), int(K), int(loss_kind)))

    def token_revealed(self, n: int, K: int, loss_kind: int, accept_first: int = 0) -> int:
        return int(self.lib.orc_token_revealed(int(n), int(K), int(loss_kind), int(accept_first)))

    def token_session(self, alpha, k_h, K: int, loss_kind: int, learner_kind: int, eta: float,
                      state, weights, sel0, accept_first: int = 0):
        """Token-level QFI-D session; alpha [H,N,B,P], k_h [H,B].  Returns
        (state, weights, sel [H,B], played [B], processed [B])."""
        alpha = _f64(alpha)
        H, N, B, P = alpha.shape
        kh = np.ascontiguousarray(k_h, dtype=np.int32)
        state, weights = _f64(state).copy(), _f64(weights).copy()
        s0 = np.ascontiguousarray(sel0, dtype=np.int32)
        sel = np.zeros((H, B), np.int32)
        played = np.zeros(B, np.float64)
        done = np.zeros(B, np.int64)
        st = self.lib.orc_token_session(_ptr(alpha), _ptr(kh), H, N, B, P, int(K), int(loss_kind),
                                        int(accept_first), int(learner_kind), float(eta),
                                        _ptr(state), _ptr(weights), _ptr(s0), _ptr(sel),
                                        _ptr(played), _ptr(done))
        if st != OK:
            raise ValueError(f"oracle token_session rejected its arguments (status {st})")
        return state, weights, sel, played, done


    # ---- App. B.5 practical heuristics --------------------------------------

    def learner_apply(self, lv, learner_kind: int, eta: float, state, weights, selected):
        """QFI-D catch-up over loss vectors lv [C,N,B] in order; new arrays."""
        lv = _f64(lv)
        C, N, B = lv.shape
        state, weights = _f64(state).copy(), _f64(weights).copy()
        sel = np.ascontiguousarray(selected, dtype=np.int32).copy()
        st = self.lib.orc_learner_apply(_ptr(lv), C, N, B, int(learner_kind), float(eta),
                                        _ptr(state), _ptr(weights), _ptr(sel))
        if st != OK:
            raise ValueError(f"oracle learner_apply rejected its arguments (status {st})")
        return state, weights, sel

    def schedule(self, warmup: int, batch_rounds: int, skip_tokens: int, hybrid_vectors: int,
                 tokens):
        """Decisions (evaluate, loss_kind, apply) for each round of a token
        sequence tokens[r] (tokens generated by round r's chunk)."""
        s = np.zeros(4, np.int64)
        act = np.zeros(3, np.int32)
        out = []
        for t in tokens:
            st = self.lib.orc_schedule_next(int(warmup), int(batch_rounds), int(skip_tokens),
                                            int(hybrid_vectors), _ptr(s), int(t), _ptr(act))
            if st != OK:
                raise ValueError(f"oracle schedule rejected its arguments (status {st})")
            out.append(tuple(int(x) for x in act))
        return out


_default: Oracle | None = None


def get() -> Oracle:
    """The oracle built from this directory's source (built on first use)."""
    global _default
    if _default is None:
        _default = Oracle()
    return _default
