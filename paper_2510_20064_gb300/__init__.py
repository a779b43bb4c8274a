"""Python binding of libhedgefb (HedgeSpec panoramic feedback on GB300).

Argument marshalling only: every entry point checks the tensors it is given
(device, dtype, shape, contiguity), allocates missing outputs with torch and
passes raw pointers to the C ABI declared in ``include/hedgefb.h``.  All
arithmetic runs in the library's CUDA kernels; there is no other code path.
Importing this module fails loudly when ``libhedgefb.so`` has not been built
(``python -m paper_2510_20064_gb300.build`` or ``__graft_entry__.build()``).
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libhedgefb.so")

HS_OK, HS_ERR_INVALID_ARG, HS_ERR_UNSUPPORTED, HS_ERR_MISALIGNED = 0, 1, 2, 3
HS_ERR_NONFINITE, HS_ERR_CUDA, HS_ERR_TIMEOUT = 4, 5, 6
HS_BF16, HS_FP16, HS_FP32 = 0, 1, 2
HS_LOSS_LENGTH, HS_LOSS_ACCEPT = 0, 1
HS_HEDGE, HS_NORMALHEDGE = 0, 1
HS_MAX_LEARNER_N = 32
HS_MAX_TREE_L = 16

_DTYPES = {torch.bfloat16: HS_BF16, torch.float16: HS_FP16, torch.float32: HS_FP32}

# argument/return types of every exported symbol (mirrors include/hedgefb.h)
_P, _I, _F, _Z = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
_L = ctypes.c_int64
SIGNATURES = {
    "hs_status_string": ([_I], ctypes.c_char_p),
    "hs_version": ([], _I),
    "hs_feedback_workspace_size": ([_I, _I, _I, _I, _I, _I], _Z),
    "hs_feedback_kernel_count": ([_I, _I, _I, _I, _I, _I], _I),
    "hs_feedback": ([_P, _P, _I, _I, _I, _I, _I, _F, _I, _P, _P, _P, _Z, _P, _P], _I),
    "hs_feedback_path": ([_P, _P, _I, _P, _I, _I, _I, _I, _I, _F, _I, _P, _P, _P, _Z, _P, _P], _I),
    "hs_feedback_static": ([_P, _P, _I, _I, _I, _I, _I, _F, _I, _P, _P, _P, _P], _I),
    "hs_test_stream_wait_timeout": ([_P, _P, _I, _I, _I, _I, _I, _F, ctypes.c_longlong, _P, _P, _P,
                                     _Z, _P, _P], _I),
    "hs_feedback_topl_workspace_size": ([_I, _I, _I, _I], _Z),
    "hs_feedback_topl_kernel_count": ([_I, _I, _I, _I], _I),
    "hs_feedback_topl": ([_P, _P, _I, _I, _I, _I, _I, _F, _I, _I, _P, _P, _P, _Z, _P, _P], _I),
    "hs_feedback_topl_path": ([_P, _P, _I, _P, _I, _I, _I, _I, _I, _F, _I, _I, _P, _P, _P, _Z,
                               _P, _P], _I),
    "hs_feedback_topl_pruned": ([_P, _P, _I, _I, _I, _I, _I, _F, _I, _I, _P, _P, _P, _P, _Z, _P,
                                 _P], _I),
    "hs_feedback_topl_pruned_path": ([_P, _P, _I, _P, _I, _I, _I, _I, _I, _F, _I, _I, _P, _P, _P,
                                      _P, _Z, _P, _P], _I),
    "hs_hedge_update": ([_P, _I, _I, _F, _P, _P, _P], _I),
    "hs_normalhedge_update": ([_P, _P, _P, _I, _I, _P, _P], _I),
    "hs_learner_step": ([_P, _P, _I, _I, _I, _I, _I, _F, _P, _P, _P, _P, _P, _P], _I),
    "hs_sample_select": ([_P, _I, _I, _P, _P, _P, _P], _I),
    "hs_chunk_learner_step": ([_P, _P, _I, _I, _I, _I, _I, _F, _P, _P, _P, _P, _P, _P, _P], _I),
    "hs_token_append": ([_P, _P, _I, _I, _I, _P, _P, _P, _I, _P, _P, _P, _P], _I),
    "hs_token_learner_step": ([_P, _P, _I, _I, _I, _P, _P, _I, _I, _L, _I, _F, _P, _P, _P, _P,
                               _P, _P], _I),
    "hs_chunk_losses": ([_P, _P, _I, _I, _I, _I, _P, _P, _P], _I),
    "hs_learner_apply": ([_P, _I, _I, _I, _I, _I, _I, _F, _P, _P, _P, _P], _I),
    "hs_schedule_next": ([_P, _P, _I, _P], _I),
}


class HedgeFBError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {hs_status_string(status)}")


_lib = None


def lib():
    """The loaded ``libhedgefb.so`` (ctypes), with argument types set."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(
                f"libhedgefb.so is missing at {LIB_PATH}: build it with "
                "`python -m paper_2510_20064_gb300.build` (needs nvcc); there is no fallback")
        handle = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in SIGNATURES.items():
            fn = getattr(handle, name)
            fn.argtypes = args
            fn.restype = res
        _lib = handle
    return _lib


def hs_status_string(status: int) -> str:
    return lib().hs_status_string(int(status)).decode()


def hs_version() -> int:
    return lib().hs_version()


def _check(status: int, where: str):
    if status != HS_OK:
        raise HedgeFBError(status, where)


def _ptr(t: torch.Tensor | None):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if isinstance(stream, torch.cuda.Stream) else int(stream))


def _need(t: torch.Tensor, name: str, dtype=None, shape=None):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype not in _DTYPES:
        raise ValueError(f"logits must be bf16, fp16 or fp32, got {t.dtype}")
    return _DTYPES[t.dtype]


def hs_feedback_workspace_size(N: int, B: int, P: int, V: int, dtype, greedy: bool) -> int:
    code = dtype if isinstance(dtype, int) else _DTYPES[dtype]
    return int(lib().hs_feedback_workspace_size(N, B, P, V, code, int(bool(greedy))))


def hs_feedback_kernel_count(N: int, B: int, P: int, V: int, dtype, greedy: bool) -> int:
    code = dtype if isinstance(dtype, int) else _DTYPES[dtype]
    return int(lib().hs_feedback_kernel_count(N, B, P, V, code, int(bool(greedy))))


def hs_feedback_topl_kernel_count(N: int, B: int, P: int, V: int) -> int:
    return int(lib().hs_feedback_topl_kernel_count(N, B, P, V))


def hs_feedback_topl_workspace_size(N: int, B: int, P: int, V: int) -> int:
    return int(lib().hs_feedback_topl_workspace_size(N, B, P, V))


def _feedback_outputs(drafter, alpha, e_len, workspace, greedy, with_workspace=True):
    N, B, P, V = drafter.shape
    dev = drafter.device
    if alpha is None:
        alpha = torch.empty((N, B, P), device=dev, dtype=torch.float32)
    if e_len is None:
        e_len = torch.empty((N, B), device=dev, dtype=torch.float32)
    _need(alpha, "alpha", torch.float32, (N, B, P))
    _need(e_len, "e_len", torch.float32, (N, B))
    if not with_workspace:
        return alpha, e_len, None, 0
    ws_bytes = hs_feedback_workspace_size(N, B, P, V, drafter.dtype, greedy)
    if workspace is None and ws_bytes > 0:
        workspace = torch.empty(ws_bytes, device=dev, dtype=torch.uint8)
    return alpha, e_len, workspace, ws_bytes


def hs_feedback(target: torch.Tensor, drafter: torch.Tensor, temperature: float = 1.0,
                greedy: bool = False, alpha=None, e_len=None, workspace=None,
                dev_status=None, stream=None):
    """alpha [N,B,P] and e_len [N,B] (fp32) from target [B,P,V] and drafter
    [N,B,P,V] logits (Thm 1 / Thm 2 with L = 1, Thm 3)."""
    _need(drafter, "drafter")
    N, B, P, V = drafter.shape
    _need(target, "target", drafter.dtype, (B, P, V))
    alpha, e_len, workspace, ws_bytes = _feedback_outputs(drafter, alpha, e_len, workspace, greedy)
    st = lib().hs_feedback(_ptr(target), _ptr(drafter), _dtype_code(drafter), N, B, P, V,
                           float(temperature), int(bool(greedy)), _ptr(alpha), _ptr(e_len),
                           _ptr(workspace), ws_bytes if workspace is not None else 0,
                           _ptr(dev_status), _stream(stream))
    _check(st, "hs_feedback")
    return alpha, e_len


def hs_feedback_static(target: torch.Tensor, drafter: torch.Tensor, temperature: float = 1.0,
                       greedy: bool = False, alpha=None, e_len=None, dev_status=None, stream=None):
    """hs_feedback with its scratch in the library's fixed device array
    (nothing is allocated by the call; see include/hedgefb.h)."""
    _need(drafter, "drafter")
    N, B, P, V = drafter.shape
    _need(target, "target", drafter.dtype, (B, P, V))
    alpha, e_len, _, _ = _feedback_outputs(drafter, alpha, e_len, None, greedy, with_workspace=False)
    st = lib().hs_feedback_static(_ptr(target), _ptr(drafter), _dtype_code(drafter), N, B, P, V,
                                  float(temperature), int(bool(greedy)), _ptr(alpha), _ptr(e_len),
                                  _ptr(dev_status), _stream(stream))
    _check(st, "hs_feedback_static")
    return alpha, e_len


def hs_feedback_path(tree_target: torch.Tensor, path_idx: torch.Tensor, drafter: torch.Tensor,
                     temperature: float = 1.0, greedy: bool = False, alpha=None, e_len=None,
                     workspace=None, dev_status=None, stream=None):
    """As hs_feedback with target row (b,k) = tree_target[b, path_idx[b,k]]."""
    _need(drafter, "drafter")
    N, B, P, V = drafter.shape
    _need(tree_target, "tree_target", drafter.dtype)
    if tree_target.dim() != 3 or tree_target.shape[0] != B or tree_target.shape[2] != V:
        raise ValueError(f"tree_target must be [B, M, V] = [{B}, M, {V}]")
    M = tree_target.shape[1]
    _need(path_idx, "path_idx", torch.int32, (B, P))
    alpha, e_len, workspace, ws_bytes = _feedback_outputs(drafter, alpha, e_len, workspace, greedy)
    st = lib().hs_feedback_path(_ptr(tree_target), _ptr(path_idx), M, _ptr(drafter),
                                _dtype_code(drafter), N, B, P, V, float(temperature),
                                int(bool(greedy)), _ptr(alpha), _ptr(e_len), _ptr(workspace),
                                ws_bytes if workspace is not None else 0, _ptr(dev_status),
                                _stream(stream))
    _check(st, "hs_feedback_path")
    return alpha, e_len


def _topl_outputs(drafter, alpha, e_len, workspace):
    alpha, e_len, _, _ = _feedback_outputs(drafter, alpha, e_len, None, False, with_workspace=False)
    N, B, P, V = drafter.shape
    ws_bytes = lib().hs_feedback_topl_workspace_size(N, B, P, V)
    if workspace is None:
        workspace = torch.empty(max(ws_bytes, 1), device=drafter.device, dtype=torch.uint8)
    return alpha, e_len, workspace, ws_bytes


def hs_feedback_topl(target: torch.Tensor, drafter: torch.Tensor, L: int,
                     temperature: float = 1.0, greedy: bool = False, alpha=None, e_len=None,
                     workspace=None, dev_status=None, stream=None):
    """Draft-tree feedback (Thm 2): alpha [N,B,P] = the target's mass on the
    drafter's top-L tokens (greedy: whether its argmax is among them), and
    e_len [N,B] (Thm 3)."""
    _need(drafter, "drafter")
    N, B, P, V = drafter.shape
    _need(target, "target", drafter.dtype, (B, P, V))
    alpha, e_len, workspace, ws_bytes = _topl_outputs(drafter, alpha, e_len, workspace)
    st = lib().hs_feedback_topl(_ptr(target), _ptr(drafter), _dtype_code(drafter), N, B, P, V,
                                float(temperature), int(bool(greedy)), int(L), _ptr(alpha),
                                _ptr(e_len), _ptr(workspace), ws_bytes, _ptr(dev_status),
                                _stream(stream))
    _check(st, "hs_feedback_topl")
    return alpha, e_len


def hs_feedback_topl_path(tree_target: torch.Tensor, path_idx: torch.Tensor,
                          drafter: torch.Tensor, L: int, temperature: float = 1.0,
                          greedy: bool = False, alpha=None, e_len=None, workspace=None,
                          dev_status=None, stream=None):
    """As hs_feedback_topl with target row (b,k) = tree_target[b, path_idx[b,k]]."""
    _need(drafter, "drafter")
    N, B, P, V = drafter.shape
    _need(tree_target, "tree_target", drafter.dtype)
    if tree_target.dim() != 3 or tree_target.shape[0] != B or tree_target.shape[2] != V:
        raise ValueError(f"tree_target must be [B, M, V] = [{B}, M, {V}]")
    M = tree_target.shape[1]
    _need(path_idx, "path_idx", torch.int32, (B, P))
    alpha, e_len, workspace, ws_bytes = _topl_outputs(drafter, alpha, e_len, workspace)
    st = lib().hs_feedback_topl_path(_ptr(tree_target), _ptr(path_idx), M, _ptr(drafter),
                                     _dtype_code(drafter), N, B, P, V, float(temperature),
                                     int(bool(greedy)), int(L), _ptr(alpha), _ptr(e_len),
                                     _ptr(workspace), ws_bytes, _ptr(dev_status), _stream(stream))
    _check(st, "hs_feedback_topl_path")
    return alpha, e_len


def hs_feedback_topl_pruned(target: torch.Tensor, drafter: torch.Tensor, L: int,
                            keep: torch.Tensor, temperature: float = 1.0, greedy: bool = False,
                            alpha=None, e_len=None, workspace=None, dev_status=None,
                            stream=None):
    """Draft-tree feedback with dynamically pruned child sets (the remark
    closing Thm 2): drafter row (i,b,k)'s candidates are the first
    keep[i,b,k] (int32 [N,B,P], 0..L) of its top-L tokens."""
    _need(drafter, "drafter")
    N, B, P, V = drafter.shape
    _need(target, "target", drafter.dtype, (B, P, V))
    _need(keep, "keep", torch.int32, (N, B, P))
    alpha, e_len, workspace, ws_bytes = _topl_outputs(drafter, alpha, e_len, workspace)
    st = lib().hs_feedback_topl_pruned(_ptr(target), _ptr(drafter), _dtype_code(drafter), N, B, P,
                                       V, float(temperature), int(bool(greedy)), int(L),
                                       _ptr(keep), _ptr(alpha), _ptr(e_len), _ptr(workspace),
                                       ws_bytes, _ptr(dev_status), _stream(stream))
    _check(st, "hs_feedback_topl_pruned")
    return alpha, e_len


def hs_feedback_topl_pruned_path(tree_target: torch.Tensor, path_idx: torch.Tensor,
                                 drafter: torch.Tensor, L: int, keep: torch.Tensor,
                                 temperature: float = 1.0, greedy: bool = False, alpha=None,
                                 e_len=None, workspace=None, dev_status=None, stream=None):
    """As hs_feedback_topl_pruned with target row (b,k) = tree_target[b, path_idx[b,k]]."""
    _need(drafter, "drafter")
    N, B, P, V = drafter.shape
    _need(tree_target, "tree_target", drafter.dtype)
    if tree_target.dim() != 3 or tree_target.shape[0] != B or tree_target.shape[2] != V:
        raise ValueError(f"tree_target must be [B, M, V] = [{B}, M, {V}]")
    M = tree_target.shape[1]
    _need(path_idx, "path_idx", torch.int32, (B, P))
    _need(keep, "keep", torch.int32, (N, B, P))
    alpha, e_len, workspace, ws_bytes = _topl_outputs(drafter, alpha, e_len, workspace)
    st = lib().hs_feedback_topl_pruned_path(_ptr(tree_target), _ptr(path_idx), M, _ptr(drafter),
                                            _dtype_code(drafter), N, B, P, V, float(temperature),
                                            int(bool(greedy)), int(L), _ptr(keep), _ptr(alpha),
                                            _ptr(e_len), _ptr(workspace), ws_bytes,
                                            _ptr(dev_status), _stream(stream))
    _check(st, "hs_feedback_topl_pruned_path")
    return alpha, e_len


def hs_hedge_update(cum_loss: torch.Tensor, eta: float, weights=None, selected=None, stream=None):
    """Hedge weights exp(-eta L)/Z and first argmin of L, per query."""
    _need(cum_loss, "cum_loss", torch.float32)
    N, B = cum_loss.shape
    if weights is None:
        weights = torch.empty_like(cum_loss)
    if selected is None:
        selected = torch.empty(B, device=cum_loss.device, dtype=torch.int32)
    _need(weights, "weights", torch.float32, (N, B))
    _need(selected, "selected", torch.int32, (B,))
    _check(lib().hs_hedge_update(_ptr(cum_loss), N, B, float(eta), _ptr(weights),
                                 _ptr(selected), _stream(stream)), "hs_hedge_update")
    return weights, selected


def hs_normalhedge_update(regret: torch.Tensor, loss: torch.Tensor, weights: torch.Tensor,
                          selected=None, stream=None):
    """One NormalHedge round in place on (regret, weights)."""
    _need(regret, "regret", torch.float32)
    N, B = regret.shape
    _need(loss, "loss", torch.float32, (N, B))
    _need(weights, "weights", torch.float32, (N, B))
    if selected is None:
        selected = torch.empty(B, device=regret.device, dtype=torch.int32)
    _need(selected, "selected", torch.int32, (B,))
    _check(lib().hs_normalhedge_update(_ptr(regret), _ptr(loss), _ptr(weights), N, B,
                                       _ptr(selected), _stream(stream)), "hs_normalhedge_update")
    return regret, weights, selected


def hs_learner_step(alpha: torch.Tensor, e_len: torch.Tensor, loss_kind: int, learner: int,
                    eta: float, state: torch.Tensor, weights: torch.Tensor,
                    selected: torch.Tensor, loss_out=None, played_loss=None, stream=None):
    """Fused loss + learner round in place on (state, weights, selected)."""
    _need(alpha, "alpha", torch.float32)
    N, B, P = alpha.shape
    _need(e_len, "e_len", torch.float32, (N, B))
    _need(state, "state", torch.float32, (N, B))
    _need(weights, "weights", torch.float32, (N, B))
    _need(selected, "selected", torch.int32, (B,))
    if loss_out is not None:
        _need(loss_out, "loss_out", torch.float32, (N, B))
    if played_loss is not None:
        _need(played_loss, "played_loss", torch.float32, (B,))
    _check(lib().hs_learner_step(_ptr(alpha), _ptr(e_len), N, B, P, int(loss_kind), int(learner),
                                 float(eta), _ptr(state), _ptr(weights), _ptr(loss_out),
                                 _ptr(selected), _ptr(played_loss), _stream(stream)),
           "hs_learner_step")
    return state, weights, selected


# ---- delayed feedback and sampled play (App. B.1, B.3, B.5; Sec. 3.2) -------------

def hs_sample_select(weights: torch.Tensor, uniforms: torch.Tensor, selected=None,
                     dev_status=None, stream=None) -> torch.Tensor:
    """Inverse-CDF draw per query from weights [N,B] with uniforms [B]."""
    _need(weights, "weights", torch.float32)
    N, B = weights.shape
    _need(uniforms, "uniforms", torch.float32, (B,))
    if selected is None:
        selected = torch.empty(B, dtype=torch.int32, device=weights.device)
    _need(selected, "selected", torch.int32, (B,))
    _check(lib().hs_sample_select(_ptr(weights), N, B, _ptr(uniforms), _ptr(selected),
                                  _ptr(dev_status), _stream(stream)), "hs_sample_select")
    return selected


def hs_chunk_learner_step(alpha: torch.Tensor, k_h: torch.Tensor, loss_kind: int, learner: int,
                          eta: float, state: torch.Tensor, weights: torch.Tensor,
                          selected: torch.Tensor, loss_out=None, played_loss=None,
                          dev_status=None, stream=None):
    """Chunk-level round with per-query chunk horizon k_h [B] int32, in place."""
    _need(alpha, "alpha", torch.float32)
    N, B, P = alpha.shape
    _need(k_h, "k_h", torch.int32, (B,))
    _need(state, "state", torch.float32, (N, B))
    _need(weights, "weights", torch.float32, (N, B))
    _need(selected, "selected", torch.int32, (B,))
    if loss_out is not None:
        _need(loss_out, "loss_out", torch.float32, (N, B))
    if played_loss is not None:
        _need(played_loss, "played_loss", torch.float32, (B,))
    _check(lib().hs_chunk_learner_step(_ptr(alpha), _ptr(k_h), N, B, P, int(loss_kind),
                                       int(learner), float(eta), _ptr(state), _ptr(weights),
                                       _ptr(loss_out), _ptr(selected), _ptr(played_loss),
                                       _ptr(dev_status), _stream(stream)),
           "hs_chunk_learner_step")
    return state, weights, selected


class TokenStream:
    """Device state of the token-level game with delay for B queries: the
    gamma ring [B,H,N], the ring of playing drafters [B,H] and the token
    counters; hs_token_append / hs_token_learner_step work on it in place."""

    def __init__(self, N: int, B: int, H: int, device):
        self.N, self.B, self.H = N, B, H
        self.gamma = torch.zeros(B, H, N, dtype=torch.float32, device=device)
        self.who = torch.zeros(B, H, dtype=torch.int32, device=device)
        self.n_tok = torch.zeros(B, dtype=torch.int64, device=device)
        self.n_done = torch.zeros(B, dtype=torch.int64, device=device)


def hs_token_append(ts: TokenStream, alpha: torch.Tensor, k_h: torch.Tensor,
                    selected: torch.Tensor, dev_status=None, stream=None) -> None:
    _need(alpha, "alpha", torch.float32)
    N, B, P = alpha.shape
    assert (N, B) == (ts.N, ts.B)
    _need(k_h, "k_h", torch.int32, (B,))
    _need(selected, "selected", torch.int32, (B,))
    _check(lib().hs_token_append(_ptr(alpha), _ptr(k_h), N, B, P, _ptr(selected),
                                 _ptr(ts.gamma), _ptr(ts.who), ts.H, _ptr(ts.n_tok),
                                 _ptr(ts.n_done), _ptr(dev_status), _stream(stream)),
           "hs_token_append")


def hs_token_learner_step(ts: TokenStream, K: int, loss_kind: int, learner: int, eta: float,
                          state: torch.Tensor, weights: torch.Tensor, selected: torch.Tensor,
                          accept_first: int = 0, played_loss=None, dev_status=None,
                          stream=None):
    """QFI-D catch-up on the revealed token losses, in place."""
    N, B = ts.N, ts.B
    _need(state, "state", torch.float32, (N, B))
    _need(weights, "weights", torch.float32, (N, B))
    _need(selected, "selected", torch.int32, (B,))
    if played_loss is not None:
        _need(played_loss, "played_loss", torch.float32, (B,))
    _check(lib().hs_token_learner_step(_ptr(ts.gamma), _ptr(ts.who), N, B, ts.H, _ptr(ts.n_tok),
                                       _ptr(ts.n_done), int(K), int(loss_kind),
                                       int(accept_first), int(learner), float(eta), _ptr(state),
                                       _ptr(weights), _ptr(selected), _ptr(played_loss),
                                       _ptr(dev_status), _stream(stream)),
           "hs_token_learner_step")
    return state, weights, selected


def hs_chunk_losses(alpha: torch.Tensor, k_h: torch.Tensor, loss_kind: int, loss_out=None,
                    dev_status=None, stream=None) -> torch.Tensor:
    """Chunk-level loss vectors [N,B] with per-query chunk horizon k_h [B]."""
    _need(alpha, "alpha", torch.float32)
    N, B, P = alpha.shape
    _need(k_h, "k_h", torch.int32, (B,))
    if loss_out is None:
        loss_out = torch.empty(N, B, dtype=torch.float32, device=alpha.device)
    _need(loss_out, "loss_out", torch.float32, (N, B))
    _check(lib().hs_chunk_losses(_ptr(alpha), _ptr(k_h), N, B, P, int(loss_kind), _ptr(loss_out),
                                 _ptr(dev_status), _stream(stream)), "hs_chunk_losses")
    return loss_out


def hs_learner_apply(queue: torch.Tensor, first: int, count: int, learner: int, eta: float,
                     state: torch.Tensor, weights: torch.Tensor, selected: torch.Tensor,
                     stream=None):
    """QFI-D catch-up over count loss vectors of queue [Q,N,B] from slot first."""
    _need(queue, "queue", torch.float32)
    Q, N, B = queue.shape
    _need(state, "state", torch.float32, (N, B))
    _need(weights, "weights", torch.float32, (N, B))
    _need(selected, "selected", torch.int32, (B,))
    _check(lib().hs_learner_apply(_ptr(queue), Q, int(first), int(count), N, B, int(learner),
                                  float(eta), _ptr(state), _ptr(weights), _ptr(selected),
                                  _stream(stream)), "hs_learner_apply")
    return state, weights, selected


class ScheduleConfig(ctypes.Structure):
    _fields_ = [("warmup_rounds", ctypes.c_int), ("batch_rounds", ctypes.c_int),
                ("skip_tokens", ctypes.c_int), ("hybrid_vectors", ctypes.c_int)]


class ScheduleState(ctypes.Structure):
    _fields_ = [("rounds", ctypes.c_int64), ("tokens_since_eval", ctypes.c_int64),
                ("vectors_made", ctypes.c_int64), ("vectors_queued", ctypes.c_int64)]


class ScheduleAction(ctypes.Structure):
    _fields_ = [("evaluate", ctypes.c_int), ("loss_kind", ctypes.c_int), ("apply", ctypes.c_int)]


class Schedule:
    """App. B.5's practical schedule (host-side, in the library): one
    next(tokens) per speculative chunk -> (evaluate, loss_kind, apply)."""

    def __init__(self, warmup_rounds: int = 6, batch_rounds: int = 12, skip_tokens: int = 6,
                 hybrid_vectors: int = 0):
        self.cfg = ScheduleConfig(warmup_rounds, batch_rounds, skip_tokens, hybrid_vectors)
        self.state = ScheduleState()

    def next(self, tokens: int) -> tuple[int, int, int]:
        act = ScheduleAction()
        _check(lib().hs_schedule_next(ctypes.byref(self.cfg), ctypes.byref(self.state),
                                      int(tokens), ctypes.byref(act)), "hs_schedule_next")
        return act.evaluate, act.loss_kind, act.apply
