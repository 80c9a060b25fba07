"""Thin Python binding of the C ABI in ``include/pr2.h`` (argument marshalling only).

Every function here has the name of the C entry point it calls and passes torch tensors as raw
device pointers; all of the layer's arithmetic runs in ``libpr2.so``.  There is no fallback:
if the library is missing the first call raises.  Output tensors are allocated by the caller
(``torch.empty`` on the GPU) - the ``alloc_*`` helpers below do just that.
"""
from __future__ import annotations

import ctypes
import os
import re
import threading
from typing import Optional

import torch

from . import build as _build

_lock = threading.Lock()
_lib: Optional[ctypes.CDLL] = None

PR2_OK = 0
PR2_FP32, PR2_BF16 = 0, 1
PR2_F_SYNC_STATUS = 0x1
PR2_F_DELTA_LOSS = 0x2
PR2_F_NORMALIZE_TOPK = 0x4
PR2_STATUS_BAD_INDEX = 0x1
PR2_STATUS_TIMEOUT = 0x2
PR2_NEAR_TIE_GAP = 1e-4
STATUS_NAMES = {0: "PR2_OK", 1: "PR2_ERR_INVALID_ARG", 2: "PR2_ERR_UNSUPPORTED", 3: "PR2_ERR_CUDA",
                4: "PR2_ERR_BAD_INDEX", 5: "PR2_ERR_TIMEOUT", 6: "PR2_ERR_WORKSPACE"}


class Pr2Error(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"{where}: {STATUS_NAMES.get(code, code)} ({pr2_strerror(code)})")
        self.code = code


class Dims(ctypes.Structure):
    """``pr2_dims``: T tokens, d, N experts, top-k, m = d_ff, n_shared, dtype, flags."""

    _fields_ = [("T", ctypes.c_int64), ("d", ctypes.c_int32), ("N", ctypes.c_int32),
                ("k", ctypes.c_int32), ("m", ctypes.c_int32), ("n_shared", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("flags", ctypes.c_uint32)]


class StageEvents(ctypes.Structure):
    """``pr2_stage_events``: cudaEvent_t handles recorded inside pr2_moe_forward."""

    _fields_ = [("start", ctypes.c_void_p), ("dispatched", ctypes.c_void_p),
                ("gate_up_done", ctypes.c_void_p), ("down_done", ctypes.c_void_p),
                ("end", ctypes.c_void_p)]


def stage_events(events) -> StageEvents:
    """Build a ``pr2_stage_events`` from five recorded ``torch.cuda.Event`` objects (or None)."""
    return StageEvents(*[None if e is None else ctypes.c_void_p(e.cuda_event) for e in events])


def dims(T: int, d: int, N: int, k: int, m: int, n_shared: int = 0, dtype: str = "bf16",
         flags: int = 0) -> Dims:
    code = {"fp32": PR2_FP32, "bf16": PR2_BF16}[dtype]
    return Dims(T, d, N, k, m, n_shared, code, flags)


def library_path() -> str:
    return _build.LIB


def load() -> ctypes.CDLL:
    """Load ``libpr2.so`` (built by ``paper_2606_00395_gb300.build``); raise if it is absent."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = library_path()
        if not os.path.exists(path):
            raise RuntimeError(
                f"libpr2.so not found at {path}: build it with "
                "`python -m paper_2606_00395_gb300.build` (there is no non-CUDA fallback)")
        lib = ctypes.CDLL(path)
        P, I32, I64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        D = ctypes.POINTER(Dims)
        lib.pr2_route_predict.argtypes = [D, P, P, P, P, P, P, P, P, P]
        lib.pr2_route_predict.restype = ctypes.c_int
        lib.pr2_route_replay.argtypes = [D, P, P, P, P, P, P, P]
        lib.pr2_route_replay.restype = ctypes.c_int
        lib.pr2_moe_workspace_bytes.argtypes = [D]
        lib.pr2_moe_workspace_bytes.restype = ctypes.c_size_t
        lib.pr2_moe_forward.argtypes = [D, P, P, P, P, P, P, P, P, P, P, P, P, P, ctypes.c_size_t,
                                        P, ctypes.POINTER(StageEvents), P]
        lib.pr2_moe_forward.restype = ctypes.c_int
        lib.pr2_strerror.argtypes = [ctypes.c_int]
        lib.pr2_strerror.restype = ctypes.c_char_p
        lib.pr2_selftest_wait_timeout.argtypes = [P, I64, P]
        lib.pr2_selftest_wait_timeout.restype = ctypes.c_int
        lib.pr2_predictor_loss_workspace_bytes.argtypes = [D]
        lib.pr2_predictor_loss_workspace_bytes.restype = ctypes.c_size_t
        lib.pr2_predictor_loss.argtypes = [D, P, P, P, P, I64, P, P, P, P, P, ctypes.c_size_t, P,
                                           P]
        lib.pr2_predictor_loss.restype = ctypes.c_int
        lib.pr2_route_diagnostics.argtypes = [D, P, P, P, P, P]
        lib.pr2_route_diagnostics.restype = ctypes.c_int
        lib.pr2_feature_cache_write.argtypes = [D, I64, P, P, P, P, P, P]
        lib.pr2_feature_cache_write.restype = ctypes.c_int
        lib.pr2_rollout_layers.argtypes = [D, I32, P, P, P, P, P, P, P, P, P, P, P, P, P, P,
                                           ctypes.c_size_t, P, P]
        lib.pr2_rollout_layers.restype = ctypes.c_int
        lib.pr2_moe_replay_forward.argtypes = [D, P, P, P, P, P, P, P, P, P, P, P, P, P, P, P,
                                               ctypes.c_size_t, P, ctypes.POINTER(StageEvents), P]
        lib.pr2_moe_replay_forward.restype = ctypes.c_int
        lib.pr2_moe_rollout_forward.argtypes = [D, P, P, P, P, P, P, P, P, P, P, P, P, P, P, P,
                                                P, P, ctypes.c_size_t, P,
                                                ctypes.POINTER(StageEvents), P]
        lib.pr2_moe_rollout_forward.restype = ctypes.c_int
        _lib = lib
        return lib


def declared_symbols() -> list:
    """Names of the functions declared in ``include/pr2.h``."""
    hdr = open(os.path.join(_build.INCLUDE, "pr2.h")).read()
    hdr = re.sub(r"/\*.*?\*/", "", hdr, flags=re.S)
    return sorted(set(re.findall(r"\b(pr2_[a-z_0-9]+)\s*\(", hdr)))


def _p(t: Optional[torch.Tensor]):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _s(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def check(code: int, where: str = "pr2") -> None:
    if code != PR2_OK:
        raise Pr2Error(code, where)


def pr2_strerror(code: int) -> str:
    return load().pr2_strerror(code).decode()


def pr2_route_predict(dm: Dims, h, W_router, W_pred, idx, gates, logits_old=None,
                      near_tie=None, status=None, stream=None) -> int:
    return load().pr2_route_predict(ctypes.byref(dm), _p(h), _p(W_router), _p(W_pred), _p(idx),
                                    _p(gates), _p(logits_old), _p(near_tie), _p(status),
                                    _s(stream))


def pr2_route_replay(dm: Dims, h, W_router, idx, gates, probs=None, status=None,
                     stream=None) -> int:
    return load().pr2_route_replay(ctypes.byref(dm), _p(h), _p(W_router), _p(idx), _p(gates),
                                   _p(probs), _p(status), _s(stream))


def pr2_moe_workspace_bytes(dm: Dims) -> int:
    return int(load().pr2_moe_workspace_bytes(ctypes.byref(dm)))


def pr2_moe_forward(dm: Dims, h, idx, gates, W_gate, W_up, W_down, Ws_gate, Ws_up, Ws_down, out,
                    counts=None, perm=None, workspace=None, ws_bytes=None, status=None,
                    events: Optional[StageEvents] = None, stream=None) -> int:
    if ws_bytes is None:
        ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    return load().pr2_moe_forward(ctypes.byref(dm), _p(h), _p(idx), _p(gates), _p(W_gate),
                                  _p(W_up), _p(W_down), _p(Ws_gate), _p(Ws_up), _p(Ws_down),
                                  _p(out), _p(counts), _p(perm), _p(workspace),
                                  ctypes.c_size_t(ws_bytes), _p(status),
                                  None if events is None else ctypes.byref(events), _s(stream))


def pr2_moe_rollout_forward(dm: Dims, h, W_router, W_pred, idx, gates, logits_old, near_tie,
                            W_gate, W_up, W_down, Ws_gate, Ws_up, Ws_down, out, counts=None,
                            perm=None, workspace=None, ws_bytes=None, status=None,
                            events: Optional[StageEvents] = None, stream=None) -> int:
    """``pr2_route_predict`` then ``pr2_moe_forward`` in one call (route, gates, optional
    logits and near-tie count written); dispatch reads the routing kernel's histograms."""
    if ws_bytes is None:
        ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    return load().pr2_moe_rollout_forward(
        ctypes.byref(dm), _p(h), _p(W_router), _p(W_pred), _p(idx), _p(gates), _p(logits_old),
        _p(near_tie), _p(W_gate), _p(W_up), _p(W_down), _p(Ws_gate), _p(Ws_up), _p(Ws_down),
        _p(out), _p(counts), _p(perm), _p(workspace), ctypes.c_size_t(ws_bytes), _p(status),
        None if events is None else ctypes.byref(events), _s(stream))


def pr2_moe_replay_forward(dm: Dims, h, W_router, idx, gates, probs, W_gate, W_up, W_down,
                           Ws_gate, Ws_up, Ws_down, out, counts=None, perm=None, workspace=None,
                           ws_bytes=None, status=None, events: Optional[StageEvents] = None,
                           stream=None) -> int:
    """``pr2_route_replay`` then ``pr2_moe_forward`` in one call (replay gates written to
    ``gates``, optional ``probs``), the routing launched behind the expert GEMMs."""
    if ws_bytes is None:
        ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    return load().pr2_moe_replay_forward(
        ctypes.byref(dm), _p(h), _p(W_router), _p(idx), _p(gates), _p(probs), _p(W_gate),
        _p(W_up), _p(W_down), _p(Ws_gate), _p(Ws_up), _p(Ws_down), _p(out), _p(counts), _p(perm),
        _p(workspace), ctypes.c_size_t(ws_bytes), _p(status),
        None if events is None else ctypes.byref(events), _s(stream))


def pr2_selftest_wait_timeout(status, timeout_ns: int, stream=None) -> int:
    return load().pr2_selftest_wait_timeout(_p(status), int(timeout_ns), _s(stream))


def pr2_predictor_loss_workspace_bytes(dm: Dims) -> int:
    return int(load().pr2_predictor_loss_workspace_bytes(ctypes.byref(dm)))


def pr2_predictor_loss(dm: Dims, h_old, p_old, W_pred, rho, loss, grad, pos=None, kl_tok=None,
                       workspace=None, ws_bytes=None, status=None, stream=None) -> int:
    """Predictive loss (Eq. pr2_loss) and W_p gradient; ``dm.T`` = number of cached tokens and
    ``dm.flags`` may hold PR2_F_DELTA_LOSS.  ``rho`` rows are addressed through ``pos``."""
    if ws_bytes is None:
        ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    T_rho = int(rho.shape[0]) if rho is not None else 0
    return load().pr2_predictor_loss(ctypes.byref(dm), _p(h_old), _p(p_old), _p(W_pred), _p(rho),
                                     T_rho, _p(pos), _p(loss), _p(kl_tok), _p(grad),
                                     _p(workspace), ctypes.c_size_t(ws_bytes), _p(status),
                                     _s(stream))


def pr2_route_diagnostics(dm: Dims, rho, idx_cached, hist, overlap_sum, stream=None) -> int:
    """Accumulate the deviation histogram (int64 [k+1]) and the overlap sum (int64 [1])."""
    return load().pr2_route_diagnostics(ctypes.byref(dm), _p(rho), _p(idx_cached), _p(hist),
                                        _p(overlap_sum), _s(stream))


def pr2_feature_cache_write(dm: Dims, Tc: int, h, logits_old, pos, cache_h, cache_p,
                            stream=None) -> int:
    return load().pr2_feature_cache_write(ctypes.byref(dm), int(Tc), _p(h), _p(logits_old),
                                          _p(pos), _p(cache_h), _p(cache_p), _s(stream))


def pr2_rollout_layers(dm: Dims, L: int, h, W_router, W_pred, W_gate, W_up, W_down, idx, gates,
                       Ws_gate=None, Ws_up=None, Ws_down=None, logits_old=None, near_tie=None,
                       workspace=None, ws_bytes=None, status=None, stream=None) -> int:
    """L rollout layers in sequence with the residual stream updated in ``h`` (in place);
    weights stacked by layer, per-layer routes in ``idx``/``gates`` [L, T, k]."""
    if ws_bytes is None:
        ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    return load().pr2_rollout_layers(ctypes.byref(dm), int(L), _p(h), _p(W_router), _p(W_pred),
                                     _p(W_gate), _p(W_up), _p(W_down), _p(Ws_gate), _p(Ws_up),
                                     _p(Ws_down), _p(idx), _p(gates), _p(logits_old),
                                     _p(near_tie), _p(workspace), ctypes.c_size_t(ws_bytes),
                                     _p(status), _s(stream))


# ---- allocation helpers (plain torch.empty on the caller's device) ---------------------------

def alloc_workspace(dm: Dims, device="cuda") -> torch.Tensor:
    n = pr2_moe_workspace_bytes(dm)
    if n == 0:
        raise Pr2Error(1, "pr2_moe_workspace_bytes")
    return torch.empty(n, dtype=torch.uint8, device=device)


def alloc_loss_workspace(dm: Dims, device="cuda") -> torch.Tensor:
    n = pr2_predictor_loss_workspace_bytes(dm)
    if n == 0:
        raise Pr2Error(1, "pr2_predictor_loss_workspace_bytes")
    return torch.empty(n, dtype=torch.uint8, device=device)


def alloc_route(dm: Dims, device="cuda", logits: bool = False):
    """idx [T,k] int32, gates [T,k] fp32, optional logits/probs [T,N] fp32."""
    T, k, N = dm.T, dm.k, dm.N
    idx = torch.empty(T, k, dtype=torch.int32, device=device)
    gates = torch.empty(T, k, dtype=torch.float32, device=device)
    aux = torch.empty(T, N, dtype=torch.float32, device=device) if logits else None
    return idx, gates, aux


# ---- workspace-free layer forward (for callers that cannot allocate device memory) -----------

_static_ready = False


def _static_lib() -> ctypes.CDLL:
    """The loaded library with the signatures of the two workspace-free entry points set."""
    global _static_ready
    lib = load()
    if not _static_ready:
        P = ctypes.c_void_p
        lib.pr2_moe_forward_static.argtypes = [ctypes.POINTER(Dims), P, P, P, P, P, P, P, P, P, P,
                                               P, P, P, P]
        lib.pr2_moe_forward_static.restype = ctypes.c_int
        lib.pr2_static_scratch_bytes.argtypes = []
        lib.pr2_static_scratch_bytes.restype = ctypes.c_size_t
        _static_ready = True
    return lib


def pr2_static_scratch_bytes() -> int:
    return int(_static_lib().pr2_static_scratch_bytes())


def pr2_moe_forward_static(dm: Dims, h, idx, gates, W_gate, W_up, W_down, Ws_gate, Ws_up,
                           Ws_down, out, counts=None, perm=None, status=None, stream=None) -> int:
    """``pr2_moe_forward`` with the library's own fixed scratch array instead of a workspace:
    for callers that cannot allocate device memory.  Calls that overlap on the GPU race."""
    return _static_lib().pr2_moe_forward_static(
        ctypes.byref(dm), _p(h), _p(idx), _p(gates), _p(W_gate), _p(W_up), _p(W_down),
        _p(Ws_gate), _p(Ws_up), _p(Ws_down), _p(out), _p(counts), _p(perm), _p(status),
        _s(stream))
