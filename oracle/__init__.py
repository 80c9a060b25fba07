"""Pr^2 oracle: ctypes wrapper over the plain fp64 C implementation in ``pr2_oracle.c``.

TEST INFRASTRUCTURE ONLY.  The tests, ``__graft_entry__.smoke()`` and the bench's CPU-baseline
and reference arms may import this package; the product package never does.  It shares no code
with the CUDA library: inputs are handed over as their stored bits (fp32, or bf16 as raw 16-bit
patterns) and every step is done in double precision by ``pr2_oracle.c``.

Functions (each cites the passage it follows in the C source):

* ``route_predict``  - Eqs. pr2_predict / pr2_route, Algorithm 1 rollout steps
* ``route_replay``   - Sec. 4.1 "Replay During Training" (Algorithm 1 replay steps, Algorithm 3)
* ``permute``        - dispatch to experts as a stable counting sort (Algorithm 1)
* ``moe_forward``    - Eqs. pr2_old_output / pr2_output with SwiGLU experts (App. E.2)

Parity status: every function is pinned by the CPU tests in ``tests/test_oracle_pins.py``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from typing import Optional

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pr2_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "libpr2_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``pr2_oracle.c`` with gcc (OpenMP when available) into ``oracle/_build``."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB)
    return _LIB


def bind(path: str):
    """Load an oracle shared library from ``path`` and declare its C signatures."""
    lib = ctypes.CDLL(path)
    P, I64, I32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
    lib.oracle_route_predict.argtypes = [I64, I32, I32, I32, I32, P, P, P, P, P, P, P, P, P]
    lib.oracle_route_predict.restype = None
    lib.oracle_route_replay.argtypes = [I64, I32, I32, I32, I32, P, P, P, P, P]
    lib.oracle_route_replay.restype = I64
    lib.oracle_permute.argtypes = [I64, I32, I32, P, P, P, P, P]
    lib.oracle_permute.restype = I64
    lib.oracle_moe_forward.argtypes = [I64, P, I64, I32, I32, I32, I32, I32, I32, P, P, P, P,
                                       P, P, P, P, P, P]
    lib.oracle_moe_forward.restype = None
    lib.oracle_num_threads.argtypes = []
    lib.oracle_num_threads.restype = I32
    return lib


def _load(lib=None):
    """The library to call: ``lib`` when given (a ``bind`` result), else the built oracle."""
    global _lib
    if lib is not None:
        return lib
    with _lock:
        if _lib is None:
            _lib = bind(build())
    return _lib


def num_threads() -> int:
    return int(_load().oracle_num_threads())


def _stored(t) -> tuple:
    """(contiguous numpy array of the stored bits, dtype code): fp32 -> 0, bf16 -> 1."""
    if isinstance(t, np.ndarray):
        a = np.ascontiguousarray(t)
        if a.dtype == np.float32:
            return a, 0
        raise TypeError(f"oracle takes fp32 or bf16 inputs, got numpy {a.dtype}")
    t = t.detach().to("cpu").contiguous()
    if t.dtype == torch.float32:
        return t.numpy(), 0
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy(), 1
    raise TypeError(f"oracle takes fp32 or bf16 inputs, got {t.dtype}")


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _same_dtype(*codes):
    codes = [c for c in codes if c is not None]
    if len(set(codes)) != 1:
        raise TypeError("oracle inputs must share one dtype")
    return codes[0]


def route_predict(h, W_router, W_pred, k: int, lib=None):
    """Rollout routing of Sec. 4.1 in fp64.  Returns a dict of numpy arrays:
    idx [T,k] int32, gates [T,k], logits [T,N] (= p_old), probs [T,N] (= rho-hat),
    margin [T] (= rho-hat_(k) - rho-hat_(k+1)), top_vals [T,k+1]."""
    hs, c0 = _stored(h)
    ws, c1 = _stored(W_router)
    ps, c2 = _stored(W_pred)
    dt = _same_dtype(c0, c1, c2)
    T, d = hs.shape
    N = ws.shape[0]
    if not (1 <= k <= N):
        raise ValueError("need 1 <= k <= N")
    out = dict(idx=np.zeros((T, k), np.int32), gates=np.zeros((T, k)),
               logits=np.zeros((T, N)), probs=np.zeros((T, N)), margin=np.zeros(T),
               top_vals=np.full((T, k + 1), np.nan))
    _load(lib).oracle_route_predict(T, d, N, k, dt, _ptr(hs), _ptr(ws), _ptr(ps), _ptr(out["idx"]),
                                 _ptr(out["gates"]), _ptr(out["logits"]), _ptr(out["probs"]),
                                 _ptr(out["margin"]), _ptr(out["top_vals"]))
    return out


def route_replay(h, W_router, idx, lib=None):
    """Replay gates of Sec. 4.1 in fp64: dict(gates [T,k], probs [T,N], bad = #invalid slots)."""
    hs, c0 = _stored(h)
    ws, c1 = _stored(W_router)
    dt = _same_dtype(c0, c1)
    ix = np.ascontiguousarray(np.asarray(idx, dtype=np.int32))
    T, d = hs.shape
    N = ws.shape[0]
    k = ix.shape[1]
    gates = np.zeros((T, k))
    probs = np.zeros((T, N))
    bad = _load(lib).oracle_route_replay(T, d, N, k, dt, _ptr(hs), _ptr(ws), _ptr(ix), _ptr(gates),
                                      _ptr(probs))
    return dict(gates=gates, probs=probs, bad=int(bad))


def permute(idx, N: int, lib=None):
    """Stable dispatch of flat slots to experts: dict(counts, offsets, perm, inv, bad)."""
    ix = np.ascontiguousarray(np.asarray(idx, dtype=np.int32))
    T, k = ix.shape
    counts = np.zeros(N, np.int32)
    offsets = np.zeros(N + 1, np.int32)
    perm = np.full(T * k, -1, np.int32)
    inv = np.full(T * k, -1, np.int32)
    bad = _load(lib).oracle_permute(T, k, N, _ptr(ix), _ptr(counts), _ptr(offsets), _ptr(perm),
                                 _ptr(inv))
    nvalid = int(offsets[N])
    return dict(counts=counts, offsets=offsets, perm=perm[:nvalid], inv=inv, bad=int(bad))


def moe_forward(h, idx, gates, W_gate, W_up, W_down, Ws_gate=None, Ws_up=None, Ws_down=None,
                tokens=None, lib=None):
    """Layer output on the given routes (Eqs. pr2_old_output / pr2_output), fp64 [n_tok, d].

    ``tokens``: optional token ids to compute (default all).  ``gates`` is read as float64.
    """
    hs, c0 = _stored(h)
    g, c1 = _stored(W_gate)
    u, c2 = _stored(W_up)
    dn, c3 = _stored(W_down)
    dt = _same_dtype(c0, c1, c2, c3)
    T, d = hs.shape
    N, m, _ = g.shape
    ix = np.ascontiguousarray(np.asarray(idx, dtype=np.int32))
    k = ix.shape[1]
    gt = np.ascontiguousarray(np.asarray(gates, dtype=np.float64))
    s = 0
    sg = su = sd = None
    if Ws_gate is not None:
        sg, c4 = _stored(Ws_gate)
        su, c5 = _stored(Ws_up)
        sd, c6 = _stored(Ws_down)
        _same_dtype(dt, c4, c5, c6)
        s = sg.shape[0]
    tok = np.arange(T, dtype=np.int64) if tokens is None else np.ascontiguousarray(
        np.asarray(tokens, dtype=np.int64))
    out = np.zeros((tok.shape[0], d))
    _load(lib).oracle_moe_forward(tok.shape[0], _ptr(tok), T, d, N, k, m, s, dt, _ptr(hs), _ptr(ix),
                               _ptr(gt), _ptr(g), _ptr(u), _ptr(dn), _ptr(sg), _ptr(su), _ptr(sd),
                               _ptr(out))
    return out
