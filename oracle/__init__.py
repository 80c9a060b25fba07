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
* ``predictor_loss`` - Eq. pr2_loss and Algorithm 3 (loss and W_p gradient), and the
  delta-matching variant of the appendix ablation
* ``route_diagnostics`` - top-k agreement and the deviation histogram (Sec. 5)
* ``feature_cache``  - the fixed-length feature cache of Algorithm 2 (evenly spaced positions)
* ``rollout_layers`` - Algorithm 2 over L stacked layers with the residual stream (composition
  of ``route_predict`` and ``moe_forward``)
* ``normalize_topk`` - the optional renormalisation of the selected gates (g / sum g, as in
  Qwen3's router).  The paper weights with the probabilities themselves (Eqs. pr2_old_output /
  pr2_output); this is the reading behind PR2_F_NORMALIZE_TOPK, not part of the method.

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
    lib.oracle_predictor_loss.argtypes = [I64, I32, I32, I32, I32, P, P, P, P, I64, P, P, P, P]
    lib.oracle_predictor_loss.restype = I64
    lib.oracle_route_diagnostics.argtypes = [I64, I32, I32, P, P, P]
    lib.oracle_route_diagnostics.restype = I64
    lib.oracle_feature_cache.argtypes = [I64, I64, I32, I32, I32, P, P, P, P, P]
    lib.oracle_feature_cache.restype = None
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


def normalize_topk(gates):
    """Selected gates divided by their sum per token (fp64); a row whose gates are all zero (every
    slot invalid) stays zero."""
    g = np.asarray(gates, dtype=np.float64)
    s = g.sum(axis=1, keepdims=True)
    return np.divide(g, s, out=np.zeros_like(g), where=s > 0)


def route_predict(h, W_router, W_pred, k: int, lib=None, normalize: bool = False):
    """Rollout routing of Sec. 4.1 in fp64.  Returns a dict of numpy arrays:
    idx [T,k] int32, gates [T,k], logits [T,N] (= p_old), probs [T,N] (= rho-hat),
    margin [T] (= rho-hat_(k) - rho-hat_(k+1)), top_vals [T,k+1].  ``normalize``: gates
    renormalised over the route (``normalize_topk``); probs, margin and top_vals are not."""
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
    if normalize:
        out["gates"] = normalize_topk(out["gates"])
    return out


def route_replay(h, W_router, idx, lib=None, normalize: bool = False):
    """Replay gates of Sec. 4.1 in fp64: dict(gates [T,k], probs [T,N], bad = #invalid slots).
    ``normalize``: gates renormalised over the valid slots (``normalize_topk``)."""
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
    if normalize:
        gates = normalize_topk(gates)
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


def _f32(a) -> np.ndarray:
    """fp32 contiguous numpy copy of a tensor / array that is stored as fp32."""
    if isinstance(a, torch.Tensor):
        if a.dtype != torch.float32:
            raise TypeError(f"expected an fp32 tensor, got {a.dtype}")
        return a.detach().to("cpu").contiguous().numpy()
    a = np.ascontiguousarray(a)
    if a.dtype != np.float32:
        raise TypeError(f"expected fp32, got {a.dtype}")
    return a


def predictor_loss(h_old, p_old, W_pred, rho, pos=None, delta: bool = False, lib=None):
    """Eq. pr2_loss for one layer (``delta``: the delta-matching variant) in fp64.

    h_old [T_c,d] (fp32 or bf16), p_old [T_c,N] fp32, W_pred [N,d] (h_old's dtype), rho
    [T_rho,N] fp32 teacher probabilities, pos [T_c] int32 rows of rho (None: row c).  Returns
    dict(loss, kl [T_c], grad [N,d], bad = #invalid pos)."""
    hs, c0 = _stored(h_old)
    ws, c1 = _stored(W_pred)
    dt = _same_dtype(c0, c1)
    po = _f32(p_old)
    rh = _f32(rho)
    Tc, d = hs.shape
    N = ws.shape[0]
    ps = None if pos is None else np.ascontiguousarray(np.asarray(pos, dtype=np.int32))
    loss = np.zeros(1)
    kl = np.zeros(max(Tc, 1))
    grad = np.zeros((N, d))
    bad = _load(lib).oracle_predictor_loss(Tc, d, N, dt, 1 if delta else 0, _ptr(hs), _ptr(po),
                                           _ptr(ws), _ptr(rh), rh.shape[0], _ptr(ps),
                                           _ptr(loss), _ptr(kl), _ptr(grad))
    return dict(loss=float(loss[0]), kl=kl[:Tc], grad=grad, bad=int(bad))


def route_diagnostics(rho, idx_cached, lib=None):
    """Top-k agreement and deviation histogram of a cached route against TopK(rho, k).
    Returns dict(hist [k+1] int64, overlap = sum_t |Î_t ∩ I_t|, agreement = overlap / (T k))."""
    rh = _f32(rho)
    ix = np.ascontiguousarray(np.asarray(idx_cached, dtype=np.int32))
    T, N = rh.shape
    k = ix.shape[1]
    hist = np.zeros(k + 1, np.int64)
    ov = _load(lib).oracle_route_diagnostics(T, N, k, _ptr(rh), _ptr(ix), _ptr(hist))
    return dict(hist=hist, overlap=int(ov), agreement=(ov / (T * k)) if T else 0.0)


def feature_cache(h, logits, Tc: int, lib=None):
    """Feature-cache rows of Algorithm 2 at evenly spaced positions: dict(pos [T_c] int32,
    h [T_c,d] (h's dtype), p [T_c,N] fp32)."""
    if isinstance(h, torch.Tensor):
        ht = h.detach().to("cpu").contiguous()
        esz = ht.element_size()
        raw = ht.view(torch.int16 if esz == 2 else torch.int32).numpy()
    else:
        raw = np.ascontiguousarray(h)
        esz = raw.dtype.itemsize
    lg = _f32(logits)
    T, d = raw.shape
    N = lg.shape[1]
    if not (0 <= Tc <= T):
        raise ValueError("need 0 <= T_c <= T")
    pos = np.zeros(max(Tc, 1), np.int32)
    ch = np.zeros((max(Tc, 1), d), raw.dtype)
    cp = np.zeros((max(Tc, 1), N), np.float32)
    _load(lib).oracle_feature_cache(T, Tc, d, N, esz, _ptr(raw), _ptr(lg), _ptr(pos), _ptr(ch),
                                    _ptr(cp))
    hc = torch.from_numpy(ch[:Tc].copy())
    if isinstance(h, torch.Tensor):
        hc = hc.view(h.dtype)
    return dict(pos=pos[:Tc], h=hc, p=cp[:Tc])


def _round_to(x: np.ndarray, dtype) -> torch.Tensor:
    """fp64 values rounded once (to nearest, ties to even) to ``dtype``, as a tensor.  bf16 is
    rounded straight from the fp64 bit pattern (no intermediate fp32 rounding): keep the top 7
    of the 52 mantissa bits, round on the other 45, carry into the exponent."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    if dtype != torch.bfloat16:
        return torch.from_numpy(x).to(dtype)
    b = x.view(np.uint64)
    sign = (b >> np.uint64(63)) & np.uint64(1)
    exp = ((b >> np.uint64(52)) & np.uint64(0x7FF)).astype(np.int64)
    man = b & np.uint64((1 << 52) - 1)
    keep = (man >> np.uint64(45)).astype(np.int64)
    rem = (man & np.uint64((1 << 45) - 1)).astype(np.int64)
    half = 1 << 44
    keep = keep + ((rem > half) | ((rem == half) & ((keep & 1) == 1))).astype(np.int64)
    e32 = exp - 1023 + 127 + (keep >> 7)
    keep &= 0x7F
    zero = exp == 0
    if np.any(~zero & ((e32 < 1) | (e32 > 254))):
        raise ValueError("value outside the normal bf16 range")
    bits = (sign.astype(np.int64) << 15) | np.where(zero, 0, (e32 << 7) | keep)
    return torch.from_numpy(bits.astype(np.uint16).view(np.int16)).view(torch.bfloat16)


def rollout_layers(h, layers, k: int, lib=None):
    """Algorithm 2 applied to layers l = 1..L in sequence (the route-recording pass of a stack of
    MoE layers): at each layer the rollout route and output of Eqs. pr2_predict / pr2_route /
    pr2_old_output, then the residual stream h <- round(h + o_old) in h's dtype (the layer's
    output is stored once in the layer dtype).  ``layers`` is a list of dicts with W_router,
    W_pred, W_gate, W_up, W_down (and optionally Ws_*).  Returns dict(h [T,d] tensor in h's
    dtype, idx [L,T,k], gates [L,T,k], logits [L,T,N], margin [L,T] (rho_(k) - rho_(k+1)),
    min_gap [L,T] (smallest gap between consecutive ones of the top k+1 probabilities, which
    also bounds how near the slot order is to a tie))."""
    cur = h.detach().to("cpu").contiguous()
    idx, gates, logits, margin, min_gap = [], [], [], [], []
    for lw in layers:
        r = route_predict(cur, lw["W_router"], lw["W_pred"], k, lib=lib)
        o = moe_forward(cur, r["idx"], r["gates"], lw["W_gate"], lw["W_up"], lw["W_down"],
                        lw.get("Ws_gate"), lw.get("Ws_up"), lw.get("Ws_down"), lib=lib)
        cur = _round_to(cur.double().numpy() + o, cur.dtype)
        idx.append(r["idx"])
        gates.append(r["gates"])
        logits.append(r["logits"])
        margin.append(r["margin"])
        tv = r["top_vals"][:, : min(k + 1, r["logits"].shape[1])]
        min_gap.append(np.min(tv[:, :-1] - tv[:, 1:], axis=1) if tv.shape[1] > 1
                       else np.full(tv.shape[0], np.inf))
    return dict(h=cur, idx=np.stack(idx), gates=np.stack(gates), logits=np.stack(logits),
                margin=np.stack(margin), min_gap=np.stack(min_gap))
