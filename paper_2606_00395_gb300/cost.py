"""Closed-form cost model of the Pr^2 layer (host logic, no GPU).

* Table 4 / App. E.2 of the paper: index cache 4*T*L*k bytes (int32 indices), feature cache
  T_c*L*(2d + 4N) bytes (bf16 hidden features + fp32 router logits), predictor FLOPs 2*L*d*N per
  token, and the FFN ratio 2*L*d*N / (6*L*(k+s)*d*m).
* Algorithmic bytes and FLOPs per kernel of this library, used as the roofline numerators.  They
  count each tensor a kernel must touch exactly once (compulsory traffic), nothing else.
"""
from __future__ import annotations

from dataclasses import dataclass


def index_cache_bytes(T: int, L: int, k: int) -> int:
    """Int32 replay indices for one response of T tokens over L layers (Table 4, App. E.2)."""
    return 4 * T * L * k


def feature_cache_bytes(T_c: int, L: int, d: int, N: int) -> int:
    """bf16 h_old [d] + fp32 p_old [N] for T_c retained positions over L layers (Table 4)."""
    return T_c * L * (2 * d + 4 * N)


def predictor_flops_per_token(L: int, d: int, N: int) -> int:
    """Extra route-recording FLOPs of the L predictor projections h W_p (App. E.2)."""
    return 2 * L * d * N


def ffn_ratio(L: int, d: int, N: int, k: int, s: int, m: int) -> float:
    """Predictor FLOPs over the active gated-MLP FLOPs 6*L*(k+s)*d*m per token (App. E.2)."""
    return predictor_flops_per_token(L, d, N) / (6 * L * (k + s) * d * m)


@dataclass(frozen=True)
class KernelWork:
    """Algorithmic work of one launch: bytes that must cross HBM and FLOPs that must be done."""

    bytes: int
    flops: int


def _esz(dtype: str) -> int:
    return 4 if dtype == "fp32" else 2


def route_predict_work(T: int, d: int, N: int, k: int, dtype: str = "bf16",
                       write_logits: bool = True) -> KernelWork:
    """Read h [T,d] and [W; W_p] [2N,d]; write idx + gates [T,k] (+ p_old [T,N] fp32)."""
    e = _esz(dtype)
    b = T * d * e + 2 * N * d * e + T * k * 8 + (T * N * 4 if write_logits else 0)
    return KernelWork(b, 2 * T * d * 2 * N)


def route_replay_work(T: int, d: int, N: int, k: int, dtype: str = "bf16",
                      write_probs: bool = False) -> KernelWork:
    """Read h, W [N,d] and idx [T,k]; write gates [T,k] (+ rho [T,N] fp32)."""
    e = _esz(dtype)
    b = T * d * e + N * d * e + T * k * 4 + T * k * 4 + (T * N * 4 if write_probs else 0)
    return KernelWork(b, 2 * T * d * N)


def dispatch_work(T: int, d: int, k: int, dtype: str = "bf16", gather: bool = False) -> KernelWork:
    """Histogram + scan + stable rank: read idx, write perm and inv.  With `gather` (the fp32
    path) also read h once and write the permuted rows X_perm [T*k, d]; the bf16 gate/up GEMM
    reads h through perm itself, so dispatch writes no rows there."""
    e = _esz(dtype)
    b = T * k * 4 + 2 * T * k * 4
    if gather:
        b += T * d * e + T * k * d * e
    return KernelWork(b, 0)


def expert_gate_up_work(rows: int, d: int, m: int, experts_hit: int,
                        dtype: str = "bf16", a_rows: int | None = None) -> KernelWork:
    """Grouped [X_e] x [W_gate; W_up]_e^T with the SwiGLU epilogue: read the A rows, the gate/up
    weights of every expert hit, write H [rows, m].  `a_rows` is the number of distinct A rows
    that must cross HBM: the T tokens of h when the GEMM gathers them (each token feeds k
    rows), `rows` when it reads a permuted copy."""
    e = _esz(dtype)
    a = rows if a_rows is None else a_rows
    return KernelWork(a * d * e + experts_hit * 2 * m * d * e + rows * m * e,
                      2 * rows * d * 2 * m)


def expert_down_work(rows: int, d: int, m: int, experts_hit: int,
                     dtype: str = "bf16") -> KernelWork:
    """Grouped H_e x W_down,e^T: read H and the down weights of every expert hit, write Y."""
    e = _esz(dtype)
    return KernelWork(rows * m * e + experts_hit * d * m * e + rows * d * e, 2 * rows * m * d)


def expert_mlp_work(rows: int, d: int, m: int, experts_hit: int, dtype: str = "bf16",
                    a_rows: int | None = None) -> KernelWork:
    """Both grouped GEMMs of the gated MLP (gate/up + SwiGLU, then down), run as one launch."""
    g = expert_gate_up_work(rows, d, m, experts_hit, dtype, a_rows)
    dn = expert_down_work(rows, d, m, experts_hit, dtype)
    return KernelWork(g.bytes + dn.bytes, g.flops + dn.flops)


def expert_mlp_algorithmic_work(rows: int, d: int, m: int, experts_hit: int,
                                dtype: str = "bf16", a_rows: int | None = None) -> KernelWork:
    """Compulsory work of the grouped gated-MLP stage (gate/up + SwiGLU + down) as a fused
    minimum: the weights of every expert hit (3*d*m each) and the distinct A rows (`a_rows`,
    default `rows`) cross HBM once; the intermediates H [rows, m] and Y [rows, d] are not
    counted (a fused layer keeps them on chip).  FLOPs 6*rows*d*m (App. E.2)."""
    e = _esz(dtype)
    a = rows if a_rows is None else a_rows
    return KernelWork(a * d * e + experts_hit * 3 * d * m * e, 6 * rows * d * m)


def combine_work(T: int, d: int, k: int, n_shared: int = 0, dtype: str = "bf16") -> KernelWork:
    """out[t] = sum_s g[t,s] Y[inv[t,s]] (+ shared rows): read Y, gates, inv; write out."""
    e = _esz(dtype)
    return KernelWork(T * k * d * e + T * k * 8 + T * n_shared * d * e + T * d * e, 0)


def predictor_loss_work(Tc: int, d: int, N: int, dtype: str = "bf16") -> KernelWork:
    """Eq. pr2_loss with its W_p gradient over T_c cached rows: read h_old, p_old, the teacher
    rows and W_p once, write the gradient and the per-token KL; FLOPs of the two products
    b = h_old W_p^T and (dKL/dz)^T h_old."""
    e = _esz(dtype)
    b = Tc * d * e + 2 * Tc * N * 4 + N * d * e + N * d * 4 + Tc * 4
    return KernelWork(b, 2 * Tc * d * N + 2 * N * d * Tc)


def route_diagnostics_work(T: int, N: int, k: int) -> KernelWork:
    """Top-k agreement / deviation histogram: read rho [T, N] fp32 and the cached route."""
    return KernelWork(T * N * 4 + T * k * 4, 0)


def feature_cache_work(Tc: int, d: int, N: int, dtype: str = "bf16") -> KernelWork:
    """Feature-cache writer: read and write T_c rows of h and p_old, write the positions."""
    e = _esz(dtype)
    return KernelWork(2 * Tc * (d * e + N * 4) + Tc * 4, 0)
