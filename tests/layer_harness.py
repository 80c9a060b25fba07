"""Shared test harness: run the layer through the C ABI and compare it with the oracle.

Tolerances (stated once, used by every parity test):
  * route indices: bit-exact, except tokens whose oracle top-k margin rho_(k) - rho_(k+1) is
    below 1e-4 (near ties).  For those the GPU's k experts must still be a valid top-k within
    the same 1e-4 band.  Slot order must match wherever adjacent oracle probabilities differ
    by at least 1e-4.
  * gates / probabilities / logits (fp32 outputs of both dtypes): |gpu - oracle| <= 1e-4 *
    max|oracle| over the row (normwise per row).
  * layer output: max|gpu - oracle| / max|oracle| <= 2e-2 for bf16 and <= 1e-4 for fp32.
  * counts and permutations: bit-exact.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2606_00395_gb300 import binding as B

TIE_GAP = 1e-4
FP32_TOL = 1e-4
OUT_TOL = {"bf16": 2e-2, "fp32": 1e-4}


def dims_of(cfg, flags=0):
    return B.dims(cfg.T, cfg.d, cfg.N, cfg.k, cfg.m, cfg.n_shared, cfg.dtype, flags)


def to_dev(L, dev="cuda"):
    return {k: (v.to(dev) if v is not None else None) for k, v in L.items()}


def gpu_predict(cfg, Ld, logits=True, stream=None, flags=0):
    dm = dims_of(cfg, flags)
    idx, gates, aux = B.alloc_route(dm, logits=logits)
    near = torch.zeros(1, dtype=torch.int64, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    B.check(B.pr2_route_predict(dm, Ld["x"], Ld["W_router"], Ld["W_pred"], idx, gates, aux, near,
                                status, stream), "pr2_route_predict")
    return dict(idx=idx, gates=gates, logits=aux, near_tie=near, status=status)


def gpu_replay(cfg, Ld, W, idx, probs=True, stream=None, flags=0):
    dm = dims_of(cfg, flags)
    gates = torch.empty(cfg.T, cfg.k, dtype=torch.float32, device="cuda")
    pr = torch.empty(cfg.T, cfg.N, dtype=torch.float32, device="cuda") if probs else None
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    B.check(B.pr2_route_replay(dm, Ld["x"], W, idx, gates, pr, status, stream),
            "pr2_route_replay")
    return dict(gates=gates, probs=pr, status=status)


def gpu_forward(cfg, Ld, idx, gates, ws=None, stream=None, flags=0):
    dm = dims_of(cfg, flags)
    if ws is None:
        ws = B.alloc_workspace(dm)
    out = torch.empty(cfg.T, cfg.d, dtype=cfg.torch_dtype, device="cuda")
    counts = torch.empty(cfg.N, dtype=torch.int32, device="cuda")
    perm = torch.full((cfg.T * cfg.k,), -1, dtype=torch.int32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    code = B.pr2_moe_forward(dm, Ld["x"], idx, gates, Ld["W_gate"], Ld["W_up"], Ld["W_down"],
                             Ld["Ws_gate"], Ld["Ws_up"], Ld["Ws_down"], out, counts, perm, ws,
                             status=status, stream=stream)
    return dict(out=out, counts=counts, perm=perm, status=status, code=code)


def check_routes(orc, idx_gpu):
    """Compare GPU top-k indices with the oracle under the near-tie rule.

    Returns the number of exempt (near-tie) tokens; asserts on everything else."""
    idx_gpu = np.asarray(idx_gpu)
    o_idx, probs, margin = orc["idx"], orc["probs"], orc["margin"]
    T, k = o_idx.shape
    exempt = 0
    for t in range(T):
        g = idx_gpu[t]
        assert len(set(g.tolist())) == k, f"token {t}: duplicate experts {g}"
        if margin[t] < TIE_GAP:
            exempt += 1
            kth = np.sort(probs[t])[::-1][k - 1]
            assert np.all(probs[t, g] >= kth - TIE_GAP), f"token {t}: {g} not a top-k"
            continue
        assert set(g.tolist()) == set(o_idx[t].tolist()), f"token {t}: {g} vs {o_idx[t]}"
        for s in range(k):
            if g[s] != o_idx[t, s]:
                # allowed only inside a near tie of adjacent slots
                assert abs(probs[t, g[s]] - probs[t, o_idx[t, s]]) < TIE_GAP, (t, s)
    return exempt


def rowwise_close(got, want, tol=FP32_TOL):
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    scale = np.maximum(np.max(np.abs(want), axis=1, keepdims=True), 1e-30)
    err = np.max(np.abs(got - want) / scale)
    assert err <= tol, f"row-normwise error {err:.3e} > {tol:.1e}"
    return err


def normwise_close(got, want, tol):
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    err = np.max(np.abs(got - want)) / max(np.max(np.abs(want)), 1e-30)
    assert err <= tol, f"normwise error {err:.3e} > {tol:.1e}"
    return err


def cpu(t):
    return t.detach().cpu()


def compact_experts(L, idx_rows, tokens=None):
    """For sampled oracle checks on very large layers: the expert weights that `idx_rows`
    reference, stacked densely, and idx remapped onto them (a relabelling, no arithmetic)."""
    used = sorted(set(int(e) for e in np.asarray(idx_rows).reshape(-1) if 0 <= e))
    remap = {e: i for i, e in enumerate(used)}
    sel = torch.tensor(used, dtype=torch.long, device=L["W_gate"].device)
    Wg = cpu(L["W_gate"].index_select(0, sel))
    Wu = cpu(L["W_up"].index_select(0, sel))
    Wd = cpu(L["W_down"].index_select(0, sel))
    new_idx = np.vectorize(lambda e: remap.get(int(e), -1))(np.asarray(idx_rows)).astype(np.int32)
    return Wg, Wu, Wd, new_idx


def oracle_forward_rows(L, toks, idx_rows, gates_rows, with_shared=True,
                        max_host_bytes=4 << 30):
    """fp64 oracle layer output for the tokens ``toks`` of a (possibly very large) layer whose
    tensors live on the GPU, with the routes ``idx_rows`` / gates ``gates_rows`` of those tokens.

    Only the experts the rows reference are copied to the host, at most ``max_host_bytes`` of
    expert weights at a time: when they do not fit at once (the DeepSeek-V3-shaped layer's 256
    experts are 22.6 GB), the referenced experts are split into groups, the oracle runs once per
    group with the other groups' slots marked invalid (the oracle skips them), and the group
    outputs are added.  Each token's slots are thereby summed in group order instead of slot
    order: a reassociation of at most k fp64 terms.  The shared experts enter with the first
    group only."""
    idx_rows = np.asarray(idx_rows)
    used = sorted(set(int(e) for e in idx_rows.reshape(-1) if 0 <= e < L["W_gate"].shape[0]))
    per_expert = 3 * L["W_gate"].shape[1] * L["W_gate"].shape[2] * L["W_gate"].element_size()
    group = max(1, int(max_host_bytes // per_expert))
    sel_t = torch.as_tensor(np.asarray(toks), dtype=torch.long, device=L["x"].device)
    x_s = cpu(L["x"].index_select(0, sel_t))
    sh = [cpu(L[n]) if (with_shared and L.get(n) is not None) else None
          for n in ("Ws_gate", "Ws_up", "Ws_down")]
    out = None
    for g0 in range(0, max(len(used), 1), group):
        chunk = used[g0:g0 + group]
        remap = {e: i for i, e in enumerate(chunk)}
        sel = torch.tensor(chunk if chunk else [0], dtype=torch.long, device=L["W_gate"].device)
        Wg = cpu(L["W_gate"].index_select(0, sel))
        Wu = cpu(L["W_up"].index_select(0, sel))
        Wd = cpu(L["W_down"].index_select(0, sel))
        idx_c = np.vectorize(lambda e: remap.get(int(e), -1))(idx_rows).astype(np.int32)
        part = oracle.moe_forward(x_s, idx_c, gates_rows, Wg, Wu, Wd,
                                  *(sh if g0 == 0 else (None, None, None)))
        out = part if out is None else out + part
        del Wg, Wu, Wd
    return out

