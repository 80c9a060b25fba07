"""GPU parity of the route-tracking diagnostics (Sec. 5) and the feature-cache writer
(Algorithm 2) through the C ABI: integer and copy outputs, compared bit-exactly with the
oracle.  Inputs are seeded and built on the CPU (never from the CUDA path)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_00395_gb300 import binding as B
from paper_2606_00395_gb300 import synth

pytestmark = pytest.mark.gpu


def _dyadic_probs(T, N, g, levels=16):
    """Probabilities on a coarse grid (many exact ties), rows normalised in fp32."""
    raw = torch.randint(0, levels, (T, N), generator=g).float() + 1
    return raw / raw.sum(1, keepdim=True)


def _cached(T, N, k, g):
    idx = torch.stack([torch.randperm(N, generator=g)[:k] for _ in range(T)]).int()
    idx[3, 1] = N           # out of range
    idx[7, k - 1] = -2      # negative
    idx[11, 1] = idx[11, 0]  # repeated in its token
    return idx


def _gpu_diag(rho, idx, dtype="bf16", reps=1):
    T, N = rho.shape
    k = idx.shape[1]
    dm = B.dims(T, 64, N, k, 64, 0, dtype)
    hist = torch.zeros(k + 1, dtype=torch.int64, device="cuda")
    ov = torch.zeros(1, dtype=torch.int64, device="cuda")
    r, ix = rho.contiguous().cuda(), idx.contiguous().cuda()
    for _ in range(reps):
        B.check(B.pr2_route_diagnostics(dm, r, ix, hist, ov), "pr2_route_diagnostics")
    torch.cuda.synchronize()
    return hist.cpu().numpy(), int(ov.item())


@pytest.mark.parametrize("T,N,k,dtype", [(4096, 128, 8, "bf16"), (700, 256, 8, "bf16"),
                                         (333, 64, 32, "fp32"), (257, 8, 2, "fp32")])
def test_diagnostics_match_oracle_with_ties_and_invalid_entries(T, N, k, dtype):
    g = torch.Generator().manual_seed(T + N + k)
    rho = _dyadic_probs(T, N, g)
    idx = _cached(T, N, k, g)
    ref = oracle.route_diagnostics(rho, idx.numpy())
    hist, ov = _gpu_diag(rho, idx, dtype)
    assert np.array_equal(hist, ref["hist"]) and ov == ref["overlap"]
    # the outputs accumulate: a second call on the same data doubles them
    hist2, ov2 = _gpu_diag(rho, idx, dtype, reps=2)
    assert np.array_equal(hist2, 2 * ref["hist"]) and ov2 == 2 * ref["overlap"]


def test_diagnostics_of_a_rollout_route_against_the_drifted_router():
    """The measurement of Sec. 5 on the qwen3 layer: the predicted route recorded at rollout
    (oracle) against TopK of the drifted current router's rho (oracle, stored fp32)."""
    cfg = synth.LayerConfig("q", T=1024, d=2048, N=128, k=8, m=768)
    L = synth.make_layer(cfg)
    W2 = synth.make_drifted_router(L["W_router"])
    rollout = oracle.route_predict(L["x"], L["W_router"], L["W_pred"], cfg.k)
    rho = torch.from_numpy(oracle.route_replay(L["x"], W2, rollout["idx"])["probs"]).float()
    ref = oracle.route_diagnostics(rho, rollout["idx"])
    hist, ov = _gpu_diag(rho, torch.from_numpy(rollout["idx"]))
    assert np.array_equal(hist, ref["hist"]) and ov == ref["overlap"]
    assert hist.sum() == cfg.T


@pytest.mark.parametrize("dtype,Tc", [("bf16", 1), ("bf16", 333), ("bf16", 1000),
                                      ("fp32", 77)])
def test_feature_cache_rows_match_oracle(dtype, Tc):
    T, d, N = 1000, 192 if dtype == "bf16" else 20, 32
    g = torch.Generator().manual_seed(Tc)
    h = torch.randn(T, d, generator=g)
    h = h.bfloat16() if dtype == "bf16" else h
    lg = torch.randn(T, N, generator=g)
    ref = oracle.feature_cache(h, lg, Tc)
    dm = B.dims(T, d, N, 2, 64, 0, dtype)
    pos = torch.full((Tc,), -7, dtype=torch.int32, device="cuda")
    ch = torch.zeros(Tc, d, dtype=h.dtype, device="cuda")
    cp = torch.zeros(Tc, N, dtype=torch.float32, device="cuda")
    B.check(B.pr2_feature_cache_write(dm, Tc, h.cuda(), lg.cuda(), pos, ch, cp),
            "pr2_feature_cache_write")
    torch.cuda.synchronize()
    assert np.array_equal(pos.cpu().numpy(), ref["pos"])
    assert torch.equal(ch.cpu(), ref["h"]) and np.array_equal(cp.cpu().numpy(), ref["p"])
