"""GPU parity at the full workload sizes (Qwen3-30B-A3B-shaped layer, its decode batch, the
Zipf-skewed long replay and the DeepSeek-V3-shaped layer).  Inputs are drawn on the GPU;
routes, counts and permutations are checked on every token, layer outputs on a seeded sample of
tokens the oracle computes one by one."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_00395_gb300 import binding as B
from paper_2606_00395_gb300 import synth
from tests import layer_harness as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_00395_gb300 import build
    build.build()
    B.load()


def _sample_output_check(cfg, L, idx, gates, out, n_tok, seed=0):
    toks = synth.make_token_sample(cfg.T, n_tok, seed).numpy()
    idx_s = np.asarray(idx)[toks]
    Wg, Wu, Wd, idx_c = H.compact_experts(L, idx_s)
    x_s = H.cpu(L["x"][torch.from_numpy(toks).to(L["x"].device)])
    sh = [H.cpu(L[n]) if L[n] is not None else None for n in ("Ws_gate", "Ws_up", "Ws_down")]
    want = oracle.moe_forward(x_s, idx_c, np.asarray(gates)[toks], Wg, Wu, Wd, *sh)
    got = H.cpu(out).float().numpy()[toks]
    return H.normwise_close(got, want, H.OUT_TOL[cfg.dtype])


def _routing_check(cfg, L, g, sample=None):
    """Full (or sampled) route comparison; returns (exempt, checked) token counts."""
    x, idx, gates, logits = L["x"], H.cpu(g["idx"]).numpy(), H.cpu(g["gates"]).numpy(), \
        H.cpu(g["logits"]).numpy()
    if sample is not None:
        sel = torch.from_numpy(sample).to(x.device)
        x = x[sel]
        idx, gates, logits = idx[sample], gates[sample], logits[sample]
    orc = oracle.route_predict(H.cpu(x), H.cpu(L["W_router"]), H.cpu(L["W_pred"]), cfg.k)
    exempt = H.check_routes(orc, idx)
    H.rowwise_close(gates, np.take_along_axis(orc["probs"], idx, 1))
    H.rowwise_close(logits, orc["logits"])
    return exempt, idx.shape[0], orc


def test_qwen3_layer_both_modes():
    cfg = synth.CONFIGS["qwen3_30b_a3b"]
    L = synth.make_layer(cfg, device="cuda")
    g = H.gpu_predict(cfg, L)
    exempt, n, orc = _routing_check(cfg, L, g)
    print(f"qwen3 rollout: {exempt}/{n} near-tie tokens")
    # replay the oracle's recorded route with the drifted router; permutation bit-exact
    W2 = synth.make_drifted_router(L["W_router"])
    idx_rec = torch.from_numpy(orc["idx"]).cuda()
    r = H.gpu_replay(cfg, L, W2, idx_rec, probs=False)
    toks = synth.make_token_sample(cfg.T, 256, 1).numpy()
    orep = oracle.route_replay(H.cpu(L["x"])[toks], H.cpu(W2), orc["idx"][toks])
    H.rowwise_close(H.cpu(r["gates"]).numpy()[toks], orep["gates"])
    f = H.gpu_forward(cfg, L, idx_rec, r["gates"])
    assert f["code"] == 0 and int(f["status"].item()) == 0
    operm = oracle.permute(orc["idx"], cfg.N)
    assert np.array_equal(H.cpu(f["counts"]).numpy(), operm["counts"])
    assert np.array_equal(H.cpu(f["perm"]).numpy(), operm["perm"])
    err = _sample_output_check(cfg, L, orc["idx"], H.cpu(r["gates"]).numpy(), f["out"], 48)
    # rollout output on the GPU's own route, sampled
    f2 = H.gpu_forward(cfg, L, g["idx"], g["gates"])
    err2 = _sample_output_check(cfg, L, H.cpu(g["idx"]).numpy(), H.cpu(g["gates"]).numpy(),
                                f2["out"], 48, seed=4)
    print(f"qwen3 output error replay {err:.2e} rollout {err2:.2e}")


def test_qwen3_shape_ragged_batch():
    """The Qwen3-shaped layer with T = 4001 (the last token tile 33 rows): every route against
    the oracle, counts and permutation bit-exact, layer outputs on a token sample."""
    cfg = synth.CONFIGS["qwen3_30b_a3b"].scaled(4001)
    L = synth.make_layer(cfg, device="cuda")
    g = H.gpu_predict(cfg, L)
    exempt, n, orc = _routing_check(cfg, L, g)
    f = H.gpu_forward(cfg, L, g["idx"], g["gates"])
    assert f["code"] == 0 and int(f["status"].item()) == 0
    gidx = H.cpu(g["idx"]).numpy()
    operm = oracle.permute(gidx, cfg.N)
    assert np.array_equal(H.cpu(f["counts"]).numpy(), operm["counts"])
    assert np.array_equal(H.cpu(f["perm"]).numpy(), operm["perm"])
    toks = np.unique(np.concatenate([synth.make_token_sample(cfg.T, 40, 7).numpy(),
                                     np.arange(cfg.T - 8, cfg.T)]))  # + the ragged tile's end
    idx_s = gidx[toks]
    Wg, Wu, Wd, idx_c = H.compact_experts(L, idx_s)
    want = oracle.moe_forward(H.cpu(L["x"])[toks], idx_c, H.cpu(g["gates"]).numpy()[toks],
                              Wg, Wu, Wd)
    err = H.normwise_close(H.cpu(f["out"]).float().numpy()[toks], want, H.OUT_TOL[cfg.dtype])
    print(f"qwen3 T=4001: {exempt}/{n} near ties, output error {err:.2e}")


def test_qwen3_decode_batch_rollout():
    cfg = synth.CONFIGS["qwen3_decode"]
    L = synth.make_layer(cfg, device="cuda")
    g = H.gpu_predict(cfg, L)
    exempt, n, orc = _routing_check(cfg, L, g)
    f = H.gpu_forward(cfg, L, g["idx"], g["gates"])
    assert f["code"] == 0
    gidx = H.cpu(g["idx"]).numpy()
    operm = oracle.permute(gidx, cfg.N)
    assert np.array_equal(H.cpu(f["perm"]).numpy(), operm["perm"])
    err = _sample_output_check(cfg, L, gidx, H.cpu(g["gates"]).numpy(), f["out"], 64)
    print(f"decode: {exempt}/{n} near ties, output error {err:.2e}")


def test_long_replay_with_zipf_routes():
    cfg = synth.CONFIGS["qwen3_long_replay"]
    L = synth.make_layer(cfg, device="cuda")
    idx = synth.make_zipf_routes(cfg.T, cfg.N, cfg.k, cfg.zipf_s)
    idx_d = idx.cuda()
    r = H.gpu_replay(cfg, L, L["W_router"], idx_d, probs=False)
    toks = synth.make_token_sample(cfg.T, 256, 2).numpy()
    orep = oracle.route_replay(H.cpu(L["x"])[toks], H.cpu(L["W_router"]), idx.numpy()[toks])
    H.rowwise_close(H.cpu(r["gates"]).numpy()[toks], orep["gates"])
    f = H.gpu_forward(cfg, L, idx_d, r["gates"])
    assert f["code"] == 0 and int(f["status"].item()) == 0
    operm = oracle.permute(idx.numpy(), cfg.N)
    counts = H.cpu(f["counts"]).numpy()
    assert np.array_equal(counts, operm["counts"])
    assert np.array_equal(H.cpu(f["perm"]).numpy(), operm["perm"])
    assert counts.max() > 50 * counts.min()  # the load really is skewed
    err = _sample_output_check(cfg, L, idx.numpy(), H.cpu(r["gates"]).numpy(), f["out"], 24)
    print(f"zipf counts {counts.min()}..{counts.max()}, output error {err:.2e}")


@pytest.mark.parametrize("T", [32768, 20001])
def test_long_batch_routing_both_modes(T):
    """T = 32768 (256 token tiles) and T = 20001 (157 tiles, the last one ragged): more tiles
    than the GPU has SMs, so routing runs two CTAs per SM with half the pipeline stages each;
    routes and gates on a token sample in both modes, the replay probabilities too."""
    cfg = synth.CONFIGS["qwen3_long_replay"].scaled(T)
    L = synth.make_layer(cfg, device="cuda")
    g = H.gpu_predict(cfg, L)
    sample = synth.make_token_sample(cfg.T, 384, 6).numpy()
    exempt, n, orc = _routing_check(cfg, L, g, sample=sample)
    W2 = synth.make_drifted_router(L["W_router"])
    r = H.gpu_replay(cfg, L, W2, g["idx"])
    orep = oracle.route_replay(H.cpu(L["x"])[sample], H.cpu(W2), H.cpu(g["idx"]).numpy()[sample])
    H.rowwise_close(H.cpu(r["gates"]).numpy()[sample], orep["gates"])
    H.rowwise_close(H.cpu(r["probs"]).numpy()[sample], orep["probs"])
    assert int(g["status"].item()) == 0 and int(r["status"].item()) == 0
    print(f"long batch routing: {exempt}/{n} near ties (sampled)")


def test_deepseek_v3_layer_with_shared_expert():
    cfg = synth.CONFIGS["deepseek_v3"]
    L = synth.make_layer(cfg, device="cuda")
    g = H.gpu_predict(cfg, L)
    sample = synth.make_token_sample(cfg.T, 512, 5).numpy()
    exempt, n, _ = _routing_check(cfg, L, g, sample=sample)
    f = H.gpu_forward(cfg, L, g["idx"], g["gates"])
    assert f["code"] == 0 and int(f["status"].item()) == 0
    gidx = H.cpu(g["idx"]).numpy()
    operm = oracle.permute(gidx, cfg.N)
    assert np.array_equal(H.cpu(f["counts"]).numpy(), operm["counts"])
    assert np.array_equal(H.cpu(f["perm"]).numpy(), operm["perm"])
    err = _sample_output_check(cfg, L, gidx, H.cpu(g["gates"]).numpy(), f["out"], 6)
    print(f"deepseek: {exempt}/{n} near ties (sampled), output error {err:.2e}")
