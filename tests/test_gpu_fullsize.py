"""GPU parity at the full workload sizes (Qwen3-30B-A3B-shaped layer, its decode batch, the
Zipf-skewed long replay and the DeepSeek-V3-shaped layer).  Inputs are drawn on the GPU.

* Qwen3-shaped layer (T = 4096): every route, gate, logit, replay gate, replay probability,
  count, permutation and layer output of both modes against the oracle.
* Decode batch (T = 256): everything, in full.
* Long replay (T = 32768) and DeepSeek-V3-shaped layer (T = 8192): every count and permutation
  (bit-exact), routes / gates / probabilities and layer outputs on a seeded sample of 512
  tokens that the oracle computes one by one.
Rollout outputs are compared with the oracle recomputed on the GPU's own route, weighted by the
oracle's probabilities there, so near-tie tokens are compared too."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_00395_gb300 import binding as B
from paper_2606_00395_gb300 import synth
from tests import layer_harness as H

pytestmark = pytest.mark.gpu

SAMPLE = 512  # tokens compared one by one on the layers too large for a full oracle pass


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_00395_gb300 import build
    build.build()
    B.load()


def _routing_check(cfg, L, g, sample=None):
    """Full (or sampled) route comparison; returns (exempt, checked, oracle result)."""
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


def _permutation_check(cfg, f, idx):
    operm = oracle.permute(np.asarray(idx), cfg.N)
    assert np.array_equal(H.cpu(f["counts"]).numpy(), operm["counts"])
    nvalid = int(operm["offsets"][-1])
    assert np.array_equal(H.cpu(f["perm"]).numpy()[:nvalid], operm["perm"])
    return operm


def _output_check(cfg, L, toks, idx_rows, gates_rows, out):
    want = H.oracle_forward_rows(L, toks, idx_rows, gates_rows)
    got = H.cpu(out).float().numpy()[np.asarray(toks)]
    return H.normwise_close(got, want, H.OUT_TOL[cfg.dtype])


def test_qwen3_layer_both_modes_in_full():
    """The bench workload, every output of both modes: rollout on the GPU's own route, then
    replay of the oracle's recorded route with the drifted router (Sec. 4.1)."""
    cfg = synth.CONFIGS["qwen3_30b_a3b"]
    L = synth.make_layer(cfg, device="cuda")
    everyone = np.arange(cfg.T)
    # ---- rollout (Eqs. pr2_predict, pr2_route, pr2_old_output)
    g = H.gpu_predict(cfg, L)
    exempt, n, orc = _routing_check(cfg, L, g)
    gidx = H.cpu(g["idx"]).numpy()
    f_roll = H.gpu_forward(cfg, L, g["idx"], g["gates"])
    assert f_roll["code"] == 0 and int(f_roll["status"].item()) == 0
    _permutation_check(cfg, f_roll, gidx)
    err_roll = _output_check(cfg, L, everyone, gidx,
                             np.take_along_axis(orc["probs"], gidx, 1), f_roll["out"])
    # ---- replay (Eq. pr2_output): gates and probabilities of every token
    W2 = synth.make_drifted_router(L["W_router"])
    idx_rec = torch.from_numpy(orc["idx"]).cuda()
    r = H.gpu_replay(cfg, L, W2, idx_rec, probs=True)
    assert int(r["status"].item()) == 0
    orep = oracle.route_replay(H.cpu(L["x"]), H.cpu(W2), orc["idx"])
    H.rowwise_close(H.cpu(r["gates"]).numpy(), orep["gates"])
    H.rowwise_close(H.cpu(r["probs"]).numpy(), orep["probs"])
    f_rep = H.gpu_forward(cfg, L, idx_rec, r["gates"])
    assert f_rep["code"] == 0 and int(f_rep["status"].item()) == 0
    _permutation_check(cfg, f_rep, orc["idx"])
    err_rep = _output_check(cfg, L, everyone, orc["idx"], orep["gates"], f_rep["out"])
    print(f"qwen3: {exempt}/{n} near ties; output error rollout {err_roll:.2e}, "
          f"replay {err_rep:.2e} (all {cfg.T} tokens)")


def test_qwen3_shape_ragged_batch():
    """The Qwen3-shaped layer with T = 4001 (the last token tile 33 rows): every route against
    the oracle, counts and permutation bit-exact, layer outputs on a token sample that includes
    the ragged tile's end."""
    cfg = synth.CONFIGS["qwen3_30b_a3b"].scaled(4001)
    L = synth.make_layer(cfg, device="cuda")
    g = H.gpu_predict(cfg, L)
    exempt, n, orc = _routing_check(cfg, L, g)
    f = H.gpu_forward(cfg, L, g["idx"], g["gates"])
    assert f["code"] == 0 and int(f["status"].item()) == 0
    gidx = H.cpu(g["idx"]).numpy()
    _permutation_check(cfg, f, gidx)
    toks = np.unique(np.concatenate([synth.make_token_sample(cfg.T, 256, 7).numpy(),
                                     np.arange(cfg.T - 40, cfg.T)]))
    err = _output_check(cfg, L, toks, gidx[toks],
                        np.take_along_axis(orc["probs"], gidx, 1)[toks], f["out"])
    print(f"qwen3 T=4001: {exempt}/{n} near ties, output error {err:.2e}")


def test_qwen3_decode_batch_rollout():
    cfg = synth.CONFIGS["qwen3_decode"]
    L = synth.make_layer(cfg, device="cuda")
    g = H.gpu_predict(cfg, L)
    exempt, n, orc = _routing_check(cfg, L, g)
    f = H.gpu_forward(cfg, L, g["idx"], g["gates"])
    assert f["code"] == 0 and int(f["status"].item()) == 0
    gidx = H.cpu(g["idx"]).numpy()
    _permutation_check(cfg, f, gidx)
    err = _output_check(cfg, L, np.arange(cfg.T), gidx,
                        np.take_along_axis(orc["probs"], gidx, 1), f["out"])
    print(f"decode: {exempt}/{n} near ties, output error {err:.2e} (all tokens)")


def test_long_replay_with_zipf_routes():
    cfg = synth.CONFIGS["qwen3_long_replay"]
    L = synth.make_layer(cfg, device="cuda")
    idx = synth.make_zipf_routes(cfg.T, cfg.N, cfg.k, cfg.zipf_s)
    idx_d = idx.cuda()
    r = H.gpu_replay(cfg, L, L["W_router"], idx_d, probs=True)
    assert int(r["status"].item()) == 0
    toks = synth.make_token_sample(cfg.T, SAMPLE, 2).numpy()
    orep = oracle.route_replay(H.cpu(L["x"])[toks], H.cpu(L["W_router"]), idx.numpy()[toks])
    H.rowwise_close(H.cpu(r["gates"]).numpy()[toks], orep["gates"])
    H.rowwise_close(H.cpu(r["probs"]).numpy()[toks], orep["probs"])
    f = H.gpu_forward(cfg, L, idx_d, r["gates"])
    assert f["code"] == 0 and int(f["status"].item()) == 0
    operm = _permutation_check(cfg, f, idx.numpy())
    counts = operm["counts"]
    assert counts.max() > 50 * counts.min()  # the load really is skewed
    err = _output_check(cfg, L, toks, idx.numpy()[toks], orep["gates"], f["out"])
    print(f"zipf counts {counts.min()}..{counts.max()}, output error {err:.2e} "
          f"({len(toks)} tokens)")


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


def test_deepseek_v3_layer_both_modes():
    """The DeepSeek-V3-shaped layer (T = 8192, d = 7168, 256 routed experts + 1 shared, top-8,
    m = 2048) in both modes: rollout on the GPU's own route, then replay of that route with the
    drifted router (Sec. 4.1; the shared expert of App. E.2 added with weight 1).  Every count
    and permutation bit-exact; routes, gates, probabilities and outputs on 512 tokens."""
    cfg = synth.CONFIGS["deepseek_v3"]
    L = synth.make_layer(cfg, device="cuda")
    sample = synth.make_token_sample(cfg.T, SAMPLE, 5).numpy()
    # ---- rollout
    g = H.gpu_predict(cfg, L)
    exempt, n, orc = _routing_check(cfg, L, g, sample=sample)
    gidx = H.cpu(g["idx"]).numpy()
    f_roll = H.gpu_forward(cfg, L, g["idx"], g["gates"])
    assert f_roll["code"] == 0 and int(f_roll["status"].item()) == 0
    _permutation_check(cfg, f_roll, gidx)
    err_roll = _output_check(cfg, L, sample, gidx[sample],
                             np.take_along_axis(orc["probs"], gidx[sample], 1), f_roll["out"])
    # ---- replay of the recorded route with the drifted router
    W2 = synth.make_drifted_router(L["W_router"])
    r = H.gpu_replay(cfg, L, W2, g["idx"], probs=True)
    assert int(r["status"].item()) == 0
    sel = torch.from_numpy(sample).cuda()
    orep = oracle.route_replay(H.cpu(L["x"][sel]), H.cpu(W2), gidx[sample])
    H.rowwise_close(H.cpu(r["gates"]).numpy()[sample], orep["gates"])
    H.rowwise_close(H.cpu(r["probs"]).numpy()[sample], orep["probs"])
    f_rep = H.gpu_forward(cfg, L, g["idx"], r["gates"])
    assert f_rep["code"] == 0 and int(f_rep["status"].item()) == 0
    _permutation_check(cfg, f_rep, gidx)
    err_rep = _output_check(cfg, L, sample, gidx[sample], orep["gates"], f_rep["out"])
    print(f"deepseek: {exempt}/{n} near ties (sampled); output error rollout {err_roll:.2e}, "
          f"replay {err_rep:.2e} ({len(sample)} tokens)")
