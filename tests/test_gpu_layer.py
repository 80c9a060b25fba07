"""GPU parity: every step of the layer through the C ABI against the CPU oracle.

Small layers are compared element by element in full (several M-tiles per expert, ragged
tails, partial N-tiles); the full-size workloads are compared on all routes and permutations
and on a seeded sample of layer outputs.  Tolerances are defined in ``layer_harness``."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_00395_gb300 import binding as B
from paper_2606_00395_gb300 import synth
from tests import layer_harness as H

pytestmark = pytest.mark.gpu

SMALL = {
    # fp32 SIMT path, the tiny workload exactly
    "tiny_fp32": synth.CONFIGS["tiny_fp32"],
    # fp32 with N = 6 experts: dispatch takes its three-kernel path (the fused cooperative
    # dispatch needs N % 4 == 0), with one and with 36 blocks of slots
    "fp32_n6": synth.LayerConfig("fp32_n6", T=300, d=64, N=6, k=3, m=96, dtype="fp32"),
    "fp32_n6_wide": synth.LayerConfig("fp32_n6_wide", T=3000, d=64, N=6, k=3, m=96,
                                      dtype="fp32"),
    # bf16, 9600 slots over 38 blocks of the fused cooperative dispatch, N = 32, m = 64
    "bf16_fused_dispatch": synth.LayerConfig("bf16_fused_dispatch", T=1200, d=128, N=32, k=8,
                                             m=64),
    # bf16, ~175 rows per expert -> 2 M-tiles per expert, 2 gate/up N-tiles, ragged T
    "bf16_multitile": synth.LayerConfig("bf16_multitile", T=700, d=256, N=16, k=4, m=256),
    # bf16, partial N-tiles in both GEMMs (m = 192 = 128 + 64, d = 320 = 256 + 64), k = 6
    "bf16_partial_n": synth.LayerConfig("bf16_partial_n", T=333, d=320, N=32, k=6, m=192),
    # bf16 with a shared expert, N = 256 routed experts (two 256-column MMAs in routing)
    "bf16_shared_n256": synth.LayerConfig("bf16_shared_n256", T=200, d=128, N=256, k=8, m=128,
                                          n_shared=1),
    # degenerate shapes: one expert (top-1 of 1: the dense SwiGLU MLP, gate 1), top-k over all
    # experts (no (k+1)-th probability, so no near ties), top-1, and a single token (one row
    # in every tile of both GEMMs, one combine block)
    "fp32_one_expert": synth.LayerConfig("fp32_one_expert", T=77, d=64, N=1, k=1, m=96,
                                         dtype="fp32"),
    "fp32_k_eq_n": synth.LayerConfig("fp32_k_eq_n", T=100, d=64, N=8, k=8, m=64, dtype="fp32"),
    "bf16_top1": synth.LayerConfig("bf16_top1", T=257, d=128, N=16, k=1, m=64),
    "bf16_one_token": synth.LayerConfig("bf16_one_token", T=1, d=256, N=32, k=8, m=128),
}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_00395_gb300 import build
    build.build()
    B.load()


def _full_layer_check(cfg, seed=0):
    L = synth.make_layer(cfg, seed=seed)
    Ld = H.to_dev(L)
    W2 = synth.make_drifted_router(L["W_router"], seed=seed)
    # ---- rollout: route prediction (Eqs. pr2_predict, pr2_route)
    g = H.gpu_predict(cfg, Ld)
    orc = oracle.route_predict(L["x"], L["W_router"], L["W_pred"], cfg.k)
    exempt = H.check_routes(orc, H.cpu(g["idx"]).numpy())
    gidx = H.cpu(g["idx"]).numpy()
    H.rowwise_close(H.cpu(g["gates"]).numpy(), np.take_along_axis(orc["probs"], gidx, 1))
    H.rowwise_close(H.cpu(g["logits"]).numpy(), orc["logits"])
    assert int(g["status"].item()) == 0
    # ---- replay of the oracle's recorded route with the drifted router (Sec. 4.1)
    idx_rec = torch.from_numpy(orc["idx"]).cuda()
    r = H.gpu_replay(cfg, Ld, W2.cuda(), idx_rec)
    orep = oracle.route_replay(L["x"], W2, orc["idx"])
    H.rowwise_close(H.cpu(r["gates"]).numpy(), orep["gates"])
    H.rowwise_close(H.cpu(r["probs"]).numpy(), orep["probs"])
    assert int(r["status"].item()) == 0
    # ---- layer output on the recorded route with replay gates (Eq. pr2_output)
    gates_rep = torch.from_numpy(orep["gates"].astype(np.float32)).cuda()
    f = H.gpu_forward(cfg, Ld, idx_rec, gates_rep)
    assert f["code"] == 0 and int(f["status"].item()) == 0
    operm = oracle.permute(orc["idx"], cfg.N)
    assert np.array_equal(H.cpu(f["counts"]).numpy(), operm["counts"])
    nvalid = int(operm["offsets"][-1])
    assert np.array_equal(H.cpu(f["perm"]).numpy()[:nvalid], operm["perm"])
    want = oracle.moe_forward(L["x"], orc["idx"], orep["gates"], L["W_gate"], L["W_up"],
                              L["W_down"], L["Ws_gate"], L["Ws_up"], L["Ws_down"])
    err = H.normwise_close(H.cpu(f["out"]).float().numpy(), want, H.OUT_TOL[cfg.dtype])
    # ---- rollout layer output on the GPU's own route (Eq. pr2_old_output), every token: a
    # near-tie token may take another (equally valid) top-k than the oracle, so the oracle is
    # recomputed on the GPU's route, weighted by the oracle's own probabilities there
    f2 = H.gpu_forward(cfg, Ld, g["idx"], g["gates"])
    want2 = oracle.moe_forward(L["x"], gidx, np.take_along_axis(orc["probs"], gidx, 1),
                               L["W_gate"], L["W_up"], L["W_down"], L["Ws_gate"], L["Ws_up"],
                               L["Ws_down"])
    H.normwise_close(H.cpu(f2["out"]).float().numpy(), want2, H.OUT_TOL[cfg.dtype])
    return exempt, err


@pytest.mark.parametrize("name", list(SMALL))
def test_small_layer_matches_oracle_everywhere(name):
    exempt, err = _full_layer_check(SMALL[name])
    print(f"{name}: near-tie tokens {exempt}, output error {err:.2e}")


@pytest.mark.parametrize("dtype,N,k", [("bf16", 64, 8), ("bf16", 256, 8), ("fp32", 6, 3),
                                       ("fp32", 8, 8)])
def test_all_zero_router_routes_to_the_lowest_experts(dtype, N, k):
    """W = W_p = 0: every logit is 0 and rho_hat is uniform, so all N probabilities tie exactly.
    The route is experts 0..k-1 in slot order (ties go to the lower expert), every gate is 1/N,
    every token is a near tie unless k = N, replay of the route gives the same gates, and the
    layer output is the uniform 1/N mix of the first k experts."""
    cfg = synth.LayerConfig("zero", T=300, d=128, N=N, k=k, m=128, dtype=dtype)
    L = synth.make_layer(cfg, seed=4)
    L["W_router"] = torch.zeros_like(L["W_router"])
    L["W_pred"] = torch.zeros_like(L["W_pred"])
    Ld = H.to_dev(L)
    g = H.gpu_predict(cfg, Ld)
    idx = H.cpu(g["idx"]).numpy()
    assert np.array_equal(idx, np.tile(np.arange(k, dtype=np.int32), (cfg.T, 1)))
    gates = H.cpu(g["gates"]).numpy().astype(np.float64)
    assert np.max(np.abs(gates * N - 1.0)) <= 1e-6
    assert np.all(H.cpu(g["logits"]).numpy() == 0.0)
    assert int(g["near_tie"].item()) == (cfg.T if k < N else 0)
    orc = oracle.route_predict(L["x"], L["W_router"], L["W_pred"], k)
    assert np.array_equal(orc["idx"], idx)
    r = H.gpu_replay(cfg, Ld, Ld["W_router"], g["idx"])
    assert torch.max(torch.abs(H.cpu(r["gates"]) - H.cpu(g["gates"]))).item() <= 1e-7
    f = H.gpu_forward(cfg, Ld, g["idx"], g["gates"])
    assert f["code"] == 0 and int(f["status"].item()) == 0
    want = oracle.moe_forward(L["x"], orc["idx"], orc["gates"], L["W_gate"], L["W_up"],
                              L["W_down"])
    H.normwise_close(H.cpu(f["out"]).float().numpy(), want, H.OUT_TOL[dtype])


def test_one_expert_layer_is_the_dense_swiglu_mlp():
    """N = k = 1: the route is expert 0 with gate exactly 1 (a softmax over one logit), and the
    layer is the dense SwiGLU MLP, checked here against fp64 matrix products directly."""
    cfg = SMALL["fp32_one_expert"]
    L = synth.make_layer(cfg, seed=6)
    Ld = H.to_dev(L)
    g = H.gpu_predict(cfg, Ld)
    assert np.all(H.cpu(g["idx"]).numpy() == 0)
    assert np.all(H.cpu(g["gates"]).numpy() == 1.0)
    f = H.gpu_forward(cfg, Ld, g["idx"], g["gates"])
    assert f["code"] == 0 and int(H.cpu(f["counts"])[0]) == cfg.T
    x = L["x"].double()
    a = x @ L["W_gate"][0].double().T
    u = x @ L["W_up"][0].double().T
    want = (a * torch.sigmoid(a) * u) @ L["W_down"][0].double().T
    H.normwise_close(H.cpu(f["out"]).double().numpy(), want.numpy(), H.OUT_TOL["fp32"])


def test_near_tie_counter_tracks_the_oracle_margin():
    cfg = synth.LayerConfig("q300", T=300, d=2048, N=128, k=8, m=768)
    L = synth.make_layer(cfg)
    Ld = H.to_dev(L)
    g = H.gpu_predict(cfg, Ld)
    orc = oracle.route_predict(L["x"], L["W_router"], L["W_pred"], cfg.k)
    H.check_routes(orc, H.cpu(g["idx"]).numpy())
    n_orc = int(np.sum(orc["margin"] < H.TIE_GAP))
    n_gpu = int(g["near_tie"].item())
    # the GPU classifies with its own fp32 probabilities: allow tokens right at the threshold
    borderline = int(np.sum(np.abs(orc["margin"] - H.TIE_GAP) < 2e-6))
    assert abs(n_gpu - n_orc) <= borderline, (n_gpu, n_orc, borderline)


@pytest.mark.parametrize("d", [192, 256])
def test_predict_routing_with_256_experts_in_two_passes(d):
    """N = 256: the router and predictor weights stream in two passes over K.  d = 256 (an even
    number of K blocks) runs them as the pass split, one pass per CTA of a 2-CTA cluster whose
    column halves meet unsummed; d = 192 (three K blocks) runs both passes in one CTA.  Routes
    under the near-tie rule, gates and p_old logits against the oracle; T = 300 leaves a ragged
    last tile."""
    cfg = synth.LayerConfig("p256", T=300, d=d, N=256, k=8, m=128)
    L = synth.make_layer(cfg, seed=d)
    Ld = H.to_dev(L)
    g = H.gpu_predict(cfg, Ld)
    assert int(g["status"].item()) == 0
    orc = oracle.route_predict(L["x"], L["W_router"], L["W_pred"], cfg.k)
    idx = H.cpu(g["idx"]).numpy()
    H.check_routes(orc, idx)
    H.rowwise_close(H.cpu(g["gates"]).numpy(), np.take_along_axis(orc["probs"], idx, 1))
    H.rowwise_close(H.cpu(g["logits"]).numpy(), orc["logits"])


def test_zero_predictor_replay_reproduces_rollout():
    """W_p = 0 and the same router: replaying the recorded route gives the rollout gates and
    the same layer output (routing replay, R2, is Pr^2 with a zero predictor)."""
    cfg = synth.LayerConfig("r2", T=260, d=512, N=64, k=8, m=256)
    L = synth.make_layer(cfg, seed=5)
    L["W_pred"] = torch.zeros_like(L["W_pred"])
    Ld = H.to_dev(L)
    g = H.gpu_predict(cfg, Ld)
    r = H.gpu_replay(cfg, Ld, Ld["W_router"], g["idx"])
    gg, rg = H.cpu(g["gates"]), H.cpu(r["gates"])
    assert torch.max(torch.abs(gg - rg)).item() <= 1e-6
    o1 = H.gpu_forward(cfg, Ld, g["idx"], g["gates"])["out"]
    o2 = H.gpu_forward(cfg, Ld, g["idx"], r["gates"])["out"]
    H.normwise_close(H.cpu(o2).float().numpy(), H.cpu(o1).float().numpy(), 1e-2)
    print("bit-exact replay gates:", torch.equal(gg, rg))


def test_layer_is_deterministic():
    cfg = synth.LayerConfig("det", T=1000, d=512, N=32, k=8, m=256)
    L = synth.make_layer(cfg, seed=11)
    Ld = H.to_dev(L)
    g = H.gpu_predict(cfg, Ld)
    a = H.gpu_forward(cfg, Ld, g["idx"], g["gates"])
    b = H.gpu_forward(cfg, Ld, g["idx"], g["gates"])
    assert torch.equal(a["out"], b["out"]) and torch.equal(a["perm"], b["perm"])


@pytest.mark.parametrize("N", [16, 64])  # one CTA per tile; a 4-CTA cluster splitting experts
def test_invalid_replay_indices_are_flagged_and_skipped(N):
    cfg = synth.LayerConfig("bad", T=130, d=256, N=N, k=4, m=128)
    L = synth.make_layer(cfg, seed=2)
    Ld = H.to_dev(L)
    orc = oracle.route_predict(L["x"], L["W_router"], L["W_pred"], cfg.k)
    idx = orc["idx"].copy()
    idx[3, 1] = N        # out of range
    idx[7, 2] = -5       # negative
    idx[129, 3] = idx[129, 0]  # duplicate within the token (last, ragged tile)
    idx_d = torch.from_numpy(idx).cuda()
    r = H.gpu_replay(cfg, Ld, Ld["W_router"], idx_d)
    orep = oracle.route_replay(L["x"], L["W_router"], idx)
    assert orep["bad"] == 3
    rg = H.cpu(r["gates"]).numpy()
    assert rg[3, 1] == 0 and rg[7, 2] == 0 and rg[129, 3] == 0
    H.rowwise_close(rg, orep["gates"])
    assert int(r["status"].item()) & B.PR2_STATUS_BAD_INDEX
    f = H.gpu_forward(cfg, Ld, idx_d, r["gates"])
    assert int(f["status"].item()) & B.PR2_STATUS_BAD_INDEX
    operm = oracle.permute(idx, cfg.N)
    assert np.array_equal(H.cpu(f["counts"]).numpy(), operm["counts"])
    assert np.array_equal(H.cpu(f["perm"]).numpy()[: operm["perm"].size], operm["perm"])
    want = oracle.moe_forward(L["x"], idx, orep["gates"], L["W_gate"], L["W_up"], L["W_down"])
    H.normwise_close(H.cpu(f["out"]).float().numpy(), want, H.OUT_TOL["bf16"])
    # with PR2_F_SYNC_STATUS the call itself reports the bad index
    f3 = H.gpu_forward(cfg, Ld, idx_d, r["gates"], flags=B.PR2_F_SYNC_STATUS)
    assert f3["code"] == 4


def test_bounded_wait_reports_timeout_instead_of_hanging():
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert B.pr2_selftest_wait_timeout(status, 20_000_000) == 0
    torch.cuda.synchronize()
    assert int(status.item()) == B.PR2_STATUS_TIMEOUT


@pytest.mark.parametrize("name", ["tiny_fp32", "bf16_multitile", "bf16_shared_n256"])
def test_normalized_gates_match_the_oracle(name):
    """PR2_F_NORMALIZE_TOPK: the same routes, gates divided by their sum over the route (replay:
    over the valid slots), in both modes; logits and probabilities are not renormalised."""
    cfg = SMALL[name]
    L = synth.make_layer(cfg, seed=3)
    Ld = H.to_dev(L)
    flag = B.PR2_F_NORMALIZE_TOPK
    g = H.gpu_predict(cfg, Ld, flags=flag)
    orc = oracle.route_predict(L["x"], L["W_router"], L["W_pred"], cfg.k, normalize=True)
    H.check_routes(orc, H.cpu(g["idx"]).numpy())
    gidx = H.cpu(g["idx"]).numpy()
    gg = H.cpu(g["gates"]).numpy()
    # every token, near ties included: the oracle's renormalisation of its own probabilities
    # at the GPU's route (equal to orc["gates"] wherever the routes agree)
    H.rowwise_close(gg, oracle.normalize_topk(np.take_along_axis(orc["probs"], gidx, 1)))
    assert np.max(np.abs(gg.sum(1) - 1.0)) < 1e-5
    H.rowwise_close(H.cpu(g["logits"]).numpy(), orc["logits"])
    idx = orc["idx"].copy()
    idx[0, 0] = cfg.N  # an invalid slot: excluded from the sum
    r = H.gpu_replay(cfg, Ld, Ld["W_router"], torch.from_numpy(idx).cuda(), flags=flag)
    orep = oracle.route_replay(L["x"], L["W_router"], idx, normalize=True)
    H.rowwise_close(H.cpu(r["gates"]).numpy(), orep["gates"])
    H.rowwise_close(H.cpu(r["probs"]).numpy(), orep["probs"])
    assert int(r["status"].item()) & B.PR2_STATUS_BAD_INDEX


@pytest.mark.parametrize("n_shared", [0, 1])
def test_all_invalid_route_gives_the_shared_experts_alone(n_shared):
    """Every cached index invalid: no routed rows (the grouped GEMM launch has no jobs, every
    combine slot carries no rows), the status flags it, counts are zero and the output is the
    shared experts' alone (zero without shared experts)."""
    cfg = synth.LayerConfig("none", T=150, d=256, N=32, k=4, m=128, n_shared=n_shared)
    L = synth.make_layer(cfg, seed=9)
    Ld = H.to_dev(L)
    idx = np.full((cfg.T, cfg.k), -1, np.int32)
    idx[:, 1] = cfg.N + 3
    gates = torch.zeros(cfg.T, cfg.k, dtype=torch.float32, device="cuda")
    f = H.gpu_forward(cfg, Ld, torch.from_numpy(idx).cuda(), gates)
    assert f["code"] == 0 and int(f["status"].item()) & B.PR2_STATUS_BAD_INDEX
    assert int(H.cpu(f["counts"]).sum().item()) == 0
    want = oracle.moe_forward(L["x"], idx, np.zeros((cfg.T, cfg.k)), L["W_gate"], L["W_up"],
                              L["W_down"], L["Ws_gate"], L["Ws_up"], L["Ws_down"])
    got = H.cpu(f["out"]).float().numpy()
    if n_shared == 0:
        assert np.all(got == 0.0)
    else:
        H.normwise_close(got, want, H.OUT_TOL["bf16"])


@pytest.mark.parametrize("name", ["tiny_fp32", "bf16_multitile", "bf16_partial_n",
                                  "bf16_shared_n256", "bf16_one_token"])
def test_replay_layer_call_equals_the_two_calls(name):
    """pr2_moe_replay_forward (replay routing launched behind the expert GEMMs) writes exactly
    what pr2_route_replay followed by pr2_moe_forward writes: gates, probabilities, counts,
    permutation and layer output, bit for bit; an invalid cached slot is flagged the same way."""
    cfg = SMALL[name]
    L = synth.make_layer(cfg, seed=11)
    Ld = H.to_dev(L)
    W2 = synth.make_drifted_router(L["W_router"], seed=11).cuda()
    g = H.gpu_predict(cfg, Ld)
    idx = g["idx"].clone()
    if cfg.T > 3:
        idx[3, 0] = cfg.N  # one invalid slot
    r = H.gpu_replay(cfg, Ld, W2, idx)
    ref = H.gpu_forward(cfg, Ld, idx, r["gates"])
    assert ref["code"] == 0
    dm = H.dims_of(cfg)
    gates = torch.full_like(r["gates"], float("nan"))
    probs = torch.full_like(r["probs"], float("nan"))
    out = torch.full_like(ref["out"], float("nan"))
    counts = torch.full_like(ref["counts"], -1)
    perm = torch.full_like(ref["perm"], -1)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    code = B.pr2_moe_replay_forward(dm, Ld["x"], W2, idx, gates, probs, Ld["W_gate"], Ld["W_up"],
                                    Ld["W_down"], Ld["Ws_gate"], Ld["Ws_up"], Ld["Ws_down"], out,
                                    counts=counts, perm=perm, workspace=B.alloc_workspace(dm),
                                    status=status)
    assert code == 0, B.pr2_strerror(code)
    torch.cuda.synchronize()
    assert torch.equal(gates, r["gates"]) and torch.equal(probs, r["probs"])
    n_valid = int(ref["counts"].sum().item())  # perm entries past sum(counts) are unspecified
    assert torch.equal(counts, ref["counts"]) and torch.equal(perm[:n_valid], ref["perm"][:n_valid])
    assert torch.equal(out, ref["out"])
    want_status = int(r["status"].item()) | int(ref["status"].item())
    assert int(status.item()) == want_status
    assert (want_status & B.PR2_STATUS_BAD_INDEX) == (B.PR2_STATUS_BAD_INDEX if cfg.T > 3 else 0)


def test_replay_layer_call_in_a_cuda_graph():
    """The replay layer captured into a CUDA graph on a side stream: replaying the graph on new
    inputs gives bit for bit what the eager call gives (the routing kernel launched behind the
    expert GEMMs, with its late dependency wait, is captured like the rest)."""
    cfg = SMALL["bf16_multitile"]
    L = synth.make_layer(cfg, seed=13)
    Ld = H.to_dev(L)
    W2 = synth.make_drifted_router(L["W_router"], seed=13).cuda()
    g = H.gpu_predict(cfg, Ld)
    dm = H.dims_of(cfg)
    ws = B.alloc_workspace(dm)
    x = Ld["x"].clone()
    gates = torch.empty(cfg.T, cfg.k, dtype=torch.float32, device="cuda")
    probs = torch.empty(cfg.T, cfg.N, dtype=torch.float32, device="cuda")
    out = torch.empty_like(x)

    def layer(stream=None):
        return B.pr2_moe_replay_forward(dm, x, W2, g["idx"], gates, probs, Ld["W_gate"],
                                        Ld["W_up"], Ld["W_down"], None, None, None, out,
                                        workspace=ws, stream=stream)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        assert layer(side) == 0  # warm-up outside the capture
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=side):
        assert layer(side) == 0
    x.copy_(torch.roll(Ld["x"], 1, 0))  # new inputs for the replay
    graph.replay()
    torch.cuda.synchronize()
    got = (gates.clone(), probs.clone(), out.clone())
    assert layer() == 0
    torch.cuda.synchronize()
    assert torch.equal(got[0], gates) and torch.equal(got[1], probs) and torch.equal(got[2], out)


@pytest.mark.parametrize("name", ["tiny_fp32", "bf16_fused_dispatch", "bf16_multitile",
                                  "bf16_partial_n", "bf16_shared_n256", "bf16_top1",
                                  "bf16_one_token"])
def test_rollout_layer_call_equals_the_two_calls(name):
    """pr2_moe_rollout_forward (dispatch from the routing kernel's per-CTA histograms) writes
    exactly what pr2_route_predict followed by pr2_moe_forward writes: route, gates, logits,
    near-tie count, counts, permutation and layer output, bit for bit."""
    cfg = SMALL[name]
    L = synth.make_layer(cfg, seed=12)
    Ld = H.to_dev(L)
    g = H.gpu_predict(cfg, Ld)
    ref = H.gpu_forward(cfg, Ld, g["idx"], g["gates"])
    assert ref["code"] == 0
    dm = H.dims_of(cfg)
    idx = torch.full_like(g["idx"], -7)
    gates = torch.full_like(g["gates"], float("nan"))
    logits = torch.full_like(g["logits"], float("nan"))
    near = torch.zeros(1, dtype=torch.int64, device="cuda")
    out = torch.full_like(ref["out"], float("nan"))
    counts = torch.full_like(ref["counts"], -1)
    perm = torch.full_like(ref["perm"], -1)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    code = B.pr2_moe_rollout_forward(dm, Ld["x"], Ld["W_router"], Ld["W_pred"], idx, gates,
                                     logits, near, Ld["W_gate"], Ld["W_up"], Ld["W_down"],
                                     Ld["Ws_gate"], Ld["Ws_up"], Ld["Ws_down"], out,
                                     counts=counts, perm=perm, workspace=B.alloc_workspace(dm),
                                     status=status)
    assert code == 0, B.pr2_strerror(code)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert torch.equal(idx, g["idx"]) and torch.equal(gates, g["gates"])
    assert torch.equal(logits, g["logits"]) and torch.equal(near, g["near_tie"])
    assert torch.equal(counts, ref["counts"]) and torch.equal(perm, ref["perm"])
    assert torch.equal(out, ref["out"])
