"""GPU parity of the multi-layer rollout decode loop (Algorithm 2 over stacked layers with the
residual stream) through pr2_rollout_layers, eager and replayed from a CUDA graph.

Inputs: seeded layers (router x4 and experts x2 the usual N(0, 0.02^2) scale, so that every
layer moves the residual stream by ~10 % while it stays O(1)); the reference is the fp64 oracle
composition, which rounds the stream to bf16 once per layer as the library does.

What is unique is checked exactly; where several answers are valid, validity is checked:
 - layer 1 sees identical inputs: every token under the usual near-tie rule;
 - a token whose top-(k+1) oracle probabilities are >= 1e-3 apart at every layer (so neither
   the top-k set nor its order is near a tie) has one trajectory: its routes
   must equal the oracle's at every layer and its gates agree row-normwise to 1e-4 at layer 1
   and 1e-2 after it (the stream entering layer l > 1 differs from the oracle's by one bf16
   ulp in the elements where the fp32 and fp64 sums round differently: ~2e-3 in the logits);
 - other tokens may legitimately follow another route after a near tie: their routes must be
   valid (in range, distinct);
 - the final stream over the unique-trajectory tokens agrees normwise to 2e-2 (the layer
   tolerance); the graph replay is bit-identical to the eager call."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_00395_gb300 import binding as B
from paper_2606_00395_gb300 import synth
from tests import layer_harness as H

pytestmark = pytest.mark.gpu

MARGIN = 1e-3


def _layers(cfg, L, seed0=40):
    out = []
    for l in range(L):
        lw = synth.make_layer(cfg, seed=seed0 + l)
        for k in ("W_router", "W_pred"):
            lw[k] = (lw[k].float() * 4).to(lw[k].dtype)
        for k in ("W_gate", "W_up", "W_down"):
            lw[k] = (lw[k].float() * 2).to(lw[k].dtype)
        out.append(lw)
    return out


def _stack(layers, key):
    return torch.stack([lw[key] for lw in layers]).contiguous().cuda()


def _run(cfg, layers, h0, stream=None):
    L = len(layers)
    dm = H.dims_of(cfg)
    h = h0.clone().cuda()
    idx = torch.full((L, cfg.T, cfg.k), -1, dtype=torch.int32, device="cuda")
    gates = torch.zeros(L, cfg.T, cfg.k, dtype=torch.float32, device="cuda")
    logits = torch.zeros(L, cfg.T, cfg.N, dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = B.alloc_workspace(dm)
    W = {k: _stack(layers, k) for k in ("W_router", "W_pred", "W_gate", "W_up", "W_down")}
    args = (dm, L, h, W["W_router"], W["W_pred"], W["W_gate"], W["W_up"], W["W_down"], idx,
            gates)
    kw = dict(logits_old=logits, workspace=ws, status=status)
    return h, idx, gates, logits, status, args, kw


@pytest.mark.parametrize("L", [1, 3])
def test_rollout_layers_match_the_oracle_composition(L):
    cfg = synth.LayerConfig("roll", T=256, d=256, N=32, k=4, m=128)
    layers = _layers(cfg, L)
    h0 = layers[0]["x"]
    ref = oracle.rollout_layers(h0, layers, cfg.k)
    h, idx, gates, logits, status, args, kw = _run(cfg, layers, h0)
    B.check(B.pr2_rollout_layers(*args, **kw), "pr2_rollout_layers")
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    gi, gg = H.cpu(idx).numpy(), H.cpu(gates).numpy()
    # layer 1: identical inputs, the single-layer rule for every token
    first = oracle.route_predict(h0, layers[0]["W_router"], layers[0]["W_pred"], cfg.k)
    H.check_routes(first, gi[0])
    H.rowwise_close(H.cpu(logits[0]).numpy(), first["logits"])
    unique = (ref["min_gap"] >= MARGIN).all(0)
    assert unique.mean() > 0.5
    for l in range(L):
        assert np.all((gi[l] >= 0) & (gi[l] < cfg.N))
        assert all(len(set(r)) == cfg.k for r in gi[l].tolist())
        assert np.array_equal(gi[l][unique], ref["idx"][l][unique]), l
        H.rowwise_close(gg[l][unique], ref["gates"][l][unique], 1e-4 if l == 0 else 1e-2)
    H.normwise_close(H.cpu(h).float().numpy()[unique], ref["h"].float().numpy()[unique],
                     H.OUT_TOL["bf16"])


def test_rollout_layers_replay_from_a_cuda_graph():
    cfg = synth.LayerConfig("roll", T=256, d=256, N=32, k=4, m=128)
    layers = _layers(cfg, 3, seed0=60)
    h0 = layers[0]["x"]
    h, idx, gates, logits, status, args, kw = _run(cfg, layers, h0)
    B.check(B.pr2_rollout_layers(*args, **kw), "eager")
    torch.cuda.synchronize()
    eager = (h.clone(), idx.clone(), gates.clone(), logits.clone())
    side = torch.cuda.Stream()
    h.copy_(h0.cuda())
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=side):
        code = B.pr2_rollout_layers(*args, **kw, stream=side)
    assert code == 0
    for _ in range(2):
        h.copy_(h0.cuda())
        idx.fill_(-1)
        gates.zero_()
        logits.zero_()
        graph.replay()
        torch.cuda.synchronize()
        assert torch.equal(h, eager[0]) and torch.equal(idx, eager[1])
        assert torch.equal(gates, eager[2]) and torch.equal(logits, eager[3])
    assert int(status.item()) == 0
