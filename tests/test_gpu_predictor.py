"""GPU parity of the predictive loss (Eq. pr2_loss, Algorithm 3, and the delta-matching
variant): loss, per-token KL and the W_p gradient through the C ABI against the fp64 oracle.

Inputs: a seeded layer; the cached rows are the evenly spaced feature-cache positions of the
batch, their features (h_old, p_old) and the teacher rho = Softmax(h W') of the drifted current
router come from the oracle (fp64, stored as fp32), never from the CUDA path.

Tolerances (derived from the arithmetic): the loss and per-token KL are computed in fp32 from
fp32 logits whose error is that of the bf16 routing GEMM (fp32 accumulation, ~1e-6); each KL
term carries a few ulp of |log rho| <= 20, so per-token KL is checked to 2e-5 absolute + 1e-4
relative and the mean loss to 1e-4 relative.  The bf16 gradient multiplies dKL/dz rounded to
bf16 (relative error 2^-9) by bf16 h_old with fp32 accumulation: normwise error ~2e-3, checked at
1e-2; the fp32 path is checked at 1e-4."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_00395_gb300 import binding as B
from paper_2606_00395_gb300 import synth

pytestmark = pytest.mark.gpu

LOSS_RTOL = 1e-4
KL_ATOL, KL_RTOL = 2e-5, 1e-4
GRAD_TOL = {"bf16": 1e-2, "fp32": 1e-4}


def _case(cfg, Tc, seed=0):
    L = synth.make_layer(cfg, seed=seed)
    W2 = synth.make_drifted_router(L["W_router"])
    rollout = oracle.route_predict(L["x"], L["W_router"], L["W_pred"], cfg.k)
    teacher = oracle.route_replay(L["x"], W2, rollout["idx"])
    fc = oracle.feature_cache(L["x"], torch.from_numpy(rollout["logits"]).float(), Tc)
    return dict(h_old=fc["h"], p_old=torch.from_numpy(fc["p"]), W_pred=L["W_pred"],
                rho=torch.from_numpy(teacher["probs"]).float(), pos=fc["pos"])


def _gpu(cfg, c, delta=False, pos=None, sync=False):
    Tc = c["h_old"].shape[0]
    flags = (B.PR2_F_DELTA_LOSS if delta else 0) | (B.PR2_F_SYNC_STATUS if sync else 0)
    dm = B.dims(Tc, cfg.d, cfg.N, cfg.k, cfg.m, 0, cfg.dtype, flags=flags)
    dev = lambda t: t.contiguous().cuda()
    loss = torch.full((1,), float("nan"), device="cuda")
    kl = torch.full((max(Tc, 1),), float("nan"), device="cuda")
    grad = torch.full((cfg.N, cfg.d), float("nan"), device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = B.alloc_loss_workspace(dm)
    p = c["pos"] if pos is None else pos
    code = B.pr2_predictor_loss(dm, dev(c["h_old"]), dev(c["p_old"]), dev(c["W_pred"]),
                                dev(c["rho"]), loss, grad,
                                pos=torch.from_numpy(np.asarray(p, np.int32)).cuda(),
                                kl_tok=kl, workspace=ws, status=status)
    torch.cuda.synchronize()
    return dict(code=code, loss=float(loss.item()), kl=kl[:Tc].cpu().numpy(),
                grad=grad.cpu().numpy(), status=int(status.item()))


def _check(cfg, c, g, delta=False, pos=None):
    ref = oracle.predictor_loss(c["h_old"], c["p_old"], c["W_pred"], c["rho"],
                                pos=c["pos"] if pos is None else pos, delta=delta)
    assert g["code"] == 0 and g["status"] == 0
    assert abs(g["loss"] - ref["loss"]) <= LOSS_RTOL * abs(ref["loss"]) + 1e-7, (g["loss"], ref["loss"])
    assert np.all(np.abs(g["kl"] - ref["kl"]) <= KL_ATOL + KL_RTOL * np.abs(ref["kl"]))
    err = np.max(np.abs(g["grad"] - ref["grad"])) / np.max(np.abs(ref["grad"]))
    assert err <= GRAD_TOL[cfg.dtype], err
    return ref


CASES = {
    # bf16, N = 32 experts: the loss routing kernel runs as 2-CTA clusters; ragged T_c = 333
    "bf16_n32": (synth.LayerConfig("l32", T=700, d=320, N=32, k=6, m=192), 333),
    # bf16, N = 128, d = 2048 (the qwen3 layer shape), T_c = 300: 8-CTA clusters, 8 d-tiles
    "bf16_qwen_shape": (synth.LayerConfig("l128", T=600, d=2048, N=128, k=8, m=768), 300),
    # bf16, N = 256 routed experts: two M-tiles in the gradient GEMM
    "bf16_n256": (synth.LayerConfig("l256", T=260, d=128, N=256, k=8, m=128), 130),
    # fp32 SIMT path
    "fp32": (synth.LayerConfig("lf", T=256, d=128, N=8, k=2, m=256, dtype="fp32"), 100),
}


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("delta", [False, True])
def test_predictor_loss_matches_oracle(name, delta):
    cfg, Tc = CASES[name]
    c = _case(cfg, Tc)
    g = _gpu(cfg, c, delta=delta)
    _check(cfg, c, g, delta=delta)


# Gradient-GEMM splits the layer cases above do not reach (inputs drawn directly): 8 CTAs per
# cluster (two 128 x 128 tiles, 8 K blocks), and one CTA per tile (N = 256, d = 4864: 76 tiles,
# too many for 2-CTA clusters to be resident at once)
DIRECT = {
    "split8": (64, 256, 512, 700),
    "split1_many_tiles": (256, 4864, 192, 300),
}


@pytest.mark.parametrize("name", list(DIRECT))
def test_predictor_loss_gradient_splits(name):
    N, d, Tc, T_rho = DIRECT[name]
    cfg = synth.LayerConfig(name, T=T_rho, d=d, N=N, k=8, m=128)
    c = synth.make_loss_inputs(N, d, Tc, T_rho, seed=11)
    c["pos"] = c["pos"].numpy()
    g = _gpu(cfg, c)
    _check(cfg, c, g)


def test_predictor_loss_full_cache_of_the_qwen3_layer():
    """T = 4096 tokens, T_c = 2048 cached (Table 4's Qwen3 cache length): the loss, every
    per-token KL and the whole gradient."""
    cfg = synth.CONFIGS["qwen3_30b_a3b"]
    c = _case(cfg, 2048)
    g = _gpu(cfg, c)
    _check(cfg, c, g)


def test_predictor_loss_invalid_rows_and_empty_cache():
    cfg, Tc = CASES["bf16_n32"]
    c = _case(cfg, Tc)
    pos = np.array(c["pos"], np.int32)
    pos[5] = cfg.T + 3
    pos[200] = -1
    g = _gpu(cfg, c, pos=pos)
    assert g["status"] & B.PR2_STATUS_BAD_INDEX
    ref = oracle.predictor_loss(c["h_old"], c["p_old"], c["W_pred"], c["rho"], pos=pos)
    assert ref["bad"] == 2 and g["kl"][5] == 0 and g["kl"][200] == 0
    assert abs(g["loss"] - ref["loss"]) <= LOSS_RTOL * abs(ref["loss"])
    err = np.max(np.abs(g["grad"] - ref["grad"])) / np.max(np.abs(ref["grad"]))
    assert err <= GRAD_TOL["bf16"]
    assert _gpu(cfg, c, pos=pos, sync=True)["code"] == 4
    e = dict(c, h_old=c["h_old"][:0], p_old=c["p_old"][:0], pos=c["pos"][:0])
    z = _gpu(cfg, e)
    assert z["code"] == 0 and z["loss"] == 0 and not np.any(z["grad"])


def test_predictor_loss_is_deterministic():
    cfg, Tc = CASES["bf16_qwen_shape"]
    c = _case(cfg, Tc, seed=3)
    a, b = _gpu(cfg, c), _gpu(cfg, c)
    assert a["loss"] == b["loss"] and np.array_equal(a["kl"], b["kl"])
    assert np.array_equal(a["grad"], b["grad"])
