"""The workspace-free layer forward (pr2_moe_forward_static), for callers that cannot allocate
device memory where they run the layer.  It must give the same output as pr2_moe_forward with a
caller-provided workspace, on two calls in a row (the second call reuses the scratch array the
first one left behind).  Collected last on purpose."""
import ctypes

import pytest
import torch

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


def test_static_scratch_forward_matches_workspace_forward_twice():
    cfg = synth.LayerConfig("decode_small", T=200, d=2048, N=128, k=8, m=768)
    dm = H.dims_of(cfg)
    assert B.pr2_moe_workspace_bytes(dm) <= B.pr2_static_scratch_bytes()
    L = H.to_dev(synth.make_layer(cfg, seed=3))
    g = H.gpu_predict(cfg, L)
    ref = H.gpu_forward(cfg, L, g["idx"], g["gates"])
    assert ref["code"] == 0
    for call in range(2):
        out = torch.full((cfg.T, cfg.d), float("nan"), dtype=torch.bfloat16, device="cuda")
        counts = torch.empty(cfg.N, dtype=torch.int32, device="cuda")
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        code = B.pr2_moe_forward_static(dm, L["x"], g["idx"], g["gates"], L["W_gate"], L["W_up"],
                                        L["W_down"], None, None, None, out, counts=counts,
                                        status=status)
        assert code == 0, B.pr2_strerror(code)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        assert torch.equal(counts, ref["counts"])
        H.normwise_close(out.float().cpu().numpy(), ref["out"].float().cpu().numpy(),
                         H.OUT_TOL["bf16"])
    # the same call with the Qwen3-shaped 4096-token batch needs far more scratch: rejected
    big = B.dims(4096, 2048, 128, 8, 768)
    fake = ctypes.c_void_p(256)
    lib = B._static_lib()
    assert lib.pr2_moe_forward_static(ctypes.byref(big), fake, fake, fake, fake, fake, fake,
                                      None, None, None, fake, None, None, None, None) == 6
