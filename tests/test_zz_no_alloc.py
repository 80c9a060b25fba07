"""The workspace-free layer forward (pr2_moe_forward_static), for callers that cannot allocate
device memory where they run the layer (a runtime whose pool owns all device memory, a hot path
that must not call cudaMalloc/cudaFree, a plug-in with a fixed memory budget).

The static entry point runs the same kernels on the same inputs as pr2_moe_forward with a
caller-provided workspace, and those kernels are deterministic, so its outputs must be
bit-identical to the workspace forward's.  The scratch array keeps whatever the previous call
left in it: the test first runs the largest Qwen3-shaped layer with a shared expert that fits
the array, then a smaller layer without one twice in a row, so that any scratch state a call
fails to reset (readiness counters, tile tables, the grid-barrier counter) would show up as a
difference.  Collected last on purpose."""
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


def _largest_T(n_shared):
    """Largest Qwen3-shaped token count whose workspace fits the static array."""
    cap = B.pr2_static_scratch_bytes()
    T = 1
    while B.pr2_moe_workspace_bytes(B.dims(T + 1, 2048, 128, 8, 768, n_shared)) <= cap:
        T += 1
    return T


def _static_forward(cfg, L, idx, gates):
    dm = H.dims_of(cfg)
    out = torch.full((cfg.T, cfg.d), float("nan"), dtype=torch.bfloat16, device="cuda")
    counts = torch.full((cfg.N,), -1, dtype=torch.int32, device="cuda")
    perm = torch.full((cfg.T * cfg.k,), -1, dtype=torch.int32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    code = B.pr2_moe_forward_static(dm, L["x"], idx, gates, L["W_gate"], L["W_up"], L["W_down"],
                                    L["Ws_gate"], L["Ws_up"], L["Ws_down"], out, counts=counts,
                                    perm=perm, status=status)
    assert code == 0, B.pr2_strerror(code)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return out, counts, perm


def _check_layer(cfg, seed, calls):
    L = H.to_dev(synth.make_layer(cfg, seed=seed))
    g = H.gpu_predict(cfg, L)
    ref = H.gpu_forward(cfg, L, g["idx"], g["gates"])
    assert ref["code"] == 0 and int(ref["status"].item()) == 0
    torch.cuda.synchronize()
    for _ in range(calls):
        out, counts, perm = _static_forward(cfg, L, g["idx"], g["gates"])
        assert torch.equal(counts, ref["counts"])
        assert torch.equal(perm, ref["perm"])
        assert torch.equal(out, ref["out"]), "static-scratch output differs from the workspace one"


def test_static_scratch_forward_is_bit_identical_after_a_larger_call():
    big_T = _largest_T(1)
    big = synth.LayerConfig("static_big", T=big_T, d=2048, N=128, k=8, m=768, n_shared=1)
    assert B.pr2_moe_workspace_bytes(H.dims_of(big)) <= B.pr2_static_scratch_bytes()
    _check_layer(big, seed=5, calls=1)
    small = synth.LayerConfig("static_small", T=200, d=2048, N=128, k=8, m=768)
    _check_layer(small, seed=3, calls=2)


def test_static_scratch_rejects_a_layer_that_does_not_fit():
    # the Qwen3-shaped 4096-token batch needs far more scratch than the array holds; the call
    # returns PR2_ERR_WORKSPACE before it touches any pointer (these are not device buffers)
    big = B.dims(4096, 2048, 128, 8, 768)
    assert B.pr2_moe_workspace_bytes(big) > B.pr2_static_scratch_bytes()
    fake = ctypes.c_void_p(256)
    lib = B._static_lib()
    assert lib.pr2_moe_forward_static(ctypes.byref(big), fake, fake, fake, fake, fake, fake,
                                      None, None, None, fake, None, None, None, None) == 6
