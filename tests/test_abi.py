"""The C-ABI library on the CPU: it builds, loads, exports every symbol include/pr2.h declares,
and rejects invalid arguments on the host before any CUDA call (no GPU needed)."""
import ctypes

import pytest

from paper_2606_00395_gb300 import binding as B
from paper_2606_00395_gb300 import build


@pytest.fixture(scope="module")
def lib():
    build.build()
    return B.load()


def test_exports_every_declared_symbol(lib):
    names = B.declared_symbols()
    assert {"pr2_route_predict", "pr2_route_replay", "pr2_moe_forward", "pr2_moe_workspace_bytes",
            "pr2_strerror"} <= set(names)
    for n in names:
        assert hasattr(lib, n), n


def test_strerror_names_every_code(lib):
    for code in range(7):
        assert B.pr2_strerror(code) and B.pr2_strerror(code) != "unknown status"
    assert B.pr2_strerror(99) == "unknown status"


def test_workspace_bytes_grow_with_the_layer(lib):
    small = B.pr2_moe_workspace_bytes(B.dims(256, 2048, 128, 8, 768))
    big = B.pr2_moe_workspace_bytes(B.dims(4096, 2048, 128, 8, 768))
    shared = B.pr2_moe_workspace_bytes(B.dims(4096, 2048, 128, 8, 768, n_shared=1))
    assert 0 < small < big < shared
    # bf16: dominated by the expert hidden activations and the expert outputs (the gate/up GEMM
    # gathers its rows from h, so there is no permuted copy); fp32 adds the permuted rows
    F = 4096 * 8
    assert 2 * F * (768 + 2048) <= big < 2 * F * (768 + 2048) + 2 * F * 2048
    big32 = B.pr2_moe_workspace_bytes(B.dims(4096, 2048, 128, 8, 768, dtype="fp32"))
    assert big32 >= 4 * F * (2048 + 768 + 2048)


@pytest.mark.parametrize("bad", [
    dict(T=-1), dict(d=0), dict(N=0), dict(k=0), dict(k=129), dict(m=0), dict(n_shared=-1),
])
def test_invalid_dims_are_rejected(lib, bad):
    kw = dict(T=64, d=2048, N=128, k=8, m=768)
    kw.update(bad)
    dm = B.dims(**kw)
    assert B.pr2_moe_workspace_bytes(dm) == 0
    fake = ctypes.c_void_p(256)
    code = lib.pr2_route_predict(ctypes.byref(dm), fake, fake, fake, fake, fake, None, None, None,
                                 None)
    assert code == 1


@pytest.mark.parametrize("kw", [
    dict(d=2000),          # bf16 needs d % 64 == 0
    dict(m=700),           # bf16 needs m % 64 == 0
    dict(N=100, k=8),      # bf16 needs N % 16 == 0
    dict(k=9),             # bf16 routing keeps at most 8 slots
    dict(N=512, k=8),      # at most 256 routed experts
])
def test_unsupported_shapes_are_rejected(lib, kw):
    base = dict(T=64, d=2048, N=128, k=8, m=768)
    base.update(kw)
    dm = B.dims(**base)
    fake = ctypes.c_void_p(256)
    assert lib.pr2_route_predict(ctypes.byref(dm), fake, fake, fake, fake, fake, None, None, None,
                                 None) == 2


def test_null_pointers_and_short_workspace_are_rejected(lib):
    dm = B.dims(64, 2048, 128, 8, 768)
    fake = ctypes.c_void_p(256)
    P = [fake] * 6
    assert lib.pr2_route_predict(ctypes.byref(dm), None, *P[:4], None, None, None, None) == 1
    assert lib.pr2_route_replay(ctypes.byref(dm), fake, fake, None, fake, None, None, None) == 1
    # misaligned device pointer
    odd = ctypes.c_void_p(258)
    assert lib.pr2_route_predict(ctypes.byref(dm), odd, *P[:4], None, None, None, None) == 1
    ws = B.pr2_moe_workspace_bytes(dm)
    args = [ctypes.byref(dm), fake, fake, fake, fake, fake, fake, None, None, None, fake, None,
            None]
    assert lib.pr2_moe_forward(*args, fake, ctypes.c_size_t(ws - 1), None, None, None) == 6
    assert lib.pr2_moe_forward(*args, None, ctypes.c_size_t(ws), None, None, None) == 6
    assert lib.pr2_moe_forward(*args, ctypes.c_void_p(512 + 16), ctypes.c_size_t(ws), None,
                               None, None) == 6
    # shared-expert weights must be given iff n_shared > 0
    dm1 = B.dims(64, 2048, 128, 8, 768, n_shared=1)
    args1 = [ctypes.byref(dm1), fake, fake, fake, fake, fake, fake, None, None, None, fake, None,
             None]
    assert lib.pr2_moe_forward(*args1, fake, ctypes.c_size_t(1 << 40), None, None, None) == 1
    # sync-status needs a status word
    dms = B.dims(64, 2048, 128, 8, 768, flags=B.PR2_F_SYNC_STATUS)
    assert lib.pr2_route_predict(ctypes.byref(dms), *P[:5], None, None, None, None) == 1


def test_empty_layer_is_a_no_op(lib):
    dm = B.dims(0, 2048, 128, 8, 768)
    assert lib.pr2_route_predict(ctypes.byref(dm), None, None, None, None, None, None, None,
                                 None, None) == 0
    ws = B.pr2_moe_workspace_bytes(dm)
    assert ws > 0
    assert lib.pr2_moe_forward(ctypes.byref(dm), *([None] * 12), None, ctypes.c_size_t(0), None,
                               None, None) == 0


def test_selftest_rejects_out_of_range_limits(lib):
    assert lib.pr2_selftest_wait_timeout(None, 1000, None) == 1
    assert lib.pr2_selftest_wait_timeout(ctypes.c_void_p(256), 10, None) == 1
    assert lib.pr2_selftest_wait_timeout(ctypes.c_void_p(256), 10 ** 10, None) == 1


def test_predictor_loss_rejects_bad_arguments_on_the_host(lib):
    dm = B.dims(256, 2048, 128, 8, 768)
    fake = ctypes.c_void_p(256)
    ws = B.pr2_predictor_loss_workspace_bytes(dm)
    assert ws > 0
    # bf16 workspace holds dKL/dz transposed (N x T_c) and the split-K gradient partials
    assert ws >= 128 * 256 * 2 + 8 * 128 * 2048 * 4
    ok = [ctypes.byref(dm), fake, fake, fake, fake, ctypes.c_int64(256), None, fake, None, fake]
    # missing output / input pointers
    bad_loss = list(ok)
    bad_loss[7] = None
    assert lib.pr2_predictor_loss(*bad_loss, fake, ctypes.c_size_t(ws), None, None) == 1
    bad_h = list(ok)
    bad_h[1] = None
    assert lib.pr2_predictor_loss(*bad_h, fake, ctypes.c_size_t(ws), None, None) == 1
    no_teacher = list(ok)
    no_teacher[5] = ctypes.c_int64(0)
    assert lib.pr2_predictor_loss(*no_teacher, fake, ctypes.c_size_t(ws), None, None) == 1
    odd = list(ok)
    odd[2] = ctypes.c_void_p(260)
    assert lib.pr2_predictor_loss(*odd, fake, ctypes.c_size_t(ws), None, None) == 1
    # workspace too small, missing or misaligned
    assert lib.pr2_predictor_loss(*ok, fake, ctypes.c_size_t(ws - 1), None, None) == 6
    assert lib.pr2_predictor_loss(*ok, None, ctypes.c_size_t(ws), None, None) == 6
    assert lib.pr2_predictor_loss(*ok, ctypes.c_void_p(512 + 16), ctypes.c_size_t(ws), None,
                                  None) == 6
    # unsupported layer shape
    dmu = B.dims(256, 2000, 128, 8, 768)
    assert lib.pr2_predictor_loss(ctypes.byref(dmu), *ok[1:], fake, ctypes.c_size_t(ws), None,
                                  None) == 2
    # sync-status needs a status word
    dms = B.dims(256, 2048, 128, 8, 768, flags=B.PR2_F_SYNC_STATUS | B.PR2_F_DELTA_LOSS)
    assert lib.pr2_predictor_loss(ctypes.byref(dms), *ok[1:], fake, ctypes.c_size_t(1 << 40),
                                  None, None) == 1


def test_diagnostics_and_feature_cache_reject_bad_arguments(lib):
    fake = ctypes.c_void_p(256)
    dm = B.dims(64, 2048, 128, 8, 768)
    assert lib.pr2_route_diagnostics(ctypes.byref(dm), fake, fake, None, fake, None) == 1
    assert lib.pr2_route_diagnostics(ctypes.byref(dm), None, fake, fake, fake, None) == 1
    assert lib.pr2_route_diagnostics(ctypes.byref(dm), ctypes.c_void_p(260), fake, fake, fake,
                                     None) == 1
    dm0 = B.dims(0, 2048, 128, 8, 768)
    assert lib.pr2_route_diagnostics(ctypes.byref(dm0), None, None, fake, fake, None) == 0
    # feature cache: T_c outside [0, T], missing buffers, half-given logits pair
    assert lib.pr2_feature_cache_write(ctypes.byref(dm), 65, fake, fake, fake, fake, fake,
                                       None) == 1
    assert lib.pr2_feature_cache_write(ctypes.byref(dm), -1, fake, fake, fake, fake, fake,
                                       None) == 1
    assert lib.pr2_feature_cache_write(ctypes.byref(dm), 8, fake, fake, None, fake, fake,
                                       None) == 1
    assert lib.pr2_feature_cache_write(ctypes.byref(dm), 8, fake, fake, fake, fake, None,
                                       None) == 1
    assert lib.pr2_feature_cache_write(ctypes.byref(dm), 0, None, None, None, None, None,
                                       None) == 0


def test_rollout_layers_rejects_bad_arguments(lib):
    fake = ctypes.c_void_p(256)
    dm = B.dims(64, 2048, 128, 8, 768)
    ws = B.pr2_moe_workspace_bytes(dm)
    # dims, L, h, W_router, W_pred, W_gate, W_up, W_down, Ws_* (3), idx, gates, logits, near_tie
    base = [ctypes.byref(dm), ctypes.c_int32(2), fake, fake, fake, fake, fake, fake, None, None,
            None, fake, fake, None, None]
    bad_L = list(base)
    bad_L[1] = ctypes.c_int32(0)
    assert lib.pr2_rollout_layers(*bad_L, fake, ctypes.c_size_t(ws), None, None) == 1
    no_idx = list(base)
    no_idx[11] = None
    assert lib.pr2_rollout_layers(*no_idx, fake, ctypes.c_size_t(ws), None, None) == 1
    no_h = list(base)
    no_h[2] = None
    assert lib.pr2_rollout_layers(*no_h, fake, ctypes.c_size_t(ws), None, None) == 1
    dms = B.dims(64, 2048, 128, 8, 768, flags=B.PR2_F_SYNC_STATUS)
    sync = list(base)
    sync[0] = ctypes.byref(dms)
    assert lib.pr2_rollout_layers(*sync, fake, ctypes.c_size_t(ws), None, None) == 1


def test_one_call_layers_reject_bad_arguments_on_the_host(lib):
    """pr2_moe_rollout_forward / pr2_moe_replay_forward check everything both of their steps
    need before launching anything (these are not device buffers: nothing may be touched)."""
    fake, odd = ctypes.c_void_p(256), ctypes.c_void_p(258)
    dm = B.dims(64, 2048, 128, 8, 768)
    ws = ctypes.c_size_t(B.pr2_moe_workspace_bytes(dm))
    tail = [None, None, fake, ws, None, None, None]  # counts, perm, workspace, ws_bytes, status, events, stream
    # rollout: dims, h, W_router, W_pred, idx, gates, logits_old, near_tie, W_gate, W_up, W_down,
    # Ws_gate, Ws_up, Ws_down, out, ...
    roll = [ctypes.byref(dm), fake, fake, fake, fake, fake, None, None, fake, fake, fake, None,
            None, None, fake]

    def rollout(**edit):
        a = list(roll)
        t = list(tail)
        for i, v in edit.get("a", {}).items():
            a[i] = v
        for i, v in edit.get("t", {}).items():
            t[i] = v
        return lib.pr2_moe_rollout_forward(*a, *t)
    assert rollout(a={2: None}) == 1             # no router
    assert rollout(a={3: None}) == 1             # no predictor
    assert rollout(a={3: odd}) == 1              # misaligned predictor
    assert rollout(a={6: odd}) == 1              # misaligned logits_old
    assert rollout(a={1: None}) == 1             # no h (checked for the forward step)
    assert rollout(a={11: fake}) == 1            # shared weights without shared experts
    assert rollout(t={3: ctypes.c_size_t(ws.value - 1)}) == 6  # short workspace
    dms = B.dims(64, 2048, 128, 8, 768, flags=B.PR2_F_SYNC_STATUS)
    assert rollout(a={0: ctypes.byref(dms)}) == 1  # sync-status needs a status word
    # replay: dims, h, W_router, idx, gates, probs, W_gate, W_up, W_down, Ws_gate, Ws_up,
    # Ws_down, out, ...
    rep = [ctypes.byref(dm), fake, fake, fake, fake, None, fake, fake, fake, None, None, None,
           fake]

    def replay(**edit):
        a = list(rep)
        t = list(tail)
        for i, v in edit.get("a", {}).items():
            a[i] = v
        for i, v in edit.get("t", {}).items():
            t[i] = v
        return lib.pr2_moe_replay_forward(*a, *t)
    assert replay(a={2: None}) == 1              # no router
    assert replay(a={2: odd}) == 1               # misaligned router
    assert replay(a={4: None}) == 1              # no gates to write
    assert replay(a={5: odd}) == 1               # misaligned probs
    assert replay(a={3: None}) == 1              # no route
    assert replay(t={2: None}) == 6              # no workspace
    # an empty layer is a no-op for both, whatever the pointers
    d0 = B.dims(0, 2048, 128, 8, 768)
    assert lib.pr2_moe_rollout_forward(ctypes.byref(d0), *([None] * 17), ctypes.c_size_t(0),
                                       None, None, None) == 0
    assert lib.pr2_moe_replay_forward(ctypes.byref(d0), *([None] * 15), ctypes.c_size_t(0),
                                      None, None, None) == 0


def test_unknown_flags_are_rejected(lib):
    ok = B.dims(64, 2048, 128, 8, 768, flags=B.PR2_F_NORMALIZE_TOPK | B.PR2_F_SYNC_STATUS)
    assert B.pr2_moe_workspace_bytes(ok) > 0
    bad = B.dims(64, 2048, 128, 8, 768, flags=0x100)
    assert B.pr2_moe_workspace_bytes(bad) == 0
    fake = ctypes.c_void_p(256)
    code = lib.pr2_route_predict(ctypes.byref(bad), fake, fake, fake, fake, fake, None, None, None,
                                 None)
    assert code == 1  # PR2_ERR_INVALID_ARG, before any launch


def test_static_scratch_holds_up_to_743_tokens_of_the_qwen3_layer(lib):
    """pr2_moe_forward_static's fixed scratch: the Qwen3-shaped layer fits up to 743 tokens (the
    limit pr2.h states); one more token is rejected with PR2_ERR_WORKSPACE before any launch."""
    scratch = B.pr2_static_scratch_bytes()
    assert B.pr2_moe_workspace_bytes(B.dims(743, 2048, 128, 8, 768)) <= scratch
    over = B.dims(744, 2048, 128, 8, 768)
    assert B.pr2_moe_workspace_bytes(over) > scratch
    fake = ctypes.c_void_p(256)
    slib = B._static_lib()
    assert slib.pr2_moe_forward_static(ctypes.byref(over), fake, fake, fake, fake, fake, fake,
                                       None, None, None, fake, None, None, None, None) == 6
