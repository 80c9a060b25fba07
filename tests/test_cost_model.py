"""The closed-form cost model against the values Table 4 (App. E.2) prints."""
import json
import os

import pytest

from paper_2606_00395_gb300 import cost

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "table4_overheads.json")))


def _printed(x, ref):
    """x rounded the way the table prints ref (same number of decimals)."""
    s = repr(ref)
    dec = len(s.split(".")[1]) if "." in s else 0
    return round(x, dec) == ref


@pytest.mark.parametrize("row", GOLDEN["rows"], ids=[r["model"] for r in GOLDEN["rows"]])
def test_table4_closed_forms(row):
    L, d, N, k, s, m, T, Tc = (row[x] for x in ("L", "d", "N", "k", "s", "m", "T", "T_c"))
    assert _printed(cost.index_cache_bytes(T, L, k) / 1e6, row["index_cache_MB"])
    assert _printed(cost.feature_cache_bytes(Tc, L, d, N) / 1e6, row["feature_cache_MB"])
    assert _printed(cost.predictor_flops_per_token(L, d, N) / 1e6, row["flops_M"])
    assert _printed(100 * cost.ffn_ratio(L, d, N, k, s, m), row["ffn_ratio_pct"])


def test_kernel_work_counts_each_tensor_once():
    w = cost.route_predict_work(4096, 2048, 128, 8)
    assert w.bytes == 4096 * 2048 * 2 + 256 * 2048 * 2 + 4096 * 8 * 8 + 4096 * 128 * 4
    assert w.flops == 2 * 4096 * 2048 * 256
    g = cost.expert_gate_up_work(32768, 2048, 768, 128)
    dn = cost.expert_down_work(32768, 2048, 768, 128)
    assert g.flops + dn.flops == 6 * 4096 * 8 * 2048 * 768
    # gathering A from h: each of the 4096 tokens crosses HBM once instead of k = 8 times
    gg = cost.expert_gate_up_work(32768, 2048, 768, 128, a_rows=4096)
    assert g.bytes - gg.bytes == (32768 - 4096) * 2048 * 2 and gg.flops == g.flops
    mlp = cost.expert_mlp_work(32768, 2048, 768, 128, a_rows=4096)
    assert mlp.bytes == gg.bytes + dn.bytes and mlp.flops == g.flops + dn.flops
    # the fused minimum of the expert stage: h once and the hit experts' weights, no H / Y
    alg = cost.expert_mlp_algorithmic_work(32768, 2048, 768, 128, a_rows=4096)
    assert alg.bytes == 4096 * 2048 * 2 + 128 * 3 * 2048 * 768 * 2 and alg.flops == mlp.flops
    assert mlp.bytes - alg.bytes == 2 * 32768 * 768 * 2 + 32768 * 2048 * 2  # H out+in, Y out
    assert cost.dispatch_work(4096, 2048, 8).bytes == 3 * 4096 * 8 * 4
    assert (cost.dispatch_work(4096, 2048, 8, "fp32", gather=True).bytes
            == 3 * 4096 * 8 * 4 + 4096 * 2048 * 4 + 32768 * 2048 * 4)


def test_tracking_and_loss_work_match_table4_sizes():
    """The feature-cache writer moves each cached byte of Table 4 twice (read and write), one
    layer at a time; the predictive loss does the predictor projection and its transpose."""
    row = next(r for r in GOLDEN["rows"] if r["model"].startswith("Qwen3"))
    Tc, d, N = row["T_c"], row["d"], row["N"]
    fc = cost.feature_cache_work(Tc, d, N)
    assert fc.bytes == 2 * cost.feature_cache_bytes(Tc, 1, d, N) + 4 * Tc
    lw = cost.predictor_loss_work(Tc, d, N)
    assert lw.flops == 2 * Tc * cost.predictor_flops_per_token(1, d, N)
    assert lw.bytes > Tc * 2 * d
    dg = cost.route_diagnostics_work(4096, N, row["k"])
    assert dg.bytes == 4096 * (4 * N + 4 * row["k"])
