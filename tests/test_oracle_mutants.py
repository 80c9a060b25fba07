"""Planted mistakes: each mutant is a copy of the oracle source with one plausible error, built
on the CPU; the pins of ``test_oracle_pins.py`` must reject every one of them.  Nothing here
touches the CUDA library."""
import inspect
import os
import subprocess

import pytest

import oracle
from tests import test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "pr2_oracle.c")

# (name, text in the oracle, replacement, occurrence to change (0-based))
MUTANTS = [
    ("predictor_sign", "z[e] = p[e] + b[e];", "z[e] = p[e] - b[e];", 0),
    ("predictor_dropped", "z[e] = p[e] + b[e];", "z[e] = p[e];", 0),
    ("router_transposed", "widen(W, (int64_t)e * d + i, dtype)", "widen(W, (int64_t)i * N + e, dtype)", 0),
    ("softmax_unnormalised", "rho[e] /= sum;", "(void)sum;", 0),
    ("tie_to_higher_index", "rho[e] > rho[best]", "rho[e] >= rho[best]", 0),
    ("margin_wrong_rank", "top_vals[k - 1] - top_vals[k]", "top_vals[0] - top_vals[k]", 0),
    ("gate_wrong_slot", "gates[t * k + s] = rho[idx[t * k + s]];", "gates[t * k + s] = rho[s];", 0),
    ("replay_no_duplicate_check",
     "for (int s2 = 0; ok && s2 < s; ++s2) if (idx[t * k + s2] == e) ok = 0;\n                gates",
     "gates", 0),
    ("replay_uses_slot_not_index", "gates[t * k + s] = ok ? rho[e] : 0.0;", "gates[t * k + s] = ok ? rho[s] : 0.0;", 0),
    ("permute_unstable", "for (int64_t f = 0; f < F; ++f) {\n        if (!valid[f])",
     "for (int64_t f = F - 1; f >= 0; --f) {\n        if (!valid[f])", 0),
    ("permute_no_invalid_skip", "if (ok) counts[e] += 1; else bad += 1;", "if (e >= 0 && e < N) counts[e] += 1; if (!ok) bad += 1;", 0),
    ("sigmoid_not_silu", "return x / (1.0 + exp(-x));", "return 1.0 / (1.0 + exp(-x));", 0),
    ("down_transposed", "widen(Wd, dn + (int64_t)c * m + j, dtype)", "widen(Wd, dn + (int64_t)j * d + c, dtype)", 0),
    ("gate_up_swapped", "a[j] = silu(g) * u;", "a[j] = silu(u) * g;", 0),
    ("expert_offset", "gu = ex * (int64_t)m * d,", "gu = ex * (int64_t)m,", 0),
    ("shared_dropped", "for (int c = 0; c < d; ++c) o[c] += y[c];", "(void)y;", 0),
    ("forward_gate_slot0", "o[c] += gates[t * k + s] * y[c];", "o[c] += gates[t * k] * y[c];", 0),
    ("bf16_widen_shift", "<< 16;", "<< 15;", 0),
    ("loss_grad_sign", "dz[c * N + j] = pred[j] - tgt[j];", "dz[c * N + j] = tgt[j] - pred[j];", 0),
    ("loss_kl_reversed", "if (tgt[j] > 0.0) acc += tgt[j] * (ltgt[j] - lpred[j]);",
     "if (pred[j] > 0.0) acc += pred[j] * (lpred[j] - ltgt[j]);", 0),
    ("loss_not_averaged", "*loss = (Tc > 0) ? tot / (double)Tc : 0.0;", "*loss = tot;", 0),
    ("loss_grad_transposed", "grad[(int64_t)j * d + i] = ", "grad[(int64_t)i * N + j] = ", 0),
    ("loss_predictor_dropped", "v[j] = (double)po[j] + b[j];", "v[j] = (double)po[j];", 0),
    ("delta_target_sign", "log((double)rho[j]) - (double)po[j]", "log((double)rho[j]) + (double)po[j]", 0),
    ("delta_predicts_with_p_old", "log_softmax(b, N, pred, lpred);", "for (int j = 0; j < N; ++j) v[j] = (double)po[j] + b[j];\n                log_softmax(v, N, pred, lpred);", 0),
    ("loss_pos_ignored", "int64_t r = pos ? (int64_t)pos[c] : c;", "int64_t r = c;", 0),
    ("diag_duplicates_counted", "for (int s2 = 0; ok && s2 < s; ++s2) if (idx_cached[t * k + s2] == e) ok = 0;", "", 0),
    ("diag_hist_by_overlap", "hist[k - ov] += 1;", "hist[ov] += 1;", 0),
    ("diag_keeps_k_plus_one", "for (int s = 0; s < k; ++s) taken[sel[s]] = 1;", "topk(r, N, k, sel, tv, taken);", 0),
    ("cache_positions_rounded_up", "int64_t p = (c * T) / Tc;", "int64_t p = (c * T + Tc - 1) / Tc;", 0),
]


def _pin_calls():
    calls = []
    for name, fn in inspect.getmembers(pins, inspect.isfunction):
        if not name.startswith("test_"):
            continue
        marks = getattr(fn, "pytestmark", [])
        params = [m for m in marks if m.name == "parametrize"]
        if not params:
            calls.append((name, fn, {}))
            continue
        argnames, values = params[0].args
        argnames = [a.strip() for a in argnames.split(",")]
        for v in values:
            v = v if isinstance(v, tuple) else (v,)
            calls.append((f"{name}{v}", fn, dict(zip(argnames, v))))
    return calls


def _replace_nth(text, old, new, n):
    pos = -1
    for _ in range(n + 1):
        pos = text.find(old, pos + 1)
        assert pos >= 0, f"mutation anchor not found: {old!r}"
    return text[:pos] + new + text[pos + len(old):]


@pytest.mark.parametrize("name,old,new,nth", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_reject_planted_mistake(name, old, new, nth, tmp_path, monkeypatch):
    src = _replace_nth(open(SRC).read(), old, new, nth)
    cpath = tmp_path / f"{name}.c"
    cpath.write_text(src)
    so = tmp_path / f"lib{name}.so"
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-o", str(so), str(cpath), "-lm"],
                   check=True, capture_output=True)
    monkeypatch.setattr(oracle, "_lib", oracle.bind(str(so)))
    caught = []
    for cname, fn, kw in _pin_calls():
        try:
            fn(**kw)
        except (AssertionError, ValueError, IndexError):
            caught.append(cname)
    assert caught, f"no pin rejects the mutant {name}"
