#!/usr/bin/env python
"""Throughput of the Pr^2 MoE layer forward (rollout predict-route + training replay) on GB300.

One step = the whole hot path over one batch of T tokens in both modes:
  rollout:  pr2_route_predict (router + predictor GEMM, softmax, top-k, route record)
            -> pr2_moe_forward (dispatch, grouped gate/up + SwiGLU GEMM, down GEMM, combine)
  replay:   pr2_route_replay on the recorded route with the drifted current router
            -> pr2_moe_forward with the replay gates.
value = tokens/s = T * ranks / (max over ranks of the summed per-step device time).
L2 is flushed (512 MiB write) before every step; the flush is outside the timed intervals.

--impl reference times the CPU oracle (the reference of this build) on a bounded token sample of
the same workload, on the host cores, and prints the same JSON line with "impl": "reference".
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import tempfile
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2606_00395_gb300 import binding as B  # noqa: E402
from paper_2606_00395_gb300 import cost, replicas, synth  # noqa: E402

METRIC = "MoE-layer tokens/s (predict-route & replay fwd) on 1 GB300; % of roofline"
FLUSH_BYTES = 512 << 20


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["pr2", "reference"], default="pr2")
    ap.add_argument("--workload", default="qwen3_30b_a3b", choices=sorted(synth.CONFIGS))
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="target CPU time of the oracle baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--extras-iters", type=int, default=50,
                    help="timed calls of each widening row (after 3 untimed)")
    ap.add_argument("--no-deepseek", action="store_true",
                    help="skip the DeepSeek-V3-shaped layer among the extras")
    return ap.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        p = json.load(open(path))
        return dict(hbm=float(p["hbm_gbs"]), bf16=float(p["bf16_tflops"]),
                    bf16_sustained=float(p.get("bf16_tflops_sustained", p["bf16_tflops"])),
                    source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sustained=1700.0, source="fallback")


def measured_traffic(kernel_key: str):
    """DRAM bytes per launch of a kernel from the committed ncu summary, or None when any source
    file the capture was taken with has changed since (the counters no longer apply)."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    entry = json.load(open(path)).get(kernel_key)
    if not entry:
        return None
    for rel, digest in entry["sources_sha256"].items():
        f = os.path.join(ROOT, rel)
        if not os.path.exists(f) or hashlib.sha256(open(f, "rb").read()).hexdigest() != digest:
            return None
    return entry["dram_bytes_per_launch"]


def workload_desc(cfg):
    return dict(workload=cfg.name, T=cfg.T, d=cfg.d, N=cfg.N, k=cfg.k, m=cfg.m,
                n_shared=cfg.n_shared, modes="rollout+replay", tokens_per_step=cfg.T,
                weights="N(0,0.02) seed 0, replay router drift N(0,0.002) seed 1",
                l2="flushed before every step (512 MiB write), flush not timed",
                parallelism="replicas")


# ----------------------------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.proc = None
        # raw samples: a scratch file (PR2_CLOCKS_DIR to keep them elsewhere); the JSON line
        # carries the summary
        self.path = os.path.join(os.environ.get("PR2_CLOCKS_DIR", tempfile.gettempdir()),
                                 f"pr2_clocks_rank{index}_{os.getpid()}.csv")
        uuid = str(getattr(torch.cuda.get_device_properties(index), "uuid", index))
        sel = uuid if uuid.startswith("GPU-") else (f"GPU-{uuid}" if "-" in uuid else str(index))
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", sel, f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.fh,
                stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.fh.close()
        rows = []
        with open(self.path) as fh:
            lines = fh.readlines()
        if "PR2_CLOCKS_DIR" not in os.environ:
            os.remove(self.path)
        for line in lines:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 7:
                continue
            try:
                rows.append((float(parts[0]), float(parts[1]), parts[3:7]))
            except ValueError:
                continue
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, fl in rows for i, v in enumerate(fl)
                          if v.lower() == "active"})
        return dict(sm_mhz=statistics.median(r[0] for r in rows), sm_max_mhz=max(r[1] for r in rows),
                    reasons=reasons, samples=len(rows))


# ----------------------------------------------------------------------------------- oracle

def oracle_layer_seconds(cfg, Lh, W2h, toks):
    """Run the CPU oracle over `toks` in both modes (rollout + replay); return seconds."""
    import oracle
    x = Lh["x"][torch.from_numpy(toks)]
    t0 = time.perf_counter()
    r = oracle.route_predict(x, Lh["W_router"], Lh["W_pred"], cfg.k)
    oracle.moe_forward(x, r["idx"], r["gates"], Lh["W_gate"], Lh["W_up"], Lh["W_down"],
                       Lh["Ws_gate"], Lh["Ws_up"], Lh["Ws_down"])
    rep = oracle.route_replay(x, W2h, r["idx"])
    oracle.moe_forward(x, r["idx"], rep["gates"], Lh["W_gate"], Lh["W_up"], Lh["W_down"],
                       Lh["Ws_gate"], Lh["Ws_up"], Lh["Ws_down"])
    return time.perf_counter() - t0


def cpu_baseline(cfg, Lh, W2h, target_s):
    """Time the oracle on a growing token sample until ~target_s seconds of CPU work."""
    import oracle
    n, spent, toks_done = 8, 0.0, 0
    while True:
        toks = synth.make_token_sample(cfg.T, n, 7 + n).numpy()
        dt = oracle_layer_seconds(cfg, Lh, W2h, toks)
        spent, toks_done = dt, len(toks)
        if dt * 2 > target_s or n >= cfg.T:
            break
        n = min(cfg.T, n * 2)
    return dict(value=toks_done / spent, unit="tokens/s", cores=oracle.num_threads(),
                kind="oracle",
                sample=f"{toks_done} seeded tokens of {cfg.name} through both modes "
                       f"(route predict + layer, route replay + layer), fp64, {spent:.1f} s")


def host_layer(cfg, L):
    return {k: (v.cpu() if v is not None else None) for k, v in L.items()}


# ----------------------------------------------------------------------------------- pr2 arm

def kernel_roofline(w, ms, pk, tc_peak):
    """Roofline of one kernel from its algorithmic work `w` and mean duration `ms`: the bound
    that allows the longer time (tensor at `tc_peak` or HBM), and measured time over it."""
    t_hbm = w.bytes / (pk["hbm"] * 1e9) * 1e3
    t_tc = w.flops / (tc_peak * 1e12) * 1e3
    if t_tc > t_hbm:
        return dict(ms=ms, bound="tensor", achieved=w.flops / (ms * 1e-3) / 1e12, peak=tc_peak,
                    unit="TFLOP/s", frac=t_tc / ms, algorithmic_flops=w.flops,
                    algorithmic_bytes=w.bytes)
    return dict(ms=ms, bound="hbm", achieved=w.bytes / (ms * 1e-3) / 1e9, peak=pk["hbm"],
                unit="GB/s", frac=t_hbm / ms, algorithmic_flops=w.flops,
                algorithmic_bytes=w.bytes)


def measure_extras(cfg, L, W2, dm, flush, pk, iters=50):
    """The rows that widen the hot path, each timed alone on the device (CUDA events around the
    call, L2 flushed before every call, median of ``iters``) against its own roofline:
    the fixed-length feature-cache writer (Algorithm 2) for T_c = min(2048, T) rows (Table 4's
    Qwen3 cache length), the predictive loss with its W_p gradient over that cache (Eq.
    pr2_loss, Algorithm 3), the route-tracking diagnostics of the rollout route against the
    drifted current router (Sec. 5), the multi-layer decode loop, the latency of one decode
    batch (routing alone, and the whole layer) and the Pr^3 step."""
    dev = "cuda"
    Tc = min(2048, cfg.T)
    idx, gates, logits = B.alloc_route(dm, logits=True)
    B.check(B.pr2_route_predict(dm, L["x"], L["W_router"], L["W_pred"], idx, gates, logits),
            "pr2_route_predict")
    rho = torch.empty(cfg.T, cfg.N, dtype=torch.float32, device=dev)
    rg = torch.empty_like(gates)
    B.check(B.pr2_route_replay(dm, L["x"], W2, idx, rg, rho), "pr2_route_replay")
    pos = torch.empty(Tc, dtype=torch.int32, device=dev)
    ch = torch.empty(Tc, cfg.d, dtype=cfg.torch_dtype, device=dev)
    cp = torch.empty(Tc, cfg.N, dtype=torch.float32, device=dev)
    dml = B.dims(Tc, cfg.d, cfg.N, cfg.k, cfg.m, 0, cfg.dtype)
    ws = B.alloc_loss_workspace(dml)
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    kl = torch.empty(Tc, dtype=torch.float32, device=dev)
    grad = torch.empty(cfg.N, cfg.d, dtype=torch.float32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    hist = torch.zeros(cfg.k + 1, dtype=torch.int64, device=dev)
    ov = torch.zeros(1, dtype=torch.int64, device=dev)

    def timed(fn, pre=None):
        evs = []
        for i in range(iters + 3):
            flush.fill_(i & 0xFF)
            if pre is not None:
                pre()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            evs.append((a, b))
        torch.cuda.synchronize()
        return statistics.median(a.elapsed_time(b) for a, b in evs[3:])

    out = {}

    def report(name, ms, w, **extra):
        t_hbm = w.bytes / (pk["hbm"] * 1e9) * 1e3
        t_tc = w.flops / (pk["bf16"] * 1e12) * 1e3
        bound = "tensor" if t_tc > t_hbm else "hbm"
        achieved = (w.flops / (ms * 1e-3) / 1e12) if bound == "tensor" else (
            w.bytes / (ms * 1e-3) / 1e9)
        out[name] = dict(ms=ms, bound=bound, achieved=achieved,
                         peak=pk["bf16"] if bound == "tensor" else pk["hbm"],
                         unit="TFLOP/s" if bound == "tensor" else "GB/s",
                         frac=max(t_hbm, t_tc) / ms, algorithmic_bytes=w.bytes,
                         algorithmic_flops=w.flops, **extra)

    ms = timed(lambda: B.check(B.pr2_feature_cache_write(dm, Tc, L["x"], logits, pos, ch, cp),
                               "pr2_feature_cache_write"))
    report("feature_cache_write", ms, cost.feature_cache_work(Tc, cfg.d, cfg.N, cfg.dtype), Tc=Tc)
    ms = timed(lambda: B.check(B.pr2_predictor_loss(dml, ch, cp, L["W_pred"], rho, loss, grad,
                                                    pos=pos, kl_tok=kl, workspace=ws,
                                                    status=status), "pr2_predictor_loss"))
    report("predictor_loss", ms, cost.predictor_loss_work(Tc, cfg.d, cfg.N, cfg.dtype), Tc=Tc,
           loss=float(loss.item()))

    def zero():
        hist.zero_()
        ov.zero_()
    ms = timed(lambda: B.check(B.pr2_route_diagnostics(dm, rho, idx, hist, ov),
                               "pr2_route_diagnostics"), pre=zero)
    report("route_diagnostics", ms, cost.route_diagnostics_work(cfg.T, cfg.N, cfg.k),
           topk_agreement=int(ov.item()) / (cfg.T * cfg.k),
           deviation_hist=[int(x) for x in hist.tolist()])

    # Multi-layer rollout decode (Algorithm 2 over L layers): a 256-token decode batch through
    # L = 4 layers of this shape (the layer's weights repeated per layer, each layer streaming
    # its own 1.2 GB copy), one pr2_rollout_layers call, eager and replayed from a CUDA graph.
    Ld, Td = 4, min(256, cfg.T)
    ddm = B.dims(Td, cfg.d, cfg.N, cfg.k, cfg.m, cfg.n_shared, cfg.dtype)
    keys = ["W_router", "W_pred", "W_gate", "W_up", "W_down"]
    keys += ["Ws_gate", "Ws_up", "Ws_down"] if cfg.n_shared else []
    Ws = {k: torch.stack([L[k]] * Ld).contiguous() for k in keys}
    h0 = L["x"][:Td].clone()
    hd = h0.clone()
    didx = torch.empty(Ld, Td, cfg.k, dtype=torch.int32, device=dev)
    dgates = torch.empty(Ld, Td, cfg.k, dtype=torch.float32, device=dev)
    dlog = torch.empty(Ld, Td, cfg.N, dtype=torch.float32, device=dev)
    dws = B.alloc_workspace(ddm)

    def loop(stream=None):
        return B.pr2_rollout_layers(ddm, Ld, hd, Ws["W_router"], Ws["W_pred"], Ws["W_gate"],
                                    Ws["W_up"], Ws["W_down"], didx, dgates,
                                    Ws_gate=Ws.get("Ws_gate"), Ws_up=Ws.get("Ws_up"),
                                    Ws_down=Ws.get("Ws_down"), logits_old=dlog,
                                    workspace=dws, status=status, stream=stream)

    eager_ms = timed(lambda: B.check(loop(), "pr2_rollout_layers"), pre=lambda: hd.copy_(h0))
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=side):
        B.check(loop(side), "pr2_rollout_layers (capture)")
    graph_ms = timed(graph.replay, pre=lambda: hd.copy_(h0))
    per_layer = [cost.route_predict_work(Td, cfg.d, cfg.N, cfg.k, cfg.dtype, True),
                 cost.dispatch_work(Td, cfg.d, cfg.k, cfg.dtype, gather=cfg.dtype == "fp32"),
                 cost.expert_mlp_algorithmic_work(Td * cfg.k, cfg.d, cfg.m, cfg.N, cfg.dtype,
                                                  a_rows=0),  # h counted by routing
                 cost.combine_work(Td, cfg.d, cfg.k, cfg.n_shared, cfg.dtype)]
    work = cost.KernelWork(Ld * sum(w.bytes for w in per_layer),
                           Ld * sum(w.flops for w in per_layer))
    report("decode_loop_graph", graph_ms, work, layers=Ld, T=Td, eager_ms=eager_ms,
           tokens_per_s=Td / (graph_ms * 1e-3))
    del Ws, graph

    # The rollout decode batch on its own (T = 256 tokens, one per sequence; rollout mode):
    # latency of the routing call and of the whole layer (routing + forward), each timed alone
    # from a flushed L2.
    xd = L["x"][:Td].contiguous()
    di, dgt, dlg = B.alloc_route(ddm, logits=True)
    do = torch.empty(Td, cfg.d, dtype=cfg.torch_dtype, device=dev)

    def route_d():
        B.check(B.pr2_route_predict(ddm, xd, L["W_router"], L["W_pred"], di, dgt, dlg),
                "pr2_route_predict")

    def layer_d():
        B.check(B.pr2_moe_rollout_forward(ddm, xd, L["W_router"], L["W_pred"], di, dgt, dlg,
                                          None, L["W_gate"], L["W_up"], L["W_down"],
                                          L["Ws_gate"], L["Ws_up"], L["Ws_down"], do,
                                          workspace=dws, status=status),
                "pr2_moe_rollout_forward")
    ms = timed(route_d)
    report("decode_route_predict", ms, per_layer[0], T=Td, latency_us=ms * 1e3)
    ms = timed(layer_d)
    report("decode_layer", ms, cost.KernelWork(sum(w.bytes for w in per_layer),
                                              sum(w.flops for w in per_layer)),
           T=Td, latency_us=ms * 1e3, tokens_per_s=Td / (ms * 1e-3))

    # Pr^3 step (App. "Predictive Rollout Routing Replay"): rollout with the predicted route,
    # the log-prob pass replaying it with the snapshot router, the gradient pass replaying it
    # with the current (drifted) router; T tokens, step-boundary events only.
    o1 = torch.empty(cfg.T, cfg.d, dtype=cfg.torch_dtype, device=dev)
    wsl = B.alloc_workspace(dm)

    def pr3():
        sh = (L["Ws_gate"], L["Ws_up"], L["Ws_down"])
        B.check(B.pr2_moe_rollout_forward(dm, L["x"], L["W_router"], L["W_pred"], idx, gates,
                                          logits, None, L["W_gate"], L["W_up"], L["W_down"],
                                          *sh, o1, workspace=wsl), "pr2_moe_rollout_forward")
        for Wr in (L["W_router"], W2):
            B.check(B.pr2_moe_replay_forward(dm, L["x"], Wr, idx, rg, None, L["W_gate"],
                                             L["W_up"], L["W_down"], *sh, o1, workspace=wsl),
                    "pr2_moe_replay_forward")
    ms = timed(pr3)
    out["pr3_step"] = dict(ms=ms, tokens_per_s=cfg.T / (ms * 1e-3), passes=3, T=cfg.T)
    del wsl

    # Training replay over long sequences (8 x 4096 = 32768 tokens) with recorded routes drawn
    # Zipf(1.2) over the experts (per-expert rows 279 ... 31034): the same layer weights, new
    # token rows; the routing call and the layer forward each timed alone.  At this size the
    # routing kernel is no longer launch-bound and the expert GEMMs are compute-bound.
    lcfg = synth.CONFIGS["qwen3_long_replay"]
    if (cfg.d, cfg.N, cfg.k, cfg.m, cfg.dtype) == (lcfg.d, lcfg.N, lcfg.k, lcfg.m, lcfg.dtype):
        Tl = lcfg.T
        ldm = B.dims(Tl, cfg.d, cfg.N, cfg.k, cfg.m, cfg.n_shared, cfg.dtype)
        gen = torch.Generator(device=dev)
        gen.manual_seed(7)
        xl = torch.randn(Tl, cfg.d, generator=gen, device=dev).to(cfg.torch_dtype)
        il = synth.make_zipf_routes(Tl, cfg.N, cfg.k, lcfg.zipf_s).to(dev)
        gl = torch.empty(Tl, cfg.k, dtype=torch.float32, device=dev)
        ol = torch.empty(Tl, cfg.d, dtype=cfg.torch_dtype, device=dev)
        wl = B.alloc_workspace(ldm)

        def route_l():
            B.check(B.pr2_route_replay(ldm, xl, W2, il, gl, None, status), "pr2_route_replay")

        def forward_l(evs=None):
            B.check(B.pr2_moe_forward(ldm, xl, il, gl, L["W_gate"], L["W_up"], L["W_down"],
                                      L["Ws_gate"], L["Ws_up"], L["Ws_down"], ol, workspace=wl,
                                      status=status, events=evs), "pr2_moe_forward")
        route_l()
        ms_r = timed(route_l)
        report("long_replay_route", ms_r,
               cost.route_replay_work(Tl, cfg.d, cfg.N, cfg.k, cfg.dtype, False), T=Tl)
        # the forward with an event at every stage boundary: the grouped GEMM launch alone too
        sets = []
        for i in range(iters + 3):
            flush.fill_(i & 0xFF)
            e = [torch.cuda.Event(enable_timing=True) for _ in range(5)]
            for x in e:
                x.record()
            forward_l(B.stage_events(e))
            sets.append(e)
        torch.cuda.synchronize()
        ms_f = statistics.median(e[0].elapsed_time(e[4]) for e in sets[3:])
        ms_g = statistics.median(e[1].elapsed_time(e[3]) for e in sets[3:])
        Fl = Tl * cfg.k
        gw = cost.expert_mlp_algorithmic_work(Fl, cfg.d, cfg.m, cfg.N, cfg.dtype, a_rows=Tl)
        fw = [cost.dispatch_work(Tl, cfg.d, cfg.k, cfg.dtype, gather=False), gw,
              cost.combine_work(Tl, cfg.d, cfg.k, cfg.n_shared, cfg.dtype)]
        report("long_replay_expert_gemm", ms_g, gw, T=Tl,
               tensor_frac_sustained=gw.flops / (ms_g * 1e-3) / 1e12 / pk["bf16_sustained"],
               routes="Zipf(1.2) over experts, seed 2; token rows N(0,1), seed 7")
        report("long_replay_forward", ms_f, cost.KernelWork(sum(w.bytes for w in fw),
                                                           sum(w.flops for w in fw)),
               T=Tl, tokens_per_s=Tl / ((ms_r + ms_f) * 1e-3))
        del wl, xl, ol
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())} in the extra rows")
    return out


def measure_layer_modes(cfg, flush, pk, iters, seed=0):
    """Both modes of one MoE layer workload timed on the device (the bench step's calls, CUDA
    events at the mode boundaries, L2 flushed before every step, median of ``iters`` after 3
    untimed), then a pass with an event at every stage boundary for the per-kernel split, each
    kernel against its roofline: routing against the tensor bound where its 4TdN FLOPs outlast
    its bytes (the DeepSeek-V3 shape), the routed + shared expert GEMMs against the larger of
    the tensor time and the weight stream."""
    dev = "cuda"
    L = synth.make_layer(cfg, seed=seed, device=dev)
    W2 = synth.make_drifted_router(L["W_router"], seed=seed)
    dm = B.dims(cfg.T, cfg.d, cfg.N, cfg.k, cfg.m, cfg.n_shared, cfg.dtype)
    ws = B.alloc_workspace(dm)
    idx, gates, logits = B.alloc_route(dm, logits=True)
    rg = torch.empty_like(gates)
    o1 = torch.empty(cfg.T, cfg.d, dtype=cfg.torch_dtype, device=dev)
    o2 = torch.empty_like(o1)
    counts = torch.empty(cfg.N, dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    sh = (L["Ws_gate"], L["Ws_up"], L["Ws_down"])

    def ev():
        e = torch.cuda.Event(enable_timing=True)
        e.record()
        return e

    def one(marks, st1=None, st2=None):
        marks[0].record()
        if len(marks) > 3:  # per-kernel pass: routing and forward as separate calls
            B.check(B.pr2_route_predict(dm, L["x"], L["W_router"], L["W_pred"], idx, gates,
                                        logits, None, status), "pr2_route_predict")
            marks[3].record()
            B.check(B.pr2_moe_forward(dm, L["x"], idx, gates, L["W_gate"], L["W_up"],
                                      L["W_down"], *sh, o1, counts=counts, workspace=ws,
                                      status=status, events=st1), "pr2_moe_forward")
        else:  # the rollout-mode layer as one call
            B.check(B.pr2_moe_rollout_forward(dm, L["x"], L["W_router"], L["W_pred"], idx,
                                              gates, logits, None, L["W_gate"], L["W_up"],
                                              L["W_down"], *sh, o1, counts=counts,
                                              workspace=ws, status=status),
                    "pr2_moe_rollout_forward")
        marks[1].record()
        if len(marks) > 3:  # per-kernel pass: routing and forward as separate calls
            B.check(B.pr2_route_replay(dm, L["x"], W2, idx, rg, None, status), "pr2_route_replay")
            marks[4].record()
            B.check(B.pr2_moe_forward(dm, L["x"], idx, rg, L["W_gate"], L["W_up"], L["W_down"],
                                      *sh, o2, workspace=ws, status=status, events=st2),
                    "pr2_moe_forward")
        else:  # the training-mode layer as one call
            B.check(B.pr2_moe_replay_forward(dm, L["x"], W2, idx, rg, None, L["W_gate"],
                                             L["W_up"], L["W_down"], *sh, o2, workspace=ws,
                                             status=status), "pr2_moe_replay_forward")
        marks[2].record()

    sets = []
    for i in range(iters + 3):
        flush.fill_(i & 0xFF)
        m = [ev() for _ in range(3)]
        one(m)
        sets.append(m)
    torch.cuda.synchronize()
    roll = statistics.median(m[0].elapsed_time(m[1]) for m in sets[3:])
    rep = statistics.median(m[1].elapsed_time(m[2]) for m in sets[3:])
    step = statistics.median(m[0].elapsed_time(m[2]) for m in sets[3:])
    # per-kernel pass: stage events inside both forwards
    per = dict(route_predict=[], route_replay=[], dispatch=[], expert_gemm=[], combine=[])
    for i in range(iters + 3):
        flush.fill_(i & 0xFF)
        m = [ev() for _ in range(5)]
        a = [ev() for _ in range(5)]
        b = [ev() for _ in range(5)]
        one(m, B.stage_events(a), B.stage_events(b))
        torch.cuda.synchronize()
        if i < 3:
            continue
        per["route_predict"].append(m[0].elapsed_time(m[3]))
        per["route_replay"].append(m[1].elapsed_time(m[4]))
        for st in (a, b):
            per["dispatch"].append(st[0].elapsed_time(st[1]))
            per["expert_gemm"].append(st[1].elapsed_time(st[3]))
            per["combine"].append(st[3].elapsed_time(st[4]))
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())} in the {cfg.name} layer")
    hit = int((counts > 0).sum().item())
    F = cfg.T * cfg.k
    gw = cost.expert_mlp_algorithmic_work(F, cfg.d, cfg.m, hit, cfg.dtype, a_rows=cfg.T)
    if cfg.n_shared:
        sw = cost.expert_mlp_algorithmic_work(cfg.T * cfg.n_shared, cfg.d, cfg.m, cfg.n_shared,
                                              cfg.dtype, a_rows=0)
        gw = cost.KernelWork(gw.bytes + sw.bytes, gw.flops + sw.flops)
    work = dict(route_predict=cost.route_predict_work(cfg.T, cfg.d, cfg.N, cfg.k, cfg.dtype,
                                                      True),
                route_replay=cost.route_replay_work(cfg.T, cfg.d, cfg.N, cfg.k, cfg.dtype),
                dispatch=cost.dispatch_work(cfg.T, cfg.d, cfg.k, cfg.dtype),
                expert_gemm=gw,
                combine=cost.combine_work(cfg.T, cfg.d, cfg.k, cfg.n_shared, cfg.dtype))
    kernels = {n: kernel_roofline(w, statistics.median(per[n]), pk, pk["bf16"])
               for n, w in work.items()}
    g = kernels["expert_gemm"]
    g["tensor_frac"] = gw.flops / (pk["bf16"] * 1e12) / (g["ms"] * 1e-3)
    out = dict(workload=cfg.name, T=cfg.T, d=cfg.d, N=cfg.N, k=cfg.k, m=cfg.m,
               n_shared=cfg.n_shared, experts_hit=hit,
               tokens_per_s=cfg.T / (step * 1e-3), ms_per_step=step,
               rollout_tokens_per_s=cfg.T / (roll * 1e-3),
               replay_tokens_per_s=cfg.T / (rep * 1e-3), kernels=kernels,
               note="both modes as in the bench step; median of per-step device times, L2 "
                    "flushed before every step")
    del L, W2, ws
    torch.cuda.empty_cache()
    return out


def run_pr2(args, rank, world, local_rank):
    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    cfg = synth.CONFIGS[args.workload]
    dev = "cuda"
    L = synth.make_layer(cfg, seed=0, device=dev)
    W2 = synth.make_drifted_router(L["W_router"])
    dm = B.dims(cfg.T, cfg.d, cfg.N, cfg.k, cfg.m, cfg.n_shared, cfg.dtype)
    ws = B.alloc_workspace(dm)
    idx, gates, logits = B.alloc_route(dm, logits=True)
    rgates = torch.empty_like(gates)
    out1 = torch.empty(cfg.T, cfg.d, dtype=cfg.torch_dtype, device=dev)
    out2 = torch.empty_like(out1)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    near = torch.zeros(1, dtype=torch.int64, device=dev)
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def ev():
        e = torch.cuda.Event(enable_timing=True)
        e.record()  # creates the underlying cudaEvent_t
        return e

    def rec(e):
        if e is not None:
            e.record()

    def step(x, evs):
        rec(evs[0])
        if evs[1] is None:
            # headline steps: the rollout-mode layer as one call (dispatch from the routing
            # kernel's histograms, same results as the two calls below)
            B.check(B.pr2_moe_rollout_forward(dm, x, L["W_router"], L["W_pred"], idx, gates,
                                              logits, near, L["W_gate"], L["W_up"], L["W_down"],
                                              L["Ws_gate"], L["Ws_up"], L["Ws_down"], out1,
                                              workspace=ws, status=status),
                    "pr2_moe_rollout_forward")
        else:
            # per-kernel breakdown pass: routing and forward as separate calls
            B.check(B.pr2_route_predict(dm, x, L["W_router"], L["W_pred"], idx, gates, logits,
                                        near, status), "pr2_route_predict")
            rec(evs[1])
            B.check(B.pr2_moe_forward(dm, x, idx, gates, L["W_gate"], L["W_up"], L["W_down"],
                                      L["Ws_gate"], L["Ws_up"], L["Ws_down"], out1,
                                      workspace=ws, status=status, events=evs[2]),
                    "pr2_moe_forward")
        rec(evs[3])
        if evs[4] is None:
            # headline steps: the training-mode layer as one call (replay routing launched
            # behind the expert GEMMs, same results as the two calls below)
            B.check(B.pr2_moe_replay_forward(dm, x, W2, idx, rgates, None, L["W_gate"],
                                             L["W_up"], L["W_down"], L["Ws_gate"], L["Ws_up"],
                                             L["Ws_down"], out2, workspace=ws, status=status),
                    "pr2_moe_replay_forward")
        else:
            # per-kernel breakdown pass: routing and forward as separate calls
            B.check(B.pr2_route_replay(dm, x, W2, idx, rgates, None, status), "pr2_route_replay")
            rec(evs[4])
            B.check(B.pr2_moe_forward(dm, x, idx, rgates, L["W_gate"], L["W_up"], L["W_down"],
                                      L["Ws_gate"], L["Ws_up"], L["Ws_down"], out2, workspace=ws,
                                      status=status, events=evs[5]), "pr2_moe_forward")
        rec(evs[6])

    def make_evs(stages):
        """Step-boundary events, plus (stages=True) an event at every stage boundary.  Events
        between kernels stop a kernel's prologue from overlapping the previous kernel's tail
        (programmatic dependent launch), so the headline steps record step boundaries only and
        the per-kernel breakdown comes from a separate pass."""
        if not stages:
            return [ev(), None, None, None, None, None, ev()]
        a = [ev() for _ in range(5)]
        b = [ev() for _ in range(5)]
        return [ev(), ev(), (B.stage_events(a), a), ev(), ev(), (B.stage_events(b), b), ev()]

    def run(n, evsets, x=None):
        for i in range(n):
            flush.fill_(i & 0xFF)
            e = evsets[i]
            step(L["x"] if x is None else x,
                 [e[0], e[1], e[2][0] if e[2] else None, e[3], e[4], e[5][0] if e[5] else None,
                  e[6]])

    # warm-up
    wev = [make_evs(False) for _ in range(args.warmup)]
    run(args.warmup, wev)
    torch.cuda.synchronize()
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())} after warm-up")
    evsets = [make_evs(False) for _ in range(args.steps)]
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(torch.cuda.current_device())
    time.sleep(0.3)
    near.zero_()
    run(args.steps, evsets)
    torch.cuda.synchronize()
    clk = clocks.stop()
    near_per_step = int(near.item()) / args.steps
    if dist is not None:
        dist.barrier()

    def el(a, b):
        return a.elapsed_time(b)  # ms

    total_ms = replicas.job_time_ms(sum(el(e[0], e[6]) for e in evsets), dist,
                                    torch.device("cuda", local_rank))
    # per-kernel breakdown: a separate pass with an event at every stage boundary
    n_break = min(args.steps, 200)
    bsets = [make_evs(True) for _ in range(n_break)]
    run(n_break, bsets)
    torch.cuda.synchronize()
    per = dict(step=[], route_predict=[], route_replay=[], dispatch=[], expert_gemm=[],
               combine=[], layer_rollout=[], layer_replay=[])
    for e in bsets:
        per["step"].append(el(e[0], e[6]))
        per["route_predict"].append(el(e[0], e[1]))
        per["route_replay"].append(el(e[3], e[4]))
        per["layer_rollout"].append(el(e[0], e[3]))
        per["layer_replay"].append(el(e[3], e[6]))
        for _, st in (e[2], e[5]):
            per["dispatch"].append(el(st[0], st[1]))
            # routed gate/up and down run as one launch (plus the shared experts' GEMMs)
            per["expert_gemm"].append(el(st[1], st[3]))
            per["combine"].append(el(st[3], st[4]))
    value = replicas.job_throughput(cfg.T * args.steps, world, total_ms)
    mean = {k: statistics.mean(v) for k, v in per.items()}

    # ---- per-kernel roofline (algorithmic work / measured duration)
    pk = peaks()
    F = cfg.T * cfg.k
    counts = torch.empty(cfg.N, dtype=torch.int32, device=dev)
    B.check(B.pr2_moe_forward(dm, L["x"], idx, gates, L["W_gate"], L["W_up"], L["W_down"],
                              L["Ws_gate"], L["Ws_up"], L["Ws_down"], out1, counts=counts,
                              workspace=ws, status=status), "pr2_moe_forward")
    hit = int((counts > 0).sum().item())
    work = {
        "route_predict": cost.route_predict_work(cfg.T, cfg.d, cfg.N, cfg.k, cfg.dtype, True),
        "route_replay": cost.route_replay_work(cfg.T, cfg.d, cfg.N, cfg.k, cfg.dtype, False),
        "dispatch": cost.dispatch_work(cfg.T, cfg.d, cfg.k, cfg.dtype, gather=cfg.dtype == "fp32"),
        # the fused minimum of the grouped GEMMs: h once and the hit experts' weights (the H
        # round trip and the Y write of this design are counted in `modeled_bytes`)
        "expert_gemm": cost.expert_mlp_algorithmic_work(
            F, cfg.d, cfg.m, hit, cfg.dtype, a_rows=cfg.T),
        "combine": cost.combine_work(cfg.T, cfg.d, cfg.k, cfg.n_shared, cfg.dtype),
    }
    modeled = cost.expert_mlp_work(F, cfg.d, cfg.m, hit, cfg.dtype,
                                   a_rows=cfg.T if cfg.dtype == "bf16" else None).bytes
    if cfg.n_shared:
        sw = cost.expert_mlp_algorithmic_work(cfg.T * cfg.n_shared, cfg.d, cfg.m, cfg.n_shared,
                                              cfg.dtype, a_rows=0)
        work["expert_gemm"] = cost.KernelWork(work["expert_gemm"].bytes + sw.bytes,
                                              work["expert_gemm"].flops + sw.flops)
        modeled += cost.expert_mlp_work(cfg.T * cfg.n_shared, cfg.d, cfg.m, cfg.n_shared,
                                        cfg.dtype).bytes
    timed_s = total_ms / 1e3 / world
    # The sustained bf16 peak (a GEMM looped for seconds under the power cap) applies only to a
    # run whose clock record shows the power cap during a timed region of seconds; otherwise
    # the burst peak (a GEMM timed alone at full clock) is the denominator.
    sustained = bool(clk and "sw_power_cap" in clk.get("reasons", []) and timed_s >= 2.0)
    tc_peak = pk["bf16_sustained"] if sustained else pk["bf16"]
    kernels = {name: kernel_roofline(w, mean[name], pk, tc_peak) for name, w in work.items()}
    dom = "expert_gemm"
    dk = kernels[dom]
    dk["modeled_bytes"] = modeled
    # The grouped GEMM is the one dense contraction of the path: its roofline is the tensor
    # pipe (FLOPs / duration against the bf16 peak); `combined_frac` is the time the tighter of
    # its two bounds allows (tensor, or HBM on h + the experts' weights) over the duration.
    w = work[dom]
    traffic = measured_traffic(f"{cfg.name}/{dom}")
    roofline = dict(kernel="expert_tc_kernel (routed gate/up + down, one launch)"
                    + (" + shared-expert GEMMs" if cfg.n_shared else ""),
                    bound="tensor", achieved=w.flops / (dk["ms"] * 1e-3) / 1e12,
                    peak=tc_peak, unit="TFLOP/s",
                    frac=w.flops / (tc_peak * 1e12) / (dk["ms"] * 1e-3),
                    traffic=traffic,
                    peak_source=(f"{pk['source']} (MEASURED_PEAKS.json "
                                 f"{'sustained' if sustained else 'burst'})"
                                 if pk["source"] == "measured" else "fallback"),
                    algorithmic="flops",
                    algorithmic_flops=w.flops, algorithmic_bytes=w.bytes,
                    combined_frac=dk["frac"], combined_bound=dk["bound"],
                    hbm_frac=w.bytes / (pk["hbm"] * 1e9) / (dk["ms"] * 1e-3),
                    traffic_over_algorithmic=(traffic / w.bytes) if traffic else None,
                    modeled_bytes=modeled,
                    per_launch_units=f"{F} token-expert rows x (d={cfg.d}, m={cfg.m})")

    extras = measure_extras(cfg, L, W2, dm, flush, pk, iters=args.extras_iters)
    if cfg.name != "deepseek_v3" and not args.no_deepseek:
        # the DeepSeek-V3-shaped layer (d = 7168, 256 routed experts + 1 shared, 22.6 GB of
        # expert weights), both modes
        extras["deepseek_v3"] = measure_layer_modes(synth.CONFIGS["deepseek_v3"], flush, pk,
                                                    iters=min(args.extras_iters, 20))

    # ---- end to end through the public API with host buffers.  Every step copies its input
    # from pinned host memory and both layer outputs and the recorded route back; the copies of
    # the next / previous step run on a second stream while this step computes (device buffers
    # double-buffered), and the whole run of steps is timed on the copy stream.  No L2 flush:
    # each step streams 1.2 GB of expert weights, ~10x the L2.
    cs = torch.cuda.Stream()
    S = torch.cuda.current_stream()
    xh = torch.empty(cfg.T, cfg.d, dtype=cfg.torch_dtype, pin_memory=True)
    xh.copy_(L["x"].cpu())
    xd = [torch.empty_like(L["x"]) for _ in range(2)]
    o1 = [torch.empty_like(out1) for _ in range(2)]
    o2 = [torch.empty_like(out1) for _ in range(2)]
    ixd = [torch.empty_like(idx) for _ in range(2)]
    o1h = [torch.empty(cfg.T, cfg.d, dtype=cfg.torch_dtype, pin_memory=True) for _ in range(2)]
    o2h = [torch.empty_like(o1h[0]) for _ in range(2)]
    ixh = [torch.empty(cfg.T, cfg.k, dtype=torch.int32, pin_memory=True) for _ in range(2)]

    def e2e_compute(b):
        x = xd[b]
        B.check(B.pr2_moe_rollout_forward(dm, x, L["W_router"], L["W_pred"], ixd[b], gates,
                                          logits, near, L["W_gate"], L["W_up"], L["W_down"],
                                          L["Ws_gate"], L["Ws_up"], L["Ws_down"], o1[b],
                                          workspace=ws, status=status),
                "pr2_moe_rollout_forward")
        B.check(B.pr2_moe_replay_forward(dm, x, W2, ixd[b], rgates, None, L["W_gate"], L["W_up"],
                                         L["W_down"], L["Ws_gate"], L["Ws_up"], L["Ws_down"],
                                         o2[b], workspace=ws, status=status),
                "pr2_moe_replay_forward")

    def d2h(b, comp_ev):
        with torch.cuda.stream(cs):
            cs.wait_event(comp_ev)
            o1h[b].copy_(o1[b], non_blocking=True)
            o2h[b].copy_(o2[b], non_blocking=True)
            ixh[b].copy_(ixd[b], non_blocking=True)
            e = torch.cuda.Event()
            e.record(cs)
        return e

    def run_e2e(n):
        torch.cuda.synchronize()
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        comp, done = [None] * n, [None] * n
        start.record(cs)
        for i in range(n):
            b = i & 1
            with torch.cuda.stream(cs):  # issued after the copy-out of step i-2 (same buffer)
                xd[b].copy_(xh, non_blocking=True)
                h2d = torch.cuda.Event()
                h2d.record(cs)
            S.wait_event(h2d)
            if i >= 2:
                S.wait_event(done[i - 2])  # step i-2's outputs have left buffer b
            e2e_compute(b)
            comp[i] = torch.cuda.Event()
            comp[i].record(S)
            if i >= 1:
                done[i - 1] = d2h((i - 1) & 1, comp[i - 1])
        done[n - 1] = d2h((n - 1) & 1, comp[n - 1])
        end.record(cs)
        end.synchronize()
        return start.elapsed_time(end)

    run_e2e(max(args.warmup, 2))
    e2e_total = replicas.job_time_ms(run_e2e(args.steps), dist, torch.device("cuda", local_rank))
    esz = 2 if cfg.dtype == "bf16" else 4
    e2e = dict(value=replicas.job_throughput(cfg.T * args.steps, world, e2e_total), unit="tokens/s",
               h2d_bytes_per_step=cfg.T * cfg.d * esz,
               d2h_bytes_per_step=2 * cfg.T * cfg.d * esz + cfg.T * cfg.k * 4,
               ms_per_step=e2e_total / args.steps,
               note="copies of neighbouring steps overlap compute on a second stream; "
                    "no L2 flush (1.2 GB of expert weights per step)")

    # per layer forward: dispatch (one fused cooperative kernel when N % 4 == 0 and the grid is
    # resident, as at every bench shape; else hist + scan + place; + a row gather on the fp32
    # path only, the bf16 gate/up GEMM gathers its A rows itself), the routed grouped GEMMs (one
    # launch for gate/up and down in bf16, two in fp32; + two for shared experts) and the
    # combine; plus one routing kernel per mode
    n_dispatch = (1 if cfg.N % 4 == 0 and cfg.N <= 256 else 3) + (cfg.dtype == "fp32")
    n_gemm = 1 if cfg.dtype == "bf16" else 2
    launches_per_step = 2 + 2 * (n_dispatch + n_gemm + 1 + (2 if cfg.n_shared else 0))
    line = dict(metric=METRIC, value=value, unit="tokens/s", n_gpus=world, steps=args.steps,
                warmup=args.warmup, ms_per_step=total_ms / args.steps, higher_is_better=True,
                scaling="weak", vs_baseline=None, dtype=cfg.dtype, data="synthetic",
                config=workload_desc(cfg), roofline=roofline, e2e=e2e,
                gpu_launches=launches_per_step * args.steps, clocks=clk,
                modes=dict(rollout_tokens_per_s=cfg.T / (mean["layer_rollout"] / 1e3),
                           replay_tokens_per_s=cfg.T / (mean["layer_replay"] / 1e3),
                           note="from the per-kernel breakdown pass (stage events)"),
                breakdown_ms_per_step=mean["step"],
                kernels=kernels, near_tie_tokens_per_step=near_per_step, extras=extras)

    if rank == 0 and not args.no_cpu_baseline:
        Lh = host_layer(cfg, L)
        line["cpu_baseline"] = cpu_baseline(cfg, Lh, W2.cpu(), args.cpu_seconds)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------------- reference

def run_reference(args, rank):
    if rank != 0:
        return
    import oracle
    cfg = synth.CONFIGS[args.workload]
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    L = synth.make_layer(cfg, seed=0, device=dev)
    W2 = synth.make_drifted_router(L["W_router"]).cpu()
    Lh = host_layer(cfg, L)
    del L
    n_tok = 8
    times = []
    for i in range(args.warmup + args.steps):
        toks = synth.make_token_sample(cfg.T, n_tok, 100 + i).numpy()
        dt = oracle_layer_seconds(cfg, Lh, W2, toks)
        if i >= args.warmup:
            times.append(dt)
    total = sum(times)
    value = n_tok * args.steps / total
    line = dict(metric=METRIC, value=value, unit="tokens/s", n_gpus=1, steps=args.steps,
                warmup=args.warmup, ms_per_step=1e3 * total / args.steps, higher_is_better=True,
                scaling="weak", vs_baseline=None, dtype="f64", data="synthetic",
                config=workload_desc(cfg), impl="reference",
                cpu_baseline=dict(value=value, unit="tokens/s", cores=oracle.num_threads(),
                                  kind="oracle",
                                  sample=f"{n_tok} seeded tokens of {cfg.name} per step, both "
                                         f"modes, fp64 CPU oracle"),
                e2e=dict(value=value, unit="tokens/s", h2d_bytes_per_step=0,
                         d2h_bytes_per_step=0))
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    rank, world, local_rank = replicas.rank_env()
    if args.impl == "reference":
        run_reference(args, rank)
        return
    from paper_2606_00395_gb300 import build
    if local_rank == 0:
        build.build()
    else:
        t0 = time.time()
        while not build.up_to_date() and time.time() - t0 < 600:
            time.sleep(1.0)
    run_pr2(args, rank, world, local_rank)


if __name__ == "__main__":
    main()
