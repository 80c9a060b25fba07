"""Seeded synthetic inputs for the Pr^2 MoE layer (both the CUDA path and the CPU oracle use them).

This module holds random draws and workload shapes only.  It contains none of the method's
arithmetic (no projection, softmax, top-k, permutation or expert math), so the oracle and the
CUDA path can both consume its tensors without sharing any computation.

Shapes follow the paper's MoE models (Sec. 5.1 and Table 4: Qwen3-30B-A3B has d=2048, N=128,
k=8, m=768) and a DeepSeek-V3-shaped layer (d=7168, N=256 routed + 1 shared, k=8, m=2048).
Weights are stored [out, in] row-major, i.e. the transpose of the paper's ``h W`` matrices:

* ``W_router[e, :]`` is column e of the router matrix W (d x N) of Sec. 4.1,
* ``W_pred[e, :]``   is column e of the evolution predictor W_p (d x N) of Sec. 4.1,
* ``W_gate[e], W_up[e]`` are [m, d] and ``W_down[e]`` is [d, m] (gated MLP of App. E.2).

Recipe (fixed draw order from one generator): x, W_router, W_pred, W_gate, W_up, W_down,
Ws_gate, Ws_up, Ws_down; x ~ N(0,1), every weight ~ N(0, 0.02^2); drawn in fp32 then cast once
to the layer dtype.  The replay-time router drift is a second generator (seed+1) adding
N(0, 0.002^2) to W_router.  Zipf-skewed recorded routes (the long-replay workload) use a third
generator (seed+2): k distinct experts per token drawn without replacement with probability
proportional to (e+1)^-s by the Gumbel-top-k construction.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Optional

import torch


@dataclasses.dataclass(frozen=True)
class LayerConfig:
    """One MoE-layer workload: T tokens, d=d_model, N routed experts, top-k, m=d_ff, s shared."""

    name: str
    T: int
    d: int
    N: int
    k: int
    m: int
    n_shared: int = 0
    dtype: str = "bf16"  # "fp32" or "bf16": the dtype of h, all weights and the layer output
    modes: tuple = ("rollout", "replay")
    zipf_s: Optional[float] = None  # recorded routes drawn Zipf(s) instead of by the router

    @property
    def torch_dtype(self) -> torch.dtype:
        return torch.float32 if self.dtype == "fp32" else torch.bfloat16

    def scaled(self, T: int) -> "LayerConfig":
        return dataclasses.replace(self, T=T)


CONFIGS: Dict[str, LayerConfig] = {
    # tiny fp32 layer: T=256, d=128, E=8, top-2, d_ff=256
    "tiny_fp32": LayerConfig("tiny_fp32", T=256, d=128, N=8, k=2, m=256, dtype="fp32"),
    # Qwen3-30B-A3B-shaped layer (Table 4 row "Qwen3"): the throughput workload
    "qwen3_30b_a3b": LayerConfig("qwen3_30b_a3b", T=4096, d=2048, N=128, k=8, m=768),
    # rollout decode batch: one token per sequence, predict-route mode only
    "qwen3_decode": LayerConfig("qwen3_decode", T=256, d=2048, N=128, k=8, m=768,
                                modes=("rollout",)),
    # training replay over 8 x 4096-token sequences with Zipf(1.2)-skewed recorded routes
    "qwen3_long_replay": LayerConfig("qwen3_long_replay", T=32768, d=2048, N=128, k=8, m=768,
                                     modes=("replay",), zipf_s=1.2),
    # DeepSeek-V3-shaped layer: 256 routed + 1 shared expert
    "deepseek_v3": LayerConfig("deepseek_v3", T=8192, d=7168, N=256, k=8, m=2048, n_shared=1),
}

WEIGHT_STD = 0.02
DRIFT_STD = 0.002


def _randn(gen: torch.Generator, shape, device) -> torch.Tensor:
    return torch.randn(*shape, generator=gen, dtype=torch.float32, device=device)


def make_layer(cfg: LayerConfig, seed: int = 0, device: str = "cpu") -> Dict[str, torch.Tensor]:
    """Draw the layer inputs of ``cfg`` in the fixed order above; returns contiguous tensors.

    ``device`` selects where the generator runs ("cpu" or "cuda"); the same seed on the same
    device always gives the same bits.  Shared-expert tensors are None when n_shared == 0.
    """
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    dt = cfg.torch_dtype
    T, d, N, m, s = cfg.T, cfg.d, cfg.N, cfg.m, cfg.n_shared
    out: Dict[str, Optional[torch.Tensor]] = {}
    out["x"] = _randn(gen, (T, d), device).to(dt)
    for name, shape in (("W_router", (N, d)), ("W_pred", (N, d)),
                        ("W_gate", (N, m, d)), ("W_up", (N, m, d)), ("W_down", (N, d, m))):
        out[name] = (_randn(gen, shape, device) * WEIGHT_STD).to(dt)
    for name, shape in (("Ws_gate", (s, m, d)), ("Ws_up", (s, m, d)), ("Ws_down", (s, d, m))):
        out[name] = (_randn(gen, shape, device) * WEIGHT_STD).to(dt) if s > 0 else None
    return out


def make_drifted_router(W_router: torch.Tensor, seed: int = 0) -> torch.Tensor:
    """Replay-time router weights: the rollout router plus N(0, 0.002^2) drift (seed+1)."""
    gen = torch.Generator(device=W_router.device)
    gen.manual_seed(seed + 1)
    noise = _randn(gen, tuple(W_router.shape), W_router.device) * DRIFT_STD
    return (W_router.float() + noise).to(W_router.dtype)


def make_zipf_routes(T: int, N: int, k: int, s: float, seed: int = 0) -> torch.Tensor:
    """[T, k] int32 recorded routes: k distinct experts per token, P(e) proportional to (e+1)^-s.

    Gumbel-top-k (sampling without replacement): keys = log w_e + Gumbel noise, take the k
    largest keys in descending order.  Drawn on the CPU with generator seed+2.
    """
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed + 2)
    logw = -s * torch.log(torch.arange(1, N + 1, dtype=torch.float64))
    u = torch.rand(T, N, generator=gen, dtype=torch.float64).clamp_(1e-300, 1.0 - 1e-16)
    keys = logw[None, :] - torch.log(-torch.log(u))
    return torch.topk(keys, k, dim=1).indices.to(torch.int32).contiguous()


def make_token_sample(T: int, n: int, seed: int = 0) -> torch.Tensor:
    """Sorted distinct token ids (int64) for sampled full-size checks; always includes 0 and T-1."""
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed + 3)
    n = min(n, T)
    pick = torch.randperm(T, generator=gen)[: max(n - 2, 0)]
    ids = torch.unique(torch.cat([pick, torch.tensor([0, T - 1])]))
    return ids[:n] if ids.numel() > n else ids


def make_loss_inputs(N: int, d: int, Tc: int, T_rho: int, seed: int = 0,
                     dtype: str = "bf16") -> Dict[str, torch.Tensor]:
    """Inputs of the predictive loss drawn directly, without a whole layer (for shapes whose
    expert weights would be needlessly large): cached features h_old [Tc, d] ~ N(0, 1), cached
    router logits p_old [Tc, N] ~ N(0, 0.5^2), predictor W_pred [N, d] ~ N(0, 0.02^2), a teacher
    distribution rho [T_rho, N] (u^4 normalised per row, u ~ U(0, 1): skewed but every entry
    positive) and cache positions pos [Tc] int32 ~ U{0, T_rho - 1}.  Generator seed+4, drawn in
    that order on the CPU; h_old and W_pred cast once to the layer dtype."""
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed + 4)
    dt = torch.bfloat16 if dtype == "bf16" else torch.float32
    h_old = torch.randn(Tc, d, generator=gen).to(dt)
    p_old = 0.5 * torch.randn(Tc, N, generator=gen)
    W_pred = (0.02 * torch.randn(N, d, generator=gen)).to(dt)
    u = torch.rand(T_rho, N, generator=gen, dtype=torch.float64) ** 4
    rho = (u / u.sum(dim=1, keepdim=True)).float()
    pos = torch.randint(0, T_rho, (Tc,), generator=gen, dtype=torch.int64).to(torch.int32)
    return dict(h_old=h_old, p_old=p_old, W_pred=W_pred, rho=rho, pos=pos)
