"""Seeded synthetic inputs for the MoE expert layer.

This module is shared by the CUDA path's tests/bench and by the CPU oracle's
tests. It draws random tensors and nothing else: it holds none of the layer's
arithmetic (no routing, no FFN, no pruning rule).

Shapes and distributions follow the workloads studied in the LAEP paper:
expert counts 64/128/256 (Table 4), 48 surviving experts out of 64 (Table 5),
stable-phase skew whose max/min load spans orders of magnitude (Sec. 3.1,
Fig. 1, Fig. 3) modelled by a Zipf-shaped gate bias, and transition-phase
volatility modelled by a log-uniform bias.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import torch


@dataclasses.dataclass(frozen=True)
class LayerConfig:
    name: str
    T: int              # tokens in the batch
    d: int              # d_model
    E: int              # experts held by the layer (before any pruning)
    k: int              # experts per token (top-k)
    F: int              # expert FFN hidden size (d_ff)
    bias: str           # "none" | "zipf" | "loguniform"
    zipf_s: float = 1.2
    backward: bool = False
    prune_lowest: int = 0      # experts masked after a first routing pass
    compact: bool = False      # pruned experts are removed from the weights


# The five workloads. Names describe what they are.
CONFIGS = {
    0: LayerConfig("tiny_fwd_T512_d256_E16_k2_F512", 512, 256, 16, 2, 512, "none"),
    1: LayerConfig("skew_fwd_T8192_d2048_E64_k6_F1408_zipf1.2", 8192, 2048, 64, 6, 1408,
                   "zipf", 1.2),
    2: LayerConfig("laep_pruned_fwdbwd_T16384_d4096_E64to48_k8_F2048_zipf1.2", 16384, 4096, 64,
                   8, 2048, "zipf", 1.2, backward=True, prune_lowest=16),
    3: LayerConfig("volatile_fwdbwd_T32768_d4096_E128_k8_F1536_loguniform", 32768, 4096, 128, 8,
                   1536, "loguniform", backward=True),
    4: LayerConfig("large_fwdbwd_T65536_d7168_E256_k8_F2048_zipf1.0", 65536, 7168, 256, 8, 2048,
                   "zipf", 1.0, backward=True, prune_lowest=85, compact=True),
}


def seed_for(cfg_id: int) -> int:
    return 1000 + int(cfg_id)


def gate_bias(E: int, kind: str, zipf_s: float, gen: torch.Generator,
              device: str = "cpu") -> torch.Tensor:
    """Per-expert additive logit bias (fp32) that sets the load skew.

    zipf: b_e = -s * ln(rank_e) with a seeded random rank permutation, so the
          softmax weight of expert e is proportional to rank_e^-s (Zipf(s)).
    loguniform: b_e ~ U[-7, 0]; the 8 smallest are then pushed to -30 so that
          at least 8 experts receive no token at all.
    none: zeros (roughly uniform load).
    """
    if kind == "none":
        return torch.zeros(E, dtype=torch.float32, device=device)
    if kind == "zipf":
        rank = 1.0 + torch.randperm(E, generator=gen, device=device).to(torch.float64)
        return (-zipf_s * torch.log(rank)).to(torch.float32)
    if kind == "loguniform":
        b = torch.rand(E, generator=gen, device=device, dtype=torch.float32) * 7.0 - 7.0
        n_dead = min(8, E // 4)
        if n_dead > 0:
            low = torch.argsort(b)[:n_dead]
            b[low] = -30.0
        return b
    raise ValueError(f"unknown bias kind {kind!r}")


def make_layer_inputs(T: int, d: int, E: int, k: int, F: int, *, bias: str = "none",
                      zipf_s: float = 1.2, seed: int = 0, device: str = "cpu",
                      backward: bool = True, weight_std: float = 0.02,
                      with_weights: bool = True) -> dict:
    """All inputs of one MoE layer step, drawn from one seeded generator.

    x ~ N(0,1) -> bf16 [T,d]; w_router ~ N(0, 1/d) fp32 [d,E]; bias fp32 [E];
    w_gate_up ~ N(0, weight_std) -> bf16 [E, 2F, d] (rows 0..F-1 gate, F..2F-1 up);
    w_down ~ N(0, weight_std) -> bf16 [E, d, F]; dy ~ N(0,1) -> bf16 [T,d].
    """
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    out = {}
    out["bias"] = gate_bias(E, bias, zipf_s, gen, device)
    out["x"] = torch.randn(T, d, generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16)
    out["w_router"] = torch.randn(d, E, generator=gen, device=device,
                                  dtype=torch.float32) * (1.0 / math.sqrt(d))
    if with_weights:
        wgu = torch.empty(E, 2 * F, d, dtype=torch.bfloat16, device=device)
        wdn = torch.empty(E, d, F, dtype=torch.bfloat16, device=device)
        for e in range(E):  # per expert keeps the fp32 temporaries small
            wgu[e] = (torch.randn(2 * F, d, generator=gen, device=device, dtype=torch.float32)
                      * weight_std).to(torch.bfloat16)
            wdn[e] = (torch.randn(d, F, generator=gen, device=device, dtype=torch.float32)
                      * weight_std).to(torch.bfloat16)
        out["w_gate_up"] = wgu
        out["w_down"] = wdn
    if backward:
        out["dy"] = torch.randn(T, d, generator=gen, device=device,
                                dtype=torch.float32).to(torch.bfloat16)
    return out


def make_config_inputs(cfg_id: int, device: str = "cpu", T: Optional[int] = None,
                       with_weights: bool = True) -> dict:
    """Inputs of one of the five workloads (optionally with fewer tokens)."""
    c = CONFIGS[cfg_id]
    return make_layer_inputs(T or c.T, c.d, c.E, c.k, c.F, bias=c.bias, zipf_s=c.zipf_s,
                             seed=seed_for(cfg_id), device=device, backward=True,
                             with_weights=with_weights)
