"""Seeded synthetic workloads for the speculative-step attention.

This module only draws inputs; it holds none of the attention or selection
arithmetic, so the CUDA path and the fp64 oracle can both be fed from it.

The paper's evaluation data (PG-19, LongBench QMSum, NarrativeQA) and models are
not available here; these shapes stand in for them: a Llama-3-8B-shaped
attention layer (32 query heads, 8 KV heads, head_dim 128) at the paper's context
lengths, its budget set {256, 512, 1024, 2048} and gamma = 5.

Recipe (per layer l and sequence b, generator seeded with base + 1000 l + b):
  K, V     [h_kv, t_cap, d]   i.i.d. N(0, 1)
  q_win    [h_q, W, d]        i.i.d. N(0, 1)   (queries of the last W context tokens)
  q_draft  [gamma, h_q, d]    i.i.d. N(0, 1)   (one query per drafter pass)
  q_verify [h_q, gamma+1, d]  i.i.d. N(0, 1)
Heavy hitters: for each KV head, u = unit vector of the sum of the group's window
queries; floor(f t_ctx) positions drawn without replacement from [0, t_ctx) get
k += hh_scale * u (fp32, then rounded to bf16 with everything else).
Rows t_ctx .. t_ctx + gamma hold the drafted / verified tokens' own K/V.
"""

from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field

import torch


@dataclass(frozen=True)
class Workload:
    name: str
    batch: int
    h_q: int
    h_kv: int
    head_dim: int
    t_ctx: int
    budget: int
    n_sink: int
    n_recent: int
    window: int = 32
    gamma: int = 5
    hh_frac: float = 0.02
    hh_frac_range: tuple | None = None      # per-layer U(lo, hi) draw when set
    hh_scale: float = 3.0
    layers: int = 1
    seed: int = 20260

    @property
    def t_cap(self) -> int:
        return self.t_ctx + self.gamma + 1

    @property
    def group(self) -> int:
        return self.h_q // self.h_kv

    def with_budget(self, budget: int, n_recent: int | None = None) -> "Workload":
        rec = budget // 4 if n_recent is None else n_recent
        return dataclasses.replace(self, budget=budget, n_recent=rec,
                                   name=f"{self.name.split('@')[0]}@B{budget}")

    def describe(self) -> dict:
        d = dataclasses.asdict(self)
        d["t_cap"] = self.t_cap
        return d


# The five evaluation workloads (tiny single layer; 4K; 8K x4; 16K x8 budget sweep;
# full 32-layer stack at 16K x16).
WORKLOADS = {
    "tiny_1k": Workload("tiny_1k", batch=1, h_q=8, h_kv=2, head_dim=64, t_ctx=1024,
                        budget=256, n_sink=4, n_recent=64, hh_frac=0.02),
    "l8b_4k": Workload("l8b_4k", batch=1, h_q=32, h_kv=8, head_dim=128, t_ctx=4096,
                       budget=512, n_sink=4, n_recent=128, hh_frac=0.02),
    "l8b_8k_b4": Workload("l8b_8k_b4", batch=4, h_q=32, h_kv=8, head_dim=128, t_ctx=8192,
                          budget=1024, n_sink=4, n_recent=256, hh_frac=0.01),
    "l8b_16k_b8": Workload("l8b_16k_b8", batch=8, h_q=32, h_kv=8, head_dim=128, t_ctx=16384,
                           budget=512, n_sink=4, n_recent=128, hh_frac=0.01),
    "l8b_32L_16k_b16": Workload("l8b_32L_16k_b16", batch=16, h_q=32, h_kv=8, head_dim=128,
                                t_ctx=16384, budget=512, n_sink=4, n_recent=128,
                                hh_frac_range=(0.005, 0.03), layers=32),
}
SWEEP_16K = (256, 512, 1024, 2048, 16384)


def layer_hh_frac(wl: Workload, layer: int) -> float:
    if wl.hh_frac_range is None:
        return wl.hh_frac
    g = torch.Generator().manual_seed(wl.seed * 7919 + layer)
    lo, hi = wl.hh_frac_range
    return float(lo + (hi - lo) * torch.rand((), generator=g).item())


@dataclass
class LayerInputs:
    k_cache: torch.Tensor      # bf16 [b, h_kv, t_cap, d]
    v_cache: torch.Tensor      # bf16 [b, h_kv, t_cap, d]
    q_win: torch.Tensor        # bf16 [b, h_q, W, d]
    q_draft: torch.Tensor      # bf16 [gamma, b, h_q, d]
    q_verify: torch.Tensor     # bf16 [b, h_q, gamma + 1, d]
    hh_pos: list = field(default_factory=list)   # per (b, kv): planted positions


def make_layer(wl: Workload, layer: int = 0, device="cpu", out: dict | None = None,
               first_seq: int = 0) -> LayerInputs:
    """Draw one layer's inputs for sequences first_seq .. first_seq + batch - 1.  If
    ``out`` holds preallocated bf16 tensors (keys k_cache, v_cache, q_win, q_draft,
    q_verify) they are filled in place."""
    b, hq, hkv, d, tc = wl.batch, wl.h_q, wl.h_kv, wl.head_dim, wl.t_cap
    dev = torch.device(device)
    bf = torch.bfloat16
    if out is None:
        out = dict(
            k_cache=torch.empty(b, hkv, tc, d, dtype=bf, device=dev),
            v_cache=torch.empty(b, hkv, tc, d, dtype=bf, device=dev),
            q_win=torch.empty(b, hq, wl.window, d, dtype=bf, device=dev),
            q_draft=torch.empty(wl.gamma, b, hq, d, dtype=bf, device=dev),
            q_verify=torch.empty(b, hq, wl.gamma + 1, d, dtype=bf, device=dev),
        )
    frac = layer_hh_frac(wl, layer)
    n_hh = int(frac * wl.t_ctx)
    hh_pos = []
    for bi in range(b):
        g = torch.Generator(device=dev).manual_seed(wl.seed + 1000 * layer + first_seq + bi)
        k = torch.randn(hkv, tc, d, generator=g, device=dev)
        v = torch.randn(hkv, tc, d, generator=g, device=dev)
        qw = torch.randn(hq, wl.window, d, generator=g, device=dev)
        qd = torch.randn(wl.gamma, hq, d, generator=g, device=dev)
        qv = torch.randn(hq, wl.gamma + 1, d, generator=g, device=dev)
        for kv in range(hkv):
            qsum = qw[kv * wl.group:(kv + 1) * wl.group].to(bf).float().sum(dim=(0, 1))
            u = qsum / qsum.norm().clamp_min(1e-30)
            pos = torch.randperm(wl.t_ctx, generator=g, device=dev)[:n_hh]
            k[kv, pos] += wl.hh_scale * u
            hh_pos.append(pos.cpu())
        out["k_cache"][bi].copy_(k)
        out["v_cache"][bi].copy_(v)
        out["q_win"][bi].copy_(qw)
        out["q_draft"][:, bi].copy_(qd)
        out["q_verify"][bi].copy_(qv)
    return LayerInputs(hh_pos=hh_pos, **out)


def tiny_workload(batch=1, h_q=4, h_kv=2, head_dim=64, t_ctx=200, budget=64, n_sink=4,
                  n_recent=16, window=32, gamma=5, hh_frac=0.02, seed=7) -> Workload:
    """A small custom workload for tests (same recipe, other shapes)."""
    return Workload(f"custom_b{batch}_t{t_ctx}_B{budget}", batch=batch, h_q=h_q, h_kv=h_kv,
                    head_dim=head_dim, t_ctx=t_ctx, budget=budget, n_sink=n_sink,
                    n_recent=n_recent, window=window, gamma=gamma, hh_frac=hh_frac, seed=seed)
