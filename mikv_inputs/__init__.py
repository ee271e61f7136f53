"""Seeded synthetic inputs for the MiKV decode path: workload shapes and random tensors.

This module holds no arithmetic of the method (no quantization, attention, balancing or selection):
it only names the workloads and draws the random tensors that both the CUDA library and the CPU
oracle consume. Values stand in for the activations of the paper's LLM backbones (Llama-2 7b/13b,
Mistral-7b, Sec. 4.1), which are not available here:

  * keys, values, queries ~ N(0, 1), rounded to bf16;
  * per (layer, KV head), 4 key channels are outliers scaled by 10: two seeded channels c < d/2 and
    their rotary partners c + d/2 (the paper observes fixed outlier channels in keys and queries that
    rotary embedding duplicates, Sec. 3.2 / Fig. 5);
  * initial importance scores (stand-ins for prefill accumulated attention) ~ LogNormal(0, 1), a
    heavy-tailed distribution like heavy-hitter scores.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
from typing import List, Optional

import torch

HEAD_DIM = 128
OUTLIER_SCALE = 10.0


@dataclass(frozen=True)
class Workload:
    """One decode workload: cache shape per layer and the mixed-precision settings."""
    name: str
    batch: int
    heads_q: int
    heads_kv: int
    context: int          # T, tokens in the cache before the first decode step
    layers: int
    bits: int             # retained-set code width
    group: int            # channels per quantization group
    ratio: float          # fraction of tokens kept in bf16 (importance ratio)
    seed: int = 0
    head_dim: int = HEAD_DIM

    @property
    def budget(self) -> int:
        """k, the number of important tokens: ratio * T rounded half up."""
        return int(self.ratio * self.context + 0.5)

    @property
    def hi_cap(self) -> int:
        return self.budget + 1  # plus one staging slot for the incoming token

    @property
    def hi_stride(self) -> int:
        return (self.hi_cap + 15) // 16 * 16

    @property
    def n_lo0(self) -> int:
        """Retained rows after the cache build."""
        return self.context - self.budget

    def lo_cap_for(self, steps: int) -> int:
        return max(16, (self.n_lo0 + steps + 15) // 16 * 16)


WORKLOADS = {
    "tiny": Workload("tiny-b1-h32-t512-int4-g32-r20", 1, 32, 32, 512, 1, 4, 32, 0.20, seed=0),
    "llama2-7b": Workload("llama2-7b-b8-l32-h32-t4096-int2-g32-r20", 8, 32, 32, 4096, 32, 2, 32, 0.20),
    "llama2-13b": Workload("llama2-13b-b16-l40-h40-t8192-int3-g64-r10", 16, 40, 40, 8192, 40, 3, 64, 0.10),
    "mistral-7b": Workload("mistral-7b-b32-l32-hq32-hkv8-t32768-int2-g32-r20", 32, 32, 8, 32768, 32, 2,
                           32, 0.20),
}


def sweep_workloads() -> List[Workload]:
    """Batch 64, 32 heads, T 4096, one layer: bits x ratio x group (30 points)."""
    out = []
    for bits in (2, 3, 4):
        for ratio in (0.0, 0.05, 0.10, 0.25, 0.50):
            for group in (32, 128):
                out.append(Workload(f"sweep-b64-h32-t4096-int{bits}-g{group}-r{int(ratio * 100)}", 64, 32,
                                    32, 4096, 1, bits, group, ratio))
    return out


def scaled(w: Workload, **kw) -> Workload:
    """The same workload with some fields replaced (smaller parity cases)."""
    return replace(w, **kw)


# ------------------------------------------------------------------ random tensors

def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def outlier_channels(w: Workload, layer: int) -> torch.Tensor:
    """int64 [Hkv, 4]: the outlier key channels of each KV head of `layer` (CPU)."""
    g = _gen("cpu", w.seed * 1000003 + 7919 * layer + 17)
    half = w.head_dim // 2
    out = torch.empty(w.heads_kv, 4, dtype=torch.int64)
    for h in range(w.heads_kv):
        c = torch.randperm(half, generator=g)[:2]
        out[h] = torch.cat([c, c + half])
    return out


def prefill_kv(w: Workload, layer: int, device="cpu", batch: Optional[int] = None,
               context: Optional[int] = None):
    """bf16 K, V [B, Hkv, T, d] of one layer's prefill, keys with 4 outlier channels per head x10."""
    B = w.batch if batch is None else batch
    T = w.context if context is None else context
    g = _gen(device, w.seed * 1000003 + 1000 * layer + 1)
    k = torch.randn(B, w.heads_kv, T, w.head_dim, generator=g, device=device)
    v = torch.randn(B, w.heads_kv, T, w.head_dim, generator=g, device=device)
    oc = outlier_channels(w, layer).to(device)
    scale = torch.ones(w.heads_kv, w.head_dim, device=device)
    scale.scatter_(1, oc, OUTLIER_SCALE)
    k.mul_(scale[None, :, None, :])
    return k.to(torch.bfloat16), v.to(torch.bfloat16)


def prefill_queries(w: Workload, layer: int, device="cpu", batch: Optional[int] = None,
                    context: Optional[int] = None):
    """bf16 Q [B, Hq, T, d] of one layer's prefill, with the query side of the outlier channels
    (the same channels as the keys of the KV head, scaled x10)."""
    B = w.batch if batch is None else batch
    T = w.context if context is None else context
    g = _gen(device, w.seed * 1000003 + 1000 * layer + 2)
    q = torch.randn(B, w.heads_q, T, w.head_dim, generator=g, device=device)
    G = w.heads_q // w.heads_kv
    oc = outlier_channels(w, layer).to(device)
    scale = torch.ones(w.heads_kv, w.head_dim, device=device)
    scale.scatter_(1, oc, OUTLIER_SCALE)
    q.mul_(scale.repeat_interleave(G, 0)[None, :, None, :])
    return q.to(torch.bfloat16)


def initial_scores(w: Workload, layer: int, device="cpu", batch: Optional[int] = None,
                   context: Optional[int] = None):
    """fp32 [B, Hkv, T] synthetic accumulated-attention scores of the prefill tokens."""
    B = w.batch if batch is None else batch
    T = w.context if context is None else context
    g = _gen(device, w.seed * 1000003 + 1000 * layer + 3)
    return torch.randn(B, w.heads_kv, T, generator=g, device=device).exp_()


def decode_inputs(w: Workload, layer: int, step: int, device="cpu", batch: Optional[int] = None):
    """(q bf16 [B, Hq, d], k_new bf16 [B, Hkv, d], v_new bf16 [B, Hkv, d]) of one decode step;
    the new key carries the layer's outlier channels like the prefill keys."""
    B = w.batch if batch is None else batch
    g = _gen(device, w.seed * 1000003 + 1000 * layer + 10 + 7 * step)
    q = torch.randn(B, w.heads_q, w.head_dim, generator=g, device=device)
    k = torch.randn(B, w.heads_kv, w.head_dim, generator=g, device=device)
    v = torch.randn(B, w.heads_kv, w.head_dim, generator=g, device=device)
    oc = outlier_channels(w, layer).to(device)
    scale = torch.ones(w.heads_kv, w.head_dim, device=device)
    scale.scatter_(1, oc, OUTLIER_SCALE)
    k.mul_(scale[None])
    return q.to(torch.bfloat16), k.to(torch.bfloat16), v.to(torch.bfloat16)


def bf16_bits(t: torch.Tensor):
    """uint16 numpy view of a bf16 tensor's bit patterns (CPU copy)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view("uint16")
