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

from dataclasses import dataclass, replace
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
    bits: int             # retained-set code width (0: no retained set, the H2O eviction baseline)
    group: int            # channels per quantization group
    ratio: float          # fraction of tokens kept in bf16 (importance ratio; each side turns it into a
                          # token count with its own budget function)
    seed: int = 0
    head_dim: int = HEAD_DIM
    hi_bits: int = 16     # important-set precision: 16 = bf16, or 8 / 4 / 2-bit codes in groups of 64
    k_channel: bool = False  # retained keys per channel over groups of 64 tokens (App. C)


WORKLOADS = {
    "tiny": Workload("tiny-b1-h32-t512-int4-g32-r20", 1, 32, 32, 512, 1, 4, 32, 0.20, seed=0),
    "llama2-7b": Workload("llama2-7b-b8-l32-h32-t4096-int2-g32-r20", 8, 32, 32, 4096, 32, 2, 32, 0.20),
    "llama2-13b": Workload("llama2-13b-b16-l40-h40-t8192-int3-g64-r10", 16, 40, 40, 8192, 40, 3, 64, 0.10),
    "mistral-7b": Workload("mistral-7b-b32-l32-hq32-hkv8-t32768-int2-g32-r20", 32, 32, 8, 32768, 32, 2,
                           32, 0.20),
}
# Table 3 settings (INT2 retained, 20 % important, groups of 64) on the Mistral-7B shape, with the
# important set itself at reduced precision (Sec. 3.3)
# the importance-based eviction baseline (H2O) on the Mistral-7B shape: the same 20 % important set,
# the other tokens dropped
WORKLOADS["mistral-7b-h2o"] = Workload("mistral-7b-b32-l32-hq32-hkv8-t32768-h2o-r20", 32, 32, 8, 32768, 32, 0, 32,
                                       0.20)
for _hb in (16, 8, 4, 2):
    WORKLOADS[f"mistral-7b-t3-hi{_hb}"] = Workload(
        f"mistral-7b-b32-l32-hq32-hkv8-t32768-int2-g64-r20-hi{_hb}", 32, 32, 8, 32768, 32, 2, 64, 0.20,
        hi_bits=_hb)
# per-channel retained keys (App. C, Table 8 settings): INT2 / INT3 retained, 20 % important, keys quantized
# per channel over groups of 64 retained tokens, values per token in groups of 64 channels
for _b in (2, 3):
    WORKLOADS[f"mistral-7b-kch-int{_b}"] = Workload(
        f"mistral-7b-b32-l32-hq32-hkv8-t32768-int{_b}-g64-r20-kch64", 32, 32, 8, 32768, 32, _b, 64, 0.20,
        k_channel=True)


def sweep_workloads() -> List[Workload]:
    """Batch 64, 32 heads, T 4096, one layer: bits x ratio x group (30 points)."""
    out = []
    for bits in (2, 3, 4):
        for ratio in (0.0, 0.05, 0.10, 0.25, 0.50):
            for group in (32, 128):
                out.append(Workload(f"sweep-b64-h32-t4096-int{bits}-g{group}-r{int(ratio * 100)}", 64, 32,
                                    32, 4096, 1, bits, group, ratio))
    return out


# every sweep point under its own short name (e.g. "sweep-int3-g128-r0"), so one point can be run alone
for _w in sweep_workloads():
    WORKLOADS[f"sweep-int{_w.bits}-g{_w.group}-r{int(_w.ratio * 100)}"] = _w


def scaled(w: Workload, **kw) -> Workload:
    """The same workload with some fields replaced (smaller parity cases)."""
    return replace(w, **kw)


# ------------------------------------------------------------------ random tensors
#
# Every tensor is drawn in independent chunks, one per (batch row, head), each from its own seeded
# generator, so any subset of rows and heads can be produced alone (the CPU oracle draws only the heads
# it checks) and equals the same slice of the full tensor drawn on the same device.

KIND_K, KIND_V, KIND_QPRE, KIND_SCORES, KIND_Q, KIND_KNEW, KIND_VNEW = range(7)
_MASK63 = (1 << 63) - 1


def _seed(w: Workload, layer: int, kind: int, b: int, h: int, step: int = 0) -> int:
    x = int(w.seed)
    for v in (layer, kind, b, h, step):
        x = (x * 6364136223846793005 + 1442695040888963407 + int(v)) & _MASK63
        x ^= x >> 29
    return x


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def outlier_channels(w: Workload, layer: int) -> torch.Tensor:
    """int64 [Hkv, 4]: the outlier key channels of each KV head of `layer` (CPU)."""
    g = _gen("cpu", _seed(w, layer, 99, 0, 0))
    half = w.head_dim // 2
    out = torch.empty(w.heads_kv, 4, dtype=torch.int64)
    for h in range(w.heads_kv):
        c = torch.randperm(half, generator=g)[:2]
        out[h] = torch.cat([c, c + half])
    return out


def _channel_scale(w: Workload, layer: int, device) -> torch.Tensor:
    """fp32 [Hkv, d]: 10 on each KV head's outlier channels, 1 elsewhere."""
    scale = torch.ones(w.heads_kv, w.head_dim)
    scale.scatter_(1, outlier_channels(w, layer), OUTLIER_SCALE)
    return scale.to(device)


def _draw(w, layer, kind, rows, heads, n, device, scale_of_head=None, step=0):
    out = torch.empty(len(rows), len(heads), *n, dtype=torch.bfloat16, device=device)
    for i, b in enumerate(rows):
        for j, h in enumerate(heads):
            x = torch.randn(*n, generator=_gen(device, _seed(w, layer, kind, b, h, step)), device=device)
            if scale_of_head is not None:
                x.mul_(scale_of_head(h))
            out[i, j] = x.to(torch.bfloat16)
    return out


def prefill_kv(w: Workload, layer: int, device="cpu", rows=None, heads=None):
    """bf16 K, V [B, Hkv, T, d] of one layer's prefill; keys carry 4 outlier channels per head x10.
    rows / heads select batch rows and KV heads (default: all)."""
    rows = range(w.batch) if rows is None else rows
    heads = range(w.heads_kv) if heads is None else heads
    sc = _channel_scale(w, layer, device)
    n = (w.context, w.head_dim)
    k = _draw(w, layer, KIND_K, rows, heads, n, device, lambda h: sc[h])
    v = _draw(w, layer, KIND_V, rows, heads, n, device)
    return k, v


def prefill_queries(w: Workload, layer: int, device="cpu", rows=None, heads=None):
    """bf16 Q [B, Hq, T, d] of one layer's prefill; query heads carry the outlier channels of their KV
    head, scaled x10. heads selects query heads."""
    rows = range(w.batch) if rows is None else rows
    heads = range(w.heads_q) if heads is None else heads
    G = w.heads_q // w.heads_kv
    sc = _channel_scale(w, layer, device)
    return _draw(w, layer, KIND_QPRE, rows, heads, (w.context, w.head_dim), device, lambda h: sc[h // G])


def initial_scores(w: Workload, layer: int, device="cpu", rows=None, heads=None):
    """fp32 [B, Hkv, T] synthetic accumulated-attention scores of the prefill tokens."""
    rows = range(w.batch) if rows is None else rows
    heads = range(w.heads_kv) if heads is None else heads
    out = torch.empty(len(rows), len(heads), w.context, dtype=torch.float32, device=device)
    for i, b in enumerate(rows):
        for j, h in enumerate(heads):
            g = _gen(device, _seed(w, layer, KIND_SCORES, b, h))
            out[i, j] = torch.randn(w.context, generator=g, device=device).exp_()
    return out


def decode_inputs(w: Workload, layer: int, step: int, device="cpu", rows=None, kv_heads=None):
    """(q bf16 [B, Hq, d], k_new bf16 [B, Hkv, d], v_new bf16 [B, Hkv, d]) of one decode step; the new
    key carries the layer's outlier channels. Drawn per batch row (all heads at once); kv_heads selects
    KV heads (and their query heads) from the drawn rows."""
    rows = range(w.batch) if rows is None else rows
    G = w.heads_q // w.heads_kv
    sc = _channel_scale(w, layer, device)
    q = torch.empty(len(rows), w.heads_q, w.head_dim, dtype=torch.bfloat16, device=device)
    k = torch.empty(len(rows), w.heads_kv, w.head_dim, dtype=torch.bfloat16, device=device)
    v = torch.empty_like(k)
    for i, b in enumerate(rows):
        q[i] = torch.randn(w.heads_q, w.head_dim, device=device,
                           generator=_gen(device, _seed(w, layer, KIND_Q, b, 0, step))).to(torch.bfloat16)
        k[i] = (torch.randn(w.heads_kv, w.head_dim, device=device,
                            generator=_gen(device, _seed(w, layer, KIND_KNEW, b, 0, step))) * sc).to(torch.bfloat16)
        v[i] = torch.randn(w.heads_kv, w.head_dim, device=device,
                           generator=_gen(device, _seed(w, layer, KIND_VNEW, b, 0, step))).to(torch.bfloat16)
    if kv_heads is not None:
        qh = [h * G + j for h in kv_heads for j in range(G)]
        q, k, v = q[:, qh].contiguous(), k[:, list(kv_heads)].contiguous(), v[:, list(kv_heads)].contiguous()
    return q, k, v


def bf16_bits(t: torch.Tensor):
    """uint16 numpy view of a bf16 tensor's bit patterns (CPU copy)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view("uint16")
