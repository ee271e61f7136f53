"""Cache build and decode steps of one attention layer, as a sequence of libmikv calls.

This is the flow a serving stack runs around the library (Fig. 4 of arxiv 2402.18096):
  prefill  -> channel balancer from prefill maxima (Eq. 2)
           -> choose the k most important tokens by accumulated attention (mikv_select_demote)
           -> keep them in high precision (mikv_gather_hi: bf16, or 8/4/2-bit codes for a reduced-
              precision important set, Sec. 3.3), quantize the rest into the retained set
              (mikv_quantize_pack, Eq. 1 with Eq. 3 key balancing)
  decode   -> per token: insert, attend, update importance, demote the least important (mikv_decode_step)
Every step runs in the library's kernels; this module only orders the calls and owns the buffers.
"""
from __future__ import annotations

import math

import torch

from . import (LayerCache, Shape, WS_BALANCER, WS_PREFILL, WS_STEP, mikv_compute_balancer, mikv_decode_attention,
               mikv_decode_step, mikv_gather_hi, mikv_prefill_scores, mikv_quantize_pack, mikv_select_demote,
               mikv_workspace_bytes)


def workspace(nbytes: int, device="cuda") -> torch.Tensor:
    """A 256-byte aligned uint8 device buffer of at least nbytes (torch allocations are aligned)."""
    return torch.zeros(max(nbytes, 256), dtype=torch.uint8, device=device)


class MixedPrecisionLayer:
    """One layer's MiKV cache plus the per-step state (free slots, retained length, workspace)."""

    def __init__(self, shape: Shape, balancer: torch.Tensor = None, device="cuda"):
        self.shape = shape
        self.cache = LayerCache(shape, device=device, balancer=balancer)
        self.slots = torch.zeros(shape.batch, shape.heads_kv, dtype=torch.int32, device=device)
        self.ws = workspace(mikv_workspace_bytes(shape, WS_STEP, shape.lo_cap), device)
        self.n_lo = 0
        self.pos = 0
        self.sm_scale = 1.0 / math.sqrt(shape.head_dim)

    @classmethod
    def from_prefill(cls, shape: Shape, k, v, scores, q_pre=None, budget: int = None, device="cuda"):
        """Build the cache from prefill K, V [B, Hkv, T, d] (bf16) and importance scores [B, Hkv, T].
        With q_pre [B, Hq, T, d] the channel balancer is computed (Eq. 2; not for per-channel keys, which
        need none); without it, b = 1. With scores
        None the importance is the prefill's accumulated causal attention (mikv_prefill_scores, q_pre
        required)."""
        B, H, T, _ = k.shape
        if scores is None:
            if q_pre is None:
                raise ValueError("prefill scores need the prefill queries")
            scores = torch.empty(B, H, T, dtype=torch.float32, device=device)
            ws = workspace(mikv_workspace_bytes(shape, WS_PREFILL, T), device)
            mikv_prefill_scores(shape, q_pre, k, scores, ws)
        k_budget = shape.hi_cap - 1 if budget is None else budget
        bal = None
        if q_pre is not None and not shape.k_channel_group:
            bal = torch.empty(H, shape.head_dim, dtype=torch.float32, device=device)
            ws = workspace(mikv_workspace_bytes(shape, WS_BALANCER, 0), device)
            mikv_compute_balancer(shape, q_pre, k, bal, ws)
        layer = cls(shape, balancer=bal, device=device)
        n_demote = T - k_budget
        demoted = torch.empty(B, H, n_demote, dtype=torch.int32, device=device)
        kept = torch.empty(B, H, k_budget, dtype=torch.int32, device=device)
        mikv_select_demote(scores, T, n_demote, demoted, kept)
        if k_budget > 0:
            mikv_gather_hi(layer.cache, k, v, kept, src_scores=scores)
        if n_demote > 0 and shape.bits:
            mikv_quantize_pack(layer.cache, k, v, demoted, 0)
        layer.n_lo = n_demote if shape.bits else 0  # bits = 0: eviction, the demoted tokens are dropped
        layer.pos = T
        layer.slots.fill_(k_budget)  # the staging slot receives the first decoded token
        return layer

    def step(self, q, k_new, v_new, out):
        """One decode step: the new token enters, attention runs, the least important slot is demoted."""
        mikv_decode_step(self.cache, self.n_lo, q, k_new, v_new, self.pos, self.slots, self.sm_scale, out,
                         self.ws)
        if self.shape.bits:
            self.n_lo += 1
        self.pos += 1


def oracle_eviction_attention(k, v, q, budget: int, sm_scale: float, out, device="cuda"):
    """Oracle eviction (Sec. 2.2, Fig. 2), the comparison baseline: attention computed over the full bf16
    cache k, v [B, Hkv, T, d] for q [B, Hq, d], then top-k sparsity imposed on the attention map. Reading:
    each query head keeps its `budget` largest attention weights (ties: the smaller token index) and the
    output is the softmax over the logits of those tokens (the kept weights renormalised). Built from the
    library's entry points only: full attention with its logits, selection of the T - budget smallest
    logits (mikv_select_demote) whose complement is kept, gather of the kept rows, and attention over them; query heads of a KV head are handled one by one
    because each keeps its own tokens. Writes out [B, Hq, d]; returns the kept token indices [B, Hq, budget]."""
    B, H, T, d = k.shape
    Hq = q.shape[1]
    G = Hq // H
    full = Shape(B, H, H, 2, 32, T, 16)  # one query head per KV head at a time; bf16 important set of T rows
    cache = LayerCache(full, device=device)
    rows = torch.arange(T, dtype=torch.int32, device=device).expand(B, H, T).contiguous()
    mikv_gather_hi(cache, k, v, rows)
    kept_all = torch.empty(B, Hq, budget, dtype=torch.int32, device=device)
    small = Shape(B, H, H, 2, 32, budget, 16)
    ws = workspace(max(mikv_workspace_bytes(full, 0, 0), mikv_workspace_bytes(small, 0, 0)), device)
    # ids T-1-t: among equal logits the larger token index is dropped first, so the smaller one is kept
    ids = torch.arange(T - 1, -1, -1, dtype=torch.int32, device=device).expand(B, H, T).contiguous()
    ids = torch.nn.functional.pad(ids, (0, full.hi_stride - T))
    for j in range(G):
        qj = q[:, j::G].contiguous()
        logits = torch.empty(B, H, full.hi_stride, dtype=torch.float32, device=device)
        tmp = torch.empty(B, H, d, dtype=torch.float32, device=device)
        mikv_decode_attention(cache, 0, qj, sm_scale, tmp, ws, hi_logits=logits)
        kept = torch.empty(B, H, budget, dtype=torch.int32, device=device)
        dropped = torch.empty(B, H, T - budget, dtype=torch.int32, device=device)
        mikv_select_demote(logits, T, T - budget, dropped, kept=kept, ids=ids)
        sel = LayerCache(small, device=device)
        mikv_gather_hi(sel, k, v, kept)
        oj = torch.empty(B, H, d, dtype=out.dtype, device=device)
        mikv_decode_attention(sel, 0, qj, sm_scale, oj, ws)
        out[:, j::G] = oj
        kept_all[:, j::G] = kept
    return kept_all
