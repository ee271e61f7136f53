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

from . import (LayerCache, Shape, WS_BALANCER, WS_STEP, mikv_compute_balancer, mikv_decode_step,
               mikv_gather_hi, mikv_quantize_pack, mikv_select_demote, mikv_workspace_bytes)


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
        With q_pre [B, Hq, T, d] the channel balancer is computed (Eq. 2); without it, b = 1."""
        B, H, T, _ = k.shape
        k_budget = shape.hi_cap - 1 if budget is None else budget
        bal = None
        if q_pre is not None:
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
        if n_demote > 0:
            mikv_quantize_pack(layer.cache, k, v, demoted, 0)
        layer.n_lo = n_demote
        layer.pos = T
        layer.slots.fill_(k_budget)  # the staging slot receives the first decoded token
        return layer

    def step(self, q, k_new, v_new, out):
        """One decode step: the new token enters, attention runs, the least important slot is demoted."""
        mikv_decode_step(self.cache, self.n_lo, q, k_new, v_new, self.pos, self.slots, self.sm_scale, out,
                         self.ws)
        self.n_lo += 1
        self.pos += 1
