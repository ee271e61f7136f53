"""Shared construction of parity cases: the same seeded raw inputs go to the CUDA library (which builds
its cache with its own kernels) and to the CPU oracle (which builds its own cache with its own code).
Nothing computed by one side is fed to the other."""
from __future__ import annotations

import math

import numpy as np
import torch

import mikv_inputs as mi
import oracle
import paper_2402_18096_gb300 as pkg
from paper_2402_18096_gb300.layer import MixedPrecisionLayer, workspace

bits16 = mi.bf16_bits


def make_shape(w: mi.Workload, steps: int = 4, batch: int = None) -> pkg.Shape:
    return pkg.Shape(w.batch if batch is None else batch, w.heads_q, w.heads_kv, w.bits, w.group, w.hi_cap,
                     w.lo_cap_for(steps), hi_bits=w.hi_bits, k_channel_group=64 if w.k_channel else 0)


def raw_inputs(w: mi.Workload, layer: int = 0, device="cpu", balanced: bool = True):
    k, v = mi.prefill_kv(w, layer, device)
    scores = mi.initial_scores(w, layer, device)
    q_pre = mi.prefill_queries(w, layer, device) if balanced else None
    return k, v, scores, q_pre


def gpu_layer(w: mi.Workload, raw, steps: int = 4) -> MixedPrecisionLayer:
    k, v, scores, q_pre = raw
    dev = torch.device("cuda")
    shape = make_shape(w, steps)
    return MixedPrecisionLayer.from_prefill(shape, k.to(dev), v.to(dev), scores.to(dev),
                                            None if q_pre is None else q_pre.to(dev), device=dev)


def oracle_layer(w: mi.Workload, raw, lo_cap: int, heads=None):
    """Oracle cache of the KV heads listed in `heads` ([(b, h), ...]; all when None), each built as a
    batch-1, one-KV-head problem. The balancer is taken over the full batch (Eq. 2 pools the batch)."""
    k, v, scores, q_pre = raw
    G = w.heads_q // w.heads_kv
    B, H = k.shape[0], k.shape[1]
    heads = [(b, h) for b in range(B) for h in range(H)] if heads is None else heads
    out = []
    for b, h in heads:
        bal = None
        if q_pre is not None:
            bal = oracle.balancer(bits16(q_pre[:, h * G:(h + 1) * G]), bits16(k[:, h:h + 1]))
        ks, vs = bits16(k[b:b + 1, h:h + 1]), bits16(v[b:b + 1, h:h + 1])
        sc = scores[b:b + 1, h:h + 1].numpy()
        T = k.shape[2]
        dem, kept = oracle.select_demote(sc, T - w.budget)
        if w.k_channel:  # per-channel retained keys (App. C): no balancer, staging for the last group
            c = oracle.empty_cache(1, 1, w.head_dim, w.bits, w.group, w.hi_cap, lo_cap, k_channel=True)
            oracle.gather_hi(c, ks, vs, kept, src_scores=sc)
            oracle.append_retained(c, ks, vs, dem, 0)
        else:
            c = oracle.empty_cache(1, 1, w.head_dim, w.bits, w.group, w.hi_cap, lo_cap, hi_bits=w.hi_bits)
            oracle.gather_hi(c, ks, vs, kept, src_scores=sc, balancer_=bal)
            oracle.quantize_pack(c, ks, vs, dem, 0, balancer_=bal)
        out.append(dict(cache=c, balancer=bal, b=b, h=h, demoted=dem[0, 0], kept=kept[0, 0]))
    return out


def vmax_per_head(v: torch.Tensor, extra=None) -> np.ndarray:
    """max |V| per (b, kv head) over the prefill values (and the new values when given)."""
    m = v.float().abs().amax(dim=(2, 3))
    if extra is not None:
        m = torch.maximum(m, extra.float().abs().amax(dim=2))
    return m.numpy()


def attention_tolerance(vmax: float, ref: np.ndarray, out_bf16: bool) -> np.ndarray:
    """max |GPU - oracle| allowed per element: 2e-3 * max|V| (fp32 accumulation); with a bf16 output,
    plus the bf16 rounding of the result itself (2^-8 relative)."""
    tol = np.full(ref.shape, 2e-3 * vmax)
    if out_bf16:
        tol = tol + np.abs(ref) * 2.0 ** -8
    return tol


def new_workspace(shape: pkg.Shape, op: int, n_lo: int) -> torch.Tensor:
    return workspace(pkg.mikv_workspace_bytes(shape, op, n_lo), "cuda")


def sm_scale(d: int = 128) -> float:
    return 1.0 / math.sqrt(d)
