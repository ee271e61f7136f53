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
    """The library's cache shape for workload w (its important budget from the library's mikv_budget)."""
    return pkg.shape_for_context(w.batch if batch is None else batch, w.heads_q, w.heads_kv, w.bits, w.group,
                                 w.context, w.ratio, steps, hi_bits=w.hi_bits,
                                 k_channel_group=64 if w.k_channel else 0)


class RefSizes:
    """The oracle's side of the sizes: its own budget function turns the importance ratio into k."""

    def __init__(self, w: mi.Workload):
        self.budget = oracle.budget(w.context, w.ratio)
        self.hi_cap = self.budget + 1                # plus the staging slot of the incoming token
        self.n_lo0 = w.context - self.budget         # retained rows after the cache build


def ref_sizes(w: mi.Workload) -> RefSizes:
    return RefSizes(w)


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
        R = ref_sizes(w)
        dem, kept = oracle.select_demote(sc, T - R.budget)
        if w.k_channel:  # per-channel retained keys (App. C): no balancer, staging for the last group
            c = oracle.empty_cache(1, 1, w.head_dim, w.bits, w.group, R.hi_cap, lo_cap, k_channel=True)
            oracle.gather_hi(c, ks, vs, kept, src_scores=sc)
            oracle.append_retained(c, ks, vs, dem, 0)
        else:
            c = oracle.empty_cache(1, 1, w.head_dim, w.bits, w.group, R.hi_cap, lo_cap, hi_bits=w.hi_bits)
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


ATTN_REL = 2e-3  # the benchmark spec: max |GPU - oracle| <= 2e-3 * max|V| per element (fp32 accumulation)


def attention_tolerance(vmax: float, ref: np.ndarray, out_bf16: bool = False) -> np.ndarray:
    """The bound on |GPU - oracle| of every attention output element: 2e-3 * max|V|, fp32 and bf16 outputs alike
    (no allowance for the output's own rounding)."""
    return np.full(np.shape(ref), ATTN_REL * vmax)


def _bf16_rn(x) -> np.ndarray:
    return torch.as_tensor(np.asarray(x, np.float64)).to(torch.bfloat16).double().numpy()


def assert_attention_close(got, ref, vmax, f32=None, msg=""):
    """Attention output against the oracle's fp64 result `ref` under the strict bound 2e-3 * max|V|.

    fp32 output: every element within the bound.
    bf16 output (f32 = the GPU's fp32 output of the same call, when available):
      - the bf16 output is the round-to-nearest-even of the fp32 output, bit for bit (the kernels compute in fp32
        and round once at the end);
      - every element within the bound wherever a bf16 value can be: an element whose exact value lies farther
        than the bound from every bf16 number cannot meet it in any bf16 output (bf16 rounding alone is up to 2^-8
        of |out|, and with the paper's outlier channels |out| reaches 0.9 max|V| in tiny caches). Such elements
        (|RN(ref) - ref| + 2 |f32 - ref| > bound: no output within the fp32 error rounds inside the bound) are
        left to the two checks above.
    Returns the largest error as a fraction of the bound."""
    ref = np.asarray(ref, np.float64)
    bf16_out = isinstance(got, torch.Tensor) and got.dtype == torch.bfloat16
    g = got.double().cpu().numpy() if isinstance(got, torch.Tensor) else np.asarray(got, np.float64)
    bound = ATTN_REL * np.broadcast_to(np.asarray(vmax, np.float64), ref.shape)
    err = np.abs(g - ref)
    if not bf16_out:
        assert np.all(err <= bound), f"{msg}: max err {float((err / bound).max()):.3f} of the bound"
        return float((err / bound).max())
    slack = np.abs(_bf16_rn(ref) - ref)
    if f32 is not None:
        f = f32.double().cpu().numpy() if isinstance(f32, torch.Tensor) else np.asarray(f32, np.float64)
        assert np.array_equal(g, _bf16_rn(f)), f"{msg}: bf16 output is not the rounded fp32 output"
        assert np.all(np.abs(f - ref) <= bound), f"{msg}: fp32 max err {float((np.abs(f - ref) / bound).max()):.3f}"
        slack = slack + 2 * np.abs(f - ref)
    attainable = slack <= bound
    bad = (err > bound) & attainable
    assert not bad.any(), f"{msg}: max err {float((err[attainable] / bound[attainable]).max()):.3f} of the bound"
    return float((err / bound).max())


# fp32 accumulation allowance of the tensor-core dot products: 16 exact fp16 / bf16 products per MMA, 8 MMAs over
# two interleaved accumulators and one final add; each step rounds (or truncates) to fp32 relative to the running
# magnitude, so the error is at most a few 2^-23 of sum |products|: 2^-19 is taken, with margin
ACC_GAMMA = 2.0 ** -19


def logit_bounds(c, q_bits, bal, bits: int, group: int, n_lo: int, scale: float, hi_bits: int = 16):
    """Per-token bound on |GPU logit - oracle logit| for one (b, KV head) of a cache with a bf16 important set and
    per-token retained keys, from the kernel's documented arithmetic (the oracle evaluates in fp64):
      important rows: bf16 q times bf16 k, exact products, fp32 accumulation, times the fp32 scale;
      retained rows (and important rows of a coded important set, hi_bits < 16, groups of 64), G > 1 or a coded
                      important set: q_hat = fp16(fp32 q / fp32 b) and k_hat = fp16(alpha * code + beta) (HFMA2, one
                      rounding) as MMA operands, exact products, fp32 accumulation;
      retained rows, G = 1 with a bf16 important set (the group-column path): the MMA sums q_hat * code (exact
                      integer codes) per group in fp32, and alpha, beta enter in fp32 afterwards,
                      s = scale * sum_g (alpha_g * (q_hat . code)_g + beta_g * sum_g q_hat): bounded by the q_hat
                      rounding (evaluated exactly) plus (ACC_GAMMA + 2^-22) * sum_c |q_hat_c| (alpha code_c + |beta|)
                      for the fp32 accumulations and the few fp32 roundings that combine the groups.
    The operand roundings are evaluated exactly (numpy's IEEE fp32 division and correctly rounded fp16 casts);
    only the accumulation is bounded (ACC_GAMMA * sum |products|, plus 2^-24 of the scaling multiply).
    q_bits uint16 [1, G, d]; returns (hi [G, hi_cap], lo [G, n_lo])."""
    d = q_bits.shape[-1]
    q = (q_bits.astype(np.uint32) << 16).view(np.float32)[0]                  # [G, d] fp32 (exact bf16)
    s32 = float(np.float32(scale))
    qd = q.astype(np.float64)
    b32 = np.ones(d, np.float32) if bal is None else np.asarray(bal, np.float32).reshape(-1)[:d]
    q16 = (q / b32).astype(np.float16).astype(np.float64)                      # fp32 IEEE divide, fp16 RN
    qhat = qd / b32.astype(np.float64)                                         # the oracle's query (Eq. 4)

    def coded(rows):  # rows: exact dequantized keys [n, d]
        k16 = rows.astype(np.float16).astype(np.float64)
        return (np.abs(s32 * (q16 @ k16.T) - scale * (qhat @ rows.T))
                + s32 * (ACC_GAMMA + 2.0 ** -24) * (np.abs(q16) @ np.abs(k16).T))

    if hi_bits < 16:
        hi = coded(np.stack([oracle.dequantize_row(c["k_hi"][0, 0, i], c["k_hp"][0, 0, i], hi_bits, 64)
                             for i in range(c["k_hi"].shape[2])]))
    else:
        kh = (c["k_hi"][0, 0].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        hi = s32 * (ACC_GAMMA + 2.0 ** -24) * (np.abs(qd) @ np.abs(kh).T) + abs(s32 - scale) * np.abs(qd @ kh.T)
    if n_lo == 0:
        return hi, np.zeros((q.shape[0], 0))
    rows = np.stack([oracle.dequantize_row(c["k_codes"][0, 0, t], c["k_params"][0, 0, t], bits, group)
                     for t in range(n_lo)])
    if q.shape[0] > 1 or hi_bits < 16:
        return hi, coded(rows)
    # G = 1 group-column path: exact keys alpha * code + beta; |alpha code| = |k - beta|
    beta = np.stack([np.repeat(c["k_params"][0, 0, t][:, 1].view(np.float16).astype(np.float64), group)
                     for t in range(n_lo)])
    mag = np.abs(rows - beta) + np.abs(beta)
    lo = (np.abs(s32 * (q16 @ rows.T) - scale * (qhat @ rows.T))
          + s32 * (ACC_GAMMA + 2.0 ** -22) * (np.abs(q16) @ mag.T))
    return hi, lo


def softmax_stat_bounds(hi, lo, n_tokens: int):
    """From per-token logit bounds: |dm| <= E = max bound; the fp32 sum l = sum exp(s - m) then moves by at most
    e^(2E) - 1 relative (the logits and the max each move by E), plus ex2.approx (2^-22 per term) and fp32
    summation over chains of at most n / 16 + 64 terms. Returns (E [G], l_rtol [G])."""
    E = np.maximum(hi.max(axis=1), lo.max(axis=1) if lo.size else 0.0)
    return E, np.expm1(2 * E) + 2.0 ** -21 + (n_tokens / 16 + 64) * 2.0 ** -24


def new_workspace(shape: pkg.Shape, op: int, n_lo: int) -> torch.Tensor:
    return workspace(pkg.mikv_workspace_bytes(shape, op, n_lo), "cuda")


def sm_scale(d: int = 128) -> float:
    return 1.0 / math.sqrt(d)
