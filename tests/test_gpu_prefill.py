"""GPU parity of the prefill importance (mikv_prefill_scores: the accumulated causal attention every prefill
token receives, summed over the query heads of its KV head) against the oracle's fp64 evaluation, on the
seeded synthetic prefill (outlier channels included), with ragged and exact tiles, one token, GQA and
MHA; and the cache build from those scores (MixedPrecisionLayer.from_prefill with scores=None) choosing
the oracle's important set."""
import math

import numpy as np
import pytest
import torch

import mikv_inputs as mi
import oracle
import paper_2402_18096_gb300 as pkg
from paper_2402_18096_gb300.layer import MixedPrecisionLayer, workspace
from _cases import bits16

pytestmark = pytest.mark.gpu


def _gpu_scores(w, q, k):
    dev = torch.device("cuda")
    shape = pkg.Shape(w.batch, w.heads_q, w.heads_kv, 2, 32, 1, 16)
    out = torch.full((w.batch, w.heads_kv, w.context), float("nan"), device=dev)
    ws = workspace(pkg.mikv_workspace_bytes(shape, pkg.WS_PREFILL, w.context), dev)
    pkg.mikv_prefill_scores(shape, q.to(dev), k.to(dev), out, ws)
    pkg.mikv_workspace_check(ws)
    return out.cpu().numpy()


def prefill_rtol(q_bits, k_bits, T: int, G: int) -> float:
    """Relative bound on every prefill score, from the kernel's fp32 arithmetic (each score is a sum of positive
    terms 2^x, x = s * log2(e) * scale - c_i, so relative errors of the terms carry over to the sum):
      - logit s: bf16 products exact, fp32 tensor-core accumulation of 128 of them: |ds| <= 2^-21 S, with
        S = scale * sum_c max_i |q_ic| max_t |k_tc| >= scale * sum_c |q_ic k_tc| for every (i, t);
      - exponent x: one fma rounding and the row normaliser c_i = r + log2(l_i), l_i a positive fp32 sum of
        chains up to 16 + T/64 terms: |dx| <= log2(e) |ds| + 2^-23 (2 + 16 + T/64) + 2^-24 |x| with |x| <= 2 S;
      - ex2.approx: 2^-22 relative; the column sum: chains up to 16 + T/64 + G terms, 2^-24 each.
    rtol = ln2 |dx| + 2^-22 + (16 + T/64 + G) 2^-24, with a factor 2 of margin."""
    qf = (q_bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    kf = (k_bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    qmax = np.abs(qf).reshape(-1, qf.shape[-1]).max(axis=0)
    kmax = np.abs(kf).reshape(-1, kf.shape[-1]).max(axis=0)
    S = float((qmax * kmax).sum()) / math.sqrt(128)
    chain = 16 + T / 64
    dx = math.log2(math.e) * 2.0 ** -21 * S + 2.0 ** -23 * (2 + chain) + 2.0 ** -24 * 2 * S
    return 2 * (math.log(2) * dx + 2.0 ** -22 + (chain + G) * 2.0 ** -24)


@pytest.mark.parametrize("B,Hq,Hkv,T", [(1, 4, 2, 300), (2, 8, 1, 64), (1, 2, 2, 1), (1, 4, 4, 130), (1, 4, 1, 2048)])
def test_prefill_scores_match_oracle(B, Hq, Hkv, T):
    w = mi.Workload("pf", B, Hq, Hkv, T, 1, 2, 32, 0.2, seed=T + 7 * Hq)
    k, _ = mi.prefill_kv(w, 0)
    q = mi.prefill_queries(w, 0)
    got = _gpu_scores(w, q, k)
    ref = oracle.prefill_scores(bits16(q), bits16(k), 1 / math.sqrt(128))
    G = Hq // Hkv
    assert np.all(np.isfinite(got))
    rtol = prefill_rtol(bits16(q), bits16(k), T, G)
    np.testing.assert_allclose(got, ref, rtol=rtol, atol=0)
    np.testing.assert_allclose(got.sum(axis=2), G * T, rtol=rtol)  # every query row's weights sum to one


@pytest.mark.parametrize("B,Hq,Hkv,T,heads", [(8, 32, 32, 4096, [(0, 0), (7, 31)]),   # Llama-2-7B shape
                                              (2, 32, 8, 8192, [(1, 5)])],           # GQA, G = 4
                         ids=["llama2-7b-t4096", "gqa4-t8192"])
def test_prefill_scores_long_rows_sampled_heads(B, Hq, Hkv, T, heads):
    """Prefill importance at the lengths it is benchmarked on: the library on the whole batch, the oracle on
    sampled KV heads (its fp64 causal softmax per query row). Rows this long reach the cases short ones do not:
    row sums far from the first tile's reference, thousands of tiles per column sum."""
    w = mi.Workload("pfl", B, Hq, Hkv, T, 1, 2, 32, 0.2, seed=T + Hq)
    dev = torch.device("cuda")
    k, _ = mi.prefill_kv(w, 0, dev)
    q = mi.prefill_queries(w, 0, dev)
    got = _gpu_scores(w, q, k)
    G = Hq // Hkv
    for b, h in heads:
        qh, kh = bits16(q[b:b + 1, h * G:(h + 1) * G]), bits16(k[b:b + 1, h:h + 1])
        ref = oracle.prefill_scores(qh, kh, 1 / math.sqrt(128))[0, 0]
        rtol = prefill_rtol(qh, kh, T, G)
        np.testing.assert_allclose(got[b, h], ref, rtol=rtol, atol=0)
        assert abs(got[b, h].sum() / (G * T) - 1) <= rtol


def test_cache_built_from_prefill_scores():
    """The important set chosen from the GPU prefill scores is the oracle's top-k (near ties excepted)."""
    w = mi.Workload("pfb", 2, 8, 2, 700, 1, 2, 32, 0.2, seed=71)
    k, v = mi.prefill_kv(w, 0)
    q = mi.prefill_queries(w, 0)
    dev = torch.device("cuda")
    shape = pkg.shape_for_context(w.batch, w.heads_q, w.heads_kv, w.bits, w.group, w.context, w.ratio, 4)
    layer = MixedPrecisionLayer.from_prefill(shape, k.to(dev), v.to(dev), None, q.to(dev), device=dev)
    ref = oracle.prefill_scores(bits16(q), bits16(k), 1 / math.sqrt(128))
    k_b = oracle.budget(w.context, w.ratio)
    assert shape.hi_cap == k_b + 1
    rtol = prefill_rtol(bits16(q), bits16(k), w.context, w.heads_q // w.heads_kv)
    for b in range(w.batch):
        for h in range(w.heads_kv):
            got = set(layer.cache.hi_tok[b, h, :k_b].tolist())
            order = np.argsort(-ref[b, h], kind="stable")
            want = set(order[:k_b].tolist())
            edge = ref[b, h][order[k_b - 1]]
            for t in got ^ want:  # only tokens whose score is within the score bound of the boundary may differ
                assert abs(ref[b, h][t] - edge) <= 2 * rtol * edge, (b, h, t)
