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


@pytest.mark.parametrize("B,Hq,Hkv,T", [(1, 4, 2, 300), (2, 8, 1, 64), (1, 2, 2, 1), (1, 4, 4, 130), (1, 4, 1, 2048)])
def test_prefill_scores_match_oracle(B, Hq, Hkv, T):
    w = mi.Workload("pf", B, Hq, Hkv, T, 1, 2, 32, 0.2, seed=T + 7 * Hq)
    k, _ = mi.prefill_kv(w, 0)
    q = mi.prefill_queries(w, 0)
    got = _gpu_scores(w, q, k)
    ref = oracle.prefill_scores(bits16(q), bits16(k), 1 / math.sqrt(128))
    G = Hq // Hkv
    assert np.all(np.isfinite(got))
    np.testing.assert_allclose(got, ref, rtol=5e-3, atol=1e-4 * G)
    np.testing.assert_allclose(got.sum(axis=2), G * T, rtol=1e-3)  # every query row's weights sum to one


def test_cache_built_from_prefill_scores():
    """The important set chosen from the GPU prefill scores is the oracle's top-k (near ties excepted)."""
    w = mi.Workload("pfb", 2, 8, 2, 700, 1, 2, 32, 0.2, seed=71)
    k, v = mi.prefill_kv(w, 0)
    q = mi.prefill_queries(w, 0)
    dev = torch.device("cuda")
    shape = pkg.Shape(w.batch, w.heads_q, w.heads_kv, w.bits, w.group, w.hi_cap, w.lo_cap_for(4))
    layer = MixedPrecisionLayer.from_prefill(shape, k.to(dev), v.to(dev), None, q.to(dev), device=dev)
    ref = oracle.prefill_scores(bits16(q), bits16(k), 1 / math.sqrt(128))
    for b in range(w.batch):
        for h in range(w.heads_kv):
            got = set(layer.cache.hi_tok[b, h, :w.budget].tolist())
            order = np.argsort(-ref[b, h], kind="stable")
            want = set(order[:w.budget].tolist())
            edge = ref[b, h][order[w.budget - 1]]
            for t in got ^ want:  # only tokens at the boundary may differ
                assert abs(ref[b, h][t] - edge) <= 5e-3 * edge + 1e-4, (b, h, t)
