"""Pins of the oracle's balancer (Eq. 2), importance policy, demotion choice and memory accounting.

References: hand-set maxima with exact square roots, a brute-force sort of (score, id) keys, the
normalisation of softmax (increments per step sum to G when every token is tracked), and the
"Cache size" columns printed in Tables 2-3 (tests/golden/cache_size_tables.json).
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from mikv_inputs import bf16_bits

D = 128
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _bf16(x):
    return torch.as_tensor(x).to(torch.bfloat16)


# ------------------------------------------------------------------ Eq. 2

def test_balancer_hand_values():
    """b = sqrt(max|q| / max|k|) with maxima chosen so that the root is exact."""
    B, Hq, Hkv, T = 2, 4, 2, 5
    q = torch.zeros(B, Hq, T, D)
    k = torch.zeros(B, Hkv, T, D)
    q[..., :] = 0.5
    k[..., :] = 0.5
    # channel 3 of KV head 0: max |q| = 8 (second query head of the group, batch 1, a negative
    # value), max |k| = 2 -> b = 2
    q[1, 1, 4, 3] = -8.0
    k[0, 0, 2, 3] = 2.0
    # channel 100 of KV head 1: max |q| = 1, max |k| = 16 -> b = 1/4
    q[0, 2, 0, 100] = 1.0
    k[1, 1, 3, 100] = -16.0
    # channel 7 of KV head 1: keys all zero -> b = 1 by definition
    k[:, 1, :, 7] = 0.0
    b = oracle.balancer(bf16_bits(_bf16(q)), bf16_bits(_bf16(k)))
    assert b.shape == (Hkv, D)
    assert b[0, 3] == 2.0
    assert b[1, 100] == 0.25
    assert b[1, 7] == 1.0
    assert b[0, 0] == 1.0 and b[1, 50] == 1.0  # equal maxima


def test_balancer_random_properties():
    rng = np.random.default_rng(4)
    B, Hq, Hkv, T = 2, 8, 2, 33
    q = _bf16(rng.standard_normal((B, Hq, T, D)) * rng.uniform(0.1, 10, (1, Hq, 1, D)))
    k = _bf16(rng.standard_normal((B, Hkv, T, D)) * rng.uniform(0.1, 10, (1, Hkv, 1, D)))
    b = oracle.balancer(bf16_bits(q), bf16_bits(k)).astype(np.float64)
    G = Hq // Hkv
    mq = q.float().abs().reshape(B, Hkv, G, T, D).amax(dim=(0, 2, 3)).double().numpy()
    mk = k.float().abs().amax(dim=(0, 2)).double().numpy()
    # sqrt is correctly rounded in fp32: b^2 reproduces the ratio to fp32 precision
    np.testing.assert_allclose(b * b, mq / mk, rtol=3e-7)
    # balanced maxima become equal: max|q / b| == max|k * b| (the point of Eq. 2)
    np.testing.assert_allclose(mq / b, mk * b, rtol=3e-7)


# ------------------------------------------------------------------ heavy-hitter policy

def _keys_sorted(scores, ids):
    return sorted(range(len(scores)), key=lambda i: (scores[i], ids[i]))


@pytest.mark.parametrize("n,n_demote", [(1, 1), (7, 1), (50, 13), (64, 0), (33, 33)])
def test_select_demote_brute_force(n, n_demote):
    rng = np.random.default_rng(n * 31 + n_demote)
    B, H = 2, 3
    scores = rng.choice(np.float32([0.5, 0.25, 1.0, 3.0, 0.0]), size=(B, H, n))  # many ties
    scores[0, 0] = rng.standard_normal(n).astype(np.float32)
    ids = np.stack([np.stack([rng.permutation(10 * n)[:n] for _ in range(H)]) for _ in range(B)])
    ids = ids.astype(np.int32)
    dem, kept = oracle.select_demote(scores, n_demote, ids)
    for b in range(B):
        for h in range(H):
            order = _keys_sorted(list(scores[b, h]), list(ids[b, h]))
            want = sorted(order[:n_demote])
            assert list(dem[b, h]) == want
            assert list(kept[b, h]) == sorted(order[n_demote:])
    # ids omitted -> the entry index breaks ties
    dem2, _ = oracle.select_demote(scores, n_demote)
    for b in range(B):
        for h in range(H):
            order = _keys_sorted(list(scores[b, h]), list(range(n)))
            assert list(dem2[b, h]) == sorted(order[:n_demote])


def test_importance_increments_sum_to_group_size():
    """When every token sits in the important set, one step adds exactly the softmax mass of the G
    query heads: the increments sum to G per KV head, and scores never decrease."""
    rng = np.random.default_rng(6)
    B, Hq, Hkv, n = 2, 8, 2, 40
    k = _bf16(rng.standard_normal((B, Hkv, n, D)))
    v = _bf16(rng.standard_normal((B, Hkv, n, D)))
    q = _bf16(rng.standard_normal((B, Hq, D)) * 3)
    cache = oracle.empty_cache(B, Hkv, D, 2, 32, n, 16)
    cache["k_hi"][:] = bf16_bits(k)
    cache["v_hi"][:] = bf16_bits(v)
    _, hl, ml = oracle.decode_attention(cache, bf16_bits(q), 0, 1 / math.sqrt(D))
    acc0 = rng.uniform(0, 5, (B, Hkv, n)).astype(np.float32)
    acc1 = oracle.update_importance(acc0, hl.astype(np.float32), ml.astype(np.float32), Hq)
    inc = acc1.astype(np.float64) - acc0
    np.testing.assert_allclose(inc.sum(-1), Hq // Hkv, rtol=1e-5)
    assert np.all(acc1 >= acc0)
    # the increment of one slot is the textbook softmax weight summed over its query heads
    s = torch.tensor(hl)
    w = torch.softmax(s, -1).reshape(B, Hkv, Hq // Hkv, n).sum(2).numpy()
    np.testing.assert_allclose(inc, w, rtol=1e-5, atol=2e-6)


def test_insert_and_gather():
    rng = np.random.default_rng(8)
    B, Hkv, hi_cap, n_src = 2, 2, 6, 11
    c = oracle.empty_cache(B, Hkv, D, 2, 32, hi_cap, 16)
    ks = rng.integers(0, 65535, (B, Hkv, n_src, D)).astype(np.uint16)
    vs = rng.integers(0, 65535, (B, Hkv, n_src, D)).astype(np.uint16)
    sc = rng.uniform(0, 1, (B, Hkv, n_src)).astype(np.float32)
    rows = np.stack([np.stack([np.sort(rng.permutation(n_src)[:5]) for _ in range(Hkv)]) for _ in range(B)])
    rows = rows.astype(np.int32)
    oracle.gather_hi(c, ks, vs, rows, src_scores=sc)
    for b in range(B):
        for h in range(Hkv):
            for i in range(5):
                assert np.array_equal(c["k_hi"][b, h, i], ks[b, h, rows[b, h, i]])
                assert c["hi_tok"][b, h, i] == rows[b, h, i] and c["acc"][b, h, i] == sc[b, h, rows[b, h, i]]
    slots = np.array([[5, 2], [0, 5]], np.int32)
    kn = rng.integers(0, 65535, (B, Hkv, D)).astype(np.uint16)
    vn = rng.integers(0, 65535, (B, Hkv, D)).astype(np.uint16)
    oracle.insert_token(c, kn, vn, 999, slots)
    for b in range(B):
        for h in range(Hkv):
            s = slots[b, h]
            assert np.array_equal(c["k_hi"][b, h, s], kn[b, h]) and np.array_equal(c["v_hi"][b, h, s], vn[b, h])
            assert c["hi_tok"][b, h, s] == 999 and c["acc"][b, h, s] == 0.0


# ------------------------------------------------------------------ memory accounting

def test_cache_fraction_matches_tables_2_and_3():
    with open(os.path.join(GOLDEN, "cache_size_tables.json")) as f:
        golden = json.load(f)
    for row in golden["rows"]:
        frac = oracle.cache_fraction(row["retained_bits"], row["group"], row["ratio"], row["importance_bits"])
        pct = math.floor(frac * 100 + 0.5)
        assert pct == row["cache_size_percent"], row


def test_cache_fraction_limits():
    assert oracle.cache_fraction(2, 64, 1.0) == 1.0                    # everything fp16
    assert oracle.cache_fraction(4, 128, 0.0) == (4 + 0.25) / 16       # uniform RTN baseline
    assert oracle.cache_fraction(8, 64, 1.0, 8) == (8 + 0.5) / 16


def test_budget_hand_values():
    """Tables 1-3 give the important set as a ratio of the tokens; the oracle's count (reading R10) is the
    nearest integer to ratio * T, halves rounded up. Hand-computed values of the benchmark shapes and ties."""
    assert oracle.budget(4096, 0.2) == 819       # 819.2
    assert oracle.budget(8192, 0.1) == 819       # 819.2
    assert oracle.budget(32768, 0.2) == 6554     # 6553.6
    assert oracle.budget(512, 0.2) == 102        # 102.4
    assert oracle.budget(4096, 0.05) == 205      # 204.8
    assert oracle.budget(10, 0.25) == 3          # 2.5: a half rounds up
    assert oracle.budget(1, 0.5) == 1            # 0.5
    assert oracle.budget(3, 0.5) == 2            # 1.5
    assert oracle.budget(6, 0.25) == 2           # 1.5
    assert oracle.budget(1, 0.2) == 0            # 0.2
    assert oracle.budget(0, 0.7) == 0
    assert oracle.budget(4096, 0.0) == 0 and oracle.budget(4096, 1.0) == 4096
    for bad in ((-1, 0.5), (10, -0.1), (10, 1.5), (10, float("nan"))):
        with pytest.raises(ValueError):
            oracle.budget(*bad)


def test_budget_brute_force_exact_ratios():
    """For ratios k/64 (exact in binary) the budget is the integer n minimising |n - ratio * T| in exact
    rational arithmetic, the larger n on a tie."""
    from fractions import Fraction
    for num in range(65):
        r = Fraction(num, 64)
        for T in (0, 1, 2, 3, 5, 7, 31, 64, 100, 127, 4095, 4096):
            x = r * T
            lo = x.numerator // x.denominator
            want = lo + 1 if x - lo >= Fraction(1, 2) else lo
            assert oracle.budget(T, num / 64) == want, (num, T)