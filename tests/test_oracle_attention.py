"""Pins of the oracle's decode attention, balancer application and demotion (CPU only).

The references are textbook softmax attention from torch (scaled_dot_product_attention and plain
matmul/softmax in fp64), exact constructions on which Eq. 1 is lossless, and invariances the paper
states (permutation invariance, Sec. 3.4; (q / b) . (k * b) = q . k, Eq. 3-4).
"""
import math

import numpy as np
import pytest
import torch

import oracle
from mikv_inputs import bf16_bits

D = 128


def _bf16(x: torch.Tensor) -> torch.Tensor:
    return x.to(torch.bfloat16)


def _textbook(q, k, v, scale):
    """q [B, Hq, d], k/v [B, Hkv, n, d] (float64) -> out [B, Hq, d], logits [B, Hq, n]."""
    B, Hq, d = q.shape
    G = Hq // k.shape[1]
    kk = k.repeat_interleave(G, 1)
    vv = v.repeat_interleave(G, 1)
    s = torch.einsum("bhd,bhnd->bhn", q, kk) * scale
    out = torch.einsum("bhn,bhnd->bhd", torch.softmax(s, -1), vv)
    return out, s


def _hi_only_cache(k, v, bits=2, g=32, lo_cap=16):
    B, Hkv, n, d = k.shape
    c = oracle.empty_cache(B, Hkv, d, bits, g, n, lo_cap)
    c["k_hi"][:] = bf16_bits(k)
    c["v_hi"][:] = bf16_bits(v)
    return c


@pytest.mark.parametrize("B,Hq,Hkv,n", [(1, 2, 2, 5), (2, 4, 1, 37), (1, 8, 2, 130)])
def test_all_important_is_textbook_attention(B, Hq, Hkv, n):
    """Importance ratio 100 %: MiKV attention is plain softmax attention over bf16 K/V."""
    g = torch.Generator().manual_seed(B * 100 + n)
    q = _bf16(torch.randn(B, Hq, D, generator=g))
    k = _bf16(torch.randn(B, Hkv, n, D, generator=g) * 2)
    v = _bf16(torch.randn(B, Hkv, n, D, generator=g))
    scale = 1 / math.sqrt(D)
    cache = _hi_only_cache(k, v)
    out, hl, ml = oracle.decode_attention(cache, bf16_bits(q), 0, scale)
    ref, s = _textbook(q.double(), k.double(), v.double(), scale)
    np.testing.assert_allclose(out, ref.numpy(), rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(hl, s.numpy(), rtol=1e-12, atol=1e-12)
    G = Hq // Hkv
    sdpa = torch.nn.functional.scaled_dot_product_attention(
        q.double()[:, :, None, :], k.double().repeat_interleave(G, 1), v.double().repeat_interleave(G, 1),
        scale=scale)[:, :, 0, :]
    np.testing.assert_allclose(out, sdpa.numpy(), rtol=1e-10, atol=1e-12)
    # softmax weights sum to one: sum_i exp(s_i - m) / l == 1, and m is the max logit
    np.testing.assert_allclose((np.exp(hl - ml[..., :1]) / ml[..., 1:]).sum(-1), 1.0, rtol=1e-12)
    np.testing.assert_allclose(ml[..., 0], hl.max(-1), rtol=0, atol=0)


def _lossless_rows(rng, n_rows, bits, g, balancer):
    """bf16 K, V rows whose balanced keys and values sit exactly on an Eq. 1 grid, so that
    quantization is lossless: per group, beta in multiples of 1/4, alpha = 1/4, codes covering 0 and
    2^N - 1. balancer: powers of two, so k * b is exact."""
    qmax = (1 << bits) - 1

    def grid_rows():
        x = np.empty((n_rows, D))
        for r in range(n_rows):
            for j in range(D // g):
                codes = rng.integers(0, qmax + 1, g)
                lo_at, hi_at = rng.permutation(g)[:2]
                codes[lo_at], codes[hi_at] = 0, qmax
                beta = rng.integers(-12, 12) / 4
                x[r, j * g:(j + 1) * g] = beta + codes / 4
        return x

    kb = grid_rows()             # balanced keys k * b
    v = grid_rows()
    k = kb / balancer[None, :]   # exact: balancer is a power of two
    return torch.tensor(k), torch.tensor(v)


@pytest.mark.parametrize("bits,g", [(2, 32), (3, 64), (4, 32), (4, 128)])
def test_retained_set_lossless_case_is_textbook(bits, g):
    """With K*b and V on an exact Eq. 1 grid the retained set loses nothing; MiKV attention must then
    equal textbook attention over the original keys. Pins dequantization (alpha*c+beta), the balancer
    direction (keys multiplied, query divided) and the union of both sets."""
    rng = np.random.default_rng(bits * 1000 + g)
    B, Hq, Hkv, n_hi, n_lo = 2, 4, 2, 7, 45
    bal = (2.0 ** rng.integers(-2, 3, size=(Hkv, D))).astype(np.float32)
    q = _bf16(torch.tensor(rng.standard_normal((B, Hq, D))))
    k_hi = _bf16(torch.tensor(rng.standard_normal((B, Hkv, n_hi, D))))
    v_hi = _bf16(torch.tensor(rng.standard_normal((B, Hkv, n_hi, D))))
    k_lo = torch.empty(B, Hkv, n_lo, D, dtype=torch.float64)
    v_lo = torch.empty_like(k_lo)
    for b in range(B):
        for h in range(Hkv):
            k_lo[b, h], v_lo[b, h] = _lossless_rows(rng, n_lo, bits, g, bal[h].astype(np.float64))
    assert torch.equal(_bf16(k_lo).double(), k_lo) and torch.equal(_bf16(v_lo).double(), v_lo)
    cache = oracle.empty_cache(B, Hkv, D, bits, g, n_hi, 48)
    cache["k_hi"][:] = bf16_bits(k_hi)
    cache["v_hi"][:] = bf16_bits(v_hi)
    rows = np.tile(np.arange(n_lo, dtype=np.int32), (B, Hkv, 1))
    oracle.quantize_pack(cache, bf16_bits(_bf16(k_lo)), bf16_bits(_bf16(v_lo)), rows, 0, balancer_=bal)
    # the stored codes reproduce the grid exactly
    for b in range(B):
        for h in range(Hkv):
            for t in range(n_lo):
                kh = oracle.dequantize_row(cache["k_codes"][b, h, t], cache["k_params"][b, h, t], bits, g)
                vh = oracle.dequantize_row(cache["v_codes"][b, h, t], cache["v_params"][b, h, t], bits, g)
                np.testing.assert_array_equal(kh, k_lo[b, h, t].numpy() * bal[h])
                np.testing.assert_array_equal(vh, v_lo[b, h, t].numpy())
    scale = 1 / math.sqrt(D)
    out, hl, ml = oracle.decode_attention(cache, bf16_bits(q), n_lo, scale, balancer_=bal)
    k_all = torch.cat([k_hi.double(), k_lo], 2)
    v_all = torch.cat([v_hi.double(), v_lo], 2)
    ref, s = _textbook(q.double(), k_all, v_all, scale)
    np.testing.assert_allclose(out, ref.numpy(), rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(hl, s[..., :n_hi].numpy(), rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(ml[..., 0], s.max(-1).values.numpy(), rtol=1e-12)
    np.testing.assert_allclose(ml[..., 1], torch.exp(s - s.max(-1, keepdim=True).values).sum(-1).numpy(),
                               rtol=1e-11)


def test_permutation_invariance():
    """Sec. 3.4: attention is permutation invariant, so reordering either set changes nothing."""
    rng = np.random.default_rng(5)
    B, Hq, Hkv, n_hi, n_lo, bits, g = 1, 4, 2, 9, 30, 3, 64
    k = _bf16(torch.tensor(rng.standard_normal((B, Hkv, n_hi + n_lo, D))))
    v = _bf16(torch.tensor(rng.standard_normal((B, Hkv, n_hi + n_lo, D))))
    q = bf16_bits(_bf16(torch.tensor(rng.standard_normal((B, Hq, D)))))
    bal = rng.uniform(0.5, 2, (Hkv, D)).astype(np.float32)

    def build(perm_hi, perm_lo):
        c = oracle.empty_cache(B, Hkv, D, bits, g, n_hi, 32)
        c["k_hi"][:] = bf16_bits(k[:, :, perm_hi])
        c["v_hi"][:] = bf16_bits(v[:, :, perm_hi])
        rows = np.tile(np.asarray(perm_lo, np.int32), (B, Hkv, 1))
        oracle.quantize_pack(c, bf16_bits(k), bf16_bits(v), rows, 0, balancer_=bal)
        return oracle.decode_attention(c, q, n_lo, 0.1, balancer_=bal)

    base = build(np.arange(n_hi), np.arange(n_hi, n_hi + n_lo))
    p_hi = rng.permutation(n_hi)
    p_lo = n_hi + rng.permutation(n_lo)
    shuf = build(p_hi, p_lo)
    np.testing.assert_allclose(shuf[0], base[0], rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(shuf[1], base[1][..., p_hi], rtol=1e-12, atol=1e-14)


def test_balancer_is_identity_without_quantization_error():
    """Eq. 3-4 cancel in exact arithmetic: for fixed keys on an exact grid, a power-of-two balancer
    keeps quantization lossless, so attention must not depend on it (a wrong direction, k / b or
    q * b, would change the logits by b^2)."""
    rng = np.random.default_rng(9)
    B, Hq, Hkv, n_lo, bits, g = 1, 2, 1, 20, 2, 32
    k_lo, v_lo = _lossless_rows(np.random.default_rng(3), n_lo, bits, g, np.ones(D))
    q = bf16_bits(_bf16(torch.tensor(rng.standard_normal((B, Hq, D)))))
    outs = []
    for e in (0, 1, -2):
        bal = np.full((Hkv, D), 2.0 ** e, np.float32)
        cache = oracle.empty_cache(B, Hkv, D, bits, g, 1, 32)
        rows = np.arange(n_lo, dtype=np.int32)[None, None]
        oracle.quantize_pack(cache, bf16_bits(_bf16(k_lo)[None, None]), bf16_bits(_bf16(v_lo)[None, None]),
                             rows, 0, balancer_=bal)
        outs.append(oracle.decode_attention(cache, q, n_lo, 0.3, balancer_=bal)[0])
    np.testing.assert_allclose(outs[1], outs[0], rtol=1e-13)
    np.testing.assert_allclose(outs[2], outs[0], rtol=1e-13)
    # and a balancer that is not a power of two only moves the result by quantization error
    bal = np.full((Hkv, D), 1.37, np.float32)
    cache = oracle.empty_cache(B, Hkv, D, bits, g, 1, 32)
    oracle.quantize_pack(cache, bf16_bits(_bf16(k_lo)[None, None]), bf16_bits(_bf16(v_lo)[None, None]),
                         np.arange(n_lo, dtype=np.int32)[None, None], 0, balancer_=bal)
    out = oracle.decode_attention(cache, q, n_lo, 0.3, balancer_=bal)[0]
    assert np.abs(out - outs[0]).max() < 0.5


def test_quantize_pack_rows_and_tokens():
    rng = np.random.default_rng(11)
    B, Hkv, n_src, bits, g = 2, 3, 10, 4, 32
    k = bf16_bits(_bf16(torch.tensor(rng.standard_normal((B, Hkv, n_src, D)))))
    v = bf16_bits(_bf16(torch.tensor(rng.standard_normal((B, Hkv, n_src, D)))))
    tok = rng.integers(0, 10000, (B, Hkv, n_src)).astype(np.int32)
    rows = rng.integers(0, n_src, (B, Hkv, 3)).astype(np.int32)
    c = oracle.empty_cache(B, Hkv, D, bits, g, 1, 16)
    oracle.quantize_pack(c, k, v, rows, 5, src_tok=tok)
    for b in range(B):
        for h in range(Hkv):
            for i in range(3):
                r = rows[b, h, i]
                xk = k[b, h, r].astype(np.uint32) << 16
                packed, params = oracle.quantize_row(xk.view(np.float32), bits, g)
                assert np.array_equal(c["k_codes"][b, h, 5 + i], packed)
                assert np.array_equal(c["k_params"][b, h, 5 + i], params)
                assert c["lo_tok"][b, h, 5 + i] == tok[b, h, r]
    with pytest.raises(ValueError):  # capacity
        oracle.quantize_pack(c, k, v, rows, 14, src_tok=tok)
