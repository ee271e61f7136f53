"""Pins of the oracle's reduced-precision important set (Sec. 3.3, Table 3), CPU only.

Constructions on which Eq. 1 is lossless (every group holds an exact fp16 grid beta + alpha * [0, 2^N - 1]
with both ends present, values exact in bf16, power-of-two balancers) tie the quantized important set to
the bf16 definitions it must reduce to: the same attention, the same demoted retained rows. The fp32
dequantization used by the demotion is checked against the exact value rounded once, and the quantized
important rows against the Eq. 1 error bound.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from mikv_inputs import bf16_bits

D = 128
HG = 64


def _grid_rows(n, bits, g, rng, alpha_exp, beta):
    """[n, D] float32 rows on the grid beta + 2^alpha_exp * c per group of g channels, c in [0, 2^N - 1],
    with codes 0 and 2^N - 1 present in every group."""
    qmax = (1 << bits) - 1
    c = rng.integers(0, qmax + 1, size=(n, D))
    for j in range(D // g):
        c[:, j * g] = 0
        c[:, j * g + 1] = qmax
    return (beta + c * 2.0 ** alpha_exp).astype(np.float32)


GRID = {8: (-5, -2.0), 4: (-2, -2.0), 2: (0, -1.5)}


def _pow2_balancer(rng, Hkv):
    return (2.0 ** rng.integers(-2, 3, size=(Hkv, D))).astype(np.float32)


def _to_bf16_bits(x):
    t = torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16)
    assert torch.equal(t.float(), torch.from_numpy(np.ascontiguousarray(x, np.float32))), "not exact in bf16"
    return bf16_bits(t)


def _lossless_case(hi_bits, n_hi, rng, B=1, Hkv=2):
    """Balanced keys y and values v on the hi_bits grid; stored keys k = y / balancer."""
    e, beta = GRID[hi_bits]
    bal = _pow2_balancer(rng, Hkv)
    y = _grid_rows(B * Hkv * n_hi, hi_bits, HG, rng, e, beta).reshape(B, Hkv, n_hi, D)
    v = _grid_rows(B * Hkv * n_hi, hi_bits, HG, rng, e, beta).reshape(B, Hkv, n_hi, D)
    k = y / bal[None, :, None, :]
    return _to_bf16_bits(k), _to_bf16_bits(v), bal


@pytest.mark.parametrize("hi_bits", [8, 4, 2])
def test_lossless_quantized_important_set_is_the_bf16_attention(hi_bits):
    rng = np.random.default_rng(hi_bits)
    B, Hkv, Hq, n_hi, n_lo, bits, g = 1, 2, 4, 37, 21, 2, 32
    kb, vb, bal = _lossless_case(hi_bits, n_hi, rng, B, Hkv)
    rows = np.tile(np.arange(n_hi, dtype=np.int32), (B, Hkv, 1))
    ref = oracle.empty_cache(B, Hkv, D, bits, g, n_hi, 32)
    oracle.gather_hi(ref, kb, vb, rows)
    quant = oracle.empty_cache(B, Hkv, D, bits, g, n_hi, 32, hi_bits=hi_bits, hi_group=HG)
    oracle.gather_hi(quant, kb, vb, rows, balancer_=bal)
    # identical retained sets on both sides
    klo = bf16_bits(torch.randn(B, Hkv, n_lo, D, generator=torch.Generator().manual_seed(5)).to(torch.bfloat16))
    vlo = bf16_bits(torch.randn(B, Hkv, n_lo, D, generator=torch.Generator().manual_seed(6)).to(torch.bfloat16))
    lrows = np.tile(np.arange(n_lo, dtype=np.int32), (B, Hkv, 1))
    for c in (ref, quant):
        oracle.quantize_pack(c, klo, vlo, lrows, 0, balancer_=bal)
    q = bf16_bits(torch.randn(B, Hq, D, generator=torch.Generator().manual_seed(7)).to(torch.bfloat16))
    o1, hl1, ml1 = oracle.decode_attention(ref, q, n_lo, 1 / math.sqrt(D), balancer_=bal)
    o2, hl2, ml2 = oracle.decode_attention(quant, q, n_lo, 1 / math.sqrt(D), balancer_=bal)
    np.testing.assert_allclose(hl2, hl1, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(o2, o1, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(ml2, ml1, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("hi_bits,bits,g", [(8, 2, 32), (4, 3, 64), (2, 4, 128), (8, 4, 32)])
def test_lossless_demotion_equals_demotion_of_the_bf16_row(hi_bits, bits, g):
    """Demoting a losslessly quantized important row gives the retained row that demoting its bf16
    original (key times the balancer, Eq. 3) gives: codes, parameters and token id bit for bit."""
    rng = np.random.default_rng(10 * hi_bits + bits)
    B, Hkv, n_hi, lo_cap = 2, 2, 9, 8
    kb, vb, bal = _lossless_case(hi_bits, n_hi, rng, B, Hkv)
    rows = np.tile(np.arange(n_hi, dtype=np.int32), (B, Hkv, 1))
    tok = rng.permutation(1000)[:B * Hkv * n_hi].reshape(B, Hkv, n_hi).astype(np.int32)
    ref = oracle.empty_cache(B, Hkv, D, bits, g, n_hi, lo_cap)
    oracle.gather_hi(ref, kb, vb, rows, src_tok=tok)
    quant = oracle.empty_cache(B, Hkv, D, bits, g, n_hi, lo_cap, hi_bits=hi_bits, hi_group=HG)
    oracle.gather_hi(quant, kb, vb, rows, src_tok=tok, balancer_=bal)
    slots = rng.integers(0, n_hi, size=(B, Hkv)).astype(np.int32)
    oracle.demote_hi(ref, slots, 5, balancer_=bal)
    oracle.demote_hi(quant, slots, 5, balancer_=bal)
    for name in ("k_codes", "v_codes", "k_params", "v_params", "lo_tok"):
        assert np.array_equal(quant[name][:, :, 5], ref[name][:, :, 5]), name
    assert np.array_equal(quant["lo_tok"][:, :, 5], np.take_along_axis(tok, slots[..., None], 2)[..., 0])


@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_fp32_dequantization_is_the_exact_value_rounded_once(bits):
    rng = np.random.default_rng(bits)
    for g in (32, 64, 128):
        codes = rng.integers(0, 1 << bits, size=D).astype(np.int32)
        packed = np.zeros(D * bits // 8, np.uint8)
        oracle._check(oracle._load().mikv_ref_pack_row(oracle._p(codes), D, bits, oracle._p(packed)), "pack")
        params = np.zeros((D // g, 2), np.uint16)
        for j in range(D // g):
            params[j, 0] = oracle.f32_to_f16(float(rng.uniform(1e-3, 2.0)))
            params[j, 1] = oracle.f32_to_f16(float(rng.uniform(-8.0, 8.0)))
        exact = np.array([oracle.f16_to_f64(int(params[i // g, 0])) * codes[i] + oracle.f16_to_f64(int(params[i // g, 1]))
                          for i in range(D)])  # fp64 holds these sums exactly
        got = oracle.dequantize_row_f32(packed, params, bits, g)
        assert np.array_equal(got, exact.astype(np.float32))


@pytest.mark.parametrize("hi_bits", [8, 4, 2])
def test_quantized_important_rows_obey_the_eq1_error_bound(hi_bits):
    """Gathered and inserted rows dequantize to within alpha16 / 2 of the balanced key / the value."""
    rng = np.random.default_rng(hi_bits + 40)
    B, Hkv, n = 1, 2, 12
    g = torch.Generator().manual_seed(hi_bits)
    k = torch.randn(B, Hkv, n, D, generator=g).to(torch.bfloat16)
    v = torch.randn(B, Hkv, n, D, generator=g).to(torch.bfloat16)
    bal = (rng.uniform(0.5, 2.0, size=(Hkv, D))).astype(np.float32)
    c = oracle.empty_cache(B, Hkv, D, 2, 32, n, 4, hi_bits=hi_bits, hi_group=HG)
    oracle.gather_hi(c, bf16_bits(k), bf16_bits(v), np.tile(np.arange(n - 1, dtype=np.int32), (B, Hkv, 1)),
                     balancer_=bal)
    oracle.insert_token(c, bf16_bits(k[:, :, n - 1]), bf16_bits(v[:, :, n - 1]), 77,
                        np.full((B, Hkv), n - 1, np.int32), balancer_=bal)
    assert np.all(c["hi_tok"][:, :, n - 1] == 77) and np.all(c["acc"][:, :, n - 1] == 0)
    kf = k.float().numpy() * bal[None, :, None, :].astype(np.float32)
    vf = v.float().numpy()
    for h in range(Hkv):
        for i in range(n):
            for src, codes, params in ((kf, c["k_hi"], c["k_hp"]), (vf, c["v_hi"], c["v_hp"])):
                x = src[0, h, i]
                xh = oracle.dequantize_row(codes[0, h, i], params[0, h, i], hi_bits, HG)
                alpha = np.repeat([oracle.f16_to_f64(int(a)) for a in params[0, h, i, :, 0]], HG)
                assert np.all(np.abs(xh - x) <= alpha / 2 + 1e-6 * np.abs(x)), (h, i)


def test_retained_only_cache_ignores_the_important_format():
    """hi_cap = 0: the reduced-precision and the bf16 important-set paths are the same retained attention."""
    B, Hkv, Hq, n_lo = 1, 1, 2, 19
    g = torch.Generator().manual_seed(3)
    klo = bf16_bits(torch.randn(B, Hkv, n_lo, D, generator=g).to(torch.bfloat16))
    vlo = bf16_bits(torch.randn(B, Hkv, n_lo, D, generator=g).to(torch.bfloat16))
    q = bf16_bits(torch.randn(B, Hq, D, generator=g).to(torch.bfloat16))
    rows = np.arange(n_lo, dtype=np.int32).reshape(1, 1, n_lo)
    outs = []
    for hb in (16, 8):
        c = oracle.empty_cache(B, Hkv, D, 3, 64, 0, n_lo, hi_bits=hb, hi_group=HG)
        oracle.quantize_pack(c, klo, vlo, rows, 0)
        outs.append(oracle.decode_attention(c, q, n_lo, 0.1)[0])
    np.testing.assert_array_equal(outs[0], outs[1])
