"""Pins of the oracle's Eq. 1 quantizer, fp16 rounding and bit packing (CPU only).

Each check ties the oracle to something other than itself: the IEEE fp16 value table (brute force),
numpy's own float32 -> float16 conversion, exact rational arithmetic (fractions), hand-worked Eq. 1
examples and the layout text of the ABI header.
"""
from fractions import Fraction

import numpy as np
import pytest

import oracle

ALL_F16 = np.arange(0, 1 << 16, dtype=np.uint32).astype(np.uint16).view(np.float16)
FINITE_F16 = np.unique(ALL_F16[np.isfinite(ALL_F16)].astype(np.float64))  # sorted, -0 merged


def _rd(x: float) -> float:
    """Largest finite fp16 value <= x (brute force over the table)."""
    i = np.searchsorted(FINITE_F16, x, side="right") - 1
    return float(FINITE_F16[i])


def _ru(x: float) -> float:
    i = np.searchsorted(FINITE_F16, x, side="left")
    return float(FINITE_F16[i])


def _val(h: int) -> float:
    return float(np.array([h], np.uint16).view(np.float16)[0])


# ------------------------------------------------------------------ fp16 conversion

def test_f16_round_nearest_matches_numpy():
    rng = np.random.default_rng(1)
    xs = np.concatenate([rng.standard_normal(4000).astype(np.float32) * 10,
                         rng.standard_normal(2000).astype(np.float32) * 1e-5,   # subnormals
                         np.float32([65519.0, 65520.0, 65504.0, -65520.0, 6.1e-5, 5.96e-8, 2.98e-8])])
    for x in xs:
        with np.errstate(over="ignore"):
            want = int(np.float16(x).view(np.uint16))
        got = oracle.f32_to_f16(x, 0)
        assert got == want or (np.isnan(_val(got)) and np.isnan(_val(want))), (x, got, want)


def test_f16_directed_rounding_brute_force():
    rng = np.random.default_rng(2)
    xs = np.concatenate([rng.standard_normal(3000).astype(np.float32) * 37,
                         rng.standard_normal(1000).astype(np.float32) * 1e-6,
                         np.float32([0.1, -0.1, 1.0, -1.0, 1.0009765625, 65504.0, -65504.0, 3.0e-8])])
    for x in xs:
        x = float(np.float32(x))
        assert _val(oracle.f32_to_f16(x, -1)) == _rd(x), x
        assert _val(oracle.f32_to_f16(x, +1)) == _ru(x), x


def test_f16_to_f64_all_patterns():
    for h in range(0, 1 << 16, 7):
        want = ALL_F16[h].astype(np.float64)
        got = oracle.f16_to_f64(h)
        assert (np.isnan(want) and np.isnan(got)) or want == got


# ------------------------------------------------------------------ Eq. 1 worked by hand

def test_eq1_hand_examples():
    # x in {0, 1, 2, 3}, N = 2: alpha = (3 - 0) / 3 = 1, beta = 0, codes equal the values.
    codes, a, b = oracle.quantize_group([0.0, 1.0, 2.0, 3.0], 2)
    assert list(codes) == [0, 1, 2, 3] and _val(a) == 1.0 and _val(b) == 0.0
    # Half-way values round to even: (0.5 - 0)/1 -> 0, 1.5 -> 2, 2.5 -> 2.
    codes, a, b = oracle.quantize_group([0.0, 0.5, 1.5, 2.5, 3.0], 2)
    assert list(codes) == [0, 0, 2, 2, 3]
    # N = 4, x = -1 .. 14 step 1: alpha = 15 / 15 = 1, beta = -1, code = x + 1.
    x = np.arange(-1.0, 15.0)
    codes, a, b = oracle.quantize_group(x, 4)
    assert list(codes) == list(range(16)) and _val(a) == 1.0 and _val(b) == -1.0
    # N = 3 on [2, 9]: alpha = 7 / 7 = 1, beta = 2.
    codes, a, b = oracle.quantize_group([9.0, 2.0, 5.25, 5.75], 3)
    assert list(codes) == [7, 0, 3, 4] and _val(b) == 2.0
    # Constant group of an fp16 value: zero span, every code 0, alpha 1.0 by definition.
    codes, a, b = oracle.quantize_group([1.5] * 8, 2)
    assert list(codes) == [0] * 8 and _val(a) == 1.0 and _val(b) == 1.5
    # beta is the minimum rounded DOWN to fp16: min = 0.1 -> 0.0999755859375.
    codes, a, b = oracle.quantize_group([0.1, 0.2], 2)
    assert _val(b) == _rd(float(np.float32(0.1))) and _val(b) <= float(np.float32(0.1))


# ------------------------------------------------------------------ Eq. 1 brute force

@pytest.mark.parametrize("bits", [2, 3, 4, 8])
@pytest.mark.parametrize("g", [4, 32, 64])
def test_eq1_brute_force(bits, g):
    rng = np.random.default_rng(100 + bits * 10 + g)
    qmax = (1 << bits) - 1
    for trial in range(40):
        scale = [1.0, 10.0, 1e-3, 300.0][trial % 4]
        x = (rng.standard_normal(g) * scale).astype(np.float32)
        if trial % 5 == 0:
            x[rng.integers(g)] *= 10  # an outlier in the group
        codes, a16, b16 = oracle.quantize_group(x, bits)
        alpha, beta = _val(a16), _val(b16)
        mn, mx = float(x.min()), float(x.max())
        # beta: the largest fp16 not above the minimum
        assert beta == _rd(mn)
        # alpha: the smallest fp16 not below the fp32 quotient (max - beta) / (2^N - 1)
        quot = float(np.float32(np.float32(mx) - np.float32(beta)) / np.float32(qmax))
        assert alpha == _ru(quot)
        assert alpha > 0
        # every code is the nearest grid point (exact rational arithmetic); ties go to even
        A, Bt = Fraction(alpha), Fraction(beta)
        for xi, c in zip(x, codes):
            X = Fraction(float(xi))
            dists = [abs(X - (A * k + Bt)) for k in range(qmax + 1)]
            best = min(dists)
            winners = [k for k, dd in enumerate(dists) if dd == best]
            if c not in winners:
                # only an fp32 rounding of the quotient can move a code off the nearest point: the
                # exact position must then sit within fp32 rounding of a half-way point
                pos = (X - Bt) / A
                assert abs(pos - (Fraction(c) + Fraction(winners[0])) / 2) < Fraction(1, 1 << 20), (xi, c)
            elif len(winners) == 2:
                assert c % 2 == 0
        # error bound implied by Eq. 1 with a covering grid: |x - x_hat| <= alpha / 2
        xhat = alpha * codes.astype(np.float64) + beta
        assert np.all(np.abs(x.astype(np.float64) - xhat) <= alpha / 2 * (1 + 1e-6) + 1e-30)


def test_eq1_grid_covers_range():
    rng = np.random.default_rng(7)
    for bits in (2, 3, 4):
        for _ in range(200):
            x = (rng.standard_normal(32) * rng.choice([0.01, 1, 50])).astype(np.float32)
            _, a16, b16 = oracle.quantize_group(x, bits)
            alpha, beta = _val(a16), _val(b16)
            top = beta + ((1 << bits) - 1) * alpha
            assert beta <= x.min() and top >= float(x.max()) * (1 - 1e-6) - 1e-6 * abs(top)


# ------------------------------------------------------------------ packing

@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_pack_roundtrip(bits):
    rng = np.random.default_rng(bits)
    for _ in range(50):
        codes = rng.integers(0, 1 << bits, 128).astype(np.int32)
        packed = oracle.pack_row(codes, bits)
        assert packed.size == 16 * bits
        assert np.array_equal(oracle.unpack_row(packed, bits), codes)


def test_pack_layout_hand_examples():
    """Bytes worked out by hand from the layout text of include/mikv.h."""
    def one(bits, c, code):
        codes = np.zeros(128, np.int32)
        codes[c] = code
        return oracle.pack_row(codes, bits)

    # N = 2: channel c = 16 m + u lives in unit u at bits [2m, 2m+2).
    p = one(2, 0, 3)                     # u 0, m 0 -> byte 0 bits 0-1
    assert p[0] == 0x03 and p.sum() == 3
    p = one(2, 17, 2)                    # u 1, m 1 -> unit 1 bits 2-3 -> byte 2 = 0x08
    assert p[2] == 0x08 and p.sum() == 8
    p = one(2, 127, 1)                   # u 15, m 7 -> unit 15 bit 14 -> byte 31 = 0x40
    assert p[31] == 0x40 and p.sum() == 0x40
    # N = 4: P = 4; unit 8*(2*(m//4) + u//8) + u%8, bits 4*(m%4).
    p = one(4, 16 * 5 + 9, 0xA)          # m 5, u 9 -> unit 8*(2+1)+1 = 25, bits 4..7 -> byte 50 = 0xA0
    assert p[50] == 0xA0 and int(p.sum()) == 0xA0
    p = one(4, 16 * 2 + 3, 0x7)          # m 2, u 3 -> unit 3, bits 8..11 -> byte 7 = 0x07
    assert p[7] == 0x07 and int(p.sum()) == 7
    # N = 3: 2-bit plane (32 bytes) then 1-bit plane: bit of c in unit u%8 at bit 2*m + u//8.
    p = one(3, 16 * 6 + 12, 0b101)      # low bits 01 -> unit 12 bits 12-13 -> byte 25 = 0x10;
    assert p[25] == 0x10                 # bit 2 -> plane 2 unit 4, bit 2*6 + 1 = 13 -> byte 32+9 bit 5 = 0x20
    assert p[41] == 0x20 and int(p.sum()) == 0x30
    p = one(3, 16 * 3 + 5, 0b110)       # low bits 10 -> unit 5 bits 6-7 -> byte 10 = 0x80;
    assert p[10] == 0x80                 # bit 2 -> plane 2 unit 5, bit 2*3 + 0 = 6 -> byte 32+10 = 0x40
    assert p[42] == 0x40 and int(p.sum()) == 0xC0
    # N = 8: P = 2; unit 8*(2*(m//2) + u//8) + u%8, bits 8*(m%2).
    p = one(8, 16 * 3 + 8, 0xC3)         # m 3, u 8 -> unit 8*(2+1)+0 = 24, high byte -> byte 49
    assert p[49] == 0xC3 and int(p.sum()) == 0xC3


@pytest.mark.parametrize("bits,g", [(2, 32), (3, 64), (4, 32), (2, 128), (4, 128)])
def test_quantize_dequantize_row(bits, g):
    rng = np.random.default_rng(bits * g)
    for _ in range(20):
        x = (rng.standard_normal(128) * 3).astype(np.float32)
        packed, params = oracle.quantize_row(x, bits, g)
        xhat = oracle.dequantize_row(packed, params, bits, g)
        for j in range(128 // g):
            codes, a16, b16 = oracle.quantize_group(x[j * g:(j + 1) * g], bits)
            assert params[j, 0] == a16 and params[j, 1] == b16
            np.testing.assert_array_equal(xhat[j * g:(j + 1) * g], _val(a16) * codes + _val(b16))
            assert np.all(np.abs(xhat[j * g:(j + 1) * g] - x[j * g:(j + 1) * g]) <= _val(a16) / 2 * (1 + 1e-6))


def test_rejects_unsupported():
    with pytest.raises(ValueError):
        oracle.pack_row(np.zeros(64, np.int32), 2, d=64)
    with pytest.raises(ValueError):
        oracle.pack_row(np.zeros(128, np.int32), 5)
