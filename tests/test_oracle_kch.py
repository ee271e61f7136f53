"""Pins of the oracle's per-channel retained keys (App. C), CPU only: the group quantizer applies Eq. 1 down
each channel of 64 tokens (orientation checked against the column definition, the alpha/2 error bound,
exact reconstruction of on-grid columns); appending retained rows one at a time gives the same cache as
appending them at once (staging, group completion, token ids); and with every channel of every group on an
exact grid, attention over important, staged and quantized rows equals textbook attention."""
import math

import numpy as np
import pytest
import torch

import oracle
from mikv_inputs import bf16_bits

D = 128


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_channel_group_orientation_and_bound(bits):
    rng = np.random.default_rng(bits)
    x = (rng.standard_normal((64, D)) * rng.uniform(0.1, 10, size=D)).astype(np.float32)  # per-channel scales
    packed, params = oracle.quantize_channel_group(x, bits)
    for c in range(D):
        codes, a16, b16 = oracle.quantize_group(x[:, c], bits)
        assert params[c, 0] == a16 and params[c, 1] == b16
        got = np.array([oracle.unpack_row(packed[t], bits)[c] for t in range(64)])
        np.testing.assert_array_equal(got, codes)
        alpha, beta = oracle.f16_to_f64(int(a16)), oracle.f16_to_f64(int(b16))
        assert np.all(np.abs(alpha * got + beta - x[:, c]) <= alpha / 2 + 1e-6 * np.abs(x[:, c]))


def test_channel_group_on_grid_is_exact():
    rng = np.random.default_rng(5)
    bits = 3
    codes = rng.integers(0, 8, size=(64, D))
    codes[0], codes[1] = 0, 7
    alpha = 2.0 ** rng.integers(-4, 2, size=D)
    beta = rng.integers(-8, 8, size=D) * 0.25
    x = (beta + alpha * codes).astype(np.float32)
    packed, params = oracle.quantize_channel_group(x, bits)
    for t in range(64):
        xh = [oracle.f16_to_f64(int(params[c, 0])) * oracle.unpack_row(packed[t], bits)[c] +
              oracle.f16_to_f64(int(params[c, 1])) for c in range(D)]
        np.testing.assert_array_equal(np.array(xh, np.float32), x[t])


def _bf16(x):
    return bf16_bits(torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16))


def test_append_one_at_a_time_equals_at_once():
    rng = np.random.default_rng(9)
    B, Hkv, n_src, hi_cap, lo_cap = 1, 2, 150, 7, 192
    k = _bf16(rng.standard_normal((B, Hkv, n_src, D)))
    v = _bf16(rng.standard_normal((B, Hkv, n_src, D)))
    rows = np.stack([rng.permutation(n_src)[:140] for _ in range(B * Hkv)]).reshape(B, Hkv, 140).astype(np.int32)
    tok = (1000 + np.arange(n_src, dtype=np.int32))[None, None].repeat(Hkv, 1)
    a = oracle.empty_cache(B, Hkv, D, 2, 32, hi_cap, lo_cap, k_channel=True)
    b = oracle.empty_cache(B, Hkv, D, 2, 32, hi_cap, lo_cap, k_channel=True)
    oracle.append_retained(a, k, v, rows, 0, src_tok=tok)
    oracle.append_retained(b, k, v, rows[..., :61], 0, src_tok=tok)
    for i in range(61, 140):
        oracle.append_retained(b, k, v, rows[..., i:i + 1], i, src_tok=tok)
    for name in ("k_codes", "v_codes", "k_params", "v_params", "lo_tok", "k_hi", "v_hi", "hi_tok"):
        np.testing.assert_array_equal(a[name], b[name], err_msg=name)
    # two complete groups quantized, 12 rows staged, in order
    np.testing.assert_array_equal(a["lo_tok"][..., :128], 1000 + rows[..., :128])
    np.testing.assert_array_equal(a["hi_tok"][..., hi_cap:hi_cap + 12], 1000 + rows[..., 128:140])
    for h in range(Hkv):  # group 1's keys are the per-channel quantization of its 64 rows
        xk = (k[0, h, rows[0, h, 64:128]].astype(np.uint32) << 16).view(np.float32)
        packed, params = oracle.quantize_channel_group(xk, 2)
        np.testing.assert_array_equal(a["k_codes"][0, h, 64:128], packed)
        np.testing.assert_array_equal(a["k_params"][0, h, 1], params)


def test_lossless_per_channel_attention_is_textbook():
    """Keys of every group exactly on a per-channel grid, values on per-token grids, staged and important
    rows in bf16: attention equals textbook softmax attention over all rows."""
    rng = np.random.default_rng(11)
    hi_cap, n_lo, Hq = 5, 64 * 2 + 9, 4
    T = hi_cap + n_lo
    keys = np.zeros((T, D), np.float32)
    vals = np.zeros((T, D), np.float32)
    for grp in range(2):
        codes = rng.integers(0, 4, size=(64, D))
        codes[0], codes[1] = 0, 3
        alpha = 2.0 ** rng.integers(-3, 1, size=D)
        beta = rng.integers(-4, 4, size=D) * 0.5
        keys[hi_cap + 64 * grp:hi_cap + 64 * grp + 64] = beta + alpha * codes
    for t in range(T):  # per-token value grids (group 32): four values per group, both ends present
        for j in range(D // 32):
            c = rng.integers(0, 4, size=32)
            c[0], c[1] = 0, 3
            vals[t, 32 * j:32 * j + 32] = -1.5 + c
    keys[:hi_cap] = rng.standard_normal((hi_cap, D))
    keys[hi_cap + 128:] = rng.standard_normal((9, D))
    kb, vb = _bf16(keys[None, None]), _bf16(vals[None, None])
    kf = (kb[0, 0].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    vf = (vb[0, 0].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    c = oracle.empty_cache(1, 1, D, 2, 32, hi_cap, 192, k_channel=True)
    oracle.gather_hi(c, kb, vb, np.arange(hi_cap, dtype=np.int32).reshape(1, 1, -1))
    oracle.append_retained(c, kb, vb, np.arange(hi_cap, T, dtype=np.int32).reshape(1, 1, -1), 0)
    q = bf16_bits(torch.randn(1, Hq, D, generator=torch.Generator().manual_seed(3)).to(torch.bfloat16))
    out, _, ml = oracle.decode_attention(c, q, n_lo, 1 / math.sqrt(D))
    qf = (q[0].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    s = qf @ kf.T / math.sqrt(D)
    p = np.exp(s - s.max(axis=1, keepdims=True))
    ref = (p / p.sum(axis=1, keepdims=True)) @ vf
    np.testing.assert_allclose(out[0], ref, rtol=1e-12, atol=1e-12)
