"""Host-side checks of the C ABI (no GPU needed): the library builds and loads, exports every function
include/mikv.h declares, validates arguments before launching anything, and its host-only helpers
agree with the paper's memory accounting."""
import ctypes
import json
import math
import os
import re

import pytest

import oracle
import paper_2402_18096_gb300 as pkg

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mikv.h")


@pytest.fixture(scope="module")
def lib():
    return pkg.load()


def _declared():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[a-z_0-9]+\s*\*?\s*(mikv_[a-z_0-9]+)\s*\(", text, re.M)))


def test_exports_every_declared_symbol(lib):
    names = _declared()
    assert len(names) >= 14, names
    for n in ["mikv_quantize_pack", "mikv_decode_attention", "mikv_update_importance", "mikv_select_demote"]:
        assert n in names
    for n in names:
        assert hasattr(lib, n), n
    # every name the header declares is a plain C symbol (no C++ mangling)
    nm = os.popen(f"nm -D --defined-only {pkg._build.LIB}").read()
    for n in names:
        assert re.search(rf"\bT {n}$", nm, re.M), n


def test_status_strings(lib):
    for code in range(7):
        assert pkg.mikv_status_string(code) not in ("", "unknown status")
    assert pkg.mikv_status_string(99) == "unknown status"


def test_cache_fraction_matches_oracle_and_tables(lib):
    for bits in (2, 3, 4, 8):
        for g in (32, 64, 128):
            for r in (0.0, 0.05, 0.2, 0.5, 1.0):
                for hb in (16, 8, 4, 2):
                    assert pkg.mikv_cache_fraction(bits, g, r, hb) == pytest.approx(
                        oracle.cache_fraction(bits, g, r, hb), rel=1e-15)
    with open(os.path.join(ROOT, "tests", "golden", "cache_size_tables.json")) as f:
        for row in json.load(f)["rows"]:
            frac = pkg.mikv_cache_fraction(row["retained_bits"], row["group"], row["ratio"], row["importance_bits"])
            assert math.floor(frac * 100 + 0.5) == row["cache_size_percent"]


def test_row_bytes(lib):
    assert pkg.mikv_retained_row_bytes(2, 32) == 32 + 16
    assert pkg.mikv_retained_row_bytes(3, 64) == 48 + 8
    assert pkg.mikv_retained_row_bytes(4, 128) == 64 + 4
    assert pkg.mikv_retained_row_bytes(2, 48) == 0  # group must divide d


def _shape(**kw):
    s = dict(batch=2, heads_q=8, heads_kv=2, head_dim=128, bits=2, group=32, hi_cap=20, hi_stride=32, lo_cap=64,
             hi_bits=0, hi_group=64, k_channel_group=0)
    s.update(kw)
    return pkg._Shape(*[s[n] for n, _ in pkg._Shape._fields_])


def _fake_cache():
    # never dereferenced: validation rejects or the test stops before any launch
    return pkg._Cache(*([0x10000] * 9 + [None, 0x10000, 0x10000]))


def test_workspace_sizes_monotone(lib):
    s = _shape()
    sizes = [lib.mikv_workspace_bytes(ctypes.byref(s), 0, n) for n in (0, 16, 100, 1000, 5000)]
    assert all(x > 0 for x in sizes)
    assert sizes == sorted(sizes)
    assert lib.mikv_workspace_bytes(ctypes.byref(s), 2, 64) >= lib.mikv_workspace_bytes(ctypes.byref(s), 0, 64)
    assert lib.mikv_workspace_bytes(ctypes.byref(_shape(head_dim=64)), 0, 16) == 0
    assert lib.mikv_workspace_bytes(ctypes.byref(_shape(bits=5)), 0, 16) == 0


@pytest.mark.parametrize("kw,code", [
    (dict(head_dim=64), 2), (dict(bits=5), 2), (dict(bits=8), 2), (dict(group=48), 2),
    (dict(heads_q=6, heads_kv=2), 2), (dict(heads_q=7), 1), (dict(hi_stride=24), 1),
    (dict(lo_cap=60), 1), (dict(batch=0), 1), (dict(hi_stride=16, hi_cap=20), 1),
    (dict(hi_bits=3), 2), (dict(hi_bits=12), 2), (dict(hi_bits=8, hi_group=32), 2), (dict(hi_bits=4, hi_group=128), 2),
    (dict(hi_bits=8), 0), (dict(hi_bits=4), 0), (dict(hi_bits=2), 0), (dict(hi_bits=16, hi_group=0), 0),
    (dict(bits=0, group=7), 0), (dict(bits=-1), 1),
    # per-channel keys: groups of 64 tokens, 64 staging rows after the important slots, bf16 important set
    (dict(k_channel_group=64, hi_stride=96), 0), (dict(k_channel_group=32, hi_stride=96), 2),
    (dict(k_channel_group=64, hi_stride=80), 1), (dict(k_channel_group=64, hi_stride=96, lo_cap=96), 1),
    (dict(k_channel_group=64, hi_stride=96, hi_bits=8), 2), (dict(k_channel_group=64, hi_stride=96, bits=0), 2),
])
def test_shape_validation(lib, kw, code):
    s = _shape(**kw)
    c = _fake_cache()
    if code == 0:  # a valid shape: check it through the pure workspace query instead of launching
        assert lib.mikv_workspace_bytes(ctypes.byref(s), 0, 16) > 0
        return
    rc = lib.mikv_quantize_pack(ctypes.byref(s), ctypes.byref(c), 0x10000, 0x10000, None, 4, 0x10000, 1, 0, None)
    assert rc == code


def test_argument_validation_before_launch(lib):
    s = _shape()
    c = _fake_cache()
    P = 0x10000
    # retained capacity: lo_start + n_rows > lo_cap
    assert lib.mikv_quantize_pack(ctypes.byref(s), ctypes.byref(c), P, P, None, 4, P, 5, 60, None) == 3
    # source rows are read in 16-byte pieces: both sources 16-byte aligned
    assert lib.mikv_quantize_pack(ctypes.byref(s), ctypes.byref(c), P + 8, P, None, 4, P, 1, 0, None) == 1
    assert lib.mikv_quantize_pack(ctypes.byref(s), ctypes.byref(c), P, P + 8, None, 4, P, 1, 0, None) == 1
    # null cache member
    bad = pkg._Cache(*([P] * 8 + [None, None, None, None]))
    assert lib.mikv_quantize_pack(ctypes.byref(s), ctypes.byref(bad), P, P, None, 4, P, 1, 0, None) == 1
    # a coded important set needs its parameter arrays (16-byte aligned)
    sq = _shape(hi_bits=8)
    no_hp = pkg._Cache(*([P] * 9 + [None, None, None]))
    assert lib.mikv_quantize_pack(ctypes.byref(sq), ctypes.byref(no_hp), P, P, None, 4, P, 1, 0, None) == 1
    odd_hp = pkg._Cache(*([P] * 9 + [None, P + 8, P]))
    assert lib.mikv_quantize_pack(ctypes.byref(sq), ctypes.byref(odd_hp), P, P, None, 4, P, 1, 0, None) == 1
    # eviction (bits = 0): there is no retained set to write, and attention takes no retained rows
    se = _shape(bits=0, lo_cap=0)
    no_lo = pkg._Cache(*([P] * 4 + [None] * 8))
    assert lib.mikv_quantize_pack(ctypes.byref(se), ctypes.byref(no_lo), P, P, None, 4, P, 1, 0, None) == 2
    assert lib.mikv_decode_attention(ctypes.byref(se), ctypes.byref(no_lo), 1, P, ctypes.c_float(1.0), P, 0, None, None,
                                     P, 1 << 20, None) == 3
    # attention: n_lo beyond capacity, bad output type, missing or misaligned workspace
    assert lib.mikv_decode_attention(ctypes.byref(s), ctypes.byref(c), 65, P, 1.0, P, 0, None, None, P, 1 << 20,
                                     None) == 3
    assert lib.mikv_decode_attention(ctypes.byref(s), ctypes.byref(c), 3, P, 1.0, P, 7, None, None, P, 1 << 20,
                                     None) == 1
    assert lib.mikv_decode_attention(ctypes.byref(s), ctypes.byref(c), 3, P, 1.0, P, 0, None, None, None, 0,
                                     None) == 5
    assert lib.mikv_decode_attention(ctypes.byref(s), ctypes.byref(c), 3, P, 1.0, P, 0, None, None, P + 8, 1 << 20,
                                     None) == 5
    assert lib.mikv_decode_attention(ctypes.byref(s), ctypes.byref(c), 3, P, 1.0, P, 0, None, None, P, 16,
                                     None) == 5
    # selection: more demoted than entries, stride below n
    assert lib.mikv_select_demote(2, 2, P, None, 10, 10, 11, P, None, None) == 1
    assert lib.mikv_select_demote(2, 2, P, None, 10, 8, 1, P, None, None) == 1
    # step: retained set full
    full = _shape(lo_cap=16)
    assert lib.mikv_decode_step(ctypes.byref(full), ctypes.byref(c), 16, P, P, P, 0, P, 1.0, P, 0, P, 1 << 30,
                                None) == 3
    # gather beyond the important capacity
    assert lib.mikv_gather_hi(ctypes.byref(s), ctypes.byref(c), P, P, None, None, 40, P, 21, None) == 3


def test_budget_on_the_boundary_matches_oracle(lib):
    """mikv_budget (the library's importance-ratio rule) against the oracle's independent budget function over
    every workload, the sweep and a grid of ratios and lengths; invalid arguments give -1."""
    import mikv_inputs as mi
    cases = [(w.context, w.ratio) for w in mi.WORKLOADS.values()]
    cases += [(T, r / 100) for T in (0, 1, 2, 3, 10, 257, 512, 611, 999, 4096, 8192, 32768) for r in range(101)]
    for T, r in cases:
        assert pkg.mikv_budget(T, r) == oracle.budget(T, r), (T, r)
    for T, r in ((-1, 0.5), (10, -0.01), (10, 1.01), (10, float("nan"))):
        assert lib.mikv_budget(T, r) == -1


def test_shape_for_context_capacities(lib):
    """The cache shape derived from a context and a ratio: hi_cap = budget + 1, hi_stride a multiple of 16, and
    retained capacity for the rest of the context plus the requested steps (multiple of 16; 64 with per-channel
    keys)."""
    for T, r in ((32768, 0.2), (4096, 0.0), (100, 1.0), (611, 0.15)):
        for steps in (0, 1, 17, 100):
            for kcg in (0, 64):
                s = pkg.shape_for_context(2, 8, 2, 2, 32, T, r, steps, k_channel_group=kcg)
                k = oracle.budget(T, r)
                assert s.hi_cap == k + 1 and s.hi_stride % 16 == 0 and s.hi_stride >= s.hi_cap + (64 if kcg else 0)
                q = 64 if kcg else 16
                assert s.lo_cap % q == 0 and s.lo_cap >= T - k + steps and s.lo_cap >= q