"""CPU oracle for the MiKV decode path (arxiv 2402.18096) — TEST INFRASTRUCTURE ONLY.

A plain, slow restatement of what the path computes, written in C (``mikv_oracle.c``) and called
through ctypes with numpy arrays. Only the tests, ``__graft_entry__.smoke()`` and the benchmark's
CPU-baseline / reference legs use it; the product library never imports, links or calls it, and the
two share no code.

Functions follow the paper:
  * ``quantize_group`` / ``quantize_row`` / ``dequantize_row``: Eq. 1 (asymmetric N-bit RTN,
    per token, groups of ``g`` channels, Sec. 3.2 uses g = d/2), fp16 alpha/beta.
  * ``balancer``: Eq. 2 channel balancer; applied to keys before quantization (Eq. 3) and divided
    out of the query (Eq. 4).
  * ``decode_attention``: softmax attention of one new query over the important (bf16) and the
    retained (low-bit) sets, which attention treats as one unordered set (Sec. 3.4).
  * ``update_importance`` / ``select_demote``: accumulated-attention (heavy-hitter) importance policy
    that decides which tokens stay in high precision (Fig. 4, Sec. 3).
  * ``cache_fraction``: the "Cache size" columns of Tables 2-3.
  * caches with ``hi_bits < 16``: the reduced-precision important set of Sec. 3.3 / Table 3
    (important rows quantized like retained rows; demotion re-quantizes their dequantized values).

Readings where the paper is silent are documented in ``mikv_oracle.c`` next to the code.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mikv_oracle.c")
_LIB = os.path.join(_HERE, "_build", "libmikv_oracle.so")
_lock = threading.Lock()
_lib = None

CFLAGS = ["-O2", "-ffp-contract=off", "-fno-fast-math", "-std=c11", "-Wall", "-shared", "-fPIC"]


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (IEEE arithmetic, no contraction, no fast-math)."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    stale = not os.path.exists(_LIB) or os.path.getmtime(_LIB) < max(
        os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "mikv_oracle.h")))
    if force or stale:
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", *CFLAGS, "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P, I, D = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
            sig = {
                "mikv_ref_f32_to_f16": (ctypes.c_uint16, [ctypes.c_float, I]),
                "mikv_ref_f16_to_f64": (D, [ctypes.c_uint16]),
                "mikv_ref_quantize_group": (I, [P, I, I, P, P, P]),
                "mikv_ref_pack_row": (I, [P, I, I, P]),
                "mikv_ref_unpack_row": (I, [P, I, I, P]),
                "mikv_ref_quantize_row": (I, [P, I, I, I, P, P]),
                "mikv_ref_dequantize_row": (I, [P, P, I, I, I, P]),
                "mikv_ref_balancer": (I, [I, I, I, I, I, P, P, P]),
                "mikv_ref_quantize_pack": (I, [I, I, I, I, I, I, P, P, P, I, P, I, I, P, P, P, P, P, P]),
                "mikv_ref_decode_attention": (I, [I, I, I, I, I, I, I, I, I, P, P, P, P, P, P, P, P, D,
                                                  P, P, P]),
                "mikv_ref_update_importance": (I, [I, I, I, I, P, P, P]),
                "mikv_ref_select_demote": (I, [I, I, I, I, P, P, P, P]),
                "mikv_ref_insert_token": (I, [I, I, I, I, P, P, I, P, P, P, P, P]),
                "mikv_ref_gather_hi": (I, [I, I, I, I, P, P, P, P, I, P, I, P, P, P, P]),
                "mikv_ref_cache_fraction": (D, [I, I, D, I]),
                "mikv_ref_budget": (I, [I, D]),
                "mikv_ref_dequantize_row_f32": (I, [P, P, I, I, I, P]),
                "mikv_ref_prefill_scores": (I, [I, I, I, I, I, P, P, D, P]),
                "mikv_ref_quantize_channel_group": (I, [P, I, I, P, P]),
                "mikv_ref_append_retained_kch": (I, [I, I, I, I, I, I, I, I, I, P, P, P, I, P, I, P, P, P, P, P, P, P,
                                                     P]),
                "mikv_ref_decode_attention_kch": (I, [I, I, I, I, I, I, I, I, I, I, P, P, P, P, P, P, P, D, P, P, P]),
                "mikv_ref_gather_hi_q": (I, [I, I, I, I, I, I, P, P, P, P, I, P, I, P, P, P, P, P, P, P]),
                "mikv_ref_insert_token_q": (I, [I, I, I, I, I, I, P, P, I, P, P, P, P, P, P, P, P]),
                "mikv_ref_decode_attention_q": (I, [I, I, I, I, I, I, I, I, I, I, I, P, P, P, P, P, P, P, P,
                                                    P, P, D, P, P, P]),
                "mikv_ref_demote_hi_q": (I, [I, I, I, I, I, I, I, I, I, P, I, P, P, P, P, P, P, P, P, P, P]),
            }
            for name, (res, args) in sig.items():
                fn = getattr(lib, name)
                fn.restype, fn.argtypes = res, args
            _lib = lib
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _arr(a, dtype):
    if a is None:
        return None
    a = np.ascontiguousarray(a)
    if a.dtype != np.dtype(dtype):
        raise TypeError(f"expected {np.dtype(dtype)}, got {a.dtype}")
    return a


def _check(rc, what):
    if rc != 0:
        raise ValueError(f"oracle {what} rejected its arguments")


# ------------------------------------------------------------------ number formats

def f32_to_f16(x: float, mode: int = 0) -> int:
    """fp16 bit pattern of fp32 ``x`` rounded to nearest-even (0), toward -inf (-1) or +inf (+1)."""
    return int(_load().mikv_ref_f32_to_f16(float(np.float32(x)), mode))


def f16_to_f64(h: int) -> float:
    return float(_load().mikv_ref_f16_to_f64(int(h)))


# ------------------------------------------------------------------ Eq. 1

def quantize_group(x, bits: int):
    """Eq. 1 on one group: returns (codes int32[g], alpha16 bits, beta16 bits)."""
    x = _arr(np.asarray(x, dtype=np.float32), np.float32)
    codes = np.zeros(x.size, np.int32)
    a = ctypes.c_uint16()
    b = ctypes.c_uint16()
    _check(_load().mikv_ref_quantize_group(_p(x), x.size, bits, _p(codes), ctypes.byref(a),
                                           ctypes.byref(b)), "quantize_group")
    return codes, int(a.value), int(b.value)


def pack_row(codes, bits: int, d: int = 128):
    codes = _arr(np.asarray(codes, dtype=np.int32), np.int32)
    out = np.zeros(d * bits // 8, np.uint8)
    _check(_load().mikv_ref_pack_row(_p(codes), d, bits, _p(out)), "pack_row")
    return out


def unpack_row(packed, bits: int, d: int = 128):
    packed = _arr(packed, np.uint8)
    out = np.zeros(d, np.int32)
    _check(_load().mikv_ref_unpack_row(_p(packed), d, bits, _p(out)), "unpack_row")
    return out


def quantize_row(x, bits: int, g: int):
    """Quantize + pack one row: returns (packed uint8[16*bits], params uint16[d/g, 2])."""
    x = _arr(np.asarray(x, dtype=np.float32), np.float32)
    d = x.size
    packed = np.zeros(d * bits // 8, np.uint8)
    params = np.zeros((d // g, 2), np.uint16)
    _check(_load().mikv_ref_quantize_row(_p(x), d, bits, g, _p(packed), _p(params)), "quantize_row")
    return packed, params


def dequantize_row(packed, params, bits: int, g: int, d: int = 128):
    packed = _arr(packed, np.uint8)
    params = _arr(params, np.uint16)
    out = np.zeros(d, np.float64)
    _check(_load().mikv_ref_dequantize_row(_p(packed), _p(params), d, bits, g, _p(out)),
           "dequantize_row")
    return out


# ------------------------------------------------------------------ Eq. 2

def balancer(q_pre, k_pre):
    """Eq. 2. q_pre bf16 bits uint16 [B, Hq, T, d], k_pre uint16 [B, Hkv, T, d] -> fp32 [Hkv, d]."""
    q_pre = _arr(q_pre, np.uint16)
    k_pre = _arr(k_pre, np.uint16)
    B, Hq, T, d = q_pre.shape
    Hkv = k_pre.shape[1]
    out = np.zeros((Hkv, d), np.float32)
    _check(_load().mikv_ref_balancer(B, Hq, Hkv, T, d, _p(q_pre), _p(k_pre), _p(out)), "balancer")
    return out


# ------------------------------------------------------------------ cache operations

def quantize_pack(cache: dict, k_src, v_src, rows, lo_start: int, src_tok=None, balancer_=None):
    """Demote rows of k_src/v_src (uint16 bf16 bits [B, Hkv, n_src, d]) into the retained arrays of
    ``cache`` (numpy dict with k_codes, v_codes, k_params, v_params, lo_tok; modified in place)."""
    k_src = _arr(k_src, np.uint16)
    v_src = _arr(v_src, np.uint16)
    rows = _arr(rows, np.int32)
    src_tok = _arr(src_tok, np.int32)
    bal = _arr(balancer_, np.float32)
    B, Hkv, n_src, d = k_src.shape
    n_rows = rows.shape[2]
    kc = cache["k_codes"]
    lo_cap, row_bytes = kc.shape[2], kc.shape[3]
    bits = row_bytes // 16
    g = d // cache["k_params"].shape[3]
    for name in ("k_codes", "v_codes", "k_params", "v_params", "lo_tok"):
        assert cache[name].flags.c_contiguous
    _check(_load().mikv_ref_quantize_pack(
        B, Hkv, d, bits, g, lo_cap, _p(k_src), _p(v_src), _p(src_tok), n_src, _p(rows), n_rows,
        lo_start, _p(bal), _p(cache["k_codes"]), _p(cache["v_codes"]), _p(cache["k_params"]),
        _p(cache["v_params"]), _p(cache["lo_tok"])), "quantize_pack")


def decode_attention(cache: dict, q, n_lo: int, sm_scale: float, balancer_=None):
    """Returns (out f64 [B, Hq, d], hi_logits f64 [B, Hq, hi_cap], ml f64 [B, Hq, 2]).

    cache: numpy dict with k_hi, v_hi (uint16 [B, Hkv, hi_cap, d]), k_codes, v_codes
    (uint8 [B, Hkv, lo_cap, 16*bits]), k_params, v_params (uint16 [B, Hkv, lo_cap, d/g, 2]).
    q: uint16 bf16 bits [B, Hq, d]."""
    if cache.get("hi_bits", 16) < 16:
        return _decode_attention_q(cache, q, n_lo, sm_scale, balancer_)
    if cache.get("kch"):
        return _decode_attention_kch(cache, q, n_lo, sm_scale)
    q = _arr(q, np.uint16)
    B, Hq, d = q.shape
    k_hi = _arr(cache["k_hi"], np.uint16)
    v_hi = _arr(cache["v_hi"], np.uint16)
    Hkv, hi_cap = k_hi.shape[1], k_hi.shape[2]
    kc = _arr(cache["k_codes"], np.uint8)
    vc = _arr(cache["v_codes"], np.uint8)
    kp = _arr(cache["k_params"], np.uint16)
    vp = _arr(cache["v_params"], np.uint16)
    lo_cap, bits = kc.shape[2], kc.shape[3] // 16
    g = d // kp.shape[3]
    bal = _arr(balancer_, np.float32)
    out = np.zeros((B, Hq, d), np.float64)
    hl = np.zeros((B, Hq, hi_cap), np.float64)
    ml = np.zeros((B, Hq, 2), np.float64)
    _check(_load().mikv_ref_decode_attention(
        B, Hq, Hkv, d, bits, g, hi_cap, lo_cap, n_lo, _p(k_hi), _p(v_hi), _p(kc), _p(vc), _p(kp),
        _p(vp), _p(bal), _p(q), float(sm_scale), _p(out), _p(hl), _p(ml)), "decode_attention")
    return out, hl, ml


def _decode_attention_q(cache: dict, q, n_lo: int, sm_scale: float, balancer_=None):
    q = _arr(q, np.uint16)
    B, Hq, d = q.shape
    hb, hg = cache["hi_bits"], cache["hi_group"]
    khc, vhc = _arr(cache["k_hi"], np.uint8), _arr(cache["v_hi"], np.uint8)
    khp, vhp = _arr(cache["k_hp"], np.uint16), _arr(cache["v_hp"], np.uint16)
    Hkv, hi_cap = khc.shape[1], khc.shape[2]
    kc = _arr(cache["k_codes"], np.uint8)
    vc = _arr(cache["v_codes"], np.uint8)
    kp = _arr(cache["k_params"], np.uint16)
    vp = _arr(cache["v_params"], np.uint16)
    lo_cap, bits = kc.shape[2], kc.shape[3] // 16
    g = d // kp.shape[3]
    bal = _arr(balancer_, np.float32)
    out = np.zeros((B, Hq, d), np.float64)
    hl = np.zeros((B, Hq, hi_cap), np.float64)
    ml = np.zeros((B, Hq, 2), np.float64)
    _check(_load().mikv_ref_decode_attention_q(
        B, Hq, Hkv, d, hb, hg, bits, g, hi_cap, lo_cap, n_lo, _p(khc), _p(vhc), _p(khp), _p(vhp), _p(kc),
        _p(vc), _p(kp), _p(vp), _p(bal), _p(q), float(sm_scale), _p(out), _p(hl), _p(ml)), "decode_attention_q")
    return out, hl, ml


def _decode_attention_kch(cache: dict, q, n_lo: int, sm_scale: float):
    """Per-channel retained keys: the important set plus the n_lo mod 64 staged tokens in bf16, the rest of
    the retained set in quantized groups. hi_logits covers the important slots and the staged rows."""
    q = _arr(q, np.uint16)
    B, Hq, d = q.shape
    k_hi = _arr(cache["k_hi"], np.uint16)
    v_hi = _arr(cache["v_hi"], np.uint16)
    Hkv, hi_rows = k_hi.shape[1], k_hi.shape[2]
    n_stage = n_lo % 64
    n_hi, n_lo_q = cache["hi_cap"] + n_stage, n_lo - n_stage
    kc = _arr(cache["k_codes"], np.uint8)
    vc = _arr(cache["v_codes"], np.uint8)
    kp = _arr(cache["k_params"], np.uint16)
    vp = _arr(cache["v_params"], np.uint16)
    lo_cap, bits = kc.shape[2], kc.shape[3] // 16
    g = d // vp.shape[3]
    out = np.zeros((B, Hq, d), np.float64)
    hl = np.zeros((B, Hq, n_hi), np.float64)
    ml = np.zeros((B, Hq, 2), np.float64)
    _check(_load().mikv_ref_decode_attention_kch(
        B, Hq, Hkv, d, bits, g, hi_rows, n_hi, lo_cap, n_lo_q, _p(k_hi), _p(v_hi), _p(kc), _p(vc), _p(kp), _p(vp),
        _p(q), float(sm_scale), _p(out), _p(hl), _p(ml)), "decode_attention_kch")
    return out, hl, ml


def quantize_channel_group(x, bits: int):
    """Per-channel quantization of 64 token rows (App. C): x fp32 [64, 128] -> (packed uint8 [64, 16*bits],
    params uint16 [128, 2] = (alpha16, beta16) per channel)."""
    x = _arr(x, np.float32)
    packed = np.zeros((64, 16 * bits), np.uint8)
    params = np.zeros((128, 2), np.uint16)
    _check(_load().mikv_ref_quantize_channel_group(_p(x), 128, bits, _p(packed), _p(params)), "quantize_channel_group")
    return packed, params


def append_retained(cache: dict, k_src, v_src, rows, n_lo: int, src_tok=None):
    """Per-channel-key cache: append rows rows[b, h, :] of k_src/v_src (uint16 [B, Hkv, n_src, d]) at retained
    positions n_lo.. (staged in bf16; quantized per group of 64 when a group completes)."""
    k_src = _arr(k_src, np.uint16)
    v_src = _arr(v_src, np.uint16)
    rows = _arr(rows, np.int32)
    src_tok = _arr(src_tok, np.int32)
    B, Hkv, n_src, d = k_src.shape
    kc = cache["k_codes"]
    lo_cap, bits = kc.shape[2], kc.shape[3] // 16
    g = d // cache["v_params"].shape[3]
    _check(_load().mikv_ref_append_retained_kch(
        B, Hkv, d, bits, g, cache["hi_cap"], cache["k_hi"].shape[2], lo_cap, n_lo, _p(k_src), _p(v_src), _p(src_tok),
        n_src, _p(rows), rows.shape[2], _p(cache["k_hi"]), _p(cache["v_hi"]), _p(cache["hi_tok"]), _p(cache["k_codes"]),
        _p(cache["v_codes"]), _p(cache["k_params"]), _p(cache["v_params"]), _p(cache["lo_tok"])), "append_retained_kch")


def update_importance(acc, hi_logits, ml, Hq: int):
    """acc fp32 [B, Hkv, hi_cap] (returned updated copy), hi_logits fp32 [B, Hq, hi_cap],
    ml fp32 [B, Hq, 2]."""
    acc = np.array(acc, dtype=np.float32, copy=True, order="C")
    hl = _arr(hi_logits, np.float32)
    ml = _arr(ml, np.float32)
    B, Hkv, hi_cap = acc.shape
    _check(_load().mikv_ref_update_importance(B, Hq, Hkv, hi_cap, _p(hl), _p(ml), _p(acc)),
           "update_importance")
    return acc


def select_demote(scores, n_demote: int, ids=None, want_kept: bool = True):
    """scores fp32 [B, Hkv, n]; returns (demoted int32 [B, Hkv, n_demote], kept or None)."""
    scores = _arr(scores, np.float32)
    ids = _arr(ids, np.int32)
    B, Hkv, n = scores.shape
    dem = np.zeros((B, Hkv, n_demote), np.int32)
    kept = np.zeros((B, Hkv, n - n_demote), np.int32) if want_kept else None
    _check(_load().mikv_ref_select_demote(B, Hkv, n, n_demote, _p(scores), _p(ids), _p(dem),
                                          _p(kept)), "select_demote")
    return dem, kept


def insert_token(cache: dict, k_new, v_new, tok: int, slots, balancer_=None):
    """Write the new token (uint16 [B, Hkv, d]) into slot ``slots[b, h]`` of the important set (quantized,
    keys balanced, when the cache's important set is reduced-precision)."""
    k_new = _arr(k_new, np.uint16)
    v_new = _arr(v_new, np.uint16)
    slots = _arr(slots, np.int32)
    if cache.get("hi_bits", 16) < 16:
        B, Hkv, hi_cap = cache["hi_tok"].shape
        d = k_new.shape[2]
        _check(_load().mikv_ref_insert_token_q(
            B, Hkv, d, hi_cap, cache["hi_bits"], cache["hi_group"], _p(k_new), _p(v_new), tok, _p(slots),
            _p(_arr(balancer_, np.float32)), _p(cache["k_hi"]), _p(cache["v_hi"]), _p(cache["k_hp"]),
            _p(cache["v_hp"]), _p(cache["hi_tok"]), _p(cache["acc"])), "insert_token_q")
        return
    B, Hkv, hi_cap, d = cache["k_hi"].shape
    _check(_load().mikv_ref_insert_token(B, Hkv, d, hi_cap, _p(k_new), _p(v_new), tok, _p(slots),
                                         _p(cache["k_hi"]), _p(cache["v_hi"]), _p(cache["hi_tok"]),
                                         _p(cache["acc"])), "insert_token")


def gather_hi(cache: dict, k_src, v_src, rows, src_tok=None, src_scores=None, balancer_=None):
    """Important-set build: slot i of (b, h) receives source row rows[b, h, i] (quantized, keys balanced,
    for a reduced-precision important set)."""
    k_src = _arr(k_src, np.uint16)
    v_src = _arr(v_src, np.uint16)
    rows = _arr(rows, np.int32)
    src_tok = _arr(src_tok, np.int32)
    src_scores = _arr(src_scores, np.float32)
    B, Hkv, n_src, d = k_src.shape
    hi_cap = cache["hi_tok"].shape[2]
    if cache.get("hi_bits", 16) < 16:
        _check(_load().mikv_ref_gather_hi_q(
            B, Hkv, d, hi_cap, cache["hi_bits"], cache["hi_group"], _p(k_src), _p(v_src), _p(src_tok),
            _p(src_scores), n_src, _p(rows), rows.shape[2], _p(_arr(balancer_, np.float32)), _p(cache["k_hi"]),
            _p(cache["v_hi"]), _p(cache["k_hp"]), _p(cache["v_hp"]), _p(cache["hi_tok"]), _p(cache["acc"])),
            "gather_hi_q")
        return
    _check(_load().mikv_ref_gather_hi(B, Hkv, d, hi_cap, _p(k_src), _p(v_src), _p(src_tok),
                                      _p(src_scores), n_src, _p(rows), rows.shape[2],
                                      _p(cache["k_hi"]), _p(cache["v_hi"]), _p(cache["hi_tok"]),
                                      _p(cache["acc"])), "gather_hi")


def demote_hi(cache: dict, slots, lo_pos: int, balancer_=None):
    """Move important slot ``slots[b, h]`` into retained position ``lo_pos`` (Eq. 1 at the retained
    precision; a bf16 important row gets the balancer on its key first, a reduced-precision one is
    re-quantized from its fp32 dequantized values)."""
    slots = _arr(slots, np.int32)
    B, Hkv, hi_cap = cache["hi_tok"].shape
    if cache.get("hi_bits", 16) >= 16:
        quantize_pack(cache, cache["k_hi"], cache["v_hi"], slots.reshape(B, Hkv, 1), lo_pos, src_tok=cache["hi_tok"],
                      balancer_=balancer_)
        return
    kc = cache["k_codes"]
    d = cache["k_hp"].shape[3] * cache["hi_group"]
    lo_cap, bits = kc.shape[2], kc.shape[3] // 16
    g = d // cache["k_params"].shape[3]
    _check(_load().mikv_ref_demote_hi_q(
        B, Hkv, d, hi_cap, cache["hi_bits"], cache["hi_group"], bits, g, lo_cap, _p(slots), lo_pos,
        _p(cache["k_hi"]), _p(cache["v_hi"]), _p(cache["k_hp"]), _p(cache["v_hp"]), _p(cache["hi_tok"]),
        _p(cache["k_codes"]), _p(cache["v_codes"]), _p(cache["k_params"]), _p(cache["v_params"]),
        _p(cache["lo_tok"])), "demote_hi_q")


def dequantize_row_f32(packed, params, bits: int, g: int, d: int = 128):
    """fp32 dequantization alpha16 * code + beta16 (exact product, one rounding) -> float32 [d]."""
    packed = _arr(packed, np.uint8)
    params = _arr(params, np.uint16)
    out = np.zeros(d, np.float32)
    _check(_load().mikv_ref_dequantize_row_f32(_p(packed), _p(params), d, bits, g, _p(out)), "dequantize_row_f32")
    return out


def prefill_scores(q_pre, k_pre, sm_scale: float):
    """Initial importance from the prefill's causal attention: q_pre uint16 [B, Hq, T, d], k_pre uint16
    [B, Hkv, T, d] (bf16 bits) -> fp64 [B, Hkv, T]."""
    q_pre = _arr(q_pre, np.uint16)
    k_pre = _arr(k_pre, np.uint16)
    B, Hq, T, d = q_pre.shape
    Hkv = k_pre.shape[1]
    out = np.zeros((B, Hkv, T), np.float64)
    _check(_load().mikv_ref_prefill_scores(B, Hq, Hkv, T, d, _p(q_pre), _p(k_pre), float(sm_scale), _p(out)),
           "prefill_scores")
    return out


def cache_fraction(bits: int, g: int, ratio: float, hi_bits: int = 16) -> float:
    return float(_load().mikv_ref_cache_fraction(bits, g, ratio, hi_bits))


def budget(T: int, ratio: float) -> int:
    """Important tokens for importance ratio `ratio` over T tokens (Tables 1-3): nearest integer to
    ratio * T, halves up (reading R10)."""
    k = int(_load().mikv_ref_budget(int(T), float(ratio)))
    if k < 0:
        raise ValueError(f"budget: invalid T={T} or ratio={ratio}")
    return k


def empty_cache(B: int, Hkv: int, d: int, bits: int, g: int, hi_cap: int, lo_cap: int, hi_bits: int = 16,
                hi_group: int = 64, k_channel: bool = False) -> dict:
    """Zero-initialised numpy arrays in the oracle's (dense) layout. With hi_bits < 16 the important set
    holds codes (k_hi, v_hi uint8 [B, Hkv, hi_cap, d*hi_bits/8]) and parameters (k_hp, v_hp). With
    k_channel the retained keys are per channel (App. C): the important arrays carry 64 staging rows
    after the hi_cap slots, and k_params is [B, Hkv, lo_cap/64, d, 2]."""
    if k_channel:
        c = empty_cache(B, Hkv, d, bits, g, hi_cap + 64, lo_cap)
        c.update({"kch": True, "hi_cap": hi_cap, "k_params": np.zeros((B, Hkv, lo_cap // 64, d, 2), np.uint16)})
        return c
    if hi_bits < 16:
        c = empty_cache(B, Hkv, d, bits, g, hi_cap, lo_cap)
        c.update({
            "hi_bits": hi_bits,
            "hi_group": hi_group,
            "k_hi": np.zeros((B, Hkv, hi_cap, d * hi_bits // 8), np.uint8),
            "v_hi": np.zeros((B, Hkv, hi_cap, d * hi_bits // 8), np.uint8),
            "k_hp": np.zeros((B, Hkv, hi_cap, d // hi_group, 2), np.uint16),
            "v_hp": np.zeros((B, Hkv, hi_cap, d // hi_group, 2), np.uint16),
        })
        return c
    return {
        "k_hi": np.zeros((B, Hkv, hi_cap, d), np.uint16),
        "v_hi": np.zeros((B, Hkv, hi_cap, d), np.uint16),
        "hi_tok": np.zeros((B, Hkv, hi_cap), np.int32),
        "acc": np.zeros((B, Hkv, hi_cap), np.float32),
        "k_codes": np.zeros((B, Hkv, lo_cap, d * bits // 8), np.uint8),
        "v_codes": np.zeros((B, Hkv, lo_cap, d * bits // 8), np.uint8),
        "k_params": np.zeros((B, Hkv, lo_cap, d // g, 2), np.uint16),
        "v_params": np.zeros((B, Hkv, lo_cap, d // g, 2), np.uint16),
        "lo_tok": np.zeros((B, Hkv, lo_cap), np.int32),
    }
