"""GB300 (sm_103a) decode path of MiKV — importance-aware mixed-precision KV cache (arxiv 2402.18096).

Thin Python binding of ``libmikv.so`` (C ABI in ``include/mikv.h``). Functions carry the C names and
only marshal arguments: torch tensors supply device memory, ``torch.cuda.current_stream()`` supplies
the stream, and every computation runs in the library's CUDA kernels. There is no CPU path: if the
library is not built or no GPU is present, calls raise.
"""
from __future__ import annotations

import ctypes
import math
import os
import threading
from dataclasses import dataclass

import torch

from . import build as _build

__all__ = [
    "MikvError", "Shape", "LayerCache", "load", "mikv_status_string", "mikv_workspace_bytes",
    "mikv_workspace_reset", "mikv_workspace_check", "mikv_compute_balancer", "mikv_quantize_pack",
    "mikv_decode_attention", "mikv_update_importance", "mikv_select_demote", "mikv_insert_token",
    "mikv_gather_hi", "mikv_decode_step", "mikv_cache_fraction", "mikv_retained_row_bytes",
    "mikv_decode_attention_noalloc", "mikv_noalloc_check", "NOALLOC_SCRATCH_BYTES", "mikv_prefill_scores",
    "mikv_budget", "shape_for_context", "mikv_debug_check", "debug_build",
    "WS_ATTENTION", "WS_BALANCER", "WS_STEP", "WS_PREFILL", "OUT_BF16", "OUT_F32", "HEAD_DIM",
]

HEAD_DIM = 128
OUT_BF16, OUT_F32 = 0, 1
WS_ATTENTION, WS_BALANCER, WS_STEP, WS_PREFILL = 0, 1, 2, 3
STATUS = {0: "MIKV_OK", 1: "MIKV_ERR_ARG", 2: "MIKV_ERR_UNSUPPORTED", 3: "MIKV_ERR_CAPACITY",
          4: "MIKV_ERR_CUDA", 5: "MIKV_ERR_WORKSPACE", 6: "MIKV_ERR_DEVICE", 7: "MIKV_ERR_SCRATCH"}
NOALLOC_SCRATCH_BYTES = 8 << 20


class MikvError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn}: {STATUS.get(code, code)}")
        self.code = code
        self.status = STATUS.get(code, str(code))


class _Shape(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("batch", "heads_q", "heads_kv", "head_dim", "bits", "group", "hi_cap", "hi_stride", "lo_cap",
                 "hi_bits", "hi_group", "k_channel_group")]


class _Cache(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("k_hi", "v_hi", "hi_tok", "acc", "k_codes", "v_codes", "k_params", "v_params", "lo_tok",
                 "balancer", "k_hi_params", "v_hi_params")]


_lib = None
_lock = threading.Lock()


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load libmikv.so (building it with nvcc first when it is missing or stale). With MIKV_DEBUG=1 in the
    environment the checked build (libmikv_debug.so, -DMIKV_DEBUG) is loaded instead."""
    global _lib
    with _lock:
        if _lib is None:
            debug = os.environ.get("MIKV_DEBUG", "") == "1"
            path = _build.LIB_DEBUG if debug else _build.LIB
            if build_if_missing and not _build.up_to_date(debug):
                _build.build(debug=debug)
            if not os.path.exists(path):
                raise RuntimeError(f"libmikv is not built ({path}); run paper_2402_18096_gb300.build")
            lib = ctypes.CDLL(path)
            P, I, Z, F = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t, ctypes.c_float
            SP = ctypes.POINTER(_Shape)
            CP = ctypes.POINTER(_Cache)
            sig = {
                "mikv_status_string": (ctypes.c_char_p, [I]),
                "mikv_workspace_bytes": (Z, [SP, I, I]),
                "mikv_workspace_reset": (I, [P, Z, P]),
                "mikv_workspace_check": (I, [P, P]),
                "mikv_compute_balancer": (I, [SP, P, P, I, P, P, Z, P]),
                "mikv_quantize_pack": (I, [SP, CP, P, P, P, I, P, I, I, P]),
                "mikv_decode_attention": (I, [SP, CP, I, P, F, P, I, P, P, P, Z, P]),
                "mikv_update_importance": (I, [SP, CP, P, P, P]),
                "mikv_select_demote": (I, [I, I, P, P, I, I, I, P, P, P]),
                "mikv_insert_token": (I, [SP, CP, P, P, I, P, P]),
                "mikv_gather_hi": (I, [SP, CP, P, P, P, P, I, P, I, P]),
                "mikv_decode_step": (I, [SP, CP, I, P, P, P, I, P, F, P, I, P, Z, P]),
                "mikv_decode_attention_noalloc": (I, [SP, CP, I, P, F, P, I, P, P, P]),
                "mikv_noalloc_check": (I, [P]),
                "mikv_budget": (I, [I, ctypes.c_double]),
                "mikv_debug_enabled": (I, []),
                "mikv_debug_check": (I, [P]),
                "mikv_prefill_scores": (I, [SP, P, P, I, F, P, P, Z, P]),
                "mikv_cache_fraction": (ctypes.c_double, [I, I, ctypes.c_double, I]),
                "mikv_retained_row_bytes": (Z, [I, I, I]),
            }
            for name, (res, args) in sig.items():
                fn = getattr(lib, name)
                fn.restype, fn.argtypes = res, args
            _lib = lib
    return _lib


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("libmikv takes device tensors")
    if not t.is_contiguous():
        raise ValueError("libmikv takes contiguous tensors")
    return t.data_ptr()


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _check(name, rc):
    if rc != 0:
        raise MikvError(name, rc)


@dataclass(frozen=True)
class Shape:
    """mikv_shape: one layer's cache geometry."""
    batch: int
    heads_q: int
    heads_kv: int
    bits: int
    group: int
    hi_cap: int
    lo_cap: int
    head_dim: int = HEAD_DIM
    hi_bits: int = 16   # important-set precision: 16 = bf16; 8, 4, 2 = codes (Sec. 3.3, Table 3)
    hi_group: int = 64  # channels per group of a coded important set
    k_channel_group: int = 0  # 64: retained keys per channel over groups of 64 tokens (App. C)

    @property
    def hi_stride(self) -> int:
        # per-channel keys: 64 staging rows of retained tokens follow the important slots
        return (self.hi_cap + (64 if self.k_channel_group else 0) + 15) // 16 * 16

    @property
    def hi_coded(self) -> bool:
        return self.hi_bits not in (0, 16)

    def c(self) -> _Shape:
        return _Shape(self.batch, self.heads_q, self.heads_kv, self.head_dim, self.bits, self.group,
                      self.hi_cap, self.hi_stride, self.lo_cap, self.hi_bits, self.hi_group, self.k_channel_group)


def shape_for_context(batch: int, heads_q: int, heads_kv: int, bits: int, group: int, context: int, ratio: float,
                      steps: int, hi_bits: int = 16, k_channel_group: int = 0) -> Shape:
    """Shape of a cache built from `context` prefill tokens with importance ratio `ratio`: k = mikv_budget(
    context, ratio) important tokens (hi_cap = k + 1 slots) and room for the other context - k tokens plus
    `steps` decode steps in the retained set (a multiple of 16 rows; of 64 with per-channel keys)."""
    k = mikv_budget(context, ratio)
    q = 64 if k_channel_group else 16
    lo_cap = max(q, (context - k + steps + q - 1) // q * q)
    return Shape(batch, heads_q, heads_kv, bits, group, k + 1, lo_cap, hi_bits=hi_bits,
                 k_channel_group=k_channel_group)


class LayerCache:
    """Device arrays of one layer's mixed-precision cache (allocated by torch; layouts of mikv_cache)."""

    def __init__(self, shape: Shape, device="cuda", balancer: torch.Tensor = None):
        s = shape
        B, H, d = s.batch, s.heads_kv, s.head_dim
        self.shape = s
        z = dict(device=device)
        if s.hi_coded:  # codes of balanced keys / values plus (alpha, beta) per group
            self.k_hi = torch.zeros(B, H, s.hi_stride, 16 * s.hi_bits, dtype=torch.uint8, **z)
            self.v_hi = torch.zeros(B, H, s.hi_stride, 16 * s.hi_bits, dtype=torch.uint8, **z)
            self.k_hi_params = torch.zeros(B, H, s.hi_stride, d // s.hi_group, 2, dtype=torch.float16, **z)
            self.v_hi_params = torch.zeros(B, H, s.hi_stride, d // s.hi_group, 2, dtype=torch.float16, **z)
        else:
            self.k_hi = torch.zeros(B, H, s.hi_stride, d, dtype=torch.bfloat16, **z)
            self.v_hi = torch.zeros(B, H, s.hi_stride, d, dtype=torch.bfloat16, **z)
            self.k_hi_params = self.v_hi_params = None
        self.hi_tok = torch.zeros(B, H, s.hi_stride, dtype=torch.int32, **z)
        self.acc = torch.zeros(B, H, s.hi_stride, dtype=torch.float32, **z)
        # (bits = 0: eviction, no retained set; its arrays are empty)
        self.k_codes = torch.zeros(B, H, s.lo_cap, 16 * s.bits, dtype=torch.uint8, **z)
        self.v_codes = torch.zeros(B, H, s.lo_cap, 16 * s.bits, dtype=torch.uint8, **z)
        npar = d // s.group if s.bits else 0
        if s.k_channel_group:  # one (alpha, beta) per channel and group of 64 retained tokens
            self.k_params = torch.zeros(B, H, s.lo_cap // s.k_channel_group, d, 2, dtype=torch.float16, **z)
        else:
            self.k_params = torch.zeros(B, H, s.lo_cap, npar, 2, dtype=torch.float16, **z)
        self.v_params = torch.zeros(B, H, s.lo_cap, npar, 2, dtype=torch.float16, **z)
        self.lo_tok = torch.zeros(B, H, s.lo_cap, dtype=torch.int32, **z)
        self.balancer = balancer
        self.n_lo = 0

    def c(self) -> _Cache:
        return _Cache(*[_ptr(getattr(self, n)) for n in
                        ("k_hi", "v_hi", "hi_tok", "acc", "k_codes", "v_codes", "k_params", "v_params",
                         "lo_tok", "balancer", "k_hi_params", "v_hi_params")])

    def nbytes_attended(self, n_lo: int) -> int:
        """Bytes of cache one decode attention reads: hi_cap important K/V rows + n_lo retained rows."""
        s = self.shape
        row_lo = 2 * mikv_retained_row_bytes(s.bits, s.group, s.head_dim)
        row_hi = 2 * mikv_retained_row_bytes(s.hi_bits, s.hi_group, s.head_dim) if s.hi_coded else 4 * s.head_dim
        if s.k_channel_group:  # keys: codes per token plus 4 bytes per channel per 64 tokens; staged rows bf16
            g = s.k_channel_group
            row_lo = 2 * s.head_dim * s.bits // 8 + 4 * s.head_dim // s.group + 4 * s.head_dim // g
            return s.batch * s.heads_kv * (s.hi_cap * row_hi + n_lo // g * g * row_lo + n_lo % g * row_hi)
        return s.batch * s.heads_kv * (s.hi_cap * row_hi + n_lo * row_lo)


# ------------------------------------------------------------------ C-ABI functions

def mikv_status_string(code: int) -> str:
    return load().mikv_status_string(code).decode()


def mikv_workspace_bytes(shape: Shape, op: int, n_lo_max: int) -> int:
    return int(load().mikv_workspace_bytes(ctypes.byref(shape.c()), op, n_lo_max))


def mikv_workspace_reset(workspace: torch.Tensor, stream=None):
    _check("mikv_workspace_reset", load().mikv_workspace_reset(_ptr(workspace), workspace.numel(), _stream(stream)))


def mikv_workspace_check(workspace: torch.Tensor, stream=None):
    _check("mikv_workspace_check", load().mikv_workspace_check(_ptr(workspace), _stream(stream)))


def mikv_compute_balancer(shape: Shape, q_pre, k_pre, out, workspace, stream=None):
    T = q_pre.shape[2]
    _check("mikv_compute_balancer", load().mikv_compute_balancer(
        ctypes.byref(shape.c()), _ptr(q_pre), _ptr(k_pre), T, _ptr(out), _ptr(workspace), workspace.numel(),
        _stream(stream)))


def mikv_quantize_pack(cache: LayerCache, k_src, v_src, rows, lo_start: int, src_tok=None, stream=None):
    n_src = k_src.shape[2]
    _check("mikv_quantize_pack", load().mikv_quantize_pack(
        ctypes.byref(cache.shape.c()), ctypes.byref(cache.c()), _ptr(k_src), _ptr(v_src), _ptr(src_tok), n_src,
        _ptr(rows), rows.shape[-1], lo_start, _stream(stream)))


def mikv_decode_attention(cache: LayerCache, n_lo: int, q, sm_scale: float, out, workspace,
                          hi_logits=None, ml=None, stream=None):
    out_dtype = OUT_F32 if out.dtype == torch.float32 else OUT_BF16
    _check("mikv_decode_attention", load().mikv_decode_attention(
        ctypes.byref(cache.shape.c()), ctypes.byref(cache.c()), n_lo, _ptr(q), float(sm_scale), _ptr(out),
        out_dtype, _ptr(hi_logits), _ptr(ml), _ptr(workspace), workspace.numel(), _stream(stream)))


def mikv_decode_attention_noalloc(cache: LayerCache, n_lo: int, q, sm_scale: float, out, hi_logits=None,
                                  ml=None, stream=None):
    """mikv_decode_attention with the library's built-in scratch buffer instead of a workspace; for
    callers that may not allocate device memory. Calls must not overlap on the GPU (one shared buffer)."""
    out_dtype = OUT_F32 if out.dtype == torch.float32 else OUT_BF16
    _check("mikv_decode_attention_noalloc", load().mikv_decode_attention_noalloc(
        ctypes.byref(cache.shape.c()), ctypes.byref(cache.c()), n_lo, _ptr(q), float(sm_scale), _ptr(out),
        out_dtype, _ptr(hi_logits), _ptr(ml), _stream(stream)))


def mikv_noalloc_check(stream=None):
    """Raise MikvError(MIKV_ERR_DEVICE) if the last mikv_decode_attention_noalloc call's kernels reported a
    failure in the built-in buffer's status word (synchronises the stream)."""
    _check("mikv_noalloc_check", load().mikv_noalloc_check(_stream(stream)))


def debug_build() -> bool:
    """Whether the loaded library is the checked build (-DMIKV_DEBUG)."""
    return bool(load().mikv_debug_enabled())


def mikv_debug_check(stream=None):
    """Raise MikvError(MIKV_ERR_DEVICE) if a kernel of a checked build found an out-of-range index since the last
    call (entry points without a workspace); clears the word. A release build always passes."""
    _check("mikv_debug_check", load().mikv_debug_check(_stream(stream)))


def mikv_update_importance(cache: LayerCache, hi_logits, ml, stream=None):
    _check("mikv_update_importance", load().mikv_update_importance(
        ctypes.byref(cache.shape.c()), ctypes.byref(cache.c()), _ptr(hi_logits), _ptr(ml), _stream(stream)))


def mikv_select_demote(scores, n: int, n_demote: int, demoted, kept=None, ids=None, stream=None):
    B, H, stride = scores.shape
    _check("mikv_select_demote", load().mikv_select_demote(
        B, H, _ptr(scores), _ptr(ids), n, stride, n_demote, _ptr(demoted), _ptr(kept), _stream(stream)))


def mikv_insert_token(cache: LayerCache, k_new, v_new, tok: int, slots, stream=None):
    _check("mikv_insert_token", load().mikv_insert_token(
        ctypes.byref(cache.shape.c()), ctypes.byref(cache.c()), _ptr(k_new), _ptr(v_new), tok, _ptr(slots),
        _stream(stream)))


def mikv_gather_hi(cache: LayerCache, k_src, v_src, rows, src_tok=None, src_scores=None, stream=None):
    _check("mikv_gather_hi", load().mikv_gather_hi(
        ctypes.byref(cache.shape.c()), ctypes.byref(cache.c()), _ptr(k_src), _ptr(v_src), _ptr(src_tok),
        _ptr(src_scores), k_src.shape[2], _ptr(rows), rows.shape[-1], _stream(stream)))


def mikv_decode_step(cache: LayerCache, n_lo: int, q, k_new, v_new, tok: int, slots, sm_scale: float, out,
                     workspace, stream=None):
    out_dtype = OUT_F32 if out.dtype == torch.float32 else OUT_BF16
    _check("mikv_decode_step", load().mikv_decode_step(
        ctypes.byref(cache.shape.c()), ctypes.byref(cache.c()), n_lo, _ptr(q), _ptr(k_new), _ptr(v_new), tok,
        _ptr(slots), float(sm_scale), _ptr(out), out_dtype, _ptr(workspace), workspace.numel(), _stream(stream)))


def mikv_prefill_scores(shape: Shape, q_pre, k_pre, scores, workspace, sm_scale: float = None, stream=None):
    """Initial importance of the prefill tokens into scores [B, Hkv, T] (fp32) from q_pre [B, Hq, T, d] and
    k_pre [B, Hkv, T, d] (bf16); workspace of mikv_workspace_bytes(shape, WS_PREFILL, T) bytes."""
    T = k_pre.shape[2]
    scale = 1.0 / math.sqrt(shape.head_dim) if sm_scale is None else sm_scale
    _check("mikv_prefill_scores", load().mikv_prefill_scores(
        ctypes.byref(shape.c()), _ptr(q_pre), _ptr(k_pre), T, float(scale), _ptr(scores), _ptr(workspace),
        workspace.numel(), _stream(stream)))


def mikv_cache_fraction(bits: int, group: int, ratio: float, hi_bits: int = 16) -> float:
    return float(load(build_if_missing=False).mikv_cache_fraction(bits, group, ratio, hi_bits))


def mikv_budget(T: int, ratio: float) -> int:
    """Important tokens k for importance ratio `ratio` over T tokens (Tables 1-3): floor(ratio * T + 0.5).
    A cache for context T then attends hi_cap = k + 1 important slots."""
    k = int(load(build_if_missing=False).mikv_budget(int(T), float(ratio)))
    if k < 0:
        raise ValueError(f"mikv_budget: invalid T={T} or ratio={ratio}")
    return k


def mikv_retained_row_bytes(bits: int, group: int, head_dim: int = HEAD_DIM) -> int:
    return int(load(build_if_missing=False).mikv_retained_row_bytes(bits, group, head_dim))
