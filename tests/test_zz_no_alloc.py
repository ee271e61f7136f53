"""The no-allocation decode attention entry point (mikv_decode_attention_noalloc), called through the C ABI.

It exists for callers that may not allocate device memory while decoding (an engine that owns every byte of
device memory, a serving loop that must not call cudaMalloc): it keeps its split partials in the library's own
fixed device buffer instead of a caller workspace. It runs the same plan and the same kernels as
mikv_decode_attention, so its outputs must be bit-identical to that entry point's, call after call on the one
shared buffer, and within the attention bound of the oracle. mikv_noalloc_check reads the buffer's status word
after each call. This file is collected last so that a run stopping at its first failure has already run every
other test; it passes alone in a fresh process too."""
import ctypes

import numpy as np
import pytest
import torch

import mikv_inputs as mi
import oracle
import paper_2402_18096_gb300 as pkg
from _cases import (assert_attention_close, bits16, gpu_layer, new_workspace, oracle_layer, raw_inputs, ref_sizes,
                    sm_scale, vmax_per_head)

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("w", [mi.Workload("gqa4", 2, 8, 2, 700, 1, 2, 32, 0.20, seed=31),
                               mi.Workload("mha", 2, 4, 4, 999, 1, 3, 64, 0.10, seed=32)],
                         ids=["gqa4-int2-g32", "mha-int3-g64"])
@pytest.mark.parametrize("out_dtype", [torch.bfloat16, torch.float32])
def test_noalloc_matches_workspace_entry_point(w, out_dtype):
    raw = raw_inputs(w)
    layer = gpu_layer(w, raw)
    dev = torch.device("cuda")
    q, k_new, v_new = mi.decode_inputs(w, 0, 0)
    q = q.to(dev)
    pkg.mikv_insert_token(layer.cache, k_new.to(dev), v_new.to(dev), w.context, layer.slots)
    s = layer.shape
    n_lo = layer.n_lo
    ref = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=out_dtype, device=dev)
    ref_hl = torch.zeros(w.batch, w.heads_q, s.hi_stride, device=dev)
    ref_ml = torch.zeros(w.batch, w.heads_q, 2, device=dev)
    ws = new_workspace(s, pkg.WS_ATTENTION, n_lo)
    pkg.mikv_decode_attention(layer.cache, n_lo, q, sm_scale(), ref, ws, hi_logits=ref_hl, ml=ref_ml)
    pkg.mikv_workspace_check(ws)
    for call in range(2):  # two calls in a row share the one built-in buffer
        out = torch.full_like(ref, float("nan"))
        hl = torch.full_like(ref_hl, float("nan"))
        ml = torch.full_like(ref_ml, float("nan"))
        pkg.mikv_decode_attention_noalloc(layer.cache, n_lo, q, sm_scale(), out, hi_logits=hl, ml=ml)
        pkg.mikv_noalloc_check()  # the buffer's status word: no kernel reported a failure
        assert torch.equal(out, ref), call
        assert torch.equal(hl[..., :s.hi_cap], ref_hl[..., :s.hi_cap]), call
        assert torch.equal(ml, ref_ml), call

    # and against the oracle, on every (b, KV head)
    R = ref_sizes(w)
    G = w.heads_q // w.heads_kv
    vmax = vmax_per_head(raw[1], v_new)
    out32 = None
    if out_dtype == torch.bfloat16:
        out32 = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.float32, device=dev)
        pkg.mikv_decode_attention_noalloc(layer.cache, n_lo, q, sm_scale(), out32)
        pkg.mikv_noalloc_check()
        out32 = out32.cpu()
    out_c = out.cpu()
    for r in oracle_layer(w, raw, s.lo_cap):
        b, h, c = r["b"], r["h"], r["cache"]
        oracle.insert_token(c, bits16(k_new[b:b + 1, h:h + 1]), bits16(v_new[b:b + 1, h:h + 1]), w.context,
                            np.array([[R.budget]], np.int32))
        ref_o, _, _ = oracle.decode_attention(c, bits16(q[b:b + 1, h * G:(h + 1) * G]), R.n_lo0, sm_scale(),
                                              balancer_=r["balancer"])
        sl = slice(h * G, (h + 1) * G)
        assert_attention_close(out_c[b, sl], ref_o[0], vmax[b, h], f32=None if out32 is None else out32[b, sl],
                               msg=f"noalloc b{b} h{h}")


def test_noalloc_rejects_problems_beyond_its_buffer():
    lib = pkg.load()
    # 16384 KV heads need about 8.5 MB of partials: more than the built-in buffer
    shape = pkg._Shape(512, 32, 32, 128, 2, 32, 17, 32, 64)
    cache = pkg._Cache(*([0x10000] * 9 + [None]))
    rc = lib.mikv_decode_attention_noalloc(ctypes.byref(shape), ctypes.byref(cache), 16, 0x10000, 1.0, 0x10000,
                                           0, None, None, None)
    assert rc == 7
    assert "scratch" in pkg.mikv_status_string(7)
