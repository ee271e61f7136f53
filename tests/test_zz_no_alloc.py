"""The no-allocation decode attention entry point (mikv_decode_attention_noalloc), called through the
C ABI: it must give what mikv_decode_attention gives with a caller workspace, call after call, while
keeping its scratch in the library's own fixed device buffer. This file is collected last so that a run
stopping at its first failure has already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

import mikv_inputs as mi
import paper_2402_18096_gb300 as pkg
from _cases import attention_tolerance, gpu_layer, new_workspace, raw_inputs, sm_scale, vmax_per_head

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("w", [mi.Workload("gqa4", 2, 8, 2, 700, 1, 2, 32, 0.20, seed=31),
                               mi.Workload("mha", 2, 4, 4, 999, 1, 3, 64, 0.10, seed=32)],
                         ids=["gqa4-int2-g32", "mha-int3-g64"])
def test_noalloc_matches_workspace_entry_point(w):
    raw = raw_inputs(w)
    layer = gpu_layer(w, raw)
    dev = torch.device("cuda")
    q, k_new, v_new = mi.decode_inputs(w, 0, 0)
    q = q.to(dev)
    pkg.mikv_insert_token(layer.cache, k_new.to(dev), v_new.to(dev), w.context, layer.slots)
    s = layer.shape
    n_lo = w.n_lo0
    ref = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.bfloat16, device=dev)
    ref_hl = torch.zeros(w.batch, w.heads_q, s.hi_stride, device=dev)
    ref_ml = torch.zeros(w.batch, w.heads_q, 2, device=dev)
    ws = new_workspace(s, pkg.WS_ATTENTION, n_lo)
    pkg.mikv_decode_attention(layer.cache, n_lo, q, sm_scale(), ref, ws, hi_logits=ref_hl, ml=ref_ml)
    pkg.mikv_workspace_check(ws)
    G = w.heads_q // w.heads_kv
    vmax = np.repeat(vmax_per_head(raw[1], v_new), G, axis=1)[..., None]  # per query head
    r = ref.float().cpu().numpy()
    tol = attention_tolerance(1.0, r, True) - 2e-3 + 2e-3 * vmax  # 2e-3 max|V| + bf16 rounding of r
    for call in range(2):  # two calls in a row share the one built-in buffer
        out = torch.full_like(ref, float("nan"))
        hl = torch.zeros_like(ref_hl)
        ml = torch.zeros_like(ref_ml)
        pkg.mikv_decode_attention_noalloc(layer.cache, n_lo, q, sm_scale(), out, hi_logits=hl, ml=ml)
        torch.cuda.synchronize()
        err = np.abs(out.float().cpu().numpy() - r)
        assert np.all(err <= tol), (call, float(err.max()))
        np.testing.assert_allclose(hl[..., :s.hi_cap].cpu().numpy(), ref_hl[..., :s.hi_cap].cpu().numpy(),
                                   rtol=1e-6, atol=1e-6)
        np.testing.assert_allclose(ml.cpu().numpy(), ref_ml.cpu().numpy(), rtol=1e-6, atol=1e-6)


def test_noalloc_rejects_problems_beyond_its_buffer():
    lib = pkg.load()
    # 16384 KV heads need about 8.5 MB of partials: more than the built-in buffer
    shape = pkg._Shape(512, 32, 32, 128, 2, 32, 17, 32, 64)
    cache = pkg._Cache(*([0x10000] * 9 + [None]))
    rc = lib.mikv_decode_attention_noalloc(ctypes.byref(shape), ctypes.byref(cache), 16, 0x10000, 1.0, 0x10000,
                                           0, None, None, None)
    assert rc == 7
    assert "scratch" in pkg.mikv_status_string(7)
