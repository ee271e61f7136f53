"""Index checks of the checked build (-DMIKV_DEBUG; the package loads it with MIKV_DEBUG=1 in the environment).

Kernels that take an index from device memory skip out-of-range ones in every build; the checked build also
records them, in the workspace status word or in the library's own word (mikv_debug_check). Every invalid index
used here lies inside the arrays' padding (an insertion slot between hi_cap and hi_stride, a source row just past
n_src of a head that is not the last one), so even a library without the checks would only skip them. These tests
run only against the checked build (tests/test_gpu_debug_build.py starts them in a process of their own)."""
import os

import numpy as np
import pytest
import torch

import mikv_inputs as mi
import paper_2402_18096_gb300 as pkg
from _cases import gpu_layer, raw_inputs, sm_scale

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True, scope="module")
def checked_build():
    if not pkg.debug_build():
        if os.environ.get("MIKV_REQUIRE_DEBUG") == "1":
            pytest.fail("MIKV_REQUIRE_DEBUG=1 but the loaded library is not the checked build")
        pytest.skip("needs the checked build (MIKV_DEBUG=1)")
    pkg.mikv_debug_check()  # start from a clear word


def _small_cache(bits=2):
    shape = pkg.Shape(2, 4, 2, bits, 32, hi_cap=13, lo_cap=32)  # hi_stride 16: rows 13..15 are padding
    assert shape.hi_stride == 16
    return shape, pkg.LayerCache(shape, device="cuda")


def test_out_of_range_insertion_slot_is_recorded_and_skipped():
    shape, cache = _small_cache()
    dev = torch.device("cuda")
    k_new = torch.randn(2, 2, 128, device=dev).to(torch.bfloat16)
    v_new = torch.randn(2, 2, 128, device=dev).to(torch.bfloat16)
    slots = torch.tensor([[13, 5], [0, 12]], dtype=torch.int32, device=dev)  # (0, 0): slot 13 >= hi_cap
    pkg.mikv_insert_token(cache, k_new, v_new, 77, slots)
    with pytest.raises(pkg.MikvError) as e:
        pkg.mikv_debug_check()
    assert e.value.status == "MIKV_ERR_DEVICE"
    assert torch.count_nonzero(cache.k_hi[0, 0, 13:]) == 0 and int(cache.hi_tok[0, 0, 13]) == 0  # skipped
    assert torch.equal(cache.k_hi[0, 1, 5], k_new[0, 1]) and torch.equal(cache.v_hi[1, 1, 12], v_new[1, 1])
    pkg.mikv_insert_token(cache, k_new, v_new, 78, torch.tensor([[1, 2], [3, 4]], dtype=torch.int32, device=dev))
    pkg.mikv_debug_check()  # valid slots: nothing recorded (the word was cleared by the previous check)


def test_out_of_range_source_rows_are_recorded_and_skipped():
    shape, cache = _small_cache()
    dev = torch.device("cuda")
    n_src = 20
    k = torch.randn(2, 2, n_src, 128, device=dev).to(torch.bfloat16)
    v = torch.randn(2, 2, n_src, 128, device=dev).to(torch.bfloat16)
    rows = torch.arange(4, dtype=torch.int32, device=dev).expand(2, 2, 4).contiguous()
    pkg.mikv_gather_hi(cache, k, v, rows)
    pkg.mikv_quantize_pack(cache, k, v, rows, 0)
    pkg.mikv_debug_check()  # in-range rows
    bad = rows.clone()
    bad[0, 0, 3] = n_src  # one past the source rows of head (0, 0): row 0 of the next head, still allocated
    pkg.mikv_gather_hi(cache, k, v, bad)
    with pytest.raises(pkg.MikvError):
        pkg.mikv_debug_check()
    pkg.mikv_quantize_pack(cache, k, v, bad, 4)
    with pytest.raises(pkg.MikvError):
        pkg.mikv_debug_check()
    assert torch.count_nonzero(cache.k_codes[0, 0, 7]) == 0  # the skipped row wrote nothing
    assert torch.count_nonzero(cache.k_codes[0, 1, 7]) > 0


def test_out_of_range_step_slot_is_recorded_in_the_workspace():
    """A decode step whose insertion slot is out of range: the attention kernel inserts nothing and reports it
    through the workspace status word."""
    w = mi.Workload("dbg", 1, 4, 2, 120, 1, 2, 32, 0.1, seed=91)
    layer = gpu_layer(w, raw_inputs(w), steps=2)
    assert layer.shape.hi_cap < layer.shape.hi_stride
    q, k_new, v_new = (x.cuda() for x in mi.decode_inputs(w, 0, 0))
    layer.slots[0, 1] = layer.shape.hi_cap  # padding row of the important arrays
    out = torch.empty(w.batch, w.heads_q, 128, device="cuda")
    layer.step(q, k_new, v_new, out)
    with pytest.raises(pkg.MikvError) as e:
        pkg.mikv_workspace_check(layer.ws)
    assert e.value.status == "MIKV_ERR_DEVICE"
    pkg.mikv_workspace_reset(layer.ws)


def test_normal_cases_record_nothing():
    """A cache build and decode steps with valid indices leave both status words clear."""
    w = mi.Workload("dbg2", 2, 8, 2, 333, 1, 3, 64, 0.2, seed=92)
    layer = gpu_layer(w, raw_inputs(w), steps=3)
    for s in range(3):
        q, k_new, v_new = (x.cuda() for x in mi.decode_inputs(w, 0, s))
        out = torch.empty(w.batch, w.heads_q, 128, device="cuda")
        layer.step(q, k_new, v_new, out)
    pkg.mikv_workspace_check(layer.ws)
    pkg.mikv_debug_check()
    assert np.isfinite(out.cpu().numpy()).all()
