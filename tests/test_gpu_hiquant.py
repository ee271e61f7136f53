"""GPU parity of the reduced-precision important set (Sec. 3.3, Table 3): the important set stored as
INT8 / INT4 / INT2 codes in groups of 64 (keys balanced, Eq. 3), against the oracle on the same seeded
inputs — cache build (codes bit for bit), insert + decode attention (outputs, important-set logits,
softmax statistics), and whole decode steps (importance update, victim choice, re-quantized demotion
bit for bit)."""
import numpy as np
import pytest
import torch

import mikv_inputs as mi
import oracle
import paper_2402_18096_gb300 as pkg
from _cases import (assert_attention_close, bits16, gpu_layer, logit_bounds, new_workspace, oracle_layer, raw_inputs,
                    ref_sizes, sm_scale, softmax_stat_bounds, vmax_per_head)

pytestmark = pytest.mark.gpu

CASES = {
    "hi8-gqa4-int2-g64": mi.Workload("h8", 2, 8, 2, 700, 1, 2, 64, 0.20, seed=31, hi_bits=8),
    "hi4-mha-int3-g32": mi.Workload("h4", 1, 4, 4, 611, 1, 3, 32, 0.25, seed=32, hi_bits=4),
    "hi2-gqa8-int4-g128": mi.Workload("h2", 1, 8, 1, 333, 1, 4, 128, 0.50, seed=33, hi_bits=2),
    "hi8-all-important": mi.Workload("h8a", 1, 4, 2, 150, 1, 2, 32, 1.00, seed=34, hi_bits=8),
    "hi4-gqa2-int4-g64-r5": mi.Workload("h4b", 2, 4, 2, 801, 1, 4, 64, 0.05, seed=35, hi_bits=4),
    "hi8-one-token": mi.Workload("h8t", 1, 2, 2, 1, 1, 2, 64, 0.2, seed=36, hi_bits=8),
}


def _u16(t: torch.Tensor) -> np.ndarray:
    return t.cpu().view(torch.int16).numpy().view(np.uint16)


def _check_hi_cache(layer, refs, w):
    R = ref_sizes(w)
    assert layer.shape.hi_cap == R.hi_cap and layer.n_lo == R.n_lo0  # library budget = oracle budget
    k_b = R.budget
    for r in refs:
        b, h, c = r["b"], r["h"], r["cache"]
        for name in ("k_hi", "v_hi"):
            np.testing.assert_array_equal(getattr(layer.cache, name)[b, h, :k_b].cpu().numpy(), c[name][0, 0, :k_b],
                                          err_msg=name)
        for gname, oname in (("k_hi_params", "k_hp"), ("v_hi_params", "v_hp")):
            np.testing.assert_array_equal(_u16(getattr(layer.cache, gname)[b, h, :k_b]), c[oname][0, 0, :k_b],
                                          err_msg=gname)
        np.testing.assert_array_equal(layer.cache.hi_tok[b, h, :k_b].cpu().numpy(), c["hi_tok"][0, 0, :k_b])
        n_lo = R.n_lo0
        for name in ("k_codes", "v_codes", "lo_tok"):
            np.testing.assert_array_equal(getattr(layer.cache, name)[b, h, :n_lo].cpu().numpy(), c[name][0, 0, :n_lo])
        for name in ("k_params", "v_params"):
            np.testing.assert_array_equal(_u16(getattr(layer.cache, name)[b, h, :n_lo]), c[name][0, 0, :n_lo])


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_coded_important_set_attention(name, out_dtype):
    w = CASES[name]
    raw = raw_inputs(w)
    layer = gpu_layer(w, raw)
    assert layer.shape.hi_coded
    refs = oracle_layer(w, raw, layer.shape.lo_cap)
    _check_hi_cache(layer, refs, w)
    R = ref_sizes(w)

    q, k_new, v_new = mi.decode_inputs(w, 0, 0)
    dev = torch.device("cuda")
    s = layer.shape
    G = w.heads_q // w.heads_kv
    pkg.mikv_insert_token(layer.cache, k_new.to(dev), v_new.to(dev), w.context, layer.slots)
    out = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=out_dtype, device=dev)
    hl = torch.full((w.batch, w.heads_q, s.hi_stride), float("nan"), device=dev)
    ml = torch.empty(w.batch, w.heads_q, 2, device=dev)
    ws = new_workspace(s, pkg.WS_ATTENTION, layer.n_lo)
    pkg.mikv_decode_attention(layer.cache, layer.n_lo, q.to(dev), sm_scale(), out, ws, hi_logits=hl, ml=ml)
    pkg.mikv_workspace_check(ws)
    out_c, hl_c, ml_c = out.cpu(), hl.cpu().numpy(), ml.cpu().numpy()
    out32 = None
    if out_dtype == torch.bfloat16:  # the same call with fp32 output: the bf16 output must be its rounding
        out32 = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.float32, device=dev)
        pkg.mikv_decode_attention(layer.cache, layer.n_lo, q.to(dev), sm_scale(), out32, ws)
        pkg.mikv_workspace_check(ws)
        out32 = out32.cpu()
    vmax = vmax_per_head(raw[1], v_new)
    for r in refs:
        b, h, c = r["b"], r["h"], r["cache"]
        oracle.insert_token(c, bits16(k_new[b:b + 1, h:h + 1]), bits16(v_new[b:b + 1, h:h + 1]), w.context,
                            np.array([[R.budget]], np.int32), balancer_=r["balancer"])
        # the inserted slot's codes are bit-exact too
        np.testing.assert_array_equal(layer.cache.k_hi[b, h, R.budget].cpu().numpy(), c["k_hi"][0, 0, R.budget])
        np.testing.assert_array_equal(_u16(layer.cache.v_hi_params[b, h, R.budget]), c["v_hp"][0, 0, R.budget])
        qb = bits16(q[b:b + 1, h * G:(h + 1) * G])
        ref_o, ref_l, ref_ml = oracle.decode_attention(c, qb, R.n_lo0, sm_scale(), balancer_=r["balancer"])
        sl = slice(h * G, (h + 1) * G)
        assert_attention_close(out_c[b, sl], ref_o[0], vmax[b, h], f32=None if out32 is None else out32[b, sl],
                               msg=f"{name} b{b} h{h}")
        hb, lb = logit_bounds(c, qb, r["balancer"], w.bits, w.group, R.n_lo0, sm_scale(), hi_bits=w.hi_bits)
        E, l_rtol = softmax_stat_bounds(hb, lb, R.hi_cap + R.n_lo0)
        assert np.all(np.abs(hl_c[b, sl, :R.hi_cap] - ref_l[0]) <= hb), "important-set logits"
        assert np.all(np.abs(ml_c[b, sl, 0] - ref_ml[0, :, 0]) <= E), "softmax max"
        assert np.all(np.abs(ml_c[b, sl, 1] / ref_ml[0, :, 1] - 1) <= l_rtol), "softmax sum"


@pytest.mark.parametrize("hi_bits,bits,group", [(8, 2, 64), (4, 3, 32), (2, 4, 128)])
def test_coded_important_set_decode_steps(hi_bits, bits, group):
    """Whole decode steps through mikv_decode_step: outputs, scores, the victims and the re-quantized
    retained rows (codes and parameters bit for bit) against the oracle's step sequence."""
    w = mi.Workload("trajq", 2, 8, 2, 420, 1, bits, group, 0.2, seed=40 + hi_bits, hi_bits=hi_bits)
    steps = 5
    raw = raw_inputs(w)
    layer = gpu_layer(w, raw, steps=steps)
    s = layer.shape
    refs = oracle_layer(w, raw, s.lo_cap)
    G = w.heads_q // w.heads_kv
    dev = torch.device("cuda")
    R = ref_sizes(w)
    slots_ref = {(r["b"], r["h"]): np.array([[R.budget]], np.int32) for r in refs}
    near_ties = 0
    acc_tol = {}
    for step in range(steps):
        q, k_new, v_new = mi.decode_inputs(w, 0, step)
        out = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.float32, device=dev)
        n_lo = R.n_lo0 + step  # the oracle's retained length; the library's must agree
        assert layer.n_lo == n_lo
        layer.step(q.to(dev), k_new.to(dev), v_new.to(dev), out)
        pkg.mikv_workspace_check(layer.ws)
        gslots = layer.slots.cpu().numpy()
        vmax = vmax_per_head(raw[1], v_new)
        for r in refs:
            b, h, c = r["b"], r["h"], r["cache"]
            slot = slots_ref[(b, h)]
            oracle.insert_token(c, bits16(k_new[b:b + 1, h:h + 1]), bits16(v_new[b:b + 1, h:h + 1]), w.context + step,
                                slot, balancer_=r["balancer"])
            qb = bits16(q[b:b + 1, h * G:(h + 1) * G])
            ref_o, hl, ml = oracle.decode_attention(c, qb, n_lo, sm_scale(), balancer_=r["balancer"])
            err = np.abs(out[b, h * G:(h + 1) * G].cpu().numpy() - ref_o[0])
            assert np.all(err <= 2e-3 * vmax[b, h]), (step, b, h, err.max())
            acc_before = c["acc"][0, 0].astype(np.float64)
            c["acc"] = oracle.update_importance(c["acc"], hl.astype(np.float32), ml.astype(np.float32), G)
            # a softmax weight's relative error: its logit's plus m's and l's (logit_bounds), plus 2^-21 for its fp32
            # roundings; the fp32 add into the score rounds once (2^-24, taken twice); errors add up over steps
            hb, lb = logit_bounds(c, qb, r["balancer"], w.bits, w.group, n_lo, sm_scale(), hi_bits=w.hi_bits)
            E, l_rtol = softmax_stat_bounds(hb, lb, R.hi_cap + n_lo)
            inc_rtol = float((np.expm1(2 * E) + l_rtol).max()) + 2.0 ** -21
            tol = acc_tol.setdefault((b, h), np.zeros(R.hi_cap))
            tol[slot[0, 0]] = 0.0
            tol += inc_rtol * np.abs(c["acc"][0, 0] - acc_before) + 2.0 ** -23 * np.abs(c["acc"][0, 0])
            acc_gpu = layer.cache.acc[b, h, :R.hi_cap].cpu().numpy()
            assert np.all(np.abs(acc_gpu - c["acc"][0, 0]) <= tol), (step, b, h)
            dem, _ = oracle.select_demote(c["acc"], 1, c["hi_tok"], want_kept=False)
            victim = int(dem[0, 0, 0])
            if gslots[b, h] != victim:
                a_sorted = np.sort(c["acc"][0, 0])
                assert abs(a_sorted[1] - a_sorted[0]) < 1e-5 * max(1.0, abs(a_sorted[0])), (step, b, h)
                near_ties += 1
                victim = int(gslots[b, h])
            oracle.demote_hi(c, np.array([[victim]], np.int32), n_lo, balancer_=r["balancer"])
            for name in ("k_codes", "v_codes", "lo_tok"):
                np.testing.assert_array_equal(getattr(layer.cache, name)[b, h, n_lo].cpu().numpy(), c[name][0, 0, n_lo],
                                              err_msg=f"{name} step {step}")
            for name in ("k_params", "v_params"):
                np.testing.assert_array_equal(_u16(getattr(layer.cache, name)[b, h, n_lo]), c[name][0, 0, n_lo])
            slots_ref[(b, h)] = np.array([[victim]], np.int32)
    assert near_ties <= 2
