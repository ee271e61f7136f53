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
from _cases import (attention_tolerance, bits16, gpu_layer, new_workspace, oracle_layer, raw_inputs, sm_scale,
                    vmax_per_head)

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
    k_b = w.budget
    for r in refs:
        b, h, c = r["b"], r["h"], r["cache"]
        for name in ("k_hi", "v_hi"):
            np.testing.assert_array_equal(getattr(layer.cache, name)[b, h, :k_b].cpu().numpy(), c[name][0, 0, :k_b],
                                          err_msg=name)
        for gname, oname in (("k_hi_params", "k_hp"), ("v_hi_params", "v_hp")):
            np.testing.assert_array_equal(_u16(getattr(layer.cache, gname)[b, h, :k_b]), c[oname][0, 0, :k_b],
                                          err_msg=gname)
        np.testing.assert_array_equal(layer.cache.hi_tok[b, h, :k_b].cpu().numpy(), c["hi_tok"][0, 0, :k_b])
        n_lo = w.n_lo0
        for name in ("k_codes", "v_codes", "lo_tok"):
            np.testing.assert_array_equal(getattr(layer.cache, name)[b, h, :n_lo].cpu().numpy(), c[name][0, 0, :n_lo])
        for name in ("k_params", "v_params"):
            np.testing.assert_array_equal(_u16(getattr(layer.cache, name)[b, h, :n_lo]), c[name][0, 0, :n_lo])


def _logit_bound(c, q_bits, bal, w, n_lo):
    """|GPU - oracle| bound for logits: fp16 rounding of q / b and of every dequantized key (2^-11 relative
    each) plus fp32 accumulation: 2^-9 * scale * max_t sum_c |q_c k_tc|, over both coded sets."""
    q = (q_bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)[0]
    qh = q / (bal[0] if bal is not None else 1.0)
    rows = [oracle.dequantize_row(c["k_hi"][0, 0, i], c["k_hp"][0, 0, i], w.hi_bits, 64) for i in range(w.hi_cap)]
    rows += [oracle.dequantize_row(c["k_codes"][0, 0, t], c["k_params"][0, 0, t], w.bits, w.group)
             for t in range(n_lo)]
    worst = (np.abs(qh) @ np.abs(np.stack(rows)).T).max(axis=1) * 2.0 ** -9
    return sm_scale() * worst + 1e-6


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_coded_important_set_attention(name, out_dtype):
    w = CASES[name]
    raw = raw_inputs(w)
    layer = gpu_layer(w, raw)
    assert layer.shape.hi_coded
    refs = oracle_layer(w, raw, layer.shape.lo_cap)
    _check_hi_cache(layer, refs, w)

    q, k_new, v_new = mi.decode_inputs(w, 0, 0)
    dev = torch.device("cuda")
    s = layer.shape
    G = w.heads_q // w.heads_kv
    pkg.mikv_insert_token(layer.cache, k_new.to(dev), v_new.to(dev), w.context, layer.slots)
    out = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=out_dtype, device=dev)
    hl = torch.full((w.batch, w.heads_q, s.hi_stride), float("nan"), device=dev)
    ml = torch.empty(w.batch, w.heads_q, 2, device=dev)
    ws = new_workspace(s, pkg.WS_ATTENTION, w.n_lo0)
    pkg.mikv_decode_attention(layer.cache, w.n_lo0, q.to(dev), sm_scale(), out, ws, hi_logits=hl, ml=ml)
    pkg.mikv_workspace_check(ws)
    out_c, hl_c, ml_c = out.float().cpu().numpy(), hl.cpu().numpy(), ml.cpu().numpy()
    vmax = vmax_per_head(raw[1], v_new)
    for r in refs:
        b, h, c = r["b"], r["h"], r["cache"]
        oracle.insert_token(c, bits16(k_new[b:b + 1, h:h + 1]), bits16(v_new[b:b + 1, h:h + 1]), w.context,
                            np.array([[w.budget]], np.int32), balancer_=r["balancer"])
        # the inserted slot's codes are bit-exact too
        np.testing.assert_array_equal(layer.cache.k_hi[b, h, w.budget].cpu().numpy(), c["k_hi"][0, 0, w.budget])
        np.testing.assert_array_equal(_u16(layer.cache.v_hi_params[b, h, w.budget]), c["v_hp"][0, 0, w.budget])
        qb = bits16(q[b:b + 1, h * G:(h + 1) * G])
        ref_o, ref_l, ref_ml = oracle.decode_attention(c, qb, w.n_lo0, sm_scale(), balancer_=r["balancer"])
        got = out_c[b, h * G:(h + 1) * G]
        tol = attention_tolerance(vmax[b, h], ref_o[0], out_dtype == torch.bfloat16)
        err = np.abs(got - ref_o[0])
        assert np.all(err <= tol), f"{name} b{b} h{h}: max err {err.max():.3e}, tol {tol.min():.3e}"
        bound = _logit_bound(c, qb, r["balancer"], w, w.n_lo0)
        np.testing.assert_allclose(hl_c[b, h * G:(h + 1) * G, :w.hi_cap], ref_l[0], atol=float(bound.max()), rtol=0)
        dm = np.abs(ml_c[b, h * G:(h + 1) * G, 0] - ref_ml[0, :, 0])
        assert np.all(dm <= bound), (dm, bound)
        np.testing.assert_allclose(ml_c[b, h * G:(h + 1) * G, 1], ref_ml[0, :, 1], rtol=4 * float(bound.max()) + 1e-5)


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
    slots_ref = {(r["b"], r["h"]): np.array([[w.budget]], np.int32) for r in refs}
    near_ties = 0
    acc_tol = {}
    for step in range(steps):
        q, k_new, v_new = mi.decode_inputs(w, 0, step)
        out = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.float32, device=dev)
        n_lo = layer.n_lo
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
            tol = acc_tol.setdefault((b, h), np.zeros(w.hi_cap))
            tol[slot[0, 0]] = 0.0
            tol += 3e-3 * np.abs(c["acc"][0, 0] - acc_before) + 2e-7 * np.abs(acc_before) + 1e-9
            acc_gpu = layer.cache.acc[b, h, :w.hi_cap].cpu().numpy()
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
