"""GPU parity of the decode path against the CPU oracle.

Each case draws the same seeded raw inputs (prefill K/V with outlier key channels, prefill queries,
importance scores, the decode token); the CUDA library and the oracle each build their own cache
from them and attend. Compared: balancer, important set and retained set bit-exact; attention output
within max|err| <= 2e-3 * max|V| (fp32 accumulation; plus bf16 rounding of the output when it is bf16);
logits and softmax statistics within bounds derived from fp16 operand rounding.
"""
import math

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
    # name: workload (ragged important / retained tails, several splits and stages)
    "tiny-int4-g32-mha": mi.WORKLOADS["tiny"],
    "gqa4-int2-g32": mi.Workload("gqa4", 2, 8, 2, 700, 1, 2, 32, 0.20, seed=1),
    "mha-int3-g64-r10": mi.Workload("int3", 2, 4, 4, 999, 1, 3, 64, 0.10, seed=2),
    "gqa8-int4-g128-r0": mi.Workload("r0", 1, 8, 1, 300, 1, 4, 128, 0.0, seed=3),
    "gqa2-int2-g128-r50": mi.Workload("r50", 2, 4, 2, 257, 1, 2, 128, 0.5, seed=4),
    "all-important": mi.Workload("r100", 1, 2, 2, 100, 1, 2, 32, 1.0, seed=5),
    "one-token": mi.Workload("t1", 1, 4, 4, 1, 1, 3, 32, 0.2, seed=6),
    "exact-16": mi.Workload("x16", 1, 4, 1, 160, 1, 4, 32, 0.09375, seed=7),  # hi_cap = 16
}
# every retained layout (bits x group): ragged lengths, several units per head
for _b in (2, 3, 4):
    for _g in (32, 64, 128):
        CASES[f"layout-int{_b}-g{_g}"] = mi.Workload(f"l{_b}{_g}", 1, 4, 2, 611, 1, _b, _g, 0.15, seed=10 * _b + _g)


def _check_cache(layer, refs, w):
    k_b = w.budget
    for r in refs:
        b, h, c = r["b"], r["h"], r["cache"]
        if r["balancer"] is not None:
            np.testing.assert_array_equal(layer.cache.balancer[h].cpu().numpy().view(np.uint32),
                                          r["balancer"][0].view(np.uint32))
        np.testing.assert_array_equal(bits16(layer.cache.k_hi[b, h, :k_b]), c["k_hi"][0, 0, :k_b])
        np.testing.assert_array_equal(bits16(layer.cache.v_hi[b, h, :k_b]), c["v_hi"][0, 0, :k_b])
        np.testing.assert_array_equal(layer.cache.hi_tok[b, h, :k_b].cpu().numpy(), c["hi_tok"][0, 0, :k_b])
        n_lo = w.n_lo0
        for name in ("k_codes", "v_codes", "lo_tok"):
            np.testing.assert_array_equal(getattr(layer.cache, name)[b, h, :n_lo].cpu().numpy(),
                                          c[name][0, 0, :n_lo], err_msg=name)
        for name in ("k_params", "v_params"):
            got = getattr(layer.cache, name)[b, h, :n_lo].cpu().view(torch.int16).numpy().view(np.uint16)
            np.testing.assert_array_equal(got, c[name][0, 0, :n_lo], err_msg=name)


def _logit_bound(c, q_bits, bal, w, n_lo):
    """Bound on |GPU - oracle| for logits: fp16 rounding of q / b and of each dequantized key (2^-11
    relative each) plus fp32 accumulation, i.e. 2^-9 * scale * max_t sum_c |q_c k_tc| with margin."""
    G = q_bits.shape[1]
    q = (q_bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)[0]  # [G, d]
    qh = q / (bal[0] if bal is not None else 1.0)
    kh = (c["k_hi"][0, 0].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    worst = (np.abs(q) @ np.abs(kh).T).max(axis=1) * 2.0 ** -20
    if n_lo:
        kl = np.stack([oracle.dequantize_row(c["k_codes"][0, 0, t], c["k_params"][0, 0, t], w.bits, w.group)
                       for t in range(n_lo)])
        worst = np.maximum(worst, (np.abs(qh) @ np.abs(kl).T).max(axis=1) * 2.0 ** -9)
    return sm_scale() * worst + 1e-6  # [G]


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_attention_matches_oracle(name, out_dtype):
    w = CASES[name]
    raw = raw_inputs(w)
    layer = gpu_layer(w, raw)
    refs = oracle_layer(w, raw, layer.shape.lo_cap)
    _check_cache(layer, refs, w)

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
                            np.array([[w.budget]], np.int32))
        qb = bits16(q[b:b + 1, h * G:(h + 1) * G])
        ref_o, ref_l, ref_ml = oracle.decode_attention(c, qb, w.n_lo0, sm_scale(), balancer_=r["balancer"])
        got = out_c[b, h * G:(h + 1) * G]
        tol = attention_tolerance(vmax[b, h], ref_o[0], out_dtype == torch.bfloat16)
        err = np.abs(got - ref_o[0])
        assert np.all(err <= tol), f"{name} b{b} h{h}: max err {err.max():.3e}, tol {tol.min():.3e}"
        bound = _logit_bound(c, qb, r["balancer"], w, w.n_lo0)
        np.testing.assert_allclose(hl_c[b, h * G:(h + 1) * G, :w.hi_cap], ref_l[0],
                                   atol=float(bound.max()), rtol=0)
        dm = np.abs(ml_c[b, h * G:(h + 1) * G, 0] - ref_ml[0, :, 0])
        assert np.all(dm <= bound), (dm, bound)
        np.testing.assert_allclose(ml_c[b, h * G:(h + 1) * G, 1], ref_ml[0, :, 1], rtol=4 * float(bound.max()) + 1e-5)


def test_decode_steps_trajectory():
    """Several whole decode steps (insert, attend, update, select, demote) through mikv_decode_step
    against the oracle's step sequence: chosen victims, appended retained rows and outputs."""
    w = mi.Workload("traj", 2, 8, 2, 500, 1, 2, 32, 0.2, seed=21)
    steps = 6
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
                                slot)
            qb = bits16(q[b:b + 1, h * G:(h + 1) * G])
            ref_o, hl, ml = oracle.decode_attention(c, qb, n_lo, sm_scale(), balancer_=r["balancer"])
            err = np.abs(out[b, h * G:(h + 1) * G].cpu().numpy() - ref_o[0])
            assert np.all(err <= 2e-3 * vmax[b, h]), (step, b, h, err.max())
            acc_before = c["acc"][0, 0].astype(np.float64)
            c["acc"] = oracle.update_importance(c["acc"], hl.astype(np.float32), ml.astype(np.float32), G)
            # each step's increment is a softmax weight whose relative error follows the logit error
            # (fp16 query / key operands, about 1e-3 at most here); errors add up over the steps
            tol = acc_tol.setdefault((b, h), np.zeros(w.hi_cap))
            tol[slot[0, 0]] = 0.0
            tol += 3e-3 * np.abs(c["acc"][0, 0] - acc_before) + 2e-7 * np.abs(acc_before) + 1e-9
            acc_gpu = layer.cache.acc[b, h, :w.hi_cap].cpu().numpy()
            dem, _ = oracle.select_demote(c["acc"], 1, c["hi_tok"], want_kept=False)
            victim = int(dem[0, 0, 0])
            if gslots[b, h] != victim:
                # both sides pick the minimum of fp32 scores computed in different orders; accept only a
                # near tie and continue from the GPU's choice
                a_sorted = np.sort(c["acc"][0, 0])
                assert abs(a_sorted[1] - a_sorted[0]) < 1e-5 * max(1.0, abs(a_sorted[0])), (step, b, h)
                near_ties += 1
                victim = int(gslots[b, h])
            assert np.all(np.abs(acc_gpu - c["acc"][0, 0]) <= tol), (step, b, h)
            oracle.quantize_pack(c, c["k_hi"], c["v_hi"], np.array([[[victim]]], np.int32), n_lo,
                                 src_tok=c["hi_tok"], balancer_=r["balancer"])
            np.testing.assert_array_equal(layer.cache.k_codes[b, h, n_lo].cpu().numpy(), c["k_codes"][0, 0, n_lo])
            np.testing.assert_array_equal(layer.cache.v_codes[b, h, n_lo].cpu().numpy(), c["v_codes"][0, 0, n_lo])
            assert int(layer.cache.lo_tok[b, h, n_lo]) == int(c["lo_tok"][0, 0, n_lo])
            slots_ref[(b, h)] = np.array([[victim]], np.int32)
    assert near_ties <= 2


@pytest.mark.parametrize("wname,heads", [("llama2-7b", [(0, 0), (3, 17), (7, 31)]),
                                        ("mistral-7b", [(0, 0), (13, 5), (31, 7)]),
                                        ("llama2-13b", [(9, 21), (15, 39)])])
def test_full_size_layer_sampled_heads(wname, heads):
    """One layer at the benchmark's full size, built and stepped in the benchmark's launch
    configuration (decode step: insert, attention, fused merge / update / select / demote); the oracle
    checks sampled (batch, KV head) pairs one by one: retained codes, output, softmax max and sum, the
    demoted slot and its packed row."""
    w = mi.WORKLOADS[wname]
    dev = torch.device("cuda")
    k, v = mi.prefill_kv(w, 0, dev)
    scores = mi.initial_scores(w, 0, dev)
    q_pre = mi.prefill_queries(w, 0, dev)
    from _cases import make_shape
    from paper_2402_18096_gb300.layer import MixedPrecisionLayer
    shape = make_shape(w, 1)
    layer = MixedPrecisionLayer.from_prefill(shape, k, v, scores, q_pre, device=dev)
    G = w.heads_q // w.heads_kv
    q, k_new, v_new = mi.decode_inputs(w, 0, 0, dev)
    # attention with statistics on a copy of the inserted state, then the real fused step
    pkg.mikv_insert_token(layer.cache, k_new, v_new, w.context, layer.slots)
    ml = torch.empty(w.batch, w.heads_q, 2, device=dev)
    out_a = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.float32, device=dev)
    ws = new_workspace(shape, pkg.WS_ATTENTION, w.n_lo0)
    pkg.mikv_decode_attention(layer.cache, w.n_lo0, q, sm_scale(), out_a, ws, ml=ml)
    out = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.bfloat16, device=dev)
    layer.step(q, k_new, v_new, out)  # re-inserts the same token into the same slot: idempotent
    pkg.mikv_workspace_check(layer.ws)
    victims = layer.slots.cpu().numpy()
    for b, h in heads:
        raw = (k[:, h:h + 1].cpu(), v[:, h:h + 1].cpu(), scores[:, h:h + 1].cpu(),
               q_pre[:, h * G:(h + 1) * G].cpu())
        sub = mi.scaled(w, heads_q=G, heads_kv=1)
        ref = oracle_layer(sub, raw, shape.lo_cap, heads=[(b, 0)])[0]
        c = ref["cache"]
        n_lo = w.n_lo0
        np.testing.assert_array_equal(layer.cache.k_codes[b, h, :n_lo].cpu().numpy(), c["k_codes"][0, 0, :n_lo])
        np.testing.assert_array_equal(layer.cache.v_params[b, h, :n_lo].cpu().view(torch.int16).numpy()
                                      .view(np.uint16), c["v_params"][0, 0, :n_lo])
        oracle.insert_token(c, bits16(k_new[b:b + 1, h:h + 1]), bits16(v_new[b:b + 1, h:h + 1]), w.context,
                            np.array([[w.budget]], np.int32))
        qb = bits16(q[b:b + 1, h * G:(h + 1) * G])
        ref_o, hl, rml = oracle.decode_attention(c, qb, n_lo, sm_scale(), balancer_=ref["balancer"])
        vmax = max(float(v[b, h].float().abs().max()), float(v_new[b, h].float().abs().max()))
        got = out[b, h * G:(h + 1) * G].float().cpu().numpy()
        tol = attention_tolerance(vmax, ref_o[0], True)
        assert np.all(np.abs(got - ref_o[0]) <= tol), np.abs(got - ref_o[0]).max()
        got_a = out_a[b, h * G:(h + 1) * G].cpu().numpy()
        assert np.all(np.abs(got_a - ref_o[0]) <= attention_tolerance(vmax, ref_o[0], False))
        # softmax statistics: every token is counted once (a lost or doubled block moves l by >= 0.1 %)
        bound = _logit_bound(c, qb, ref["balancer"], w, n_lo)
        gm = ml[b, h * G:(h + 1) * G].cpu().numpy()
        assert np.all(np.abs(gm[:, 0] - rml[0, :, 0]) <= bound)
        np.testing.assert_allclose(gm[:, 1], rml[0, :, 1], rtol=4 * float(bound.max()) + 1e-5)
        # the demoted slot and its packed rows
        acc = oracle.update_importance(c["acc"], hl.astype(np.float32), rml.astype(np.float32), G)
        dem, _ = oracle.select_demote(acc, 1, c["hi_tok"], want_kept=False)
        if int(dem[0, 0, 0]) == int(victims[b, h]):
            oracle.quantize_pack(c, c["k_hi"], c["v_hi"], dem, n_lo, src_tok=c["hi_tok"], balancer_=ref["balancer"])
            np.testing.assert_array_equal(layer.cache.v_codes[b, h, n_lo].cpu().numpy(), c["v_codes"][0, 0, n_lo])
            assert int(layer.cache.lo_tok[b, h, n_lo]) == int(c["lo_tok"][0, 0, n_lo])
        else:  # only a near tie of fp32 scores may pick another slot
            a_sorted = np.sort(acc[0, 0])
            assert abs(a_sorted[1] - a_sorted[0]) < 1e-5 * max(1.0, abs(a_sorted[0]))


@pytest.mark.parametrize("w", mi.sweep_workloads(), ids=lambda w: f"int{w.bits}-g{w.group}-r{int(w.ratio * 100)}")
def test_sweep_points_one_step(w):
    """Every point of the batch-64 sweep (bits x importance ratio x group) at batch 2: one whole decode
    step (insert, attention, importance update, demotion) against the oracle on one sampled KV head."""
    w = mi.scaled(w, batch=2, seed=w.bits * 100 + w.group + int(w.ratio * 1000))
    raw = raw_inputs(w)
    layer = gpu_layer(w, raw, steps=2)
    b, h = 1, (w.bits * 7 + w.group) % w.heads_kv
    ref = oracle_layer(w, raw, layer.shape.lo_cap, heads=[(b, h)])[0]
    c = ref["cache"]
    q, k_new, v_new = mi.decode_inputs(w, 0, 0)
    dev = torch.device("cuda")
    out = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.float32, device=dev)
    n_lo = layer.n_lo
    layer.step(q.to(dev), k_new.to(dev), v_new.to(dev), out)
    pkg.mikv_workspace_check(layer.ws)
    oracle.insert_token(c, bits16(k_new[b:b + 1, h:h + 1]), bits16(v_new[b:b + 1, h:h + 1]), w.context,
                        np.array([[w.budget]], np.int32))
    ref_o, hl, ml = oracle.decode_attention(c, bits16(q[b:b + 1, h:h + 1]), n_lo, sm_scale(), balancer_=ref["balancer"])
    vmax = max(float(raw[1][b, h].float().abs().max()), float(v_new[b, h].float().abs().max()))
    err = np.abs(out[b, h:h + 1].cpu().numpy() - ref_o[0])
    assert np.all(err <= 2e-3 * vmax), err.max()
    acc = oracle.update_importance(c["acc"], hl.astype(np.float32), ml.astype(np.float32), 1)
    dem, _ = oracle.select_demote(acc, 1, c["hi_tok"], want_kept=False)
    victim = int(layer.slots[b, h])
    if victim == int(dem[0, 0, 0]):
        oracle.quantize_pack(c, c["k_hi"], c["v_hi"], dem, n_lo, src_tok=c["hi_tok"], balancer_=ref["balancer"])
        np.testing.assert_array_equal(layer.cache.k_codes[b, h, n_lo].cpu().numpy(), c["k_codes"][0, 0, n_lo])
        np.testing.assert_array_equal(layer.cache.k_params[b, h, n_lo].cpu().view(torch.int16).numpy().view(np.uint16),
                                      c["k_params"][0, 0, n_lo])
    else:
        a_sorted = np.sort(acc[0, 0])
        assert abs(a_sorted[1] - a_sorted[0]) < 1e-5 * max(1.0, abs(a_sorted[0]))
