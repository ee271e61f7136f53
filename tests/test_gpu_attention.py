"""GPU parity of the decode path against the CPU oracle.

Each case draws the same seeded raw inputs (prefill K/V with outlier key channels, prefill queries,
importance scores, the decode token); the CUDA library and the oracle each build their own cache
from them and attend. Compared: balancer, important set and retained set bit-exact; attention output
within max|err| <= 2e-3 * max|V| (a bf16 output also equal to the rounding of the fp32 one); logits, softmax
statistics and accumulated scores within per-token bounds derived from the kernel's arithmetic (logit_bounds).
"""
import math

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
# every retained layout (bits x group): ragged lengths, several units per head; with two query heads per KV head
# and with one (the group-column path of G = 1)
for _b in (2, 3, 4):
    for _g in (32, 64, 128):
        CASES[f"layout-int{_b}-g{_g}"] = mi.Workload(f"l{_b}{_g}", 1, 4, 2, 611, 1, _b, _g, 0.15, seed=10 * _b + _g)
        CASES[f"layout-mha-int{_b}-g{_g}"] = mi.Workload(f"m{_b}{_g}", 1, 3, 3, 611, 1, _b, _g, 0.15,
                                                         seed=100 + 10 * _b + _g)


def _check_cache(layer, refs, w):
    R = ref_sizes(w)
    assert layer.shape.hi_cap == R.hi_cap and layer.n_lo == R.n_lo0  # library budget = oracle budget
    k_b = R.budget
    for r in refs:
        b, h, c = r["b"], r["h"], r["cache"]
        if r["balancer"] is not None:
            np.testing.assert_array_equal(layer.cache.balancer[h].cpu().numpy().view(np.uint32),
                                          r["balancer"][0].view(np.uint32))
        np.testing.assert_array_equal(bits16(layer.cache.k_hi[b, h, :k_b]), c["k_hi"][0, 0, :k_b])
        np.testing.assert_array_equal(bits16(layer.cache.v_hi[b, h, :k_b]), c["v_hi"][0, 0, :k_b])
        np.testing.assert_array_equal(layer.cache.hi_tok[b, h, :k_b].cpu().numpy(), c["hi_tok"][0, 0, :k_b])
        n_lo = R.n_lo0
        for name in ("k_codes", "v_codes", "lo_tok"):
            np.testing.assert_array_equal(getattr(layer.cache, name)[b, h, :n_lo].cpu().numpy(),
                                          c[name][0, 0, :n_lo], err_msg=name)
        for name in ("k_params", "v_params"):
            got = getattr(layer.cache, name)[b, h, :n_lo].cpu().view(torch.int16).numpy().view(np.uint16)
            np.testing.assert_array_equal(got, c[name][0, 0, :n_lo], err_msg=name)


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_attention_matches_oracle(name, out_dtype):
    w = CASES[name]
    raw = raw_inputs(w)
    layer = gpu_layer(w, raw)
    refs = oracle_layer(w, raw, layer.shape.lo_cap)
    _check_cache(layer, refs, w)
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
                            np.array([[R.budget]], np.int32))
        qb = bits16(q[b:b + 1, h * G:(h + 1) * G])
        ref_o, ref_l, ref_ml = oracle.decode_attention(c, qb, R.n_lo0, sm_scale(), balancer_=r["balancer"])
        sl = slice(h * G, (h + 1) * G)
        assert_attention_close(out_c[b, sl], ref_o[0], vmax[b, h], f32=None if out32 is None else out32[b, sl],
                               msg=f"{name} b{b} h{h}")
        hb, lb = logit_bounds(c, qb, r["balancer"], w.bits, w.group, R.n_lo0, sm_scale())
        E, l_rtol = softmax_stat_bounds(hb, lb, R.hi_cap + R.n_lo0)
        assert np.all(np.abs(hl_c[b, sl, :R.hi_cap] - ref_l[0]) <= hb), "important-set logits"
        assert np.all(np.abs(ml_c[b, sl, 0] - ref_ml[0, :, 0]) <= E), "softmax max"
        assert np.all(np.abs(ml_c[b, sl, 1] / ref_ml[0, :, 1] - 1) <= l_rtol), "softmax sum"


@pytest.mark.parametrize("w", [mi.Workload("traj", 2, 8, 2, 500, 1, 2, 32, 0.2, seed=21),
                               mi.Workload("traj-mha", 2, 4, 4, 500, 1, 3, 64, 0.1, seed=22)], ids=lambda w: w.name)
def test_decode_steps_trajectory(w):
    """Several whole decode steps (insert, attend, update, select, demote) through mikv_decode_step
    against the oracle's step sequence: chosen victims, appended retained rows and outputs (G = 4, and G = 1 on
    the group-column path)."""
    steps = 6
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
                                slot)
            qb = bits16(q[b:b + 1, h * G:(h + 1) * G])
            ref_o, hl, ml = oracle.decode_attention(c, qb, n_lo, sm_scale(), balancer_=r["balancer"])
            err = np.abs(out[b, h * G:(h + 1) * G].cpu().numpy() - ref_o[0])
            assert np.all(err <= 2e-3 * vmax[b, h]), (step, b, h, err.max())
            acc_before = c["acc"][0, 0].astype(np.float64)
            c["acc"] = oracle.update_importance(c["acc"], hl.astype(np.float32), ml.astype(np.float32), G)
            # each step adds the softmax weight exp(s_i - m) / l of every query head: its relative error is at most
            # that of s_i plus those of m and l (logit_bounds), plus the fp32 roundings of the weight (2^-21); the
            # fp32 add into the score rounds once (2^-24 of the new score, taken twice). Errors add up over steps.
            hb, lb = logit_bounds(c, qb, r["balancer"], w.bits, w.group, n_lo, sm_scale())
            E, l_rtol = softmax_stat_bounds(hb, lb, R.hi_cap + n_lo)
            inc_rtol = float((np.expm1(2 * E) + l_rtol).max()) + 2.0 ** -21
            tol = acc_tol.setdefault((b, h), np.zeros(R.hi_cap))
            tol[slot[0, 0]] = 0.0
            tol += inc_rtol * np.abs(c["acc"][0, 0] - acc_before) + 2.0 ** -23 * np.abs(c["acc"][0, 0])
            acc_gpu = layer.cache.acc[b, h, :R.hi_cap].cpu().numpy()
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
    ws = new_workspace(shape, pkg.WS_ATTENTION, layer.n_lo)
    pkg.mikv_decode_attention(layer.cache, layer.n_lo, q, sm_scale(), out_a, ws, ml=ml)
    out = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.bfloat16, device=dev)
    layer.step(q, k_new, v_new, out)  # re-inserts the same token into the same slot: idempotent
    pkg.mikv_workspace_check(layer.ws)
    victims = layer.slots.cpu().numpy()
    R = ref_sizes(w)
    for b, h in heads:
        raw = (k[:, h:h + 1].cpu(), v[:, h:h + 1].cpu(), scores[:, h:h + 1].cpu(),
               q_pre[:, h * G:(h + 1) * G].cpu())
        sub = mi.scaled(w, heads_q=G, heads_kv=1)
        ref = oracle_layer(sub, raw, shape.lo_cap, heads=[(b, 0)])[0]
        c = ref["cache"]
        n_lo = R.n_lo0
        np.testing.assert_array_equal(layer.cache.k_codes[b, h, :n_lo].cpu().numpy(), c["k_codes"][0, 0, :n_lo])
        np.testing.assert_array_equal(layer.cache.v_params[b, h, :n_lo].cpu().view(torch.int16).numpy()
                                      .view(np.uint16), c["v_params"][0, 0, :n_lo])
        oracle.insert_token(c, bits16(k_new[b:b + 1, h:h + 1]), bits16(v_new[b:b + 1, h:h + 1]), w.context,
                            np.array([[R.budget]], np.int32))
        qb = bits16(q[b:b + 1, h * G:(h + 1) * G])
        ref_o, hl, rml = oracle.decode_attention(c, qb, n_lo, sm_scale(), balancer_=ref["balancer"])
        vmax = max(float(v[b, h].float().abs().max()), float(v_new[b, h].float().abs().max()))
        sl = slice(h * G, (h + 1) * G)
        assert_attention_close(out[b, sl].cpu(), ref_o[0], vmax, f32=out_a[b, sl].cpu(), msg=f"{wname} b{b} h{h}")
        assert_attention_close(out_a[b, sl].cpu(), ref_o[0], vmax, msg=f"{wname} b{b} h{h} fp32")
        # softmax statistics: every token is counted once (a lost or doubled block moves l far more than the bound)
        hb, lb = logit_bounds(c, qb, ref["balancer"], w.bits, w.group, n_lo, sm_scale())
        E, l_rtol = softmax_stat_bounds(hb, lb, R.hi_cap + n_lo)
        gm = ml[b, h * G:(h + 1) * G].cpu().numpy()
        assert np.all(np.abs(gm[:, 0] - rml[0, :, 0]) <= E)
        assert np.all(np.abs(gm[:, 1] / rml[0, :, 1] - 1) <= l_rtol)
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
                        np.array([[ref_sizes(w).budget]], np.int32))
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


_FULL_SWEEP = [w for w in mi.sweep_workloads() if w.ratio in (0.0, 0.5)]


@pytest.mark.parametrize("w", _FULL_SWEEP, ids=lambda w: f"int{w.bits}-g{w.group}-r{int(w.ratio * 100)}")
def test_sweep_full_batch_sampled_heads(w):
    """A sweep point at its own size (batch 64, 32 heads, T 4096) in the benchmark's launch configuration: the
    cache built by the library, then one fused decode step (bf16 output) and one attention with fp32 output and
    softmax statistics. At this size the persistent grid's equal warp shares (about 1.1 heads per warp) start
    inside most heads, so the sampled heads are split between warps; the oracle checks each sampled (b, KV head)
    one by one: retained codes, output, softmax max and sum, the demoted slot and its packed row."""
    dev = torch.device("cuda")
    from _cases import make_shape
    from paper_2402_18096_gb300.layer import MixedPrecisionLayer
    k, v = mi.prefill_kv(w, 0, dev)
    scores = mi.initial_scores(w, 0, dev)
    q_pre = mi.prefill_queries(w, 0, dev)
    shape = make_shape(w, 1)
    layer = MixedPrecisionLayer.from_prefill(shape, k, v, scores, q_pre, device=dev)
    q, k_new, v_new = mi.decode_inputs(w, 0, 0, dev)
    pkg.mikv_insert_token(layer.cache, k_new, v_new, w.context, layer.slots)
    ml = torch.empty(w.batch, w.heads_q, 2, device=dev)
    out_a = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.float32, device=dev)
    ws = new_workspace(shape, pkg.WS_ATTENTION, layer.n_lo)
    pkg.mikv_decode_attention(layer.cache, layer.n_lo, q, sm_scale(), out_a, ws, ml=ml)
    out = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.bfloat16, device=dev)
    layer.step(q, k_new, v_new, out)  # re-inserts the same token into the same slot: idempotent
    pkg.mikv_workspace_check(layer.ws)
    pkg.mikv_workspace_check(ws)
    victims = layer.slots.cpu().numpy()
    R = ref_sizes(w)
    n_lo = R.n_lo0
    sampled = [(b, h) for b in (0, 21, 42, 63) for h in (0, 11, 22, 31)]
    by_head = {}
    for b, h in sampled:
        by_head.setdefault(h, []).append(b)
    for h, rows in by_head.items():
        raw = (k[:, h:h + 1].cpu(), v[:, h:h + 1].cpu(), scores[:, h:h + 1].cpu(), q_pre[:, h:h + 1].cpu())
        sub = mi.scaled(w, heads_q=1, heads_kv=1)
        for ref in oracle_layer(sub, raw, shape.lo_cap, heads=[(b, 0) for b in rows]):
            b, c = ref["b"], ref["cache"]
            np.testing.assert_array_equal(layer.cache.k_codes[b, h, :n_lo].cpu().numpy(), c["k_codes"][0, 0, :n_lo])
            oracle.insert_token(c, bits16(k_new[b:b + 1, h:h + 1]), bits16(v_new[b:b + 1, h:h + 1]), w.context,
                                np.array([[R.budget]], np.int32))
            qb = bits16(q[b:b + 1, h:h + 1])
            ref_o, hl, rml = oracle.decode_attention(c, qb, n_lo, sm_scale(), balancer_=ref["balancer"])
            vmax = max(float(v[b, h].float().abs().max()), float(v_new[b, h].float().abs().max()))
            assert_attention_close(out[b, h:h + 1].cpu(), ref_o[0], vmax, f32=out_a[b, h:h + 1].cpu())
            assert_attention_close(out_a[b, h:h + 1].cpu(), ref_o[0], vmax)
            hb, lb = logit_bounds(c, qb, ref["balancer"], w.bits, w.group, n_lo, sm_scale())
            E, l_rtol = softmax_stat_bounds(hb, lb, R.hi_cap + n_lo)
            gm = ml[b, h:h + 1].cpu().numpy()
            assert np.all(np.abs(gm[:, 0] - rml[0, :, 0]) <= E)
            assert np.all(np.abs(gm[:, 1] / rml[0, :, 1] - 1) <= l_rtol)
            acc = oracle.update_importance(c["acc"], hl.astype(np.float32), rml.astype(np.float32), 1)
            dem, _ = oracle.select_demote(acc, 1, c["hi_tok"], want_kept=False)
            if int(dem[0, 0, 0]) == int(victims[b, h]):
                oracle.quantize_pack(c, c["k_hi"], c["v_hi"], dem, n_lo, src_tok=c["hi_tok"], balancer_=ref["balancer"])
                np.testing.assert_array_equal(layer.cache.k_codes[b, h, n_lo].cpu().numpy(), c["k_codes"][0, 0, n_lo])
                np.testing.assert_array_equal(layer.cache.v_codes[b, h, n_lo].cpu().numpy(), c["v_codes"][0, 0, n_lo])
                assert int(layer.cache.lo_tok[b, h, n_lo]) == int(c["lo_tok"][0, 0, n_lo])
            else:  # only a near tie of fp32 scores may pick another slot
                a_sorted = np.sort(acc[0, 0])
                assert abs(a_sorted[1] - a_sorted[0]) < 1e-5 * max(1.0, abs(a_sorted[0]))
