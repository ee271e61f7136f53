"""GPU parity of per-channel retained keys with token buffering (App. C): keys quantized per channel over
groups of 64 retained tokens (no balancer), values per token, the tokens of an incomplete group staged in
bf16 after the important slots. Against the oracle on the same seeded inputs: the cache build (group codes
and parameters, staged rows and token ids bit for bit), insert + decode attention, and whole decode steps
across a group boundary (the completed group quantized bit for bit)."""
import numpy as np
import pytest
import torch

import mikv_inputs as mi
import oracle
import paper_2402_18096_gb300 as pkg
from _cases import (assert_attention_close, bits16, gpu_layer, new_workspace, oracle_layer, raw_inputs, ref_sizes,
                    sm_scale, vmax_per_head)

pytestmark = pytest.mark.gpu


def _u16(t):
    return t.cpu().view(torch.int16).numpy().view(np.uint16)


def _check_kch_cache(layer, refs, w, n_lo):
    R = ref_sizes(w)
    assert layer.shape.hi_cap == R.hi_cap
    n_q, n_st = n_lo // 64 * 64, n_lo % 64
    for r in refs:
        b, h, c = r["b"], r["h"], r["cache"]
        for name in ("k_codes", "v_codes", "lo_tok"):
            np.testing.assert_array_equal(getattr(layer.cache, name)[b, h, :n_q].cpu().numpy(), c[name][0, 0, :n_q],
                                          err_msg=name)
        np.testing.assert_array_equal(_u16(layer.cache.k_params[b, h, :n_q // 64]), c["k_params"][0, 0, :n_q // 64])
        np.testing.assert_array_equal(_u16(layer.cache.v_params[b, h, :n_q]), c["v_params"][0, 0, :n_q])
        rows = slice(R.hi_cap, R.hi_cap + n_st)  # the staged retained tokens
        np.testing.assert_array_equal(bits16(layer.cache.k_hi[b, h, rows]), c["k_hi"][0, 0, rows])
        np.testing.assert_array_equal(bits16(layer.cache.v_hi[b, h, rows]), c["v_hi"][0, 0, rows])
        np.testing.assert_array_equal(layer.cache.hi_tok[b, h, rows].cpu().numpy(), c["hi_tok"][0, 0, rows])


def _kch_logit_bound(c, q_bits, w, n_lo):
    """Bound on |GPU - oracle| for logits, from the kernel's arithmetic: a per-channel key logit is
    sum_c fp16(q_c alpha_c) code_tc + sum_c q_c beta_c, fp16 operands and fp32 accumulation, so the rounded
    products q_c alpha_c (2^-11 relative each) dominate; bf16 rows (important and staged) have exact products
    and fp32 sums. 2^-9 (4x margin) of max_t sum_c |q_c alpha_c code_tc| plus 2^-20 of the exact parts."""
    q = np.abs((q_bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)[0])  # [G, d]
    n_q, n_st = n_lo // 64 * 64, n_lo % 64
    kh = (c["k_hi"][0, 0, :ref_sizes(w).hi_cap + n_st].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    worst = (q @ np.abs(kh).T).max(axis=1) * 2.0 ** -20
    for j in range(n_q // 64):
        par = c["k_params"][0, 0, j].view(np.float16).astype(np.float64)  # [d, 2]: alpha, beta
        codes = np.stack([oracle.unpack_row(c["k_codes"][0, 0, t], w.bits) for t in range(64 * j, 64 * j + 64)])
        prod = (q * np.abs(par[:, 0])) @ codes.T.astype(np.float64)  # [G, 64]
        worst = np.maximum(worst, prod.max(axis=1) * 2.0 ** -9 + (q @ np.abs(par[:, 1])) * 2.0 ** -20)
    return sm_scale() * worst + 1e-6  # [G]


CASES = {
    "kch-int2-g32-gqa4": mi.Workload("kc2", 2, 8, 2, 403, 1, 2, 32, 0.2, seed=81, k_channel=True),
    "kch-int3-g64-mha": mi.Workload("kc3", 1, 4, 4, 700, 1, 3, 64, 0.1, seed=82, k_channel=True),
    "kch-int4-g128-gqa8": mi.Workload("kc4", 1, 8, 1, 331, 1, 4, 128, 0.3, seed=83, k_channel=True),
    "kch-int2-exact-groups": mi.Workload("kc5", 1, 4, 2, 160, 1, 2, 32, 0.2, seed=84, k_channel=True),  # 128 retained
}


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_kch_attention(name, out_dtype):
    w = CASES[name]
    raw = raw_inputs(w)
    layer = gpu_layer(w, raw)
    refs = oracle_layer(w, raw, layer.shape.lo_cap)
    R = ref_sizes(w)
    _check_kch_cache(layer, refs, w, R.n_lo0)
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
        ref_o, ref_l, ref_ml = oracle.decode_attention(c, qb, R.n_lo0, sm_scale())
        sl = slice(h * G, (h + 1) * G)
        assert_attention_close(out_c[b, sl], ref_o[0], vmax[b, h], f32=None if out32 is None else out32[b, sl],
                               msg=f"{name} b{b} h{h}")
        bound = _kch_logit_bound(c, qb, w, R.n_lo0)
        np.testing.assert_allclose(hl_c[b, h * G:(h + 1) * G, :R.hi_cap], ref_l[0, :, :R.hi_cap],
                                   atol=float(bound.max()), rtol=0)
        dm = np.abs(ml_c[b, h * G:(h + 1) * G, 0] - ref_ml[0, :, 0])
        assert np.all(dm <= bound), (dm, bound)
        np.testing.assert_allclose(ml_c[b, h * G:(h + 1) * G, 1], ref_ml[0, :, 1], rtol=4 * float(bound.max()) + 1e-5)


@pytest.mark.parametrize("bits,group", [(2, 32), (3, 64), (4, 128)])
def test_kch_decode_steps_across_a_group(bits, group):
    """61 staged tokens after the build: the third step completes the group, which is quantized per channel
    from the staged rows bit for bit; outputs, scores and victims follow the oracle's steps."""
    w = mi.Workload("kct", 2, 8, 2, 396, 1, bits, group, 0.2, seed=85 + bits, k_channel=True)
    R = ref_sizes(w)
    assert R.n_lo0 % 64 == 61
    steps = 6
    raw = raw_inputs(w)
    layer = gpu_layer(w, raw, steps=steps)
    refs = oracle_layer(w, raw, layer.shape.lo_cap)
    G = w.heads_q // w.heads_kv
    dev = torch.device("cuda")
    slots_ref = {(r["b"], r["h"]): np.array([[R.budget]], np.int32) for r in refs}
    near_ties = 0
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
            oracle.insert_token(c, bits16(k_new[b:b + 1, h:h + 1]), bits16(v_new[b:b + 1, h:h + 1]), w.context + step,
                                slots_ref[(b, h)])
            qb = bits16(q[b:b + 1, h * G:(h + 1) * G])
            ref_o, hl, ml = oracle.decode_attention(c, qb, n_lo, sm_scale())
            err = np.abs(out[b, h * G:(h + 1) * G].cpu().numpy() - ref_o[0])
            assert np.all(err <= 2e-3 * vmax[b, h]), (step, b, h, err.max())
            acc = c["acc"][:, :, :R.hi_cap]
            acc = oracle.update_importance(acc, hl[:, :, :R.hi_cap].astype(np.float32), ml.astype(np.float32), G)
            c["acc"][:, :, :R.hi_cap] = acc
            dem, _ = oracle.select_demote(acc, 1, c["hi_tok"][:, :, :R.hi_cap], want_kept=False)
            victim = int(dem[0, 0, 0])
            if gslots[b, h] != victim:
                a_sorted = np.sort(acc[0, 0])
                assert abs(a_sorted[1] - a_sorted[0]) < 1e-5 * max(1.0, abs(a_sorted[0])), (step, b, h)
                near_ties += 1
                victim = int(gslots[b, h])
            oracle.append_retained(c, c["k_hi"], c["v_hi"], np.array([[[victim]]], np.int32), n_lo,
                                   src_tok=c["hi_tok"])
            slots_ref[(b, h)] = np.array([[victim]], np.int32)
        _check_kch_cache(layer, refs, w, n_lo + 1)
    assert near_ties <= 2
