"""The fused decode step (mikv_decode_step: insert, attention, then one kernel that merges, updates the
importance scores, picks the victim and demotes it) against the same step through the separate entry
points (mikv_insert_token, mikv_decode_attention, mikv_update_importance, mikv_select_demote,
mikv_quantize_pack) on two copies of one cache: outputs, scores, victims and demoted rows bit for bit,
over several steps."""
import pytest
import torch

import mikv_inputs as mi
import paper_2402_18096_gb300 as pkg
from _cases import gpu_layer, new_workspace, raw_inputs, sm_scale

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("w", [
    mi.Workload("fz4", 2, 8, 2, 900, 1, 2, 32, 0.2, seed=51),     # GQA G = 4, several hi units
    mi.Workload("fz1", 1, 4, 4, 333, 1, 3, 64, 0.1, seed=52),     # MHA, INT3
    mi.Workload("fz8", 1, 8, 1, 5000, 1, 4, 128, 0.35, seed=53),  # G = 8, hi_cap beyond one round of slots
], ids=lambda w: w.name)
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_fused_step_equals_separate_calls(w, out_dtype):
    steps = 4
    raw = raw_inputs(w)
    fused = gpu_layer(w, raw, steps=steps)
    sep = gpu_layer(w, raw, steps=steps)
    s = sep.shape
    dev = torch.device("cuda")
    ws = new_workspace(s, pkg.WS_ATTENTION, s.lo_cap)
    for step in range(steps):
        q, k_new, v_new = (x.to(dev) for x in mi.decode_inputs(w, 0, step))
        n_lo, pos = sep.n_lo, sep.pos
        out_f = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=out_dtype, device=dev)
        fused.step(q, k_new, v_new, out_f)
        pkg.mikv_workspace_check(fused.ws)

        out_s = torch.empty_like(out_f)
        hl = torch.zeros(w.batch, w.heads_q, s.hi_stride, device=dev)
        ml = torch.empty(w.batch, w.heads_q, 2, device=dev)
        pkg.mikv_insert_token(sep.cache, k_new, v_new, pos, sep.slots)
        pkg.mikv_decode_attention(sep.cache, n_lo, q, sm_scale(), out_s, ws, hi_logits=hl, ml=ml)
        pkg.mikv_update_importance(sep.cache, hl, ml)
        victim = torch.empty(w.batch, w.heads_kv, 1, dtype=torch.int32, device=dev)
        pkg.mikv_select_demote(sep.cache.acc, s.hi_cap, 1, victim, ids=sep.cache.hi_tok)
        pkg.mikv_quantize_pack(sep.cache, sep.cache.k_hi, sep.cache.v_hi, victim, n_lo, src_tok=sep.cache.hi_tok)
        pkg.mikv_workspace_check(ws)
        sep.slots.copy_(victim[..., 0])
        sep.n_lo += 1
        sep.pos += 1

        assert torch.equal(out_f, out_s), step
        assert torch.equal(fused.cache.acc[..., :s.hi_cap], sep.cache.acc[..., :s.hi_cap]), step
        assert torch.equal(fused.slots, sep.slots), step
        for name in ("k_codes", "v_codes", "k_params", "v_params", "lo_tok"):
            assert torch.equal(getattr(fused.cache, name)[:, :, n_lo], getattr(sep.cache, name)[:, :, n_lo]), (name, step)
