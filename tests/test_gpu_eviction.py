"""The eviction baselines the paper compares against (Sec. 2.2, Fig. 2), run in the library's kernels:

* importance-based eviction (H2O): the MiKV step with no retained set (shape.bits = 0) — the least
  important token is dropped instead of quantized. Checked over several decode steps against the oracle's
  sequence (insert, attention over the important set only, importance update, victim choice);
* oracle eviction: attention over the full cache with top-k sparsity imposed on the attention map
  (layer.oracle_eviction_attention), against the oracle's full attention logits, its top-k choice and
  its attention over the kept tokens; with k = T it is plain attention, with k = 1 the argmax's value."""
import numpy as np
import pytest
import torch

import mikv_inputs as mi
import oracle
import paper_2402_18096_gb300 as pkg
from paper_2402_18096_gb300.layer import oracle_eviction_attention
from _cases import bits16, gpu_layer, raw_inputs, ref_sizes, sm_scale, vmax_per_head

pytestmark = pytest.mark.gpu


def _oracle_h2o(w, raw, b, h):
    k, v, scores, _ = raw
    ks, vs = bits16(k[b:b + 1, h:h + 1]), bits16(v[b:b + 1, h:h + 1])
    sc = scores[b:b + 1, h:h + 1].numpy()
    R = ref_sizes(w)
    _, kept = oracle.select_demote(sc, w.context - R.budget)
    c = oracle.empty_cache(1, 1, w.head_dim, 2, 32, R.hi_cap, 16)
    oracle.gather_hi(c, ks, vs, kept, src_scores=sc)
    return c


@pytest.mark.parametrize("w", [mi.Workload("h2o4", 2, 8, 2, 600, 1, 0, 32, 0.2, seed=61),
                               mi.Workload("h2o1", 1, 4, 4, 300, 1, 0, 32, 0.5, seed=62)], ids=lambda w: w.name)
def test_h2o_eviction_steps(w):
    steps = 5
    raw = raw_inputs(w, balanced=False)
    layer = gpu_layer(w, raw, steps=steps)
    assert layer.shape.bits == 0 and layer.n_lo == 0
    G = w.heads_q // w.heads_kv
    dev = torch.device("cuda")
    refs = {(b, h): _oracle_h2o(w, raw, b, h) for b in range(w.batch) for h in range(w.heads_kv)}
    R = ref_sizes(w)
    assert layer.shape.hi_cap == R.hi_cap
    slots_ref = {key: np.array([[R.budget]], np.int32) for key in refs}
    near_ties = 0
    for step in range(steps):
        q, k_new, v_new = mi.decode_inputs(w, 0, step)
        out = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.float32, device=dev)
        layer.step(q.to(dev), k_new.to(dev), v_new.to(dev), out)
        pkg.mikv_workspace_check(layer.ws)
        assert layer.n_lo == 0
        gslots = layer.slots.cpu().numpy()
        vmax = vmax_per_head(raw[1], v_new)
        for (b, h), c in refs.items():
            slot = slots_ref[(b, h)]
            oracle.insert_token(c, bits16(k_new[b:b + 1, h:h + 1]), bits16(v_new[b:b + 1, h:h + 1]), w.context + step,
                                slot)
            # the important set holds exactly the oracle's tokens
            assert sorted(layer.cache.hi_tok[b, h, :R.hi_cap].tolist()) == sorted(c["hi_tok"][0, 0].tolist())
            qb = bits16(q[b:b + 1, h * G:(h + 1) * G])
            ref_o, hl, ml = oracle.decode_attention(c, qb, 0, sm_scale())
            err = np.abs(out[b, h * G:(h + 1) * G].cpu().numpy() - ref_o[0])
            assert np.all(err <= 2e-3 * vmax[b, h]), (step, b, h, err.max())
            c["acc"] = oracle.update_importance(c["acc"], hl.astype(np.float32), ml.astype(np.float32), G)
            dem, _ = oracle.select_demote(c["acc"], 1, c["hi_tok"], want_kept=False)
            victim = int(dem[0, 0, 0])
            if gslots[b, h] != victim:
                a_sorted = np.sort(c["acc"][0, 0])
                assert abs(a_sorted[1] - a_sorted[0]) < 1e-5 * max(1.0, abs(a_sorted[0])), (step, b, h)
                near_ties += 1
                victim = int(gslots[b, h])
            slots_ref[(b, h)] = np.array([[victim]], np.int32)
    assert near_ties <= 2


def _oracle_topk(k, v, q, budget, b, h, G):
    """Oracle eviction on the CPU oracle for KV head h of batch row b: full attention logits, the budget
    largest per query head (ties: smaller token index), attention over those tokens."""
    T = k.shape[2]
    ks, vs = bits16(k[b:b + 1, h:h + 1]), bits16(v[b:b + 1, h:h + 1])
    full = oracle.empty_cache(1, 1, 128, 2, 32, T, 16)
    oracle.gather_hi(full, ks, vs, np.arange(T, dtype=np.int32).reshape(1, 1, T))
    outs, kept_all, logits_all = [], [], []
    for j in range(G):
        qb = bits16(q[b:b + 1, h * G + j:h * G + j + 1])
        _, logit, _ = oracle.decode_attention(full, qb, 0, sm_scale())
        ids = (T - 1 - np.arange(T, dtype=np.int32)).reshape(1, 1, T)
        _, kept = oracle.select_demote(logit.astype(np.float32), T - budget, ids)
        sel = oracle.empty_cache(1, 1, 128, 2, 32, budget, 16)
        oracle.gather_hi(sel, ks, vs, kept)
        o, _, _ = oracle.decode_attention(sel, qb, 0, sm_scale())
        outs.append(o[0, 0])
        kept_all.append(kept[0, 0])
        logits_all.append(logit[0, 0])
    return np.stack(outs), kept_all, logits_all


@pytest.mark.parametrize("B,Hq,Hkv,T,budget", [(1, 4, 2, 300, 60), (2, 8, 2, 777, 100), (1, 2, 2, 64, 64),
                                               (1, 4, 4, 128, 1)])
def test_oracle_eviction(B, Hq, Hkv, T, budget):
    w = mi.Workload("oe", B, Hq, Hkv, T, 1, 2, 32, 1.0, seed=B * 1000 + T)
    k, v = mi.prefill_kv(w, 0)
    q, _, _ = mi.decode_inputs(w, 0, 0)
    dev = torch.device("cuda")
    out = torch.empty(B, Hq, 128, dtype=torch.float32, device=dev)
    kept = oracle_eviction_attention(k.to(dev), v.to(dev), q.to(dev), budget, sm_scale(), out).cpu().numpy()
    out = out.cpu().numpy()
    G = Hq // Hkv
    vmax = vmax_per_head(v)
    for b in range(B):
        for h in range(Hkv):
            ref, kept_ref, logits = _oracle_topk(k, v, q, budget, b, h, G)
            for j in range(G):
                got = set(kept[b, h * G + j].tolist())
                want = set(kept_ref[j].tolist())
                if got != want:
                    # both sides rank fp32 logits computed in different orders: only near ties may differ
                    edge = np.sort(logits[j])[::-1][budget - 1]
                    diff = got ^ want
                    assert all(abs(logits[j][t] - edge) < 1e-4 for t in diff), (b, h, j)
                    continue
                err = np.abs(out[b, h * G + j] - ref[j])
                assert np.all(err <= 2e-3 * vmax[b, h]), (b, h, j, err.max())
                if budget == 1:  # the kept token's value alone
                    t = kept_ref[j][0]
                    vt = v[b, h, t].float().numpy()
                    assert np.all(np.abs(out[b, h * G + j] - vt) <= 2e-3 * vmax[b, h])
