"""The seeded input recipe (keys, values, queries N(0, 1) in bf16; four outlier key channels per KV head
scaled by 10, two seeded channels below d/2 and their rotary partners c + d/2, shared by the query heads of
the KV head; LogNormal(0, 1) initial scores; k = ratio * T rounded half up), and the generators'
determinism: any subset of rows and heads equals the same slice of the full draw."""
import torch

import mikv_inputs as mi

W = mi.scaled(mi.WORKLOADS["mistral-7b"], batch=2, context=2048, layers=2)  # GQA, G = 4


def test_draws_are_deterministic_and_sliceable():
    k1, v1 = mi.prefill_kv(W, 1)
    k2, v2 = mi.prefill_kv(W, 1)
    assert torch.equal(k1, k2) and torch.equal(v1, v2)
    ks, vs = mi.prefill_kv(W, 1, rows=[1], heads=[3, 5])
    assert torch.equal(ks, k1[1:2, [3, 5]]) and torch.equal(vs, v1[1:2, [3, 5]])
    q = mi.prefill_queries(W, 1)
    assert torch.equal(mi.prefill_queries(W, 1, rows=[0], heads=[7]), q[0:1, [7]])
    s = mi.initial_scores(W, 1)
    assert torch.equal(mi.initial_scores(W, 1, rows=[1], heads=[2]), s[1:2, [2]])
    qd, kd, vd = mi.decode_inputs(W, 1, 5)
    qs, kss, vss = mi.decode_inputs(W, 1, 5, rows=[1], kv_heads=[2])
    assert torch.equal(qs, qd[1:2, 8:12]) and torch.equal(kss, kd[1:2, [2]]) and torch.equal(vss, vd[1:2, [2]])
    # another layer or step draws other numbers
    assert not torch.equal(mi.prefill_kv(W, 0)[0], k1)
    assert not torch.equal(mi.decode_inputs(W, 1, 6)[0], qd)


def test_shapes_and_dtypes():
    k, v = mi.prefill_kv(W, 0)
    assert k.shape == v.shape == (2, 8, 2048, 128) and k.dtype == v.dtype == torch.bfloat16
    assert mi.prefill_queries(W, 0).shape == (2, 32, 2048, 128)
    assert mi.initial_scores(W, 0).shape == (2, 8, 2048)
    q, kn, vn = mi.decode_inputs(W, 0, 0)
    assert q.shape == (2, 32, 128) and kn.shape == vn.shape == (2, 8, 128)


def test_outlier_channels_and_their_rotary_partners():
    for layer in range(3):
        oc = mi.outlier_channels(W, layer)
        assert oc.shape == (8, 4)
        for h in range(8):
            c = sorted(oc[h, :2].tolist())
            assert len(set(c)) == 2 and all(0 <= x < 64 for x in c)
            assert oc[h, 2:].tolist() == [x + 64 for x in oc[h, :2].tolist()]
    k, v = mi.prefill_kv(W, 1)
    q = mi.prefill_queries(W, 1)
    oc = mi.outlier_channels(W, 1)
    ksd = k.float().std(dim=(0, 2))  # [Hkv, d]
    vsd = v.float().std(dim=(0, 2))
    qsd = q.float().std(dim=(0, 2))  # [Hq, d]
    for h in range(8):
        mask = torch.zeros(128, dtype=torch.bool)
        mask[oc[h]] = True
        assert torch.allclose(ksd[h, mask], torch.full((4,), 10.0), rtol=0.05)
        assert torch.allclose(ksd[h, ~mask], torch.ones(124), rtol=0.08)
        assert torch.allclose(vsd[h], torch.ones(128), rtol=0.08)  # values have no outliers
        for j in range(4):  # the G query heads of KV head h share its outlier channels
            assert torch.allclose(qsd[4 * h + j, mask], torch.full((4,), 10.0), rtol=0.05)
            assert torch.allclose(qsd[4 * h + j, ~mask], torch.ones(124), rtol=0.08)
    # decode-time keys carry the same channels
    kn = torch.stack([mi.decode_inputs(W, 1, s)[1] for s in range(64)]).float()  # [steps, B, Hkv, d]
    knsd = kn.std(dim=(0, 1))
    for h in range(8):
        assert knsd[h, oc[h]].min() > 5 * knsd[h].median()


def test_normal_draws_and_lognormal_scores():
    _, v = mi.prefill_kv(W, 0)
    assert abs(v.float().mean().item()) < 0.01 and abs(v.float().std().item() - 1.0) < 0.01
    logs = mi.initial_scores(W, 0).log()
    assert abs(logs.mean().item()) < 0.02 and abs(logs.std().item() - 1.0) < 0.02
    assert bool((mi.initial_scores(W, 0) > 0).all())


def test_workload_table():
    assert len(mi.sweep_workloads()) == 30
    for w in mi.sweep_workloads():  # every sweep point is also reachable by its short name
        assert mi.WORKLOADS[f"sweep-int{w.bits}-g{w.group}-r{int(w.ratio * 100)}"] == w
    assert not hasattr(mi.Workload, "budget")  # the ratio -> token count rule lives on each side, not here
