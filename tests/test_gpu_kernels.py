"""GPU parity of the small kernels against the CPU oracle: quantize/pack (bit-exact codes, fp16 alpha
and beta, token ids), the Eq. 2 balancer (bit-exact), demotion choice (bit-exact index sets),
importance update (fp32 tolerance), insertion and important-set build (bit-exact)."""
import numpy as np
import pytest
import torch

import mikv_inputs as mi
import oracle
import paper_2402_18096_gb300 as pkg
from _cases import bits16, new_workspace

pytestmark = pytest.mark.gpu
D = 128


def _rand_bf16(*shape, gen, scale=1.0):
    return (torch.randn(*shape, generator=gen) * scale).to(torch.bfloat16)


@pytest.mark.parametrize("bits", [2, 3, 4])
@pytest.mark.parametrize("group", [32, 64, 128])
def test_quantize_pack_bit_exact(bits, group):
    gen = torch.Generator().manual_seed(bits * 100 + group)
    B, Hq, Hkv, n_src, n_rows, lo_start = 2, 8, 4, 37, 21, 5
    shape = pkg.Shape(B, Hq, Hkv, bits, group, hi_cap=1, lo_cap=32)
    k = _rand_bf16(B, Hkv, n_src, D, gen=gen, scale=3.0)
    k[..., 7] *= 10  # an outlier channel
    v = _rand_bf16(B, Hkv, n_src, D, gen=gen)
    k[0, 1, 3] = 1.5   # a constant row (zero span in every group)
    v[1, 2, 4, :64] = 0.0
    bal = (torch.rand(Hkv, D, generator=gen) * 3 + 0.2).float()
    tok = torch.randint(0, 1 << 30, (B, Hkv, n_src), generator=gen, dtype=torch.int32)
    rows = torch.randint(0, n_src, (B, Hkv, n_rows), generator=gen, dtype=torch.int32)
    rows[0, 0, 0] = 3
    rows[0, 1, 0] = 3
    rows[1, 2, 1] = 4

    dev = torch.device("cuda")
    cache = pkg.LayerCache(shape, device=dev, balancer=bal.to(dev))
    pkg.mikv_quantize_pack(cache, k.to(dev), v.to(dev), rows.to(dev), lo_start, src_tok=tok.to(dev))
    torch.cuda.synchronize()

    ref = oracle.empty_cache(B, Hkv, D, bits, group, 1, 32)
    oracle.quantize_pack(ref, bits16(k), bits16(v), rows.numpy(), lo_start, src_tok=tok.numpy(),
                         balancer_=bal.numpy())
    sl = slice(lo_start, lo_start + n_rows)
    for name in ("k_codes", "v_codes", "lo_tok"):
        got = getattr(cache, name)[:, :, sl].cpu().numpy()
        np.testing.assert_array_equal(got, ref[name][:, :, sl], err_msg=name)
    for name in ("k_params", "v_params"):
        got = getattr(cache, name)[:, :, sl].cpu().view(torch.int16).numpy().view(np.uint16)
        np.testing.assert_array_equal(got, ref[name][:, :, sl], err_msg=name)
    # rows outside the written range stay untouched
    assert int(cache.k_codes[:, :, :lo_start].abs().sum()) == 0


@pytest.mark.parametrize("bits", [2, 3, 4])
@pytest.mark.parametrize("group", [32, 128])
def test_quantize_pack_exact_ties(bits, group):
    """Every quotient (x - beta) / alpha an exact half-integer (beta = -s, alpha = s / 4 with s a power of
    two, x = beta + alpha (m + 1/2)): the codes must round half to even exactly as the IEEE quotient does,
    which the kernel's reciprocal product only decides after falling back to the division."""
    qmax = (1 << bits) - 1
    B, Hkv, n_src = 1, 2, 24
    shape = pkg.Shape(B, 2, Hkv, bits, group, hi_cap=1, lo_cap=32)
    rows_ = []
    for r in range(B * Hkv * n_src):
        s = 2.0 ** ((r % 7) - 3)
        beta, alpha = -s, s / 4
        m = np.arange(D) % group
        x = beta + alpha * ((m * 5 + r) % qmax + 0.5)
        x[m == 0] = beta                   # the group's minimum
        x[m == 1] = beta + alpha * qmax    # and maximum: alpha = span / qmax exactly
        rows_.append(x)
    kv = torch.tensor(np.array(rows_), dtype=torch.float32).reshape(B, Hkv, n_src, D).to(torch.bfloat16)
    assert torch.equal(kv.float().reshape(-1, D), torch.tensor(np.array(rows_), dtype=torch.float32))  # exact
    k, v = kv, kv.flip(2).contiguous()
    rows = torch.arange(n_src, dtype=torch.int32).expand(B, Hkv, n_src).contiguous()[..., :20].contiguous()
    dev = torch.device("cuda")
    cache = pkg.LayerCache(shape, device=dev)
    pkg.mikv_quantize_pack(cache, k.to(dev), v.to(dev), rows.to(dev), 0)
    torch.cuda.synchronize()
    ref = oracle.empty_cache(B, Hkv, D, bits, group, 1, 32)
    oracle.quantize_pack(ref, bits16(k), bits16(v), rows.numpy(), 0)
    for name in ("k_codes", "v_codes"):
        np.testing.assert_array_equal(getattr(cache, name)[:, :, :20].cpu().numpy(), ref[name][:, :, :20],
                                      err_msg=name)
    for name in ("k_params", "v_params"):
        got = getattr(cache, name)[:, :, :20].cpu().view(torch.int16).numpy().view(np.uint16)
        np.testing.assert_array_equal(got, ref[name][:, :, :20], err_msg=name)


def test_quantize_pack_without_balancer_and_skips_bad_rows():
    gen = torch.Generator().manual_seed(3)
    B, Hkv, n_src = 1, 2, 8
    shape = pkg.Shape(B, 2, Hkv, 2, 32, hi_cap=1, lo_cap=16)
    k = _rand_bf16(B, Hkv, n_src, D, gen=gen)
    v = _rand_bf16(B, Hkv, n_src, D, gen=gen)
    rows = torch.tensor([[[1, 9], [0, -1]]], dtype=torch.int32)  # 9 and -1 are out of range: skipped
    dev = torch.device("cuda")
    cache = pkg.LayerCache(shape, device=dev)
    cache.k_codes.fill_(0xAB)
    pkg.mikv_quantize_pack(cache, k.to(dev), v.to(dev), rows.to(dev), 0)
    ref = oracle.empty_cache(B, Hkv, D, 2, 32, 1, 16)
    ok_rows = torch.tensor([[[1], [0]]], dtype=torch.int32)
    oracle.quantize_pack(ref, bits16(k), bits16(v), ok_rows.numpy(), 0)
    got = cache.k_codes.cpu().numpy()
    np.testing.assert_array_equal(got[:, :, 0], ref["k_codes"][:, :, 0])
    assert np.all(got[:, :, 1] == 0xAB)  # skipped rows are not written


@pytest.mark.parametrize("B,Hq,Hkv,T", [(2, 8, 2, 300), (3, 4, 4, 1), (1, 32, 8, 1000)])
def test_balancer_bit_exact(B, Hq, Hkv, T):
    gen = torch.Generator().manual_seed(B * 7 + T)
    q_pre = _rand_bf16(B, Hq, T, D, gen=gen, scale=2.0)
    k_pre = _rand_bf16(B, Hkv, T, D, gen=gen, scale=2.0)
    k_pre[:, :, :, 5] = 0.0          # a channel with zero keys -> balancer 1
    q_pre[:, :, :, 9] *= 50          # query outliers
    shape = pkg.Shape(B, Hq, Hkv, 2, 32, hi_cap=1, lo_cap=16)
    dev = torch.device("cuda")
    out = torch.empty(Hkv, D, dtype=torch.float32, device=dev)
    ws = new_workspace(shape, pkg.WS_BALANCER, 0)
    pkg.mikv_compute_balancer(shape, q_pre.to(dev), k_pre.to(dev), out, ws)
    ref = oracle.balancer(bits16(q_pre), bits16(k_pre))
    np.testing.assert_array_equal(out.cpu().numpy().view(np.uint32), ref.view(np.uint32))


@pytest.mark.parametrize("n,n_demote,with_ids", [(1, 1, True), (7, 1, True), (130, 1, False), (6555, 1, True),
                                                 (200, 0, True), (200, 200, False), (512, 410, False),
                                                 (4096, 3277, True), (33, 17, True), (3000, 1500, True)])
def test_select_demote_bit_exact(n, n_demote, with_ids):
    gen = torch.Generator().manual_seed(n * 3 + n_demote)
    B, H = 2, 3
    stride = (n + 15) // 16 * 16 + 16
    scores = torch.rand(B, H, stride, generator=gen)
    scores[0, 0, : n // 2] = torch.tensor([0.5, 0.25, 0.0, -0.0, 1.0])[torch.arange(n // 2) % 5]  # ties, -0
    scores[1, 1] = torch.randn(stride, generator=gen)  # negative scores too
    ids = torch.stack([torch.randperm(10 * stride, generator=gen)[:stride] for _ in range(B * H)])
    ids = ids.reshape(B, H, stride).to(torch.int32)
    dev = torch.device("cuda")
    dem = torch.full((B, H, n_demote), -7, dtype=torch.int32, device=dev)
    kept = torch.full((B, H, n - n_demote), -7, dtype=torch.int32, device=dev)
    pkg.mikv_select_demote(scores.to(dev), n, n_demote, dem, kept, ids=ids.to(dev) if with_ids else None)
    rd, rk = oracle.select_demote(scores[..., :n].numpy(), n_demote, ids[..., :n].numpy() if with_ids else None)
    np.testing.assert_array_equal(dem.cpu().numpy(), rd)
    np.testing.assert_array_equal(kept.cpu().numpy(), rk)


@pytest.mark.parametrize("Hq,Hkv,hi_cap", [(32, 32, 103), (32, 8, 6555), (8, 1, 17)])
def test_update_importance(Hq, Hkv, hi_cap):
    gen = torch.Generator().manual_seed(hi_cap)
    B = 2
    shape = pkg.Shape(B, Hq, Hkv, 2, 32, hi_cap=hi_cap, lo_cap=16)
    dev = torch.device("cuda")
    cache = pkg.LayerCache(shape, device=dev)
    acc0 = torch.rand(B, Hkv, shape.hi_stride, generator=gen) * 5
    cache.acc.copy_(acc0)
    logits = torch.randn(B, Hq, shape.hi_stride, generator=gen) * 3
    m = logits[..., :hi_cap].amax(-1) + torch.rand(B, Hq, generator=gen)
    l = torch.rand(B, Hq, generator=gen) * 100 + 1
    ml = torch.stack([m, l], -1).contiguous()
    pkg.mikv_update_importance(cache, logits.to(dev), ml.to(dev))
    ref = oracle.update_importance(acc0[..., :hi_cap].numpy(), logits[..., :hi_cap].numpy(), ml.numpy(), Hq)
    np.testing.assert_allclose(cache.acc[..., :hi_cap].cpu().numpy(), ref, rtol=2e-6, atol=1e-7)
    # padding slots past hi_cap are not touched
    np.testing.assert_array_equal(cache.acc[..., hi_cap:].cpu().numpy(), acc0[..., hi_cap:].numpy())


def test_insert_and_gather_bit_exact():
    gen = torch.Generator().manual_seed(11)
    B, Hq, Hkv, n_src, hi_cap = 2, 4, 2, 40, 13
    shape = pkg.Shape(B, Hq, Hkv, 2, 32, hi_cap=hi_cap, lo_cap=16)
    dev = torch.device("cuda")
    k = _rand_bf16(B, Hkv, n_src, D, gen=gen)
    v = _rand_bf16(B, Hkv, n_src, D, gen=gen)
    sc = torch.rand(B, Hkv, n_src, generator=gen)
    tok = torch.randint(0, 100000, (B, Hkv, n_src), generator=gen, dtype=torch.int32)
    rows = torch.stack([torch.randperm(n_src, generator=gen)[:hi_cap - 1] for _ in range(B * Hkv)])
    rows = rows.reshape(B, Hkv, hi_cap - 1).to(torch.int32)
    cache = pkg.LayerCache(shape, device=dev)
    pkg.mikv_gather_hi(cache, k.to(dev), v.to(dev), rows.to(dev), src_tok=tok.to(dev), src_scores=sc.to(dev))
    slots = torch.tensor([[hi_cap - 1, 3], [0, hi_cap - 1]], dtype=torch.int32)
    kn = _rand_bf16(B, Hkv, D, gen=gen)
    vn = _rand_bf16(B, Hkv, D, gen=gen)
    pkg.mikv_insert_token(cache, kn.to(dev), vn.to(dev), 777, slots.to(dev))
    ref = oracle.empty_cache(B, Hkv, D, 2, 32, hi_cap, 16)
    oracle.gather_hi(ref, bits16(k), bits16(v), rows.numpy(), src_tok=tok.numpy(), src_scores=sc.numpy())
    oracle.insert_token(ref, bits16(kn), bits16(vn), 777, slots.numpy())
    np.testing.assert_array_equal(bits16(cache.k_hi[:, :, :hi_cap]), ref["k_hi"])
    np.testing.assert_array_equal(bits16(cache.v_hi[:, :, :hi_cap]), ref["v_hi"])
    np.testing.assert_array_equal(cache.hi_tok[:, :, :hi_cap].cpu().numpy(), ref["hi_tok"])
    np.testing.assert_array_equal(cache.acc[:, :, :hi_cap].cpu().numpy(), ref["acc"])
