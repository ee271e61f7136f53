"""Pins of the oracle's prefill importance (accumulated causal attention of every prefill token), CPU only:
uniform attention (q = 0) gives the closed form H_T - H_t (harmonic numbers) per query head; every query
row's weights sum to one, so the scores of a KV head sum to G * T; a single token scores G; and random
inputs match a textbook masked-softmax attention map (torch, fp64) summed over queries and query heads."""
import math

import numpy as np
import pytest
import torch

import oracle
from mikv_inputs import bf16_bits

D = 128


def _bf16(x):
    return x.to(torch.bfloat16)


@pytest.mark.parametrize("T,G", [(1, 1), (7, 2), (33, 1)])
def test_uniform_attention_harmonic_closed_form(T, G):
    q = torch.zeros(1, G, T, D)
    k = torch.randn(1, 1, T, D, generator=torch.Generator().manual_seed(T))
    s = oracle.prefill_scores(bf16_bits(_bf16(q)), bf16_bits(_bf16(k)), 0.1)
    H = np.concatenate([[0.0], np.cumsum(1.0 / np.arange(1, T + 1))])  # H[n] = 1 + 1/2 + ... + 1/n
    want = G * (H[T] - H[np.arange(T)])  # query i spreads 1/(i+1) over keys 0..i
    np.testing.assert_allclose(s[0, 0], want, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("B,Hq,Hkv,T", [(1, 2, 1, 40), (2, 4, 2, 17)])
def test_rows_sum_to_one_and_textbook_map(B, Hq, Hkv, T):
    g = torch.Generator().manual_seed(B * 100 + T)
    q = _bf16(torch.randn(B, Hq, T, D, generator=g) * 1.5)
    k = _bf16(torch.randn(B, Hkv, T, D, generator=g))
    scale = 1 / math.sqrt(D)
    s = oracle.prefill_scores(bf16_bits(q), bf16_bits(k), scale)
    G = Hq // Hkv
    np.testing.assert_allclose(s.sum(axis=2), G * T, rtol=1e-12)
    kk = k.double().repeat_interleave(G, 1)
    logits = torch.einsum("bhid,bhtd->bhit", q.double(), kk) * scale
    mask = torch.ones(T, T, dtype=torch.bool).tril()
    p = torch.softmax(logits.masked_fill(~mask, float("-inf")), dim=-1)  # [B, Hq, i, t]
    want = p.sum(dim=2).reshape(B, Hkv, G, T).sum(dim=2)
    np.testing.assert_allclose(s, want.numpy(), rtol=1e-10, atol=1e-12)


def test_single_token():
    q = _bf16(torch.randn(1, 4, 1, D))
    k = _bf16(torch.randn(1, 2, 1, D))
    np.testing.assert_array_equal(oracle.prefill_scores(bf16_bits(q), bf16_bits(k), 0.3), np.full((1, 2, 1), 2.0))
