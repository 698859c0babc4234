"""Pins of the oracle's decode attention: closed forms, invariances and a
cross-check with PyTorch's scaled_dot_product_attention in float64."""

import numpy as np
import pytest
import torch

from oracle import attention, quant


def _head(rng, L, bk=2, bv=2, R=128, const_keys=False, scale_k=1.0):
    k = (rng.standard_normal((L, 128)) * scale_k).astype(np.float16)
    if const_keys:
        k[:] = k[0]
    v = rng.standard_normal((L, 128)).astype(np.float16)
    return quant.quantize_head(k, v, bk, bv, R)


@pytest.mark.parametrize("L", [1, 40, 300])
def test_constant_keys_give_mean_of_values(L):
    rng = np.random.default_rng(L)
    qh = _head(rng, L, const_keys=True)
    khat, vhat = quant.dequantize_head(qh)
    assert np.all(khat == khat[0])  # constant keys survive quantization (scale 0)
    q = rng.standard_normal((4, 128)).astype(np.float16)
    o = attention.attend_head(q, khat, vhat, 1 / np.sqrt(128))
    assert np.allclose(o, vhat.mean(axis=0)[None], rtol=0, atol=1e-12)


def test_single_token_returns_its_value():
    rng = np.random.default_rng(2)
    qh = _head(rng, 1)
    khat, vhat = quant.dequantize_head(qh)
    q = rng.standard_normal((5, 128)).astype(np.float16)
    o = attention.attend_head(q, khat, vhat, 1 / np.sqrt(128))
    assert np.array_equal(o, np.repeat(vhat[:1], 5, axis=0))


def test_dominant_key_selects_its_value():
    rng = np.random.default_rng(3)
    L = 500
    k = (rng.standard_normal((L, 128)) * 0.01).astype(np.float16)
    k[123] = 8.0
    v = rng.standard_normal((L, 128)).astype(np.float16)
    qh = quant.quantize_head(k, v, 4, 4, 128)
    khat, vhat = quant.dequantize_head(qh)
    q = np.full((1, 128), 8.0)
    s = (q @ khat.T)[0] / np.sqrt(128)
    assert s[123] - np.delete(s, 123).max() > 50
    o = attention.attend_head(q, khat, vhat, 1 / np.sqrt(128))
    assert np.allclose(o[0], vhat[123], rtol=0, atol=1e-12)


@pytest.mark.parametrize("bits", [1, 2, 4, 8])
def test_matches_torch_sdpa_on_dequantized_cache(bits):
    rng = np.random.default_rng(10 + bits)
    hkv, gq, L = 2, 4, 333
    heads = [_head(rng, L, bits, bits, scale_k=3.0) for _ in range(hkv)]
    q = rng.standard_normal((hkv * gq, 128)).astype(np.float16)
    o = attention.decode_attention(q, heads)
    K = torch.tensor(np.stack([quant.dequantize_head(h)[0] for h in heads]))
    V = torch.tensor(np.stack([quant.dequantize_head(h)[1] for h in heads]))
    K = K.repeat_interleave(gq, dim=0)[:, None]  # [Hq, 1, L, d]... as batch of heads
    V = V.repeat_interleave(gq, dim=0)[:, None]
    Q = torch.tensor(q.astype(np.float64))[:, None, None, :]
    ref = torch.nn.functional.scaled_dot_product_attention(Q, K, V)[:, 0, 0].numpy()
    assert np.allclose(o, ref, rtol=0, atol=1e-12)


def test_gqa_mapping_uses_contiguous_query_groups():
    hkv, gq, L = 3, 4, 50
    heads = []
    for h in range(hkv):
        k = np.zeros((L, 128), np.float16)
        v = np.full((L, 128), float(h + 1), np.float16)
        heads.append(quant.quantize_head(k, v, 2, 2, 32))
    q = np.random.default_rng(0).standard_normal((hkv * gq, 128)).astype(np.float16)
    o = attention.decode_attention(q, heads)
    for i in range(hkv * gq):
        assert np.allclose(o[i], float(i // gq + 1), rtol=0, atol=1e-12)


def test_split_merge_equals_unsplit():
    rng = np.random.default_rng(4)
    qh = _head(rng, 777, scale_k=4.0)
    khat, vhat = quant.dequantize_head(qh)
    q = rng.standard_normal((4, 128))
    scale = 1 / np.sqrt(128)
    full = attention.attend_head(q, khat, vhat, scale)
    for bounds in ([0, 777], [0, 1, 777], [0, 100, 333, 700, 777]):
        parts = attention.lse_partials(q, khat, vhat, scale, bounds)
        assert np.allclose(attention.lse_merge(parts), full, rtol=0, atol=1e-12)


def test_token_permutation_invariance():
    rng = np.random.default_rng(5)
    qh = _head(rng, 250)
    khat, vhat = quant.dequantize_head(qh)
    q = rng.standard_normal((4, 128))
    perm = rng.permutation(250)
    a = attention.attend_head(q, khat, vhat, 0.1)
    b = attention.attend_head(q, khat[perm], vhat[perm], 0.1)
    assert np.allclose(a, b, rtol=0, atol=1e-12)


def test_short_context_is_plain_fp16_attention():
    rng = np.random.default_rng(6)
    k = rng.standard_normal((100, 128)).astype(np.float16)
    v = rng.standard_normal((100, 128)).astype(np.float16)
    qh = quant.quantize_head(k, v, 1, 1, 128)
    assert qh["Lq"] == 0
    q = rng.standard_normal((2, 128))
    a = attention.attend_head(q, *quant.dequantize_head(qh), 0.2)
    b = attention.attend_head(q, k.astype(np.float64), v.astype(np.float64), 0.2)
    assert np.array_equal(a, b)


def test_empty_cache_gives_zero():
    qh = quant.quantize_head(np.zeros((0, 128), np.float16), np.zeros((0, 128), np.float16),
                             2, 2, 128)
    o = attention.decode_attention(np.ones((4, 128), np.float16), [qh])
    assert np.array_equal(o, np.zeros((4, 128)))
