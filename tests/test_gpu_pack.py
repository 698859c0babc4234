"""kvq_pack (CUDA, through the C ABI) against the oracle quantizer: packed
codes, scales, zeros and the fp16 residual window must be bit-identical."""

import numpy as np
import pytest
import torch

import _util
from oracle import quant
from paper_2607_16248_gb300 import kvq, synth

pytestmark = pytest.mark.gpu

BIT_PAIRS = [(1, 1), (2, 2), (4, 4), (8, 8), (2, 1), (1, 2), (8, 1)]


@pytest.mark.parametrize("bk,bv", BIT_PAIRS)
def test_prefill_ragged_batch(kvq_lib, bk, bv):
    lengths = [1, 31, 128, 159, 160, 161, 193, 1000, 4096, 0]
    cfg = kvq.CacheConfig(batch=len(lengths), n_q_heads=8, n_kv_heads=2, bits_k=bk, bits_v=bv,
                          max_len=4352)
    cache, kv = _util.make_cache(cfg, lengths, seed=bk * 10 + bv)
    assert cache.seq_lens().cpu().tolist() == lengths
    assert cache.flags() == 0
    for b, L in enumerate(lengths):
        k, v = kv[b]
        for h in range(cfg.n_kv_heads):
            want = quant.quantize_head(k[h].numpy(), v[h].numpy(), bk, bv, cfg.residual)
            _util.assert_head_equal(_util.head_arrays(cache, b, h, L), want)


@pytest.mark.parametrize("bk,bv", [(1, 1), (2, 2), (4, 8)])
def test_decode_appends_cross_flush_boundaries(kvq_lib, bk, bv):
    cfg = kvq.CacheConfig(batch=3, n_q_heads=4, n_kv_heads=1, bits_k=bk, bits_v=bv,
                          max_len=512, residual=64)
    L0 = [0, 90, 95]
    total = 200
    cache = kvq.QuantKVCache(cfg)
    ks, vs = synth.kv_heads(7, 3, total + 10)  # [3 sequences as heads, T, 128]
    for b, L in enumerate(L0):
        if L:
            kvq.kvq_pack(cache, ks[b:b + 1, :L][None].cuda(), vs[b:b + 1, :L][None].cuda(),
                         batch_begin=b)
    lens = list(L0)
    for step in range(total - 95):
        kn = torch.stack([ks[b, lens[b]] for b in range(3)])[:, None, None].cuda()
        vn = torch.stack([vs[b, lens[b]] for b in range(3)])[:, None, None].cuda()
        kvq.kvq_pack(cache, kn.contiguous(), vn.contiguous())
        lens = [x + 1 for x in lens]
        if step % 9 == 0 or step > total - 100:
            torch.cuda.synchronize()
            assert cache.seq_lens().cpu().tolist() == lens
            for b in range(3):
                L = lens[b]
                want = quant.quantize_head(ks[b, :L].numpy(), vs[b, :L].numpy(), bk, bv, 64)
                _util.assert_head_equal(_util.head_arrays(cache, b, 0, L), want)


def test_multi_token_appends_match_one_shot_prefill(kvq_lib):
    cfg = kvq.CacheConfig(batch=1, n_q_heads=4, n_kv_heads=2, bits_k=2, bits_v=4, max_len=1024)
    k, v = synth.kv_heads(11, 2, 700)
    cache = kvq.QuantKVCache(cfg)
    pos = 0
    for n in (5, 33, 1, 64, 200, 31, 32, 100, 234):
        kvq.kvq_pack(cache, k[:, pos:pos + n][None].contiguous().cuda(),
                     v[:, pos:pos + n][None].contiguous().cuda())
        pos += n
    assert pos == 700
    torch.cuda.synchronize()
    for h in range(2):
        want = quant.quantize_head(k[h].numpy(), v[h].numpy(), 2, 4, 128)
        _util.assert_head_equal(_util.head_arrays(cache, 0, h, 700), want)


def test_overflow_sets_flag_and_leaves_cache(kvq_lib):
    cfg = kvq.CacheConfig(batch=2, n_q_heads=4, n_kv_heads=1, bits_k=1, bits_v=1, max_len=256)
    k, v = synth.kv_heads(3, 1, 300)
    cache = kvq.QuantKVCache(cfg)
    kvq.kvq_pack(cache, k[:, :250][None].cuda(), v[:, :250][None].cuda(), batch_begin=0)
    before = cache.buffer.clone()
    kvq.kvq_pack(cache, k[:, 250:260][None].cuda(), v[:, 250:260][None].cuda(), batch_begin=0)
    torch.cuda.synchronize()
    assert cache.flags() & kvq.FLAG_OVERFLOW
    assert cache.seq_lens().cpu().tolist() == [250, 0]
    diff = (cache.buffer != before).nonzero().flatten().cpu()
    flag_byte = cache.offsets[3] + 4 * cfg.batch
    assert all(flag_byte <= int(i) < flag_byte + 4 for i in diff)
    cache.reset()
    torch.cuda.synchronize()
    assert cache.flags() == 0 and cache.seq_lens().cpu().tolist() == [0, 0]


def test_constant_and_grid_groups_reach_exact_codes(kvq_lib):
    cfg = kvq.CacheConfig(batch=1, n_q_heads=1, n_kv_heads=1, bits_k=8, bits_v=2, max_len=256)
    L = 192
    k = torch.zeros(1, L, 128, dtype=torch.float16)
    k[0, :, :64] = 3.5  # constant key groups -> scale 0, code 0
    k[0, :, 64:] = torch.arange(L, dtype=torch.float16)[:, None] % 32 * 8  # grid 0, 8, .. 240
    k[0, 31::32, 64:] = 255.0  # with 255 on top: range 255, scale 1, codes = values
    v = (torch.arange(128) % 4).to(torch.float16).repeat(1, L, 1) * 0.25 - 1.0  # grid on 0.25
    cache = kvq.QuantKVCache(cfg)
    kvq.kvq_pack(cache, k[None].cuda(), v[None].cuda())
    torch.cuda.synchronize()
    got = _util.head_arrays(cache, 0, 0, L)
    want = quant.quantize_head(k[0].numpy(), v[0].numpy(), 8, 2, 128)
    _util.assert_head_equal(got, want)
    assert np.all(got["k_scale"][:, :64] == 0)
    assert np.all(got["k_scale"][:, 64:] == 1)
    assert np.all(got["v_scale"].astype(np.float64) == 0.25)


@pytest.mark.parametrize("bits", [1, 2, 4, 8])
def test_exact_ties_round_to_even(kvq_lib, bits):
    # Every group holds 0, 3 * levels and values 1.5 (2m + 1): scale 3 (not a
    # power of two), so (x - zero) / scale = m + 0.5 exactly and each code is
    # a tie that rounds to even.  RN32(1 / 3) times such an x lands just off
    # the half-integer, so only the exact quotient gives these codes.
    levels = (1 << bits) - 1

    def pattern(i, c):
        if i == 0:
            return 0.0
        if i == 1:
            return 3.0 * levels
        return 1.5 * (2 * ((7 * i + c) % levels) + 1)

    L = 160
    k = torch.empty(1, L, 128, dtype=torch.float16)
    v = torch.empty(1, L, 128, dtype=torch.float16)
    for t in range(L):
        for c in range(128):
            k[0, t, c] = pattern(t % 32, c)
            v[0, t, c] = pattern(c % 32, t + c // 32)
    cfg = kvq.CacheConfig(batch=1, n_q_heads=1, n_kv_heads=1, bits_k=bits, bits_v=bits,
                          max_len=256)
    cache = kvq.QuantKVCache(cfg)
    kvq.kvq_pack(cache, k[None].cuda(), v[None].cuda())
    torch.cuda.synchronize()
    got = _util.head_arrays(cache, 0, 0, L)
    want = quant.quantize_head(k[0].numpy(), v[0].numpy(), bits, bits, 128)
    assert np.all(want["k_scale"].astype(np.float64) == 3.0)
    assert np.all(want["v_scale"].astype(np.float64) == 3.0)
    _util.assert_head_equal(got, want)


def test_tie_where_a_reciprocal_product_misrounds(kvq_lib):
    # 2-bit groups of range 0.6650390625 = 3 x 0.2216796875 (scale
    # 0.2216796875): 0.33251953125 / scale is exactly 1.5 (code 2), while
    # 0.33251953125 * RN32(1 / scale) rounds to 1.4999999 (code 1).
    pat = [0.0, 0.6650390625, 0.11083984375, 0.33251953125, 0.55419921875]

    def pattern(i, c):
        return pat[i] if i < 2 else pat[2 + (i + c) % 3]

    L = 160
    k = torch.empty(1, L, 128, dtype=torch.float16)
    v = torch.empty(1, L, 128, dtype=torch.float16)
    for t in range(L):
        for c in range(128):
            k[0, t, c] = pattern(t % 32, c)
            v[0, t, c] = pattern(c % 32, t)
    cfg = kvq.CacheConfig(batch=1, n_q_heads=1, n_kv_heads=1, bits_k=2, bits_v=2, max_len=256)
    cache = kvq.QuantKVCache(cfg)
    kvq.kvq_pack(cache, k[None].cuda(), v[None].cuda())
    torch.cuda.synchronize()
    got = _util.head_arrays(cache, 0, 0, L)
    want = quant.quantize_head(k[0].numpy(), v[0].numpy(), 2, 2, 128)
    assert np.all(want["k_scale"].astype(np.float64) == 0.2216796875)
    _util.assert_head_equal(got, want)


def _one_tie_per_group(rng, L, bits):
    """[L, 128] fp16 keys and values whose every quantization group (keys: 32
    tokens of a channel; values: 32 channels of a token) holds its min -1,
    its max -1 + levels * 0.1875 (so the scale is 0.1875, not a power of two),
    one exact tie -1 + (m + 0.5) * 0.1875 and 29 uniform values in between,
    at random places."""
    levels = (1 << bits) - 1
    lo, s = -1.0, 0.1875

    def groups(n):
        g = rng.uniform(lo, lo + levels * s, (n, 32))
        pos = np.argsort(rng.random((n, 32)), axis=1)[:, :3]
        r = np.arange(n)
        g[r, pos[:, 0]] = lo
        g[r, pos[:, 1]] = lo + levels * s
        g[r, pos[:, 2]] = lo + (rng.integers(0, levels, n) + 0.5) * s
        return g.astype(np.float16)

    nb = L // 32
    k = groups(nb * 128).reshape(nb, 128, 32).transpose(0, 2, 1).reshape(L, 128)
    v = groups(L * 4).reshape(L, 128)
    return torch.from_numpy(np.ascontiguousarray(k)), torch.from_numpy(v)


@pytest.mark.parametrize("bits", [1, 2, 4, 8])
def test_one_tie_among_random_values_per_group(kvq_lib, bits):
    # The tie's code comes from the exact quotient while the other 31 codes
    # of its words come from the fused rounding: the tie's field is replaced
    # in place, through kvq_pack and through the decode step's flush.
    rng = np.random.default_rng(500 + bits)
    L, L0 = 320, 150
    cfg = kvq.CacheConfig(batch=2, n_q_heads=8, n_kv_heads=2, bits_k=bits, bits_v=bits,
                          max_len=512)
    kv = [[_one_tie_per_group(rng, L, bits) for _ in range(2)] for _ in range(2)]
    k_all = [torch.stack([kv[b][h][0] for h in range(2)]) for b in range(2)]  # [Hkv, L, 128]
    v_all = [torch.stack([kv[b][h][1] for h in range(2)]) for b in range(2)]
    packed = kvq.QuantKVCache(cfg)
    stepped = kvq.QuantKVCache(cfg)
    for b in range(2):
        kvq.kvq_pack(packed, k_all[b][None].cuda(), v_all[b][None].cuda(), batch_begin=b)
        kvq.kvq_pack(stepped, k_all[b][None, :, :L0].cuda(), v_all[b][None, :, :L0].cuda(),
                     batch_begin=b)
    q = torch.zeros(2, 8, 128, dtype=torch.float16, device="cuda")
    for t in range(L0, L):  # flushes at 160, 192, ..., 288
        kn = torch.stack([k_all[b][:, t] for b in range(2)]).cuda()
        vn = torch.stack([v_all[b][:, t] for b in range(2)]).cuda()
        kvq.kvq_decode_step(stepped, kn, vn, q)
    torch.cuda.synchronize()
    assert packed.seq_lens().cpu().tolist() == [L, L]
    assert stepped.seq_lens().cpu().tolist() == [L, L]
    for b in range(2):
        for h in range(2):
            want = quant.quantize_head(k_all[b][h].numpy(), v_all[b][h].numpy(), bits, bits,
                                       cfg.residual)
            assert np.all(want["k_scale"].astype(np.float64) == 0.1875)
            assert np.all(want["v_scale"].astype(np.float64) == 0.1875)
            _util.assert_head_equal(_util.head_arrays(packed, b, h, L), want)
            _util.assert_head_equal(_util.head_arrays(stepped, b, h, L), want)
