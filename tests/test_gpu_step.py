"""kvq_decode_step (append one token and attend, one kernel) through the C ABI:
over a run of decode steps its caches stay bit-identical to kvq_pack(n_new = 1)
followed by kvq_decode_attn, its outputs match that pair and the float64
oracle, and a sequence at max_len is left unchanged with the overflow flag."""

import numpy as np
import pytest
import torch

import _util


def pair_tol(cfg):
    """How far the fused step may sit from pack-then-attend on the same
    split count: fp32 summation order only (1e-5 x rms) for wider value
    codes; for 1-bit values the fp16 softmax weights are rounded relative to
    each warp's running maximum, which the flushed block (folded from shared
    memory at the end of its warp's range) can change, so 2^-12-relative
    rounding differences of single weights show (3e-4 x rms)."""
    return 3e-4 if cfg.bits_v == 1 else 1e-5
from oracle import attention
from paper_2607_16248_gb300 import kvq, synth

pytestmark = pytest.mark.gpu


def _cache_state(cache, lengths):
    cfg = cache.cfg
    return [[_util.head_arrays(cache, b, h, L) for h in range(cfg.n_kv_heads)]
            for b, L in enumerate(lengths)]


def _steps(cfg, lengths, n_steps, seed, check_oracle_every=0, n_splits=0):
    a, kv = _util.make_cache(cfg, lengths, seed)
    b_, _ = _util.make_cache(cfg, lengths, seed)
    g = synth.generator(seed + 5)
    hist = [(k.clone(), v.clone()) for k, v in kv]  # host fp16 [Hkv, L, 128]
    lens = list(lengths)
    worst_pair, worst_oracle = 0.0, 0.0
    for step in range(n_steps):
        kn = torch.randn(cfg.batch, cfg.n_kv_heads, 128, generator=g).half()
        vn = torch.randn(cfg.batch, cfg.n_kv_heads, 128, generator=g).half()
        q = torch.randn(cfg.batch, cfg.n_q_heads, 128, generator=g).half()
        out_a = kvq.kvq_decode_step(a, kn.cuda(), vn.cuda(), q.cuda(), n_splits=n_splits,
                                    out_dtype=torch.float32)
        kvq.kvq_pack(b_, kn[:, :, None].cuda(), vn[:, :, None].cuda())
        out_b = kvq.kvq_decode_attn(b_, q.cuda(), n_splits=n_splits, out_dtype=torch.float32)
        torch.cuda.synchronize()
        oa, ob = out_a.cpu().numpy(), out_b.cpu().numpy()
        for s in range(cfg.batch):
            hist[s] = (torch.cat([hist[s][0], kn[s][:, None]], 1),
                       torch.cat([hist[s][1], vn[s][:, None]], 1))
            lens[s] += 1
            rms = np.sqrt((ob[s] ** 2).mean(axis=-1))
            worst_pair = max(worst_pair, float((np.abs(oa[s] - ob[s]).max(axis=-1) / rms).max()))
            if check_oracle_every and step % check_oracle_every == check_oracle_every - 1:
                heads = _util.oracle_heads(cfg, hist[s][0], hist[s][1])
                ref = attention.decode_attention(q[s].numpy(), heads)
                worst_oracle = max(worst_oracle, float(_util.attn_rel_err(oa[s], ref).max()))
    assert a.seq_lens().cpu().tolist() == lens
    assert b_.seq_lens().cpu().tolist() == lens
    sa, sb = _cache_state(a, lens), _cache_state(b_, lens)
    for s in range(cfg.batch):
        for h in range(cfg.n_kv_heads):
            _util.assert_head_equal(sa[s][h], sb[s][h])
    return worst_pair, worst_oracle


@pytest.mark.parametrize("bk,bv", [(1, 1), (2, 2), (4, 4), (8, 8), (1, 2), (4, 1)])
def test_steps_equal_pack_then_attention(kvq_lib, bk, bv):
    lengths = [1, 127, 159, 160, 190, 700]
    cfg = kvq.CacheConfig(batch=len(lengths), n_q_heads=8, n_kv_heads=2, bits_k=bk, bits_v=bv,
                          max_len=1024)
    pair, oracle = _steps(cfg, lengths, 36, seed=bk * 7 + bv, check_oracle_every=12)
    assert pair <= pair_tol(cfg), pair
    assert oracle <= _util.ATTN_TOL, oracle


@pytest.mark.parametrize("gq", [5, 8])
def test_wide_query_groups(kvq_lib, gq):
    # groups of 5..8 heads take the wide MMA layout; the lengths cross the
    # flush at 160
    cfg = kvq.CacheConfig(batch=3, n_q_heads=2 * gq, n_kv_heads=2, bits_k=1, bits_v=2,
                          max_len=1024)
    pair, oracle = _steps(cfg, [158, 400, 159], 5, seed=21 + gq, check_oracle_every=5)
    assert pair <= pair_tol(cfg), pair
    assert oracle <= _util.ATTN_TOL, oracle


@pytest.mark.parametrize("residual,n_splits,bk,bv", [(32, 1, 1, 2), (96, 2, 2, 1), (160, 2, 1, 1),
                                                    (512, 4, 1, 1), (512, 3, 4, 2)])
def test_flush_workers_for_window_sizes(kvq_lib, residual, n_splits, bk, bv):
    # The group leaving the window is quantized by the window warps of the
    # CTA that folds it in: 1, 3, 5 and 12 of them here, and none for a
    # 512-token window over 4 splits, where the folding warp does it alone.
    R = residual
    lengths = [R - 1, R + 30, R + 63, 3 * R + 5]
    cfg = kvq.CacheConfig(batch=len(lengths), n_q_heads=8, n_kv_heads=2, bits_k=bk, bits_v=bv,
                          max_len=4 * R + 128, residual=R)
    pair, oracle = _steps(cfg, lengths, 34, seed=R + n_splits, check_oracle_every=17,
                          n_splits=n_splits)
    assert pair <= pair_tol(cfg), pair
    assert oracle <= _util.ATTN_TOL, oracle


def test_split_counts_and_llama_shape(kvq_lib):
    cfg = kvq.CacheConfig(batch=1, n_q_heads=32, n_kv_heads=8, bits_k=1, bits_v=1, max_len=8192)
    for ns in (1, 7, 19):
        a, kv = _util.make_cache(cfg, [4095], 33)
        g = synth.generator(34)
        kn = torch.randn(1, 8, 128, generator=g).half()
        vn = torch.randn(1, 8, 128, generator=g).half()
        q = torch.randn(1, 32, 128, generator=g).half()
        out = kvq.kvq_decode_step(a, kn.cuda(), vn.cuda(), q.cuda(), n_splits=ns).cpu().numpy()
        k, v = kv[0]
        heads = _util.oracle_heads(cfg, torch.cat([k, kn[0][:, None]], 1),
                                   torch.cat([v, vn[0][:, None]], 1))
        ref = attention.decode_attention(q[0].numpy(), heads)
        assert _util.attn_rel_err(out[0], ref).max() <= _util.ATTN_TOL
        assert a.seq_lens().cpu().tolist() == [4096]


def test_full_sequence_is_not_appended(kvq_lib):
    cfg = kvq.CacheConfig(batch=2, n_q_heads=8, n_kv_heads=2, bits_k=2, bits_v=2, max_len=256)
    a, kv = _util.make_cache(cfg, [256, 100], 8)
    g = synth.generator(9)
    kn = torch.randn(2, 2, 128, generator=g).half()
    vn = torch.randn(2, 2, 128, generator=g).half()
    q = torch.randn(2, 8, 128, generator=g).half()
    out = kvq.kvq_decode_step(a, kn.cuda(), vn.cuda(), q.cuda()).cpu().numpy()
    assert a.seq_lens().cpu().tolist() == [256, 101]
    assert a.flags() & kvq.FLAG_OVERFLOW
    k, v = kv[0]
    ref = attention.decode_attention(q[0].numpy(), _util.oracle_heads(cfg, k, v))
    assert _util.attn_rel_err(out[0], ref).max() <= _util.ATTN_TOL
