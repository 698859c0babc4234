"""kvq_decode_attn (CUDA, through the C ABI) against the float64 oracle:
max |o_gpu - o_oracle| <= 2e-3 * rms(o_oracle) for every (sequence, head)."""

import numpy as np
import pytest
import torch

import _util
from oracle import attention
from paper_2607_16248_gb300 import kvq, synth

pytestmark = pytest.mark.gpu


def _run(cfg, lengths, seed, n_splits=0, scale=0.0):
    cache, kv = _util.make_cache(cfg, lengths, seed)
    q = synth.queries(seed + 99, cfg.batch, cfg.n_q_heads)
    out = kvq.kvq_decode_attn(cache, q.cuda(), softmax_scale=scale, n_splits=n_splits)
    torch.cuda.synchronize()
    got = out.float().cpu().numpy()
    errs = []
    for b, L in enumerate(lengths):
        k, v = kv[b]
        heads = _util.oracle_heads(cfg, k, v)
        ref = attention.decode_attention(q[b].numpy(), heads,
                                         scale=None if scale == 0 else scale)
        errs.append(_util.attn_rel_err(got[b], ref))
    return np.array(errs), got


@pytest.mark.parametrize("bk,bv", [(1, 1), (2, 2), (4, 4), (8, 8), (2, 1), (1, 2)])
def test_lengths_around_block_and_window_edges(kvq_lib, bk, bv):
    lengths = [1, 31, 32, 33, 127, 128, 159, 160, 161, 191, 1000, 4096]
    cfg = kvq.CacheConfig(batch=len(lengths), n_q_heads=8, n_kv_heads=2, bits_k=bk, bits_v=bv,
                          max_len=4096)
    errs, _ = _run(cfg, lengths, seed=bk * 10 + bv)
    assert errs.max() <= _util.ATTN_TOL, errs.max(axis=1)


@pytest.mark.parametrize("gq", [1, 4, 5, 8])
def test_gqa_group_sizes(kvq_lib, gq):
    cfg = kvq.CacheConfig(batch=2, n_q_heads=2 * gq, n_kv_heads=2, bits_k=1, bits_v=1,
                          max_len=2048)
    errs, _ = _run(cfg, [2000, 777], seed=40 + gq)
    assert errs.max() <= _util.ATTN_TOL


@pytest.mark.parametrize("gq", [1, 2, 3, 5, 6, 7])
@pytest.mark.parametrize("n_splits", [3, 5, 19])
def test_group_widths_with_odd_split_counts(kvq_lib, gq, n_splits):
    # narrow (1..3) and wide (5..7) query groups with an odd number of
    # splits: the final merge stages gq * S partial rows
    cfg = kvq.CacheConfig(batch=2, n_q_heads=2 * gq, n_kv_heads=2, bits_k=2, bits_v=1,
                          max_len=4096)
    errs, _ = _run(cfg, [4000, 1111], seed=60 + gq, n_splits=n_splits)
    assert errs.max() <= _util.ATTN_TOL


@pytest.mark.parametrize("n_splits", [1, 2, 7, 64, 200])
def test_split_count_invariance(kvq_lib, n_splits):
    cfg = kvq.CacheConfig(batch=2, n_q_heads=8, n_kv_heads=2, bits_k=2, bits_v=2, max_len=4096)
    errs, got = _run(cfg, [4096, 1500], seed=50, n_splits=n_splits)
    assert errs.max() <= _util.ATTN_TOL
    _, one = _run(cfg, [4096, 1500], seed=50, n_splits=1)
    assert np.abs(got - one).max() <= 2e-3 * np.sqrt((one ** 2).mean())


def test_tiny_workload_shape(kvq_lib):
    """Tiny single-layer decode step: 32/8 heads, context 4096, K2V2."""
    cfg = kvq.CacheConfig(batch=1, n_q_heads=32, n_kv_heads=8, bits_k=2, bits_v=2,
                          max_len=4096)
    errs, _ = _run(cfg, [4096], seed=1)
    assert errs.max() <= _util.ATTN_TOL


def test_custom_softmax_scale(kvq_lib):
    cfg = kvq.CacheConfig(batch=1, n_q_heads=4, n_kv_heads=1, bits_k=4, bits_v=4, max_len=1024)
    errs, _ = _run(cfg, [900], seed=60, scale=0.02)
    assert errs.max() <= _util.ATTN_TOL


def test_empty_sequence_gives_zero(kvq_lib):
    cfg = kvq.CacheConfig(batch=2, n_q_heads=4, n_kv_heads=1, bits_k=2, bits_v=2, max_len=512)
    errs, got = _run(cfg, [0, 300], seed=61)
    assert np.all(got[0] == 0)
    assert errs[1].max() <= _util.ATTN_TOL


def test_decode_steps_pack_then_attend(kvq_lib):
    """The decode loop: append the step's token, then attend over all of it."""
    cfg = kvq.CacheConfig(batch=2, n_q_heads=8, n_kv_heads=2, bits_k=1, bits_v=1, max_len=1024)
    k, v = synth.kv_heads(70, 2, 400)
    cache = kvq.QuantKVCache(cfg)
    start = [150, 10]
    for b in range(2):
        kvq.kvq_pack(cache, k[:, :start[b]][None].contiguous().cuda(),
                     v[:, :start[b]][None].contiguous().cuda(), batch_begin=b)
    ws = kvq.attn_workspace(cfg)
    for step in range(45):
        L = [s + step + 1 for s in start]
        kn = torch.stack([k[:, L[b] - 1] for b in range(2)])[:, :, None].contiguous().cuda()
        vn = torch.stack([v[:, L[b] - 1] for b in range(2)])[:, :, None].contiguous().cuda()
        kvq.kvq_pack(cache, kn, vn)
        q = synth.queries(1000 + step, 2, 8)
        out = kvq.kvq_decode_attn(cache, q.cuda(), workspace=ws).float().cpu().numpy()
        if step % 4 == 0 or step > 40:
            for b in range(2):
                heads = _util.oracle_heads(cfg, k[:, :L[b]], v[:, :L[b]])
                ref = attention.decode_attention(q[b].numpy(), heads)
                assert _util.attn_rel_err(out[b], ref).max() <= _util.ATTN_TOL
