"""The C-ABI library builds, loads and exports every symbol include/kvq.h
declares; host-side validation returns the documented status codes.

No call here launches a kernel: every compute entry point is given an
argument that the host-side checks reject first.
"""

import ctypes
import re
from pathlib import Path

import pytest

from paper_2607_16248_gb300 import build, kvq

HEADER = Path(__file__).resolve().parents[1] / "include" / "kvq.h"


@pytest.fixture(scope="module")
def L():
    build.build()
    return kvq.lib()


def _declared():
    text = re.sub(r"/\*.*?\*/", "", HEADER.read_text(), flags=re.S)
    return sorted(set(re.findall(r"\b((?:kvq|dgap)_[a-z_0-9]+)\s*\(", text)))


def test_header_and_binding_agree():
    assert _declared() == sorted(kvq.EXPORTS)


def test_every_declared_symbol_is_exported(L):
    for name in _declared():
        assert hasattr(L, name), name


def _cfg(**kw):
    base = dict(batch=2, n_q_heads=32, n_kv_heads=8, bits_k=2, bits_v=2, max_len=4096)
    base.update(kw)
    return kvq.CacheConfig(**base)


def test_validate_config(L):
    _cfg().validate()
    bad = [dict(bits_k=3), dict(bits_v=0), dict(head_dim=64), dict(group=16), dict(residual=100),
           dict(max_len=100), dict(n_q_heads=30), dict(n_q_heads=72), dict(batch=0),
           dict(residual=0)]
    codes = {3: [dict(bits_k=3), dict(bits_v=0), dict(head_dim=64), dict(group=16),
                 dict(residual=100), dict(n_q_heads=72), dict(residual=0)]}
    for kw in bad:
        with pytest.raises(kvq.KvqError) as e:
            _cfg(**kw).validate()
        want = 3 if kw in codes[3] else 2
        assert e.value.status == want, (kw, e.value)


def test_layout_sizes(L):
    cfg = _cfg(bits_k=1, bits_v=4)
    total, offs = cfg.layout()
    pages = 2 * 8 * (4096 // 32) * (512 * 5 + 1024)
    assert offs[0] == 0 and offs[1] >= pages and offs[1] % 256 == 0
    resid = 2 * 8 * 160 * 128 * 2
    assert offs[2] - offs[1] >= resid and offs[3] - offs[2] >= resid
    assert total >= offs[3] + 4 * (2 * 2 + 2)
    c = cfg.c()
    assert L.kvq_page_bytes(ctypes.byref(c)) == 512 * 5 + 1024


def test_paged_layout_and_bind(L):
    cfg = _cfg(bits_k=1, bits_v=4)
    c = cfg.c()
    total, offs = cfg.layout()
    tot = ctypes.c_size_t()
    po = (ctypes.c_size_t * 4)()
    assert L.kvq_paged_cache_layout(ctypes.byref(c), ctypes.byref(tot), ctypes.byref(po)) == 0
    # the rings and lengths only: the page region of the contiguous layout is gone
    assert po[0] == 0 and po[1] == 0
    assert tot.value == total - offs[1]
    assert L.kvq_page_pool_bytes(ctypes.byref(c), 10) == 10 * 8 * (512 * 5 + 1024)
    assert L.kvq_page_pool_bytes(ctypes.byref(c), 0) == 0
    cache = kvq._Cache()
    base, pool, tbl = ctypes.c_void_p(0x10000), ctypes.c_void_p(0x20000), ctypes.c_void_p(0x30000)
    assert L.kvq_paged_cache_bind(ctypes.byref(c), base, pool, 10, tbl, ctypes.byref(cache)) == 0
    assert cache.pages == 0x20000 and cache.block_table == 0x30000 and cache.n_pages == 10
    assert cache.k_resid == 0x10000 + po[1] and cache.seq_len == 0x10000 + po[3]
    nul = ctypes.c_void_p(None)
    assert L.kvq_paged_cache_bind(ctypes.byref(c), base, pool, 10, nul, ctypes.byref(cache)) == 1
    assert L.kvq_paged_cache_bind(ctypes.byref(c), base, pool, 0, tbl, ctypes.byref(cache)) == 1
    assert L.kvq_paged_cache_bind(ctypes.byref(c), base, ctypes.c_void_p(0x20008), 10, tbl,
                                  ctypes.byref(cache)) == 5
    assert L.kvq_paged_cache_bind(ctypes.byref(c), base, pool, 10, ctypes.c_void_p(0x30002),
                                  ctypes.byref(cache)) == 5
    # the contiguous bind clears the paged fields
    assert L.kvq_cache_bind(ctypes.byref(c), base, ctypes.byref(cache)) == 0
    assert not cache.block_table and cache.n_pages == 0
    # a paged cache with n_pages < 1 is rejected before any launch
    bad = kvq._Cache(pool, base, base, base, tbl, 0)
    fake = ctypes.c_void_p(0x1000)
    assert L.kvq_pack(ctypes.byref(c), ctypes.byref(bad), fake, fake, 1, 0, 2, nul) == 1


def test_paged_helpers():
    # 4096 tokens: Lq = 32 * floor(3968 / 32) = 3968, blocks 0 .. 123
    assert list(kvq.blocks_written(0, 4096)) == list(range(0, 124))
    assert list(kvq.blocks_written(159, 1)) == [0]      # 160 tokens: the first group leaves
    assert list(kvq.blocks_written(160, 1)) == []
    assert list(kvq.blocks_written(190, 1)) == []
    assert list(kvq.blocks_written(191, 1)) == [1]      # 192 - 128 = 64: the second group
    assert list(kvq.blocks_written(100, 45)) == []
    assert list(kvq.blocks_written(100, 92)) == [0, 1]   # 192 tokens: Lq = 64


def test_workspace_sizes(L):
    cfg = _cfg()
    c = cfg.c()
    s = L.kvq_attn_default_splits(ctypes.byref(c))
    assert 1 <= s <= 1024
    n = L.kvq_attn_workspace_bytes(ctypes.byref(c), 7)
    # split plan, 7 CTAs per (sequence, kv-head): a partial (m, l and a
    # 128-channel row) per (sequence, query head, CTA) and a ticket per pair
    assert n >= 2 * 32 * 7 * (128 + 2) * 4 + 2 * 8 * 4
    # flat plan (0): a partial per CTA and two per pair, gq heads each, a
    # ticket per pair and one counter
    pairs, gq = 2 * 8, 32 // 8
    flat = L.kvq_attn_workspace_bytes(ctypes.byref(c), 0)
    assert flat >= (1 + 2 * pairs) * gq * (128 + 2) * 4 + (pairs + 1) * 4
    assert L.kvq_attn_workspace_bytes(ctypes.byref(c), 5000) == 0
    p = kvq._DgapParams(32, 64, 0.6, *([None] * 8))
    assert L.dgap_workspace_bytes(4, 128256, ctypes.byref(p)) > 4 * 32 * 33 * 8
    p.K = 1
    assert L.dgap_workspace_bytes(4, 128256, ctypes.byref(p)) == 0
    p.K = 65
    assert L.dgap_workspace_bytes(4, 128256, ctypes.byref(p)) == 0
    p.K = 32
    assert L.dgap_workspace_bytes(4, 32, ctypes.byref(p)) == 0  # K must be < vocab


def test_splits_for_lengths(L):
    def n(cfg, lengths):
        c = cfg.c()
        return L.kvq_attn_splits_for_lengths(ctypes.byref(c), (ctypes.c_int32 * cfg.batch)(*lengths))

    def default(cfg):
        return L.kvq_attn_default_splits(ctypes.byref(cfg.c()))

    # batch 1 (8 pairs): the split plan, one wave of 19 CTAs per pair
    one = kvq.CacheConfig(batch=1, n_q_heads=32, n_kv_heads=8, bits_k=1, bits_v=1, max_len=32800)
    assert default(one) * 8 >= 0.9 * 152 and n(one, [32768]) == default(one)
    # 64 pairs (Qwen-14B shape, batch 8): one wave of 2 splits leaves SMs idle,
    # so the flat plan (0)
    qwen = kvq.CacheConfig(batch=8, n_q_heads=40, n_kv_heads=8, bits_k=1, bits_v=1, max_len=65664)
    assert default(qwen) == 2 and n(qwen, [65536] * 8) == 0
    big = kvq.CacheConfig(batch=16, n_q_heads=32, n_kv_heads=8, bits_k=2, bits_v=2, max_len=32800)
    assert n(big, [20000] * 16) == 0
    assert n(big, [8192 + 1500 * i for i in range(16)]) == 0
    assert n(big, [20000] * 15 + [40000]) == -1  # beyond max_len
    assert n(big, [-1] + [20000] * 15) == -1


def test_compute_entry_points_reject_bad_arguments(L):
    cfg = _cfg()
    c = cfg.c()
    fake = ctypes.c_void_p(0x1000)  # never dereferenced: validation fails first
    cache = kvq._Cache(fake, fake, fake, fake)
    nul = ctypes.c_void_p(None)
    # kvq_pack: NULL inputs, bad n_new, bad batch range, misaligned input
    assert L.kvq_pack(ctypes.byref(c), ctypes.byref(cache), nul, fake, 1, 0, 2, nul) == 1
    assert L.kvq_pack(ctypes.byref(c), ctypes.byref(cache), fake, fake, 0, 0, 2, nul) == 1
    assert L.kvq_pack(ctypes.byref(c), ctypes.byref(cache), fake, fake, 1, 1, 2, nul) == 2
    assert L.kvq_pack(ctypes.byref(c), ctypes.byref(cache), fake, fake, 5000, 0, 2, nul) == 4
    assert L.kvq_pack(ctypes.byref(c), ctypes.byref(cache), ctypes.c_void_p(0x1002), fake, 1, 0,
                      2, nul) == 5
    bad_cache = kvq._Cache(fake, nul, fake, fake)
    assert L.kvq_pack(ctypes.byref(c), ctypes.byref(bad_cache), fake, fake, 1, 0, 2, nul) == 1
    c3 = _cfg(bits_k=3).c()
    assert L.kvq_pack(ctypes.byref(c3), ctypes.byref(cache), fake, fake, 1, 0, 2, nul) == 3
    # kvq_decode_attn: workspace too small, bad splits, misaligned q, bad scale
    ws_need = L.kvq_attn_workspace_bytes(ctypes.byref(c), 4)
    assert L.kvq_decode_attn(ctypes.byref(c), ctypes.byref(cache), fake, fake, 0.0, 4, fake,
                             ws_need - 1, nul) == 4
    assert L.kvq_decode_attn(ctypes.byref(c), ctypes.byref(cache), fake, fake, 0.0, -1, fake,
                             ws_need, nul) == 1
    assert L.kvq_decode_attn(ctypes.byref(c), ctypes.byref(cache), ctypes.c_void_p(0x1008), fake,
                             0.0, 4, fake, ws_need, nul) == 5
    assert L.kvq_decode_attn(ctypes.byref(c), ctypes.byref(cache), fake, fake, -1.0, 4, fake,
                             ws_need, nul) == 1
    assert L.kvq_decode_attn(ctypes.byref(c), ctypes.byref(cache), fake, fake, 0.0, 4, nul,
                             ws_need, nul) == 1
    assert "workspace" in kvq.last_error()
    # dgap_restore: bad K, NULL weight, small workspace, misaligned logits
    p = kvq._DgapParams(32, 64, 0.6, *([fake] * 8))
    args = [fake, 1, 1000, fake, fake, fake, fake, nul, nul, fake]
    need = L.dgap_workspace_bytes(1, 1000, ctypes.byref(p))
    assert L.dgap_restore(ctypes.byref(p), *args, need - 1, nul) == 4
    p.det_w2 = None
    assert L.dgap_restore(ctypes.byref(p), *args, need, nul) == 1
    p.det_w2 = fake
    p.K = 1000
    assert L.dgap_restore(ctypes.byref(p), *args, need, nul) == 3
    p.K = 32
    args[0] = ctypes.c_void_p(0x1004)
    assert L.dgap_restore(ctypes.byref(p), *args, need, nul) == 5
    p.tau = float("nan")
    assert L.dgap_restore(ctypes.byref(p), *args, need, nul) == 1


def test_binding_rejects_cpu_tensors(L):
    import torch
    with pytest.raises(TypeError):
        kvq._dev(torch.zeros(4), torch.float32, "x")
