"""Paged KV blocks (a block table over a shared pool of page sets), through
the C ABI, against the contiguous layout and the float64 oracle.

The page order changes nothing in the arithmetic: the same logical blocks are
quantized by the same quantizer (Sec. 3.1) and attended in the same order, so
a paged cache whose blocks land in a shuffled set of pages holds bit-identical
pages and gives bit-identical fp32 attention outputs to the contiguous cache,
and both match the oracle.  Decode steps flush groups into the page sets the
caller assigns; blocks mapped outside the pool are never touched and raise
KVQ_FLAG_BAD_PAGE; a sequence at max_len is not appended (KVQ_FLAG_OVERFLOW).
"""

import numpy as np
import pytest
import torch

import _util
from oracle import attention
from paper_2607_16248_gb300 import kvq, synth

pytestmark = pytest.mark.gpu


class Pool:
    """A caller-side allocator: free page sets handed out in a seeded
    shuffled order."""

    def __init__(self, n_pages, seed):
        g = np.random.default_rng(seed)
        self.free = list(g.permutation(n_pages))

    def take(self, n):
        out, self.free = self.free[:n], self.free[n:]
        assert len(out) == n, "pool exhausted"
        return [int(x) for x in out]


def _paged_twin(cfg, lengths, seed, spare=8):
    """A contiguous cache and a paged one prefilled with the same tokens; the
    paged cache's pool holds the blocks up to max_len of every sequence plus
    `spare` sets, in shuffled order."""
    need = sum(cfg.max_blocks for _ in lengths)
    n_pages = need + spare
    pool = Pool(n_pages, seed)
    a, kv = _util.make_cache(cfg, lengths, seed)
    p = kvq.QuantKVCache(cfg, n_pages=n_pages)
    for b, L in enumerate(lengths):
        blocks = list(kvq.blocks_written(0, L, cfg.residual))
        if blocks:
            p.map_blocks(b, blocks, pool.take(len(blocks)))
        if L:
            k, v = kv[b]
            kvq.kvq_pack(p, k[None].cuda(), v[None].cuda(), batch_begin=b)
    torch.cuda.synchronize()
    return a, p, kv, pool


def _same_state(a, p, lengths):
    cfg = a.cfg
    for b, L in enumerate(lengths):
        for h in range(cfg.n_kv_heads):
            _util.assert_head_equal(_util.head_arrays(p, b, h, L), _util.head_arrays(a, b, h, L))


@pytest.mark.parametrize("bk,bv,gq", [(1, 1, 4), (1, 1, 5), (2, 2, 4), (4, 8, 2), (2, 1, 8)])
def test_prefill_and_attention_match_contiguous(kvq_lib, bk, bv, gq):
    lengths = [4096, 1500, 159, 700, 33, 0, 2049]
    cfg = kvq.CacheConfig(batch=len(lengths), n_q_heads=2 * gq, n_kv_heads=2, bits_k=bk,
                          bits_v=bv, max_len=4096)
    a, p, kv, _ = _paged_twin(cfg, lengths, seed=400 + 10 * bk + bv + gq)
    assert p.flags() == 0
    _same_state(a, p, lengths)
    q = synth.queries(401, cfg.batch, cfg.n_q_heads).cuda()
    for ns in (1, 3, 11, 0):  # split plan counts, then the flat plan
        oa = kvq.kvq_decode_attn(a, q, n_splits=ns, out_dtype=torch.float32)
        op = kvq.kvq_decode_attn(p, q, n_splits=ns, out_dtype=torch.float32)
        torch.cuda.synchronize()
        assert torch.equal(oa.view(torch.int32), op.view(torch.int32)), f"splits {ns}"
    got = kvq.kvq_decode_attn(p, q).cpu().numpy()
    for b, L in enumerate(lengths):
        if L == 0:
            assert np.all(got[b] == 0)
            continue
        ref = attention.decode_attention(q[b].cpu().numpy(), _util.oracle_heads(cfg, *kv[b]))
        assert _util.attn_rel_err(got[b], ref).max() <= _util.ATTN_TOL
    assert p.flags() == 0


@pytest.mark.parametrize("bk,bv,gq,ns", [(1, 1, 4, 4), (1, 1, 5, 4), (2, 4, 4, 4), (1, 1, 5, 0),
                                         (2, 4, 4, 0)])
def test_decode_steps_flush_into_assigned_pages(kvq_lib, bk, bv, gq, ns):
    # lengths that cross the flush point (L + 1 - 128 a multiple of 32)
    # within a few steps; pages for the flushed groups are assigned by the
    # caller just before the step that writes them
    lengths = [158, 159, 190, 1000, 130]
    cfg = kvq.CacheConfig(batch=len(lengths), n_q_heads=2 * gq, n_kv_heads=2, bits_k=bk,
                          bits_v=bv, max_len=2048)
    a, p, kv, pool = _paged_twin(cfg, lengths, seed=410 + bk + gq)
    hist = [(k.clone(), v.clone()) for k, v in kv]
    lens = list(lengths)
    g = synth.generator(411)
    ws_a = kvq.attn_workspace(cfg, ns)  # ns = 0: the flat plan
    ws_p = kvq.attn_workspace(cfg, ns)
    flushed = 0
    for step in range(40):
        for b, L in enumerate(lens):
            blocks = list(kvq.blocks_written(L, 1, cfg.residual))
            if blocks:
                p.map_blocks(b, blocks, pool.take(len(blocks)))
                flushed += 1
        kn = torch.randn(cfg.batch, 2, 128, generator=g).half()
        vn = torch.randn(cfg.batch, 2, 128, generator=g).half()
        q = torch.randn(cfg.batch, cfg.n_q_heads, 128, generator=g).half()
        oa = kvq.kvq_decode_step(a, kn.cuda(), vn.cuda(), q.cuda(), n_splits=ns, workspace=ws_a,
                                 out_dtype=torch.float32)
        op = kvq.kvq_decode_step(p, kn.cuda(), vn.cuda(), q.cuda(), n_splits=ns, workspace=ws_p,
                                 out_dtype=torch.float32)
        torch.cuda.synchronize()
        assert torch.equal(oa.view(torch.int32), op.view(torch.int32)), f"step {step}"
        for b in range(cfg.batch):
            hist[b] = (torch.cat([hist[b][0], kn[b][:, None]], 1),
                       torch.cat([hist[b][1], vn[b][:, None]], 1))
            lens[b] += 1
        if step % 13 == 12:
            out = op.cpu().numpy()
            for b in range(cfg.batch):
                ref = attention.decode_attention(q[b].numpy(),
                                                 _util.oracle_heads(cfg, *hist[b]))
                assert _util.attn_rel_err(out[b], ref).max() <= _util.ATTN_TOL
    assert flushed >= 5
    assert p.seq_lens().cpu().tolist() == lens
    assert p.flags() == 0
    _same_state(a, p, lens)


def test_pack_steps_into_assigned_pages(kvq_lib):
    # kvq_pack with n_new = 1 and with n_new = 45 on a paged cache
    cfg = kvq.CacheConfig(batch=2, n_q_heads=8, n_kv_heads=2, bits_k=1, bits_v=2, max_len=1024)
    lengths = [100, 157]
    a, p, kv, pool = _paged_twin(cfg, lengths, seed=420)
    g = synth.generator(421)
    lens = list(lengths)
    for n_new in (1, 1, 45, 1, 33, 1):
        for b, L in enumerate(lens):
            blocks = list(kvq.blocks_written(L, n_new, cfg.residual))
            if blocks:
                p.map_blocks(b, blocks, pool.take(len(blocks)))
        for b in range(2):
            kn = torch.randn(1, 2, n_new, 128, generator=g).half().cuda()
            vn = torch.randn(1, 2, n_new, 128, generator=g).half().cuda()
            kvq.kvq_pack(a, kn, vn, batch_begin=b)
            kvq.kvq_pack(p, kn, vn, batch_begin=b)
            lens[b] += n_new
    torch.cuda.synchronize()
    assert p.flags() == 0
    _same_state(a, p, lens)


def test_unmapped_blocks_are_skipped_and_flagged(kvq_lib):
    cfg = kvq.CacheConfig(batch=3, n_q_heads=8, n_kv_heads=2, bits_k=2, bits_v=2, max_len=1024)
    lengths = [800, 600, 300]
    a, p, kv, pool = _paged_twin(cfg, lengths, seed=430)
    q = synth.queries(431, cfg.batch, cfg.n_q_heads).cuda()
    # attention: sequence 1's block 3 mapped past the pool, then unmapped
    for bad in (p.n_pages + 7, -1):
        keep = int(p.block_table[1, 3].item())
        p.block_table[1, 3] = bad
        p.seq_region()[cfg.batch] = 0
        out = kvq.kvq_decode_attn(p, q, n_splits=5, out_dtype=torch.float32)
        torch.cuda.synchronize()
        assert p.flags() & kvq.FLAG_BAD_PAGE
        ref = kvq.kvq_decode_attn(a, q, n_splits=5, out_dtype=torch.float32)
        torch.cuda.synchronize()
        for b in (0, 2):  # the other sequences are untouched
            assert torch.equal(out[b].view(torch.int32), ref[b].view(torch.int32))
        p.block_table[1, 3] = keep
    # a decode step whose flush block is unmapped: the step's output is still
    # right (the group is attended from shared memory), the write is skipped
    p.seq_region()[cfg.batch] = 0
    L = lengths[2]
    while (L + 1 - cfg.residual) % 32:
        L += 1
    g = synth.generator(432)
    for step in range(L - lengths[2] + 1):
        for b, Lb in enumerate([lengths[0] + step, lengths[1] + step]):
            blocks = list(kvq.blocks_written(Lb, 1, cfg.residual))
            if blocks:
                p.map_blocks(b, blocks, pool.take(len(blocks)))
        kn = torch.randn(3, 2, 128, generator=g).half().cuda()
        vn = torch.randn(3, 2, 128, generator=g).half().cuda()
        qq = torch.randn(3, 8, 128, generator=g).half().cuda()
        oa = kvq.kvq_decode_step(a, kn, vn, qq, n_splits=2, out_dtype=torch.float32)
        op = kvq.kvq_decode_step(p, kn, vn, qq, n_splits=2, out_dtype=torch.float32)
        torch.cuda.synchronize()
        assert torch.equal(oa.view(torch.int32), op.view(torch.int32))
    assert p.flags() & kvq.FLAG_BAD_PAGE  # sequence 2's last step had no page
    assert p.seq_lens().cpu().tolist() == a.seq_lens().cpu().tolist()


def test_overflow_on_a_paged_cache(kvq_lib):
    cfg = kvq.CacheConfig(batch=2, n_q_heads=8, n_kv_heads=2, bits_k=1, bits_v=1, max_len=256)
    a, p, kv, pool = _paged_twin(cfg, [256, 100], seed=440)
    g = synth.generator(441)
    kn = torch.randn(2, 2, 128, generator=g).half().cuda()
    q = torch.randn(2, 8, 128, generator=g).half().cuda()
    out = kvq.kvq_decode_step(p, kn, kn, q)
    torch.cuda.synchronize()
    assert p.seq_lens().cpu().tolist() == [256, 101]
    assert p.flags() & kvq.FLAG_OVERFLOW and not p.flags() & kvq.FLAG_BAD_PAGE
    ref = attention.decode_attention(q[0].cpu().numpy(), _util.oracle_heads(cfg, *kv[0]))
    assert _util.attn_rel_err(out[0].cpu().numpy(), ref).max() <= _util.ATTN_TOL
