"""The fp16 output of kvq_decode_attn / kvq_decode_step (the boundary's out
is fp16, the fp32 accumulation rounded once to nearest even).

Two checks per case, through the C ABI: the fp16 output is within the
attention tolerance of the float64 oracle (Sec. 1, softmax(QK^T/sqrt(d_k))V
over the dequantized cache), and it equals, bit for bit, the fp32 output of
kvq_decode_attn_f32 / kvq_decode_step_f32 on the same inputs rounded to fp16.
Split counts 1 (the CTA writes the output directly) and > 1 (the last CTA's
merge writes it) are both covered, for narrow (4-head) and wide (5-head)
query groups."""

import numpy as np
import pytest
import torch

import _util
from oracle import attention
from paper_2607_16248_gb300 import kvq, synth

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("gq,bk,bv", [(4, 1, 1), (5, 1, 1), (4, 2, 4), (1, 8, 8)])
@pytest.mark.parametrize("n_splits", [1, 6])
def test_attn_f16_is_rounded_f32_and_matches_oracle(kvq_lib, gq, bk, bv, n_splits):
    cfg = kvq.CacheConfig(batch=2, n_q_heads=2 * gq, n_kv_heads=2, bits_k=bk, bits_v=bv,
                          max_len=4096)
    lengths = [3001, 190]
    cache, kv = _util.make_cache(cfg, lengths, seed=300 + gq + bk)
    q = synth.queries(301 + gq, cfg.batch, cfg.n_q_heads).cuda()
    o16 = kvq.kvq_decode_attn(cache, q, n_splits=n_splits)
    o32 = kvq.kvq_decode_attn(cache, q, n_splits=n_splits, out_dtype=torch.float32)
    torch.cuda.synchronize()
    assert o16.dtype == torch.float16 and o32.dtype == torch.float32
    rn = o32.half()  # IEEE round to nearest even
    assert torch.equal(o16.view(torch.int16), rn.view(torch.int16))
    got = o16.cpu().numpy()
    for b, L in enumerate(lengths):
        k, v = kv[b]
        ref = attention.decode_attention(q[b].cpu().numpy(), _util.oracle_heads(cfg, k, v))
        assert _util.attn_rel_err(got[b], ref).max() <= _util.ATTN_TOL


@pytest.mark.parametrize("gq", [4, 5])
def test_step_f16_is_rounded_f32(kvq_lib, gq):
    cfg = kvq.CacheConfig(batch=2, n_q_heads=2 * gq, n_kv_heads=2, bits_k=1, bits_v=1,
                          max_len=1024)
    lengths = [159, 700]  # the first sequence's step flushes a group
    a, kv = _util.make_cache(cfg, lengths, seed=310 + gq)
    b_, _ = _util.make_cache(cfg, lengths, seed=310 + gq)
    g = synth.generator(311)
    kn = torch.randn(2, 2, 128, generator=g).half().cuda()
    vn = torch.randn(2, 2, 128, generator=g).half().cuda()
    q = torch.randn(2, 2 * gq, 128, generator=g).half().cuda()
    o16 = kvq.kvq_decode_step(a, kn, vn, q, n_splits=3)
    o32 = kvq.kvq_decode_step(b_, kn, vn, q, n_splits=3, out_dtype=torch.float32)
    torch.cuda.synchronize()
    assert torch.equal(o16.view(torch.int16), o32.half().view(torch.int16))
    assert a.seq_lens().cpu().tolist() == [L + 1 for L in lengths]
    got = o16.cpu().numpy()
    for s, L in enumerate(lengths):
        k, v = kv[s]
        k = torch.cat([k, kn[s].cpu()[:, None]], 1)
        v = torch.cat([v, vn[s].cpu()[:, None]], 1)
        ref = attention.decode_attention(q[s].cpu().numpy(), _util.oracle_heads(cfg, k, v))
        assert _util.attn_rel_err(got[s], ref).max() <= _util.ATTN_TOL


def test_out_dtype_is_checked(kvq_lib):
    cfg = kvq.CacheConfig(batch=1, n_q_heads=4, n_kv_heads=1, bits_k=2, bits_v=2, max_len=512)
    cache, _ = _util.make_cache(cfg, [200], seed=320)
    q = synth.queries(321, 1, 4).cuda()
    with pytest.raises(TypeError):
        kvq.kvq_decode_attn(cache, q, out=torch.empty(1, 4, 128, dtype=torch.bfloat16,
                                                      device="cuda"))
    out = torch.empty(1, 4, 128, dtype=torch.float16, device="cuda")
    assert kvq.kvq_decode_attn(cache, q, out=out) is out
    assert np.isfinite(out.float().cpu().numpy()).all()
