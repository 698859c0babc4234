"""Failure detection without a fault: a bounded wait on a copy that never
arrives gives up, reports KVQ_FLAG_WAIT_TIMEOUT through the flag word, and
the context keeps working (an attention call afterwards matches the oracle)."""

import time

import pytest
import torch

import _util
from oracle import attention
from paper_2607_16248_gb300 import kvq, synth

pytestmark = pytest.mark.gpu


def test_wait_gives_up_and_reports(kvq_lib):
    t0 = time.perf_counter()
    flag = kvq.selftest_wait_timeout()
    torch.cuda.synchronize()
    assert int(flag.item()) & kvq.FLAG_WAIT_TIMEOUT
    assert time.perf_counter() - t0 < 30.0
    # the context is still usable
    cfg = kvq.CacheConfig(batch=1, n_q_heads=8, n_kv_heads=2, bits_k=2, bits_v=2, max_len=1024)
    cache, kv = _util.make_cache(cfg, [700], 3)
    q = synth.queries(4, 1, 8)
    out = kvq.kvq_decode_attn(cache, q.cuda()).cpu().numpy()
    ref = attention.decode_attention(q[0].numpy(), _util.oracle_heads(cfg, *kv[0]))
    assert _util.attn_rel_err(out[0], ref).max() <= _util.ATTN_TOL
    assert cache.flags() & kvq.FLAG_WAIT_TIMEOUT == 0
