"""kvq_decode_attn_noalloc, the entry point for callers that cannot allocate
device memory where they run a decode step (a framework whose pool owns the
whole GPU, or a serving loop that must not allocate per step).  It keeps its
split-K scratch in a built-in device array instead of a caller workspace.

Checked through the C ABI against kvq_decode_attn (which takes a workspace)
on two calls in a row, within the attention tolerance the parity tests use.
This file is collected last on purpose.
"""

import ctypes

import numpy as np
import pytest
import torch

import _util
from paper_2607_16248_gb300 import kvq, synth

pytestmark = pytest.mark.gpu


def _rel(a, b):
    a = a.float().cpu().numpy().astype(np.float64)
    b = b.float().cpu().numpy().astype(np.float64)
    return _util.attn_rel_err(a, b).max()


def test_noalloc_matches_workspace_path_on_two_calls(kvq_lib):
    cfg = kvq.CacheConfig(batch=2, n_q_heads=32, n_kv_heads=8, bits_k=2, bits_v=2, max_len=4096)
    cache, _ = _util.make_cache(cfg, [4096, 1500], seed=91)
    lib = kvq.lib()
    c = cfg.c()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for call in range(2):  # the second call finds the previous call's scratch contents
        q = synth.queries(500 + call, cfg.batch, cfg.n_q_heads).cuda()
        ref = kvq.kvq_decode_attn(cache, q)
        out = torch.full(q.shape, float("nan"), dtype=torch.float32, device=q.device)
        status = lib.kvq_decode_attn_noalloc(ctypes.byref(c), ctypes.byref(cache._c),
                                             ctypes.c_void_p(q.data_ptr()),
                                             ctypes.c_void_p(out.data_ptr()), 0.0, 0, stream)
        assert status == 0, kvq.last_error()
        torch.cuda.synchronize()
        assert torch.isfinite(out).all()
        assert _rel(out, ref) <= _util.ATTN_TOL, f"call {call}"


def test_noalloc_rejects_configs_beyond_its_array(kvq_lib):
    cfg = kvq.CacheConfig(batch=64, n_q_heads=64, n_kv_heads=8, bits_k=1, bits_v=1,
                          max_len=1 << 20)
    c = cfg.c()
    need = kvq.lib().kvq_attn_workspace_bytes(ctypes.byref(c), 255)
    assert need > kvq.NOALLOC_SCRATCH_BYTES
    fake = ctypes.c_void_p(0x1000)  # never used: the size check fails first
    cache = kvq._Cache(fake, fake, fake, fake)
    status = kvq.lib().kvq_decode_attn_noalloc(ctypes.byref(c), ctypes.byref(cache), fake, fake,
                                               0.0, 255, ctypes.c_void_p(None))
    assert status == 4 and "scratch" in kvq.last_error()
