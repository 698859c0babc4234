"""kvq_decode_attn_noalloc, the entry point for callers that cannot allocate
device memory where they run a decode step (a framework whose pool owns the
whole GPU, or a serving loop that must not allocate per step).  It keeps its
split-K scratch in a built-in device array instead of a caller workspace.

Checked through the C ABI on two calls in a row (the second finds the first
call's scratch contents), against the workspace path kvq_decode_attn_f32 and
against the float64 oracle, within the attention tolerance the parity tests
use.  Split counts: 1 (no partials, no tickets), the default, and the
largest count whose scratch fits the array (the partials reach the end of
the array's used part and the tickets sit right after them).
This file is collected last on purpose.
"""

import ctypes

import numpy as np
import pytest
import torch

import _util
from oracle import attention
from paper_2607_16248_gb300 import kvq, synth

pytestmark = pytest.mark.gpu


def _rel(a, b):
    a = a.float().cpu().numpy().astype(np.float64)
    b = b.float().cpu().numpy().astype(np.float64)
    return _util.attn_rel_err(a, b).max()


def _largest_fitting_splits(cfg):
    c = cfg.c()
    best = 0
    for n in range(1, 256):
        if kvq.lib().kvq_attn_workspace_bytes(ctypes.byref(c), n) <= kvq.NOALLOC_SCRATCH_BYTES:
            best = n
    return best


@pytest.mark.parametrize("which", ["one", "default", "largest"])
def test_noalloc_matches_workspace_path_and_oracle_on_two_calls(kvq_lib, which):
    cfg = kvq.CacheConfig(batch=2, n_q_heads=32, n_kv_heads=8, bits_k=2, bits_v=2, max_len=4096)
    n_splits = {"one": 1, "default": 0, "largest": _largest_fitting_splits(cfg)}[which]
    if which == "largest":
        c = cfg.c()
        need = kvq.lib().kvq_attn_workspace_bytes(ctypes.byref(c), n_splits)
        more = kvq.lib().kvq_attn_workspace_bytes(ctypes.byref(c), n_splits + 1)
        assert need <= kvq.NOALLOC_SCRATCH_BYTES < more or n_splits == 255
    lengths = [4096, 1500]
    cache, kv = _util.make_cache(cfg, lengths, seed=91)
    heads = [_util.oracle_heads(cfg, k, v) for k, v in kv]
    lib = kvq.lib()
    c = cfg.c()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for call in range(2):
        q = synth.queries(500 + call, cfg.batch, cfg.n_q_heads).cuda()
        ref = kvq.kvq_decode_attn(cache, q, n_splits=n_splits, out_dtype=torch.float32)
        out = torch.full(q.shape, float("nan"), dtype=torch.float32, device=q.device)
        status = lib.kvq_decode_attn_noalloc(ctypes.byref(c), ctypes.byref(cache._c),
                                             ctypes.c_void_p(q.data_ptr()),
                                             ctypes.c_void_p(out.data_ptr()), 0.0, n_splits,
                                             stream)
        assert status == 0, kvq.last_error()
        torch.cuda.synchronize()
        assert torch.isfinite(out).all()
        assert _rel(out, ref) <= _util.ATTN_TOL, f"call {call}"
        got = out.cpu().numpy()
        for b in range(cfg.batch):
            want = attention.decode_attention(q[b].cpu().numpy(), heads[b])
            assert _util.attn_rel_err(got[b], want).max() <= _util.ATTN_TOL, f"call {call} seq {b}"


def test_noalloc_wrapper_requires_out(kvq_lib):
    cfg = kvq.CacheConfig(batch=1, n_q_heads=4, n_kv_heads=1, bits_k=2, bits_v=2, max_len=512)
    cache, _ = _util.make_cache(cfg, [300], seed=92)
    q = synth.queries(93, 1, 4).cuda()
    with pytest.raises(ValueError):
        kvq.kvq_decode_attn_noalloc(cache, q, None)


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
