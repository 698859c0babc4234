"""Attention is a sum over tokens (Sec. 1): permuting the fp16 window's
tokens, keys and values together, changes kvq_decode_attn's output only by
the order of its fp32 sums."""

import numpy as np
import pytest
import torch

import _util
from paper_2607_16248_gb300 import kvq, synth

pytestmark = pytest.mark.gpu


def test_window_token_permutation_invariance(kvq_lib):
    cfg = kvq.CacheConfig(batch=2, n_q_heads=8, n_kv_heads=2, bits_k=2, bits_v=2, max_len=512)
    lengths = [300, 150]  # 140 window tokens after 160 packed; an all-window sequence
    cache, _ = _util.make_cache(cfg, lengths, 62)
    q = synth.queries(63, cfg.batch, cfg.n_q_heads).cuda()
    before = kvq.kvq_decode_attn(cache, q, out_dtype=torch.float32).cpu().numpy()
    kr, vr = cache.resid()  # views of the cache's fp16 rings
    g = torch.Generator().manual_seed(64)
    for b, L in enumerate(lengths):
        slots = torch.arange(kvq.packed_len(L), L) % cfg.ring
        perm = slots[torch.randperm(slots.numel(), generator=g)]
        assert not torch.equal(perm, slots)
        slots, perm = slots.cuda(), perm.cuda()
        kr[b, :, slots] = kr[b, :, perm]
        vr[b, :, slots] = vr[b, :, perm]
    torch.cuda.synchronize()
    after = kvq.kvq_decode_attn(cache, q, out_dtype=torch.float32).cpu().numpy()
    rms = np.sqrt((before ** 2).mean(axis=-1))
    assert (np.abs(after - before).max(axis=-1) / rms).max() <= 1e-4
