"""Parity at the benchmark workloads' full sizes, in the launch configuration
bench.py times (kvq_decode_step with the split count kvq.splits_for_lengths
gives for the prefill lengths, one layer of each shape; dgap_restore on the
full logit rows).  The oracle recomputes
sampled (sequence, kv-head) pairs one by one (all 8 kv-heads of the Llama
layer); DGAP rows are all checked.

Workloads: Llama-8B K1V1 at 32768 tokens; the bit-width sweep (K1V1..K8V8) at
131072 tokens; Mistral-7B K2V2, batch 16, ragged 8K-32K; Qwen-14B K1V1, batch
8, 40/8 heads (query groups of 5), 65536 tokens."""

import numpy as np
import pytest
import torch

import _util
from oracle import attention, quant
from paper_2607_16248_gb300 import kvq, synth

pytestmark = pytest.mark.gpu


def _one_layer(cfg, lengths, seed, samples):
    """Prefill, one decode step, and the oracle on sampled (sequence, kv-head)."""
    dev = "cuda"
    cache = kvq.QuantKVCache(cfg, dev)
    kv = {}
    for b, L in enumerate(lengths):
        k, v = synth.kv_heads(seed * 1000 + b, cfg.n_kv_heads, L, device=dev)
        kvq.kvq_pack(cache, k[None], v[None], batch_begin=b)
        for (sb, h) in samples:
            if sb == b:
                kv[(b, h)] = (k[h].cpu(), v[h].cpu())
        del k, v
    g = synth.generator(seed + 17)
    kn = torch.randn(cfg.batch, cfg.n_kv_heads, 128, generator=g).half()
    vn = torch.randn(cfg.batch, cfg.n_kv_heads, 128, generator=g).half()
    q = torch.randn(cfg.batch, cfg.n_q_heads, 128, generator=g).half()
    ns = kvq.splits_for_lengths(cfg, lengths)
    ws = kvq.attn_workspace(cfg, ns)
    out = kvq.kvq_decode_step(cache, kn.cuda(), vn.cuda(), q.cuda(), n_splits=ns,
                              workspace=ws).cpu().numpy()
    assert cache.seq_lens().cpu().tolist() == [L + 1 for L in lengths]
    assert cache.flags() == 0
    gq = cfg.n_q_heads // cfg.n_kv_heads
    assert len(kv) == len(samples)
    worst = 0.0
    for (b, h), (k, v) in kv.items():
        k = torch.cat([k, kn[b, h][None]], 0).numpy()
        v = torch.cat([v, vn[b, h][None]], 0).numpy()
        hd = quant.quantize_head(k, v, cfg.bits_k, cfg.bits_v, cfg.residual)
        K_, V_ = quant.dequantize_head(hd)
        ref = attention.attend_head(q[b, h * gq:(h + 1) * gq].numpy(), K_, V_, 1 / np.sqrt(128))
        worst = max(worst, float(_util.attn_rel_err(out[b, h * gq:(h + 1) * gq], ref).max()))
    return worst


def test_llama8b_k1v1_32k(kvq_lib):
    cfg = kvq.CacheConfig(batch=1, n_q_heads=32, n_kv_heads=8, bits_k=1, bits_v=1,
                          max_len=32768 + 64)
    # every kv-head of the layer: the 19 CTAs of each head cover different
    # block ranges, window chunks and the final merge
    assert _one_layer(cfg, [32768], 2, [(0, h) for h in range(8)]) <= _util.ATTN_TOL


@pytest.mark.parametrize("bits", [1, 2, 4, 8])
def test_sweep_131k(kvq_lib, bits):
    cfg = kvq.CacheConfig(batch=1, n_q_heads=32, n_kv_heads=8, bits_k=bits, bits_v=bits,
                          max_len=131072 + 64)
    assert _one_layer(cfg, [131072], 3 * 1000 + bits, [(0, 3)]) <= _util.ATTN_TOL


def test_mistral7b_k2v2_ragged_batch16(kvq_lib):
    lengths = synth.ragged_lengths(4, 16, 8192, 32768)
    cfg = kvq.CacheConfig(batch=16, n_q_heads=32, n_kv_heads=8, bits_k=2, bits_v=2,
                          max_len=32768 + 64)
    assert _one_layer(cfg, lengths, 4, [(0, 2), (7, 2), (15, 6)]) <= _util.ATTN_TOL


def test_qwen14b_k1v1_64k_batch8(kvq_lib):
    cfg = kvq.CacheConfig(batch=8, n_q_heads=40, n_kv_heads=8, bits_k=1, bits_v=1,
                          max_len=65536 + 64)
    assert _one_layer(cfg, [65536] * 8, 5, [(0, 0), (5, 7)]) <= _util.ATTN_TOL


@pytest.mark.parametrize("B,V,tau,seed", [(1, 128256, 0.6, 2), (8, 152064, 0.6, 5),
                                          (1, 32000, 0.6, 1)])
def test_dgap_full_rows(kvq_lib, B, V, tau, seed):
    from test_gpu_dgap import _run, _compare
    zin, out, zout, det, cor = _run(B, V, 32, tau, seed=seed)
    _compare(zin, out, zout, 32, tau, det, cor)
