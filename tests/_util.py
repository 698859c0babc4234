"""Helpers for the GPU parity tests: read the CUDA cache back into the
oracle's canonical arrays, build caches from seeded inputs, and compare."""

import numpy as np
import torch

from oracle import quant
from paper_2607_16248_gb300 import kvq

ATTN_TOL = 2e-3     # max |o_gpu - o_oracle| / rms(o_oracle), per (sequence, head)
LOGIT_TOL = 1e-4    # corrected logits, absolute
RISK_TOL = 1e-5     # r, absolute
GATE_BAND = 1e-4    # |f - logit(tau)| inside which the gate may differ


def head_arrays(cache, b, h, L):
    """The GPU cache of (sequence b, kv-head h) holding L tokens, in the
    layout quant.quantize_head returns."""
    cfg = cache.cfg
    Lq = kvq.packed_len(L, cfg.residual)
    nb = Lq // 32
    bk, bv = cfg.bits_k, cfg.bits_v
    pages = cache.pages()[b, h, :nb].cpu().numpy()

    def sl(a, c):
        return np.ascontiguousarray(pages[:, a:c])

    kw = sl(0, 512 * bk).view(np.uint32).reshape(nb, 128, bk)
    # key metadata: 128 scales, then 128 zeros (one per channel)
    km = sl(512 * bk, 512 * bk + 512).view(np.float16).reshape(nb, 2, 128)
    # value groups are stored group-major: [nb][4 group][32 token]; the 128
    # scales precede the 128 zeros
    vw = sl(512 * bk + 512, 512 * (bk + bv) + 512).view(np.uint32).reshape(nb, 4, 32, bv)
    vw = np.ascontiguousarray(vw.transpose(0, 2, 1, 3))
    vm = sl(512 * (bk + bv) + 512, 512 * (bk + bv) + 1024).view(np.float16).reshape(nb, 2, 4, 32)
    vm = np.ascontiguousarray(vm.transpose(0, 1, 3, 2))
    kr, vr = cache.resid()
    slots = torch.tensor([p % cfg.ring for p in range(Lq, L)], dtype=torch.long)
    k_res = kr[b, h].cpu()[slots].numpy()
    v_res = vr[b, h].cpu()[slots].numpy()
    return dict(k_words=kw, k_scale=km[:, 0], k_zero=km[:, 1], v_words=vw,
                v_scale=vm[:, 0], v_zero=vm[:, 1], k_res=k_res, v_res=v_res,
                bits_k=bk, bits_v=bv, L=L, Lq=Lq)


def assert_head_equal(got, want):
    """Codes bit-exact; scales, zeros and the residual window equal."""
    assert got["Lq"] == want["Lq"]
    for key in ("k_words", "v_words"):
        assert got[key].shape == want[key].shape, key
        bad = np.argwhere(got[key] != want[key])
        assert bad.size == 0, f"{key} differs at {bad[:5].tolist()}"
    for key in ("k_scale", "v_scale"):
        assert np.array_equal(got[key].view(np.uint16), want[key].view(np.uint16)), key
    for key in ("k_zero", "v_zero", "k_res", "v_res"):
        assert np.array_equal(got[key].astype(np.float64), want[key].astype(np.float64)), key


def make_cache(cfg, lengths, seed, device="cuda"):
    """Prefill sequence b with lengths[b] seeded tokens.  Returns the cache
    and the host fp16 K/V [Hkv, L_b, 128] per sequence."""
    from paper_2607_16248_gb300 import synth
    cache = kvq.QuantKVCache(cfg, device)
    kv = []
    for b, L in enumerate(lengths):
        k, v = synth.kv_heads(seed * 1000 + b, cfg.n_kv_heads, L)
        kv.append((k, v))
        if L:
            kvq.kvq_pack(cache, k[None].to(device), v[None].to(device), batch_begin=b)
    torch.cuda.synchronize()
    return cache, kv


def oracle_heads(cfg, k, v):
    return [quant.quantize_head(k[h].numpy(), v[h].numpy(), cfg.bits_k, cfg.bits_v, cfg.residual)
            for h in range(cfg.n_kv_heads)]


def attn_rel_err(o_gpu, o_ref):
    """Per query head: max |diff| / rms(reference)."""
    o_gpu = np.asarray(o_gpu, dtype=np.float64)
    rms = np.sqrt((o_ref ** 2).mean(axis=-1))
    err = np.abs(o_gpu - o_ref).max(axis=-1)
    return np.where(rms > 0, err / np.maximum(rms, 1e-300), err)
