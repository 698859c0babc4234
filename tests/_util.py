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


def key1_bit(t, c):
    """Bit index of the 1-bit key code (token t, channel c) in a page's
    512-byte code area (fragment order, as documented in include/kvq.h)."""
    gid, j, ks, tig = t >> 2, t & 3, c >> 4, (c >> 2) & 3
    h, e = (c >> 1) & 1, c & 1
    r = 2 * (ks & 1) + h
    return (16 * gid + 4 * tig + (ks >> 1)) * 32 + ((10 + 16 * e + j - 4 * r) & 31)


def val1_bit(t, c):
    """Bit index of the 1-bit value code (token t, channel c)."""
    w, gid, j = c >> 5, (c >> 2) & 7, c & 3
    tig, r, e = t >> 3, t & 3, (t >> 2) & 1
    return (16 * gid + 4 * tig + w) * 32 + ((10 + 16 * e + j - 4 * r) & 31)


def vmeta_index(g, t):
    """Position of the value scale (or zero) of (group g, token t)."""
    return 32 * g + 8 * (t >> 3) + 2 * (t & 3) + ((t >> 2) & 1)


_T, _C = np.meshgrid(np.arange(32), np.arange(128), indexing="ij")  # [token, channel]
_KBIT = key1_bit(_T, _C)
_VBIT = val1_bit(_T, _C)
_G, _TT = np.meshgrid(np.arange(4), np.arange(32), indexing="ij")    # [group, token]
_VMI = vmeta_index(_G, _TT)


def _bits_of(area, bit_index):
    """area [nb, 512] uint8 -> codes [nb, *bit_index.shape] at those bits."""
    words = area.view(np.uint32)                                        # [nb, 128]
    return (words[:, bit_index >> 5] >> (bit_index & 31).astype(np.uint32)) & 1


def _pack_rows(codes):
    """codes [..., 32] of 0/1 -> one little-endian uint32 per row."""
    return (codes.astype(np.uint64) << np.arange(32, dtype=np.uint64)).sum(-1).astype(np.uint32)


def head_arrays(cache, b, h, L):
    """The GPU cache of (sequence b, kv-head h) holding L tokens, in the
    layout quant.quantize_head returns."""
    cfg = cache.cfg
    Lq = kvq.packed_len(L, cfg.residual)
    nb = Lq // 32
    bk, bv = cfg.bits_k, cfg.bits_v
    pages = cache.head_pages(b, h, nb).cpu().numpy()

    def sl(a, c):
        return np.ascontiguousarray(pages[:, a:c])

    if bk == 1:  # fragment order: canonical word of channel c has token t at bit t
        kc = _bits_of(sl(0, 512), _KBIT)                                # [nb, tok, ch]
        kw = _pack_rows(kc.transpose(0, 2, 1))[..., None]               # [nb, 128, 1]
    else:
        kw = sl(0, 512 * bk).view(np.uint32).reshape(nb, 128, bk)
    # key metadata: 128 scales, then 128 zeros (one per channel)
    km = sl(512 * bk, 512 * bk + 512).view(np.float16).reshape(nb, 2, 128)
    if bv == 1:  # canonical word of (token t, group g) has channel 32g + i at bit i
        vc = _bits_of(sl(512 * bk + 512, 512 * bk + 1024), _VBIT)      # [nb, tok, ch]
        vw = _pack_rows(vc.reshape(nb, 32, 4, 32))[..., None]           # [nb, 32, 4, 1]
    else:
        # value groups are stored group-major: [nb][4 group][32 token]
        vw = sl(512 * bk + 512, 512 * (bk + bv) + 512).view(np.uint32).reshape(nb, 4, 32, bv)
        vw = np.ascontiguousarray(vw.transpose(0, 2, 1, 3))
    # value metadata: 128 scales, then 128 zeros, at vmeta_index(group, token)
    vm = sl(512 * (bk + bv) + 512, 512 * (bk + bv) + 1024).view(np.float16).reshape(nb, 2, 128)
    vm = np.ascontiguousarray(vm[:, :, _VMI].transpose(0, 1, 3, 2))    # [nb, 2, 32, 4]
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
