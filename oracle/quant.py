"""Oracle: asymmetric b-bit KV quantizer, bit packing and the residual window.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

The paper names the cache precisions "KbVb" (b-bit keys, b-bit values,
Sec. 3.1 Methodology) and follows KIVI-style asymmetric quantization with keys
grouped per channel and values per token (Sec. 1, Sec. 2).  It does not print
the quantizer, so the readings below are this library's definition of it:

* a group is 32 fp16 numbers: for keys, 32 consecutive tokens of one channel;
  for values, 32 consecutive channels of one token;
* zero = min of the group (exact fp16);
* scale = RU16( RU32( RU32(max - min) / (2^b - 1) ) ), RU = round toward +inf,
  stored as fp16; rounding up keeps (2^b - 1) * scale >= max - min, so no
  element is clamped;
* code = clamp( rint_half_even( RN32( RN32(x - zero) / scale ) ), 0, 2^b - 1 ),
  each RN32 one IEEE float32 operation; a zero scale gives code 0;
* dequantized value = zero + scale * code (exact in float64);
* the codes of one group occupy b little-endian uint32 words; element i sits
  in bits [(i*b) mod 32, +b) of word floor(i*b/32);
* token groups are aligned to absolute position 0; of L tokens,
  Lq = 32 * floor(max(L - R, 0) / 32) are quantized and the last L - Lq stay
  fp16 in the residual window (R <= L - Lq <= R + 31 once L >= R).
"""

import numpy as np

GROUP = 32
HEAD_DIM = 128
SUPPORTED_BITS = (1, 2, 4, 8)

# ---------------------------------------------------------------------------
# Directed rounding, written from the IEEE-754 definition: RU(x) is the
# smallest representable number >= x.
# ---------------------------------------------------------------------------


def _all_finite_f16_sorted():
    bits = np.arange(0x10000, dtype=np.uint32).astype(np.uint16)
    finite = (bits & 0x7C00) != 0x7C00  # exponent field not all ones
    vals = bits[finite].view(np.float16).astype(np.float64)
    vals = np.unique(vals + 0.0)  # sorted; x + 0.0 turns -0 into +0
    assert not np.signbit(vals[vals == 0]).any()
    return vals


_F16_TABLE = _all_finite_f16_sorted()


def round_up_f16(x):
    """RU16: smallest finite fp16 >= x (float64 input, exact), +inf above 65504.

    Defined by search over the table of every finite fp16 value, so it does
    not depend on any library conversion routine.
    """
    x = np.asarray(x, dtype=np.float64)
    idx = np.searchsorted(_F16_TABLE, x, side="left")
    out = np.full(x.shape, np.inf)
    ok = idx < _F16_TABLE.size
    out[ok] = _F16_TABLE[idx[ok]]
    return out.astype(np.float16)


def round_up_f32(x):
    """RU32 of an exactly known float64 value: smallest float32 >= x."""
    x = np.asarray(x, dtype=np.float64)
    f = x.astype(np.float32)  # round to nearest
    below = f.astype(np.float64) < x
    f[below] = np.nextafter(f[below], np.float32(np.inf))
    return f


def div_round_up_f32(num, n):
    """RU32(num / n) for float32 num >= 0 and a small positive integer n.

    q = RN32(num / n) is the correctly rounded quotient; q * n is exact in
    float64 (24 + 8 significant bits), so comparing it with num tells on which
    side of the exact quotient q lies.
    """
    num = np.asarray(num, dtype=np.float32)
    q = (num / np.float32(n)).astype(np.float32)
    below = q.astype(np.float64) * float(n) < num.astype(np.float64)
    q[below] = np.nextafter(q[below], np.float32(np.inf))
    return q


# ---------------------------------------------------------------------------
# Group quantizer (KbVb, Sec. 3.1) — acts on the last axis (length 32).
# ---------------------------------------------------------------------------


def quantize_groups(x, bits):
    """Quantize groups of 32 fp16 values along the last axis.

    Returns (codes uint8 [..., 32], scale fp16 [...], zero fp16 [...]).
    Raises ValueError when a group's range is not fp16-representable as a
    scale (max - min > 65504 * (2^b - 1)).
    """
    if bits not in SUPPORTED_BITS:
        raise ValueError(f"bits must be one of {SUPPORTED_BITS}")
    x = np.asarray(x, dtype=np.float16)
    if x.shape[-1] != GROUP:
        raise ValueError("last axis must hold one group of 32 values")
    levels = (1 << bits) - 1
    lo = x.min(axis=-1)
    hi = x.max(axis=-1)
    zero = lo.astype(np.float16)
    rng = round_up_f32(hi.astype(np.float64) - lo.astype(np.float64))
    scale32 = div_round_up_f32(rng, levels)
    scale = round_up_f16(scale32.astype(np.float64))
    if not np.all(np.isfinite(scale)):
        raise ValueError("group range too large for an fp16 scale")

    diff = x.astype(np.float32) - zero.astype(np.float32)[..., None]  # RN32
    s32 = scale.astype(np.float32)[..., None]
    safe = np.where(s32 > 0, s32, np.float32(1.0))
    ratio = diff / safe  # RN32
    codes = np.rint(ratio)  # ties to even
    codes = np.clip(codes, 0, levels)
    codes = np.where(s32 > 0, codes, 0)
    return codes.astype(np.uint8), scale, zero


def dequantize_groups(codes, scale, zero):
    """x_hat = zero + scale * code, exact in float64."""
    return (zero.astype(np.float64)[..., None]
            + scale.astype(np.float64)[..., None] * codes.astype(np.float64))


# ---------------------------------------------------------------------------
# Bit packing: b little-endian uint32 words per 32-element group.
# ---------------------------------------------------------------------------


def pack_codes(codes, bits):
    """uint8 [..., 32] -> uint32 [..., bits]; element i at bit (i*b) % 32 of
    word (i*b) // 32."""
    codes = np.asarray(codes, dtype=np.uint64)
    out = np.zeros(codes.shape[:-1] + (bits,), dtype=np.uint64)
    for i in range(GROUP):
        word, shift = divmod(i * bits, 32)
        out[..., word] |= (codes[..., i] & ((1 << bits) - 1)) << shift
    return out.astype(np.uint32)


def unpack_codes(words, bits):
    """uint32 [..., bits] -> uint8 [..., 32] (inverse of pack_codes)."""
    words = np.asarray(words, dtype=np.uint64)
    out = np.zeros(words.shape[:-1] + (GROUP,), dtype=np.uint8)
    for i in range(GROUP):
        word, shift = divmod(i * bits, 32)
        out[..., i] = (words[..., word] >> shift) & ((1 << bits) - 1)
    return out


# ---------------------------------------------------------------------------
# One (sequence, kv-head) cache: packed blocks + fp16 residual window.
# ---------------------------------------------------------------------------


def packed_len(L, residual):
    """Lq: tokens held in quantized 32-token blocks when L tokens are cached."""
    return GROUP * (max(L - residual, 0) // GROUP)


def quantize_head(k, v, bits_k, bits_v, residual):
    """Quantize one kv-head's keys and values.

    k, v: fp16 [L, 128].  Keys are grouped per channel over 32 tokens, values
    per token over 32 channels (KIVI-style asymmetric layout, Sec. 2).
    Returns a dict with
      k_words [nb, 128, bits_k] uint32, k_scale/k_zero [nb, 128] fp16,
      v_words [nb, 32, 4, bits_v] uint32, v_scale/v_zero [nb, 32, 4] fp16,
      k_res, v_res [L - Lq, 128] fp16 (the residual window, oldest first).
    """
    k = np.asarray(k, dtype=np.float16)
    v = np.asarray(v, dtype=np.float16)
    L, d = k.shape
    if d != HEAD_DIM or v.shape != k.shape:
        raise ValueError("k and v must both be [L, 128]")
    Lq = packed_len(L, residual)
    nb = Lq // GROUP
    kb = k[:Lq].reshape(nb, GROUP, d).transpose(0, 2, 1)  # [nb, ch, tok]
    kc, ks, kz = quantize_groups(kb, bits_k)
    vb = v[:Lq].reshape(nb, GROUP, d // GROUP, GROUP)  # [nb, tok, grp, ch]
    vc, vs, vz = quantize_groups(vb, bits_v)
    return dict(
        k_words=pack_codes(kc, bits_k), k_scale=ks, k_zero=kz,
        v_words=pack_codes(vc, bits_v), v_scale=vs, v_zero=vz,
        k_res=k[Lq:].copy(), v_res=v[Lq:].copy(),
        bits_k=bits_k, bits_v=bits_v, L=L, Lq=Lq)


def dequantize_head(qh):
    """Rebuild float64 K_hat, V_hat [L, 128] from quantize_head's output."""
    bk, bv = qh["bits_k"], qh["bits_v"]
    kc = unpack_codes(qh["k_words"], bk)  # [nb, ch, tok]
    khat = dequantize_groups(kc, qh["k_scale"], qh["k_zero"])
    khat = khat.transpose(0, 2, 1).reshape(-1, HEAD_DIM)
    vc = unpack_codes(qh["v_words"], bv)  # [nb, tok, grp, ch]
    vhat = dequantize_groups(vc, qh["v_scale"], qh["v_zero"])
    vhat = vhat.reshape(-1, HEAD_DIM)
    khat = np.concatenate([khat, qh["k_res"].astype(np.float64)])
    vhat = np.concatenate([vhat, qh["v_res"].astype(np.float64)])
    return khat, vhat
