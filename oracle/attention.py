"""Oracle: one GQA decode step of softmax attention over the low-bit cache.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Attention weights are softmax(Q K^T / sqrt(d_k)) V (Sec. 1; the same form is
the starting point of the analysis in Sec. 3.2).  Readings taken where the
paper is silent:

* grouped-query mapping: query head i reads kv-head floor(i / (Hq / Hkv));
* the scale is 1 / sqrt(128) unless the caller overrides it;
* the current token is appended to the cache before attention, so the query
  attends to all L cached tokens (no mask);
* an empty cache (L = 0) gives a zero output.

Everything is float64 on the dequantized cache (``quant.dequantize_head``).
"""

import numpy as np

from . import quant


def attend_head(q, khat, vhat, scale):
    """q [G, 128] (any float), khat/vhat [L, 128] float64 -> o [G, 128] f64."""
    q = np.asarray(q, dtype=np.float64)
    if khat.shape[0] == 0:
        return np.zeros((q.shape[0], khat.shape[1]))
    s = (q @ khat.T) * scale  # [G, L]
    s = s - s.max(axis=1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=1, keepdims=True)
    return p @ vhat


def decode_attention(q, heads, scale=None):
    """One sequence's decode step.

    q: fp16 [Hq, 128]; heads: list of Hkv ``quant.quantize_head`` dicts.
    Returns float64 [Hq, 128].
    """
    q = np.asarray(q)
    hq, d = q.shape
    hkv = len(heads)
    if hq % hkv:
        raise ValueError("n_q_heads must be a multiple of n_kv_heads")
    gq = hq // hkv
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    out = np.zeros((hq, d))
    for h, qh in enumerate(heads):
        khat, vhat = quant.dequantize_head(qh)
        out[h * gq:(h + 1) * gq] = attend_head(q[h * gq:(h + 1) * gq],
                                               khat, vhat, scale)
    return out


def lse_partials(q, khat, vhat, scale, bounds):
    """Split the token range at ``bounds`` and return per-split
    (m, l, o_unnormalised); the merge of these is the unsplit result.  Used
    only to pin the merge algebra the split-K path relies on."""
    q = np.asarray(q, dtype=np.float64)
    parts = []
    for a, b in zip(bounds[:-1], bounds[1:]):
        s = (q @ khat[a:b].T) * scale
        m = s.max(axis=1)
        e = np.exp(s - m[:, None])
        parts.append((m, e.sum(axis=1), e @ vhat[a:b]))
    return parts


def lse_merge(parts):
    """out = sum_s e^{m_s - M} o_s / sum_s e^{m_s - M} l_s."""
    M = np.max(np.stack([p[0] for p in parts]), axis=0)
    num = sum(np.exp(m - M)[:, None] * o for m, _, o in parts)
    den = sum(np.exp(m - M) * l for m, l, _ in parts)
    return num / den[:, None]
