"""The quantizer's codes (Sec. 3.1): code = clamp(rint(RN32(d / s)), 0, levels)
with d = RN32(x - zero) and s the stored fp16 scale.  The CUDA quantizer forms
q = RN32(d * RN32(1 / s)) and takes the exact quotient only when q lies within
1/8192 of a half-integer; this test checks that argument in IEEE float32
arithmetic (numpy), on random fp16 scales and differences and on differences
placed at and next to every half-integer multiple of the scale."""

import numpy as np
import pytest

TOL = np.float32(1.0 / 8192.0)


def _guarded(d, s):
    r = np.float32(1.0) / s                      # RN32(1 / s)
    q = (d * r).astype(np.float32)               # RN32(d * r)
    t = np.rint(q)
    near = np.abs(np.abs(q - t) - np.float32(0.5)) < TOL
    exact = np.rint((d / s).astype(np.float32))  # RN32(d / s), then ties to even
    return np.where(near, exact, t), exact, near


@pytest.mark.parametrize("bits", [1, 2, 4, 8])
def test_random_scales_and_differences(bits):
    levels = (1 << bits) - 1
    rng = np.random.default_rng(bits)
    s = rng.uniform(2.0 ** -12, 64.0, 200_000).astype(np.float16).astype(np.float32)
    s = s[s > 0]
    d = (rng.uniform(0.0, 1.0, s.size) * levels * s).astype(np.float16).astype(np.float32)
    got, exact, _ = _guarded(d, s)
    assert np.array_equal(got, exact)


@pytest.mark.parametrize("bits", [2, 8])
def test_differences_at_and_beside_half_integers(bits):
    levels = (1 << bits) - 1
    rng = np.random.default_rng(100 + bits)
    s = np.unique(rng.uniform(2.0 ** -10, 32.0, 3000).astype(np.float16)).astype(np.float32)
    m = np.arange(levels, dtype=np.float32) + np.float32(0.5)
    base = (m[None, :] * s[:, None]).astype(np.float16)
    cands = [base]
    for step in (1, 2):
        up, dn = base.copy(), base.copy()
        for _ in range(step):
            up = np.nextafter(up, np.float16(np.inf))
            dn = np.nextafter(dn, np.float16(-np.inf))
        cands += [up, dn]
    d = np.concatenate([c.astype(np.float32) for c in cands], axis=1)
    ss = np.broadcast_to(s[:, None], d.shape)
    keep = (d >= 0) & (d <= levels * ss)
    got, exact, near = _guarded(d[keep], ss[keep])
    assert np.array_equal(got, exact)
    # the bare product would misround some of these: the guard is needed
    r = np.float32(1.0) / ss[keep]
    bare = np.rint((d[keep] * r).astype(np.float32))
    assert np.any(bare != exact) and np.all(near[bare != exact])


def test_error_bound_of_the_product():
    # |RN32(d * RN32(1 / s)) - RN32(d / s)| <= 3 * 2^-24 * (d / s) <= 4.6e-5
    # for d / s <= 255, a third of the guard band
    rng = np.random.default_rng(7)
    s = rng.uniform(2.0 ** -12, 64.0, 300_000).astype(np.float16).astype(np.float32)
    s = s[s > 0]
    d = (rng.uniform(0.0, 1.0, s.size) * 255 * s).astype(np.float16).astype(np.float32)
    q = (d * (np.float32(1.0) / s)).astype(np.float32).astype(np.float64)
    e = (d / s).astype(np.float32).astype(np.float64)
    ratio = d.astype(np.float64) / s.astype(np.float64)
    assert np.all(np.abs(q - e) <= 3 * 2.0 ** -24 * ratio + 1e-12)
    assert np.abs(q - e).max() < float(TOL) / 2
