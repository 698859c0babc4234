"""The two arithmetic shortcuts of the CUDA quantizer (csrc/common.cuh),
checked against the oracle's definition (oracle/quant.py, Sec. 3.1 reading)
on the host.  The GPU parity tests compare the kernels with the oracle; this
pins the arguments the kernels rest on, on inputs that reach the cases the
arguments are about (ties, subnormal steps, wide ranges).

* Codes: y = RN32(d * r + 1536.5), d = RN32(x - zero), r = RN32(1 / scale).
  Bits 13 and up of y hold 0x22600 + floor(q + 0.5), q being d * r on the
  2^-13 grid; an element whose 13 low bits are zero takes the exact quotient.
  The result must equal clamp(rint(RN32(d / scale))) for every element.  The
  fused multiply-add is emulated exactly: d * r has at most 48 significant
  bits and d * r + 1536.5 spans bits 2^10 .. 2^-40, so float64 holds it
  before the one rounding to float32.
* Scale: RU32(x / L) for L = 3, 15, 255 from q = RN32(x * RN32(1 / L)),
  moved up while q * L < x and down while (q - ulp) * L >= x (q * L - x is
  exact in float64).
"""

import numpy as np

from oracle import quant

F32 = np.float32


def _codes_shortcut(x, bits):
    levels = (1 << bits) - 1
    _, scale, zero = quant.quantize_groups(x, bits)
    lo = zero.astype(F32)[..., None]
    s = scale.astype(F32)[..., None]
    r = np.where(s > 0, (F32(1) / np.where(s > 0, s, F32(1))).astype(F32), F32(0))
    d = (x.astype(F32) - lo).astype(F32)
    y = (d.astype(np.float64) * r.astype(np.float64) + 1536.5).astype(F32).view(np.uint32)
    code = (y >> 13).astype(np.int64) - 0x22600
    near = (y & 0x1FFF) == 0
    exact = np.clip(np.rint((d / np.where(s > 0, s, F32(1))).astype(F32)), 0, levels)
    exact = np.where(s > 0, exact, 0).astype(np.int64)
    return np.where(near, exact, code), near


def _groups(rng, bits, n):
    levels = (1 << bits) - 1
    parts = [
        rng.standard_normal((n, 32)) * 10 ** rng.uniform(-6, 3, (n, 1)),
        rng.uniform(-5, 5, (n, 1))
        + 10 ** rng.uniform(-4, 1, (n, 1)) * (rng.integers(0, 2 * levels + 1, (n, 32)) / 2.0),
        rng.integers(-60, 60, (n, 32)) * 2.0 ** -24,
        rng.standard_normal((n, 32)) * 1000,
    ]
    return np.clip(np.concatenate(parts), -60000, 60000).astype(np.float16)


def test_fused_code_rounding_matches_the_definition():
    rng = np.random.default_rng(11)
    for bits in (1, 2, 4, 8):
        x = _groups(rng, bits, 20000)
        want, _, _ = quant.quantize_groups(x, bits)
        got, near = _codes_shortcut(x, bits)
        assert np.array_equal(got, want.astype(np.int64)), bits
        assert near.any()  # the tie grids reach the exact path


def _ru_div(x, L):
    def up(q):
        return (q.view(np.uint32) + np.uint32(1)).view(F32)

    def down(q):
        return (q.view(np.uint32) - np.uint32(1)).view(F32)

    q = (x * (F32(1) / F32(L))).astype(F32)
    for _ in range(2):
        q = np.where(q.astype(np.float64) * L - x.astype(np.float64) < 0, up(q), q)
    for _ in range(2):
        p = down(q)
        q = np.where((q > 0) & (p.astype(np.float64) * L - x.astype(np.float64) >= 0), p, q)
    return q


def test_round_up_division_by_levels_matches_the_definition():
    rng = np.random.default_rng(12)
    for L in (3, 15, 255):
        x = np.concatenate([rng.uniform(0, 70000, 300000), np.arange(0, 50000) * 2.0 ** -24,
                            10 ** rng.uniform(-7, 5, 300000),
                            L * (np.arange(1, 50000) * 2.0 ** -20)]).astype(F32)
        x = np.concatenate([x, (x.view(np.uint32) + np.uint32(1)).view(F32)])
        want = quant.div_round_up_f32(x, L)
        assert np.array_equal(_ru_div(x, L).view(np.uint32), want.view(np.uint32)), L
