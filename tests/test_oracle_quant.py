"""Pins of the oracle's quantizer, bit packing and residual-window policy.

Each test checks the oracle against something other than itself: exact
rational arithmetic, closed forms, hand-derived bit patterns, brute force.
"""

from fractions import Fraction
from pathlib import Path

import numpy as np
import pytest

from oracle import quant

GOLDEN = Path(__file__).resolve().parent / "golden"
BITS = (1, 2, 4, 8)


def _groups(rng, n, kind):
    if kind == "normal":
        x = rng.standard_normal((n, 32))
    elif kind == "outlier":
        x = rng.standard_normal((n, 32)) * 10.0
    elif kind == "uniform":
        x = rng.uniform(-3, 7, (n, 32))
    else:  # wide: up to +-2000
        x = rng.standard_normal((n, 32)) * 500.0
    return x.astype(np.float16)


def _prev16(h):
    return np.nextafter(np.float16(h), np.float16(-np.inf))


def test_round_up_f16_is_least_upper_fp16():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.uniform(0, 70000, 2000), rng.uniform(0, 1e-3, 2000),
                        rng.uniform(0, 1, 2000) * 6e-8])
    r = quant.round_up_f16(x)
    for xv, rv in zip(x, r):
        if xv > 65504:
            assert np.isinf(rv)
            continue
        assert Fraction(float(rv)) >= Fraction(float(xv))
        if rv > 0:
            assert Fraction(float(_prev16(rv))) < Fraction(float(xv))
    # an exact zero rounds to +0, whatever order the table was built in
    z = quant.round_up_f16(np.array([0.0, -0.0]))
    assert z.view(np.uint16).tolist() == [0, 0]
    # fp16 values map to themselves
    h = rng.standard_normal(1000).astype(np.float16)
    h = np.abs(h)
    assert np.array_equal(quant.round_up_f16(h.astype(np.float64)), h)


def test_round_up_f32_against_exact_rationals():
    rng = np.random.default_rng(1)
    a = rng.standard_normal(3000).astype(np.float16)
    b = rng.standard_normal(3000).astype(np.float16) * np.float16(100)
    exact = np.abs(a.astype(np.float64) - b.astype(np.float64))  # exact in float64
    r = quant.round_up_f32(exact)
    for e, rv in zip(exact, r):
        fe = Fraction(float(e))
        assert Fraction(float(rv)) >= fe
        assert Fraction(float(np.nextafter(rv, np.float32(-np.inf)))) < fe or rv == 0


@pytest.mark.parametrize("n", [1, 3, 15, 255])
def test_div_round_up_f32_against_exact_rationals(n):
    rng = np.random.default_rng(n)
    num = np.abs(rng.standard_normal(3000) * 50).astype(np.float32)
    num[:5] = [0.0, 1.0, 3.0, 15.0, 255.0]
    q = quant.div_round_up_f32(num, n)
    for a, qv in zip(num, q):
        exact = Fraction(float(a)) / n
        assert Fraction(float(qv)) >= exact
        if qv > 0:
            assert Fraction(float(np.nextafter(qv, np.float32(-np.inf)))) < exact


@pytest.mark.parametrize("bits", BITS)
@pytest.mark.parametrize("kind", ["normal", "outlier", "uniform", "wide"])
def test_round_trip_bound_and_no_clamping(bits, kind):
    rng = np.random.default_rng(bits * 7 + len(kind))
    x = _groups(rng, 500, kind)
    c, s, z = quant.quantize_groups(x, bits)
    xh = quant.dequantize_groups(c, s, z)
    lo = x.astype(np.float64).min(axis=1)
    hi = x.astype(np.float64).max(axis=1)
    s64 = s.astype(np.float64)
    assert np.all(((1 << bits) - 1) * s64 >= hi - lo)
    err = np.abs(x.astype(np.float64) - xh)
    assert np.all(err <= (s64[:, None] / 2) * (1 + 2.0 ** -22))
    assert np.array_equal(z.astype(np.float64), lo)


def test_one_bit_dyadic_groups_reconstruct_min_and_max_exactly():
    rng = np.random.default_rng(5)
    for _ in range(200):
        e = rng.integers(-6, 4)
        k = rng.integers(-64, 64, 32)
        x = (k * 2.0 ** e).astype(np.float16)
        assert np.array_equal(x.astype(np.float64), k * 2.0 ** e)  # representable
        c, s, z = quant.quantize_groups(x[None], 1)
        xh = quant.dequantize_groups(c, s, z)[0]
        lo, hi = float(x.min()), float(x.max())
        assert set(np.unique(xh)) <= {lo, lo + float(s[0])}
        assert lo + float(s[0]) == hi


def test_one_bit_random_groups_overshoot_at_most_one_ulp():
    rng = np.random.default_rng(6)
    x = _groups(rng, 1000, "normal")
    c, s, z = quant.quantize_groups(x, 1)
    xh = quant.dequantize_groups(c, s, z)
    lo = x.astype(np.float64).min(axis=1)
    hi = x.astype(np.float64).max(axis=1)
    s64 = s.astype(np.float64)
    for i in range(len(x)):
        assert set(np.unique(xh[i])) <= {lo[i], lo[i] + s64[i]}
    ulp = np.spacing(s.astype(np.float16)).astype(np.float64)
    over = (lo + s64) - hi
    assert np.all(over >= 0) and np.all(over <= ulp)


@pytest.mark.parametrize("bits", BITS)
def test_constant_group(bits):
    x = np.full((3, 32), [[1.5], [-7.25], [0.0]], dtype=np.float16)
    c, s, z = quant.quantize_groups(x, bits)
    assert np.all(s.view(np.uint16) == 0) and np.all(c == 0)  # scale is +0
    assert np.array_equal(quant.dequantize_groups(c, s, z), x.astype(np.float64))


@pytest.mark.parametrize("bits", BITS)
def test_grid_inputs_give_exact_codes(bits):
    rng = np.random.default_rng(bits)
    L = (1 << bits) - 1
    for e in (-4, -1, 0, 2):
        k = rng.integers(0, L + 1, 32)
        k[0], k[1] = 0, L
        lo = -3.0
        x = (lo + k * 2.0 ** e).astype(np.float16)
        assert np.array_equal(x.astype(np.float64), lo + k * 2.0 ** e)
        c, s, z = quant.quantize_groups(x[None], bits)
        assert float(s[0]) == 2.0 ** e
        assert np.array_equal(c[0], k)


def test_eight_bit_integers_are_their_own_codes():
    rng = np.random.default_rng(8)
    k = rng.integers(0, 256, 32)
    k[3], k[9] = 0, 255
    c, s, z = quant.quantize_groups(k.astype(np.float16)[None], 8)
    assert float(s[0]) == 1.0 and float(z[0]) == 0.0
    assert np.array_equal(c[0], k)


@pytest.mark.parametrize("bits", BITS)
def test_codes_are_nearest_levels_by_brute_force(bits):
    rng = np.random.default_rng(20 + bits)
    x = _groups(rng, 200, "normal")
    c, s, z = quant.quantize_groups(x, bits)
    levels = np.arange(1 << bits, dtype=np.float64)
    for g in range(len(x)):
        cand = z[g].astype(np.float64) + s[g].astype(np.float64) * levels
        for i in range(32):
            d = np.abs(x[g, i].astype(np.float64) - cand)
            slack = float(s[g]) * 2.0 ** -22
            assert d[c[g, i]] <= d.min() + slack


def _golden_rows():
    rows = []
    for line in (GOLDEN / "pack_words.txt").read_text().splitlines():
        if not line.strip() or line.startswith("#"):
            continue
        b, codes, words = (p.strip() for p in line.split("|"))
        rows.append((int(b), [int(v) for v in codes.split()], [int(w, 16) for w in words.split()]))
    return rows


@pytest.mark.parametrize("bits,codes,words", _golden_rows())
def test_pack_matches_hand_derived_words(bits, codes, words):
    got = quant.pack_codes(np.array(codes, dtype=np.uint8)[None], bits)[0]
    assert [int(w) for w in got] == words
    back = quant.unpack_codes(np.array(words, dtype=np.uint32)[None], bits)[0]
    assert [int(v) for v in back] == codes


@pytest.mark.parametrize("bits", BITS)
def test_pack_unpack_identity_brute_force(bits):
    rng = np.random.default_rng(30 + bits)
    codes = rng.integers(0, 1 << bits, (300, 32)).astype(np.uint8)
    assert np.array_equal(quant.unpack_codes(quant.pack_codes(codes, bits), bits), codes)
    words = rng.integers(0, 2 ** 32, (300, bits), dtype=np.uint64).astype(np.uint32)
    assert np.array_equal(quant.pack_codes(quant.unpack_codes(words, bits), bits), words)


def test_residual_policy():
    R = 128
    assert quant.packed_len(4096, R) == 3968
    assert quant.packed_len(32768, R) == 32640
    assert quant.packed_len(65536, R) == 65408
    assert quant.packed_len(131072, R) == 130944
    for L in range(0, 700):
        Lq = quant.packed_len(L, R)
        assert Lq % 32 == 0 and 0 <= Lq <= L
        if L >= R:
            assert R <= L - Lq <= R + 31
        else:
            assert Lq == 0


def test_head_grouping_keys_per_channel_values_per_token():
    rng = np.random.default_rng(40)
    k = rng.standard_normal((200, 128)).astype(np.float16)
    v = rng.standard_normal((200, 128)).astype(np.float16)
    base = quant.quantize_head(k, v, 2, 2, 128)
    assert base["Lq"] == 64 and base["k_res"].shape == (136, 128)
    k2, v2 = k.copy(), v.copy()
    k2[5, 7] = 40.0  # token 5 of channel 7: only key group (block 0, channel 7) changes
    v2[37, 70] = 40.0  # token 37, channel 70: only value group (block 1, token 5, group 2)
    mod = quant.quantize_head(k2, v2, 2, 2, 128)
    dk = np.argwhere(mod["k_scale"] != base["k_scale"])
    assert dk.tolist() == [[0, 7]]
    dv = np.argwhere(mod["v_scale"] != base["v_scale"])
    assert dv.tolist() == [[1, 5, 2]]
    khat, vhat = quant.dequantize_head(mod)
    assert khat.shape == (200, 128) and vhat.shape == (200, 128)
    assert np.array_equal(khat[64:], k2[64:].astype(np.float64))  # residual stays fp16
