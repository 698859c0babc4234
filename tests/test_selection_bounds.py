"""The two lower bounds the top-(K+1) selection of the DGAP epilogue (Eqs. 2,
11) relies on, checked on ranking keys (value descending, then index
ascending) in numpy:

* chunk phase: 8 warps of 32 threads, E keys per thread; the smallest over
  the warps of each warp's q-th largest per-thread maximum, q = ceil(n / 8),
  bounds the n-th best key from below (8 q >= n keys reach it);
* finalize: chunk lists sorted best first; the n-th best of the first
  r0 = ceil(n / lists) entries of every list bounds the n-th best of all
  lists from below (r0 * lists >= n entries reach it).

Every key at or above a bound is a survivor; the n best are among them."""

import numpy as np
import pytest


def _rank_keys(values):
    # (value, -index) as one sortable float pair -> rank order, best first
    idx = np.arange(values.size)
    return np.lexsort((idx, -values))


def _nth_best_value(values, n):
    return values[_rank_keys(values)[n - 1]]


@pytest.mark.parametrize("seed", range(8))
@pytest.mark.parametrize("n", [2, 9, 33, 65])
def test_per_warp_bound(seed, n):
    rng = np.random.default_rng(seed)
    E = 16
    if seed % 2:
        vals = rng.integers(0, 30, 256 * E).astype(np.float64)  # heavy ties
    else:
        vals = rng.standard_normal(256 * E) * 3
    per_thread = vals.reshape(E, 256).T          # element i * 256 + tid
    tmax = per_thread.max(axis=1)                # per-thread maximum
    q = -(-n // 8)
    warp_q = [np.sort(tmax[32 * w:32 * w + 32])[::-1][q - 1] for w in range(8)]
    T0 = min(warp_q)
    assert _nth_best_value(vals, n) >= T0
    best = _rank_keys(vals)[:n]
    assert np.all(vals[best] >= T0)


@pytest.mark.parametrize("seed", range(8))
@pytest.mark.parametrize("lists,n", [(1, 33), (8, 33), (32, 33), (38, 33), (120, 65), (3, 2)])
def test_leader_bound_on_sorted_lists(seed, lists, n):
    rng = np.random.default_rng(100 + seed)
    chunk = 4096
    vals = (rng.integers(0, 40, lists * chunk).astype(np.float64) if seed % 2
            else rng.standard_normal(lists * chunk) * 3)
    # each chunk's n best, sorted best first (value descending, index ascending)
    cand = []
    for c in range(lists):
        v = vals[c * chunk:(c + 1) * chunk]
        order = _rank_keys(v)[:n]
        cand.append([(v[i], c * chunk + i) for i in order])
    r0 = -(-n // lists)
    leaders = np.array([cand[c][r][0] for c in range(lists) for r in range(r0)])
    T0 = _nth_best_value(leaders, n)
    overall = _nth_best_value(vals, n)
    assert overall >= T0
    flat = np.array([v for lst in cand for v, _ in lst])
    survivors = int(np.sum(flat >= T0))
    assert survivors >= n
    if seed % 2 == 0 and lists >= 8:
        # continuous values: the leader bound leaves few candidates to rank
        assert survivors <= 2 * n + lists


@pytest.mark.parametrize("lists", [8, 32, 38])
def test_both_bounds_leave_few_candidates_on_lists_of_leaders(lists):
    # sorted lists of 33 (32 lists: the finalize of a 128256-token row), held
    # as the finalize holds them (candidate i in thread i mod 256): either
    # bound keeps the n best and leaves at most 4 n candidates to rank
    n, chunk = 33, 4096
    for seed in range(10):
        rng = np.random.default_rng(seed)
        vals = rng.standard_normal(lists * chunk) * 3
        flat = []
        for c in range(lists):
            v = vals[c * chunk:(c + 1) * chunk]
            flat += [v[i] for i in _rank_keys(v)[:n]]
        flat = np.array(flat)
        regs = np.full((256, 16), -np.inf)
        for i, x in enumerate(flat):
            regs[i % 256, i // 256] = x
        tmax = regs.max(axis=1)
        q = -(-n // 8)
        T_warp = min(np.sort(tmax[32 * w:32 * w + 32])[::-1][q - 1] for w in range(8))
        r0 = -(-n // lists)
        leaders = np.array([flat[c * n + r] for c in range(lists) for r in range(r0)])
        T_lead = _nth_best_value(leaders, n)
        best = np.sort(flat)[::-1][n - 1]
        for T in (T_warp, T_lead):
            assert best >= T and n <= int(np.sum(flat >= T)) <= 4 * n
