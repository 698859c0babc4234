"""Pins of the oracle's drift metrics (Sec. 4.1 recovery-window calibration,
Sec. 4.2 offline labels): a hand-computed step, brute-force minimal candidate
sets, tie order, shift invariance, degenerate windows and the K_b rule."""

import itertools
from math import log, sqrt

import numpy as np
import pytest

from oracle import drift


def _logp(p):
    return np.log(np.asarray(p, dtype=np.float64))


def test_hand_computed_step():
    # p_fp = [.5, .2, .15, .1, .05], p_q = [.1, .4, .3, .15, .05]; alpha = 0.8:
    # FP16 prefix masses .5, .7, .85 -> C = {0, 1, 2}, M = 3.
    # S = TopK(z_q, 2) = {1, 2}; c = .2 + .15 = .35.
    # U = C: a = [10, 4, 3] / 17, b = [1, 4, 3] / 8;
    # d^2 = (63/136)^2 + (36/136)^2 + (27/136)^2 = 5994 / 18496.
    # Coverage over TopK(z_q) order [1, 2, 3, 0, 4]: .2, .35, .35, .85, .85.
    r = drift.step_metrics(_logp([.5, .2, .15, .1, .05]), _logp([.1, .4, .3, .15, .05]),
                           alpha=0.8, K=2, eps=0.5, rho_c=0.3, k_max=5)
    assert r["M"] == 3 and sorted(r["C"].tolist()) == [0, 1, 2]
    assert sorted(r["S"].tolist()) == [1, 2]
    assert abs(r["c"] - 0.35) < 1e-15
    assert abs(r["d_loc"] - sqrt(5994 / 18496)) < 1e-15
    assert r["y"]  # 0.569 > 0.5 and 0.35 >= 0.3
    assert np.allclose(r["cov"], [.2, .35, .35, .85, .85], rtol=0, atol=1e-15)
    # raising either threshold clears the label
    assert not drift.step_metrics(_logp([.5, .2, .15, .1, .05]), _logp([.1, .4, .3, .15, .05]),
                                  0.8, 2, 0.6, 0.3)["y"]
    assert not drift.step_metrics(_logp([.5, .2, .15, .1, .05]), _logp([.1, .4, .3, .15, .05]),
                                  0.8, 2, 0.5, 0.36)["y"]


def test_roles_are_not_symmetric():
    # the same step with FP16 and low-bit logits exchanged gives another c:
    # prefix masses .4, .7, .85 -> C = {1, 2, 3}; S = TopK = {0, 1}; c = .4
    r = drift.step_metrics(_logp([.1, .4, .3, .15, .05]), _logp([.5, .2, .15, .1, .05]),
                           0.8, 2, 0.5, 0.3)
    assert sorted(r["C"].tolist()) == [1, 2, 3] and sorted(r["S"].tolist()) == [0, 1]
    assert abs(r["c"] - 0.4) < 1e-15


@pytest.mark.parametrize("seed", range(6))
def test_candidate_set_is_the_smallest_set_reaching_alpha(seed):
    rng = np.random.default_rng(seed)
    V = 7
    z = rng.normal(0, 1.5, V)
    p = np.exp(z - z.max())
    p /= p.sum()
    for alpha in (0.2, 0.5, 0.77, 0.9, 0.99):
        _, m = drift.candidate_set(p, drift.order_desc(z), alpha)
        best = min(len(T) for n in range(1, V + 1) for T in itertools.combinations(range(V), n)
                   if p[list(T)].sum() >= alpha)
        assert m == best
        C, _ = drift.candidate_set(p, drift.order_desc(z), alpha)
        assert p[C].sum() >= alpha and p[C[:-1]].sum() < alpha
        assert p[C].min() >= np.delete(p, C).max(initial=0.0)


def test_ties_take_lowest_index_first():
    z = np.zeros(10)
    r = drift.step_metrics(z, z, alpha=0.35, K=3, eps=0.0, rho_c=0.0, k_max=10)
    assert r["C"].tolist() == [0, 1, 2, 3]  # 4 x 0.1 reaches 0.35
    assert r["S"].tolist() == [0, 1, 2]
    assert abs(r["c"] - 0.3) < 1e-15 and r["d_loc"] == 0.0 and not r["y"]


def test_shift_invariance_and_equal_steps():
    rng = np.random.default_rng(3)
    z = rng.normal(0, 3, 500)
    r = drift.step_metrics(z, z + 7.25, 0.9, 32, 1e-9, 0.0, k_max=64)
    assert r["d_loc"] < 1e-12 and not r["y"]
    # S = TopK(z_fp, 32): coverage is the mass of the first min(M, 32) candidates
    p = drift.softmax(z)
    o = drift.order_desc(z)
    assert abs(r["c"] - p[o[:min(r["M"], 32)]].sum()) < 1e-12


def test_full_window_and_tiny_alpha():
    rng = np.random.default_rng(5)
    zf, zq = rng.normal(0, 2, 40), rng.normal(0, 2, 40)
    pf, pq = drift.softmax(zf), drift.softmax(zq)
    r = drift.step_metrics(zf, zq, 0.9, 40, 0.1, 0.5)  # S = everything, U = everything
    assert abs(r["c"] - pf[r["C"]].sum()) < 1e-15 and r["c"] >= 0.9
    assert abs(r["d_loc"] - np.sqrt(((pf - pq) ** 2).sum())) < 1e-15
    r = drift.step_metrics(zf, zq, pf.max() / 2, 1, 0.1, 0.5)
    assert r["M"] == 1 and r["C"].tolist() == [int(np.argmax(zf))]


def test_alpha_one_with_underflow_takes_everything_reached():
    # p of the last two entries underflows to 0 in float64: mass 1 is reached
    # before the end, and alpha slightly above the rounded total takes all
    z = np.array([0.0, log(3.0), -800.0, -900.0])
    p = drift.softmax(z)
    _, m = drift.candidate_set(p, drift.order_desc(z), 1.0)
    assert m == 2
    _, m = drift.candidate_set(p, drift.order_desc(z), 1.0 + 1e-9)
    assert m == 4


def test_coverage_curve_matches_window_metric_and_is_monotone():
    rng = np.random.default_rng(8)
    zf = rng.normal(0, 3, 300)
    zq = zf + rng.normal(0, 0.7, 300)
    r = drift.step_metrics(zf, zq, 0.95, 8, 0.05, 0.5, k_max=64)
    cov = r["cov"]
    assert np.all(np.diff(cov) >= 0)
    for K in (1, 5, 8, 20, 64):
        assert abs(drift.step_metrics(zf, zq, 0.95, K, 0.05, 0.5)["c"] - cov[K - 1]) < 1e-14


def test_permutation_equivariance():
    rng = np.random.default_rng(11)
    zf = rng.normal(0, 3, 200)
    zq = zf + rng.normal(0, 1, 200)
    perm = rng.permutation(200)
    a = drift.step_metrics(zf, zq, 0.9, 16, 0.05, 0.5)
    b = drift.step_metrics(zf[perm], zq[perm], 0.9, 16, 0.05, 0.5)
    assert a["M"] == b["M"] and abs(a["c"] - b["c"]) < 1e-14
    assert abs(a["d_loc"] - b["d_loc"]) < 1e-14


def test_calibrate_window():
    cov = np.array([[0.25, 0.5, 0.75, 1.0],
                    [0.25, 0.75, 0.75, 1.0]])
    k, mean = drift.calibrate_window(cov, 0.625)
    assert k == 2 and mean.tolist() == [0.25, 0.625, 0.75, 1.0]
    assert drift.calibrate_window(cov, 0.75)[0] == 3
    assert drift.calibrate_window(cov, 1.5)[0] == 0


def test_rows_api():
    rng = np.random.default_rng(2)
    zf = rng.normal(0, 2, (3, 50))
    zq = zf + rng.normal(0, 0.5, (3, 50))
    M, c, d, y, cov = drift.metrics(zf, zq, 0.9, 4, 0.05, 0.5, 10)
    assert M.shape == (3,) and cov.shape == (3, 10)
    for i in range(3):
        r = drift.step_metrics(zf[i], zq[i], 0.9, 4, 0.05, 0.5, 10)
        assert M[i] == r["M"] and c[i] == r["c"] and d[i] == r["d_loc"] and y[i] == r["y"]
