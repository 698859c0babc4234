"""kvq_drift_metrics / kvq_drift_window (CUDA, through the C ABI) against the
float64 oracle of Sec. 4.1-4.2's drift metrics.

The GPU takes p from fp32 exponentials summed in fixed point, the oracle from
fp64 throughout, so M_t (an integer decided by a mass threshold) may differ
only where the FP16 prefix mass at both candidate lengths is within BAND of
alpha.  Every row is compared: c_t, d_loc, cov and y_t against the oracle
evaluated with the GPU's candidate set (the first M_t indices of the FP16
order), which is the oracle's own result whenever M_t agrees.  c_t and cov
within 2e-6 absolute, d_loc within 2e-6 + 1e-5 relative, y_t exactly unless
d_loc or c_t is within BAND of eps or rho_c.  ``require`` is the fraction of
rows whose M_t must equal the oracle's exactly."""

import numpy as np
import pytest
import torch

from oracle import drift
from paper_2607_16248_gb300 import kvq, synth

pytestmark = pytest.mark.gpu
BAND = 1e-6
TOL = 2e-6


def _run(zf, zq, alpha, window, k_max, eps, rho_c):
    out = kvq.drift_metrics(zf.cuda(), zq.cuda(), alpha, window, k_max, eps, rho_c)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def _compare(zf, zq, alpha, window, k_max, eps, rho_c, rows=None, require=0.95):
    g = _run(zf, zq, alpha, window, k_max, eps, rho_c)
    # the parameters reach the kernel as float32
    alpha, eps, rho_c = (float(np.float32(x)) for x in (alpha, eps, rho_c))
    zf64, zq64 = zf.double().numpy(), zq.double().numpy()
    rows = range(zf.shape[0]) if rows is None else rows
    exact = 0
    for r in rows:
        o = drift.step_metrics(zf64[r], zq64[r], alpha, window, eps, rho_c, k_max)
        order = drift.order_desc(zf64[r])
        csum = np.cumsum(drift.softmax(zf64[r])[order])
        mg, mo = int(g["m_t"][r]), o["M"]
        # a length "at the boundary": its prefix mass, or the one before it,
        # within BAND of alpha
        near = lambda m: abs(csum[m - 1] - alpha) < BAND or (m >= 2 and abs(csum[m - 2] - alpha) < BAND)
        if mg == mo:
            exact += 1
        else:
            # only rows in the band may differ, and then both lengths are there
            assert near(mg) and near(mo), f"row {r}: M {mg} vs {mo}"
            o = drift.metrics_given_candidates(zf64[r], zq64[r], order[:mg], window, eps, rho_c,
                                               k_max)
        assert abs(g["c_t"][r] - o["c"]) <= TOL, f"row {r}: c {g['c_t'][r]} vs {o['c']}"
        assert abs(g["d_loc"][r] - o["d_loc"]) <= TOL + 1e-5 * o["d_loc"], f"row {r}: d"
        np.testing.assert_allclose(g["cov"][r], o["cov"], rtol=0, atol=TOL, err_msg=f"row {r}")
        if abs(o["d_loc"] - eps) > BAND and abs(o["c"] - rho_c) > BAND:
            assert bool(g["y_t"][r]) == o["y"], f"row {r}: y"
    assert exact >= require * len(rows), f"M_t equal on {exact} of {len(rows)} rows"
    return g


@pytest.mark.parametrize("V", [33, 1000, 4097, 32000, 128256, 152064])
def test_vocab_sizes(kvq_lib, V):
    zf, zq = synth.paired_logits(V % 89, 4, V)
    _compare(zf, zq, 0.9, 8, min(64, V), 0.02, 0.5)


@pytest.mark.parametrize("alpha", [0.3, 0.9, 0.99, 0.999])
@pytest.mark.parametrize("window,k_max", [(1, 1), (32, 32), (32, 256)])
def test_parameters(kvq_lib, alpha, window, k_max):
    zf, zq = synth.paired_logits(7, 6, 20000, sigma=2.0, noise=0.5)
    _compare(zf, zq, alpha, window, k_max, 0.05, 0.5)


@pytest.mark.parametrize("sigma", [0.002, 0.05, 0.5])
def test_flat_rows_narrow_the_boundary_bin(kvq_lib, sigma):
    # thousands of logits per depth bin: the boundary set is narrowed by
    # histograms of its key range before it is sorted
    zf, zq = synth.paired_logits(3, 3, 50000, sigma=sigma, noise=sigma / 4)
    _compare(zf, zq, 0.6, 16, 128, 0.01, 0.3)


def test_equal_logits_take_lowest_indices(kvq_lib):
    V = 30000
    zf = torch.zeros(3, V)
    zq = torch.zeros(3, V)
    zq[1, 777] = 1.0  # one standout in the low-bit row
    zf[2, ::3] = -0.0
    # 15000.3 of 30000 equal masses: the first 15001 indices
    g = _compare(zf, zq, 0.50001, 4, 16, 0.0, 0.0, require=1.0)
    assert g["m_t"][0] == 15001 and g["m_t"][2] == 15001


def test_integer_logits_with_heavy_ties(kvq_lib):
    gen = synth.generator(5)
    zf = torch.randint(-3, 4, (4, 40000), generator=gen).float()
    zq = zf + torch.randint(-1, 2, (4, 40000), generator=gen).float()
    _compare(zf, zq, 0.8, 32, 256, 0.01, 0.5, require=1.0)


def test_masked_logits(kvq_lib):
    zf, zq = synth.paired_logits(9, 3, 10000)
    zf[:, 5000:] = -float("inf")
    zq[:, ::2] = -float("inf")
    zf[2, :] = -float("inf")
    zf[2, 123] = 0.5
    _compare(zf, zq, 0.95, 8, 32, 0.02, 0.5)


def test_alpha_one_takes_the_reached_prefix(kvq_lib):
    # alpha = 1: where the float64 prefix mass reaches 1 is decided by
    # rounding, so M_t may differ from the oracle's; _compare then checks
    # that both lengths sit within BAND of full mass and compares c_t, d_loc,
    # cov and y_t on every row at the GPU's M_t
    zf, zq = synth.paired_logits(2, 2, 3000, sigma=1.0)
    g = _compare(zf, zq, 1.0, 8, 32, 0.02, 0.5, require=0.0)
    assert (g["m_t"] >= 2900).all()
    zf64 = zf.double().numpy()
    for r in range(2):
        csum = np.cumsum(drift.softmax(zf64[r])[drift.order_desc(zf64[r])])
        assert abs(csum[int(g["m_t"][r]) - 1] - 1.0) < BAND


def test_window_rule(kvq_lib):
    zf, zq = synth.paired_logits(4, 64, 32000, sigma=2.5, noise=0.6)
    g = _run(zf, zq, 0.9, 16, 128, 0.02, 0.5)
    cov = torch.from_numpy(g["cov"]).cuda()
    for rho in (0.3, 0.6, 0.85, 2.0):
        kb, mean = kvq.drift_window(cov, rho)
        torch.cuda.synchronize()
        k_o, mean_o = drift.calibrate_window(g["cov"].astype(np.float64), float(np.float32(rho)))
        np.testing.assert_allclose(mean.cpu().numpy(), mean_o, rtol=1e-6, atol=0)
        if np.all(np.abs(mean_o - rho) > BAND):
            assert int(kb.item()) == k_o


def test_fullsize_sampled_rows(kvq_lib):
    # the bench workload: 256 steps of a 128256-token vocabulary
    zf, zq = synth.paired_logits(11, 256, 128256, sigma=3.0, noise=0.4)
    _compare(zf, zq, 0.9, 32, 256, 0.02, 0.5, rows=[0, 1, 77, 128, 200, 255])


def test_argument_checks(kvq_lib):
    zf, zq = synth.paired_logits(1, 2, 100)
    with pytest.raises(kvq.KvqError):
        kvq.drift_metrics(zf.cuda(), zq.cuda(), 0.0, 1, 8, 0.1, 0.5)
    with pytest.raises(kvq.KvqError):
        kvq.drift_metrics(zf.cuda(), zq.cuda(), 0.9, 9, 8, 0.1, 0.5)
    with pytest.raises(kvq.KvqError):
        kvq.drift_metrics(zf.cuda(), zq.cuda(), 0.9, 1, 101, 0.1, 0.5)
    big = torch.zeros(1, kvq.lib().kvq_drift_max_vocab() + 1, device="cuda")
    with pytest.raises(kvq.KvqError):
        kvq.drift_metrics(big, big, 0.9, 1, 8, 0.1, 0.5)
