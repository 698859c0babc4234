"""Pins of the oracle's DGAP epilogue: a hand-computed row, closed forms,
brute-force top-K, shift invariance (softmax(z + c) = softmax(z), Sec. 3.2),
gate semantics of the sparse merge (Eq. 13) and MLP closed forms."""

from math import log

import numpy as np
import pytest
import scipy.stats
import torch

from oracle import dgap
from paper_2607_16248_gb300 import synth


def _weights(seed=0, K=4, hidden=16):
    return synth.split_weights(synth.dgap_weights(seed, K=K, hidden=hidden))


def test_hand_computed_row():
    # z = [0, ln2, 0, ln3, 0, 0]: e^z = [1, 2, 1, 3, 1, 1], sum 9.
    # p = [1, 2, 1, 3, 1, 1] / 9; window (K = 2) = [3, 1], z_(K) at index 0.
    z = np.array([0.0, log(2), 0.0, log(3), 0.0, 0.0])
    phi, win = dgap.risk_features(z, 2)
    assert win.tolist() == [3, 1, 0]
    expect = [
        4 / 9 * log(9) + 2 / 9 * log(9 / 2) + 1 / 3 * log(3),  # entropy
        5 / 9,                                                  # top-K mass
        1 / 3,                                                  # top-1 probability
        log(3) - log(2),                                        # margin
        log(3) - log(2),                                        # mean gap, K - 1 = 1
        log(3) - log(2),                                        # least adjacent gap
        (log(3) - log(2)) / 2,                                  # population std of 2 values
        -(0.6 * log(0.6) + 0.4 * log(0.4)),                     # window entropy, q = [3, 2]/5
    ]
    assert np.allclose(phi, expect, rtol=0, atol=1e-14)
    xi = dgap.candidate_features(z, win, 2)
    expect_xi = [[0.0, log(1 / 3), 0.0, 0.0, log(3) - log(2)],
                 [log(2) - log(3), log(2 / 9), 1.0, log(3) - log(2), log(2)]]
    assert np.allclose(xi, expect_xi, rtol=0, atol=1e-14)


def test_uniform_row_closed_forms():
    V, K = 1000, 32
    z = np.full(V, 2.5)
    phi, win = dgap.risk_features(z, K)
    assert win.tolist() == list(range(K + 1))
    assert np.allclose(phi, [log(V), K / V, 1 / V, 0, 0, 0, 0, log(K)], rtol=0, atol=1e-12)
    xi = dgap.candidate_features(z, win, K)
    assert np.allclose(xi[:, 0], 0) and np.allclose(xi[:, 1], -log(V))
    assert np.allclose(xi[:, 2], np.arange(K) / (K - 1))
    assert np.allclose(xi[:, 3:], 0)


def test_entropy_matches_scipy():
    rng = np.random.default_rng(0)
    z = rng.standard_normal(5000) * 3
    phi, _ = dgap.risk_features(z, 32)
    assert abs(phi[0] - scipy.stats.entropy(dgap.softmax(z))) < 1e-10


@pytest.mark.parametrize("seed", range(20))
def test_topk_brute_force_with_ties(seed):
    rng = np.random.default_rng(seed)
    V = int(rng.integers(3, 65))
    K = int(rng.integers(1, V))
    z = rng.integers(0, 6, V).astype(np.float64)
    want = sorted(range(V), key=lambda i: (-z[i], i))[:K + 1]
    assert dgap.topk_window(z, K).tolist() == want


def test_topk_special_rows():
    assert dgap.topk_window(np.zeros(100), 32).tolist() == list(range(33))
    z = np.arange(100, dtype=np.float64)
    assert dgap.topk_window(z, 32).tolist() == list(range(99, 66, -1))
    z = np.array([0.0, -0.0, 0.0, -0.0])  # signed zeros compare equal
    assert dgap.topk_window(z, 2).tolist() == [0, 1, 2]


def test_shift_invariance():
    rng = np.random.default_rng(1)
    det, cor = _weights(3, K=8, hidden=32)
    z = rng.standard_normal(3000) * 3
    a = dgap.restore_row(z, 8, -1.0, det, cor)
    b = dgap.restore_row(z + 7.25, 8, -1.0, det, cor)
    assert a["idx"].tolist() == b["idx"].tolist()
    assert np.allclose(a["phi"], b["phi"], rtol=0, atol=1e-9)
    assert abs(a["f"] - b["f"]) < 1e-9 and a["gate"] == b["gate"]
    assert np.allclose(a["delta"], b["delta"], rtol=0, atol=1e-9)
    assert np.allclose(b["val"], z[b["idx"]] + 7.25 + b["delta"], rtol=0, atol=1e-9)


def test_zero_weights():
    det, cor = _weights(4, K=8, hidden=32)
    for d in (det, cor):
        for k in ("w1", "b1", "w2"):
            d[k] = np.zeros_like(d[k])
    z = np.random.default_rng(2).standard_normal(500)
    out = dgap.restore_row(z, 8, -1.0, det, cor)
    assert out["gate"] and np.allclose(out["delta"], cor["b2"])
    assert out["r"] == pytest.approx(1 / (1 + np.exp(-det["b2"][0])), abs=1e-15)


def test_gate_bypass_and_sparse_merge():
    det, cor = _weights(5, K=8, hidden=32)
    z = np.random.default_rng(3).standard_normal(400) * 3
    never = dgap.restore_row(z, 8, 1.0, det, cor)
    assert not never["gate"] and np.array_equal(never["z_tilde"], z)
    always = dgap.restore_row(z, 8, -1.0, det, cor)
    assert always["gate"]
    mask = np.ones(400, bool)
    mask[always["idx"]] = False
    assert np.array_equal(always["z_tilde"][mask], z[mask])  # non-selected unchanged
    assert np.allclose(always["z_tilde"][always["idx"]], z[always["idx"]] + always["delta"])
    r = always["r"]
    assert dgap.restore_row(z, 8, r - 1e-9, det, cor)["gate"]
    assert not dgap.restore_row(z, 8, r, det, cor)["gate"]  # strict: r > tau


def test_mlp_closed_forms():
    # Detector picks +-entropy: f = relu(H) + relu(-H) - 2 = H - 2.
    K, H = 4, 2
    det = dict(w1=np.zeros((H, 8)), b1=np.zeros(H), w2=np.ones((1, H)), b2=np.array([-2.0]))
    det["w1"][0, 0], det["w1"][1, 0] = 1.0, -1.0
    # Corrector: identity hidden layer, output k reads xi[k, 4] = z_(k) - z_(k+1) >= 0.
    nin = 5 * K + 8
    cor = dict(w1=np.eye(nin), b1=np.zeros(nin), w2=np.zeros((K, nin)), b2=np.zeros(K))
    for k in range(K):
        cor["w2"][k, 5 * k + 4] = 1.0
    z = np.random.default_rng(4).standard_normal(300) * 2
    out = dgap.restore_row(z, K, -1.0, det, cor)
    zs = z[dgap.topk_window(z, K)]
    assert out["f"] == pytest.approx(out["phi"][0] - 2.0, abs=1e-14)
    assert np.allclose(out["delta"], zs[:K] - zs[1:], rtol=0, atol=1e-14)
    assert np.allclose(out["val"], 2 * zs[:K] - zs[1:], rtol=0, atol=1e-14)


def test_mlp_orientation_with_permuted_first_layer():
    # A square first layer that is a permutation: hidden unit j reads input
    # perm[j] (W1[j, perm[j]] = 1).  Output k reads the hidden unit that
    # holds xi[k, 4] = z_(k) - z_(k+1) >= 0, so Delta_k equals that gap; a
    # transposed W1 (unit j reading the input whose image is j) picks other
    # inputs and fails.
    K = 4
    nin = 5 * K + 8
    perm = np.random.default_rng(9).permutation(nin)
    inv = np.argsort(perm)
    cor = dict(w1=np.zeros((nin, nin)), b1=np.zeros(nin), w2=np.zeros((K, nin)), b2=np.zeros(K))
    cor["w1"][np.arange(nin), perm] = 1.0
    for k in range(K):
        cor["w2"][k, inv[5 * k + 4]] = 1.0
    det = dict(w1=np.zeros((2, 8)), b1=np.zeros(2), w2=np.zeros((1, 2)), b2=np.array([1.0]))
    z = np.random.default_rng(10).standard_normal(300) * 2
    out = dgap.restore_row(z, K, 0.5, det, cor)  # r = sigmoid(1) > 0.5: gated
    assert out["gate"]
    zs = z[dgap.topk_window(z, K)]
    assert np.allclose(out["delta"], zs[:K] - zs[1:], rtol=0, atol=1e-14)
    # the same weights transposed read other inputs
    cor_t = dict(cor, w1=cor["w1"].T.copy())
    assert not np.allclose(dgap.restore_row(z, K, 0.5, det, cor_t)["delta"], zs[:K] - zs[1:])


def test_next_token_is_argmax_of_merged_row():
    det, cor = _weights(6, K=8, hidden=32)
    rng = np.random.default_rng(5)
    for _ in range(10):
        z = rng.standard_normal(700) * 3
        out = dgap.restore_row(z, 8, -1.0, det, cor)
        zt = out["z_tilde"]
        assert out["next_token"] == int(np.flatnonzero(zt == zt.max())[0])


def test_weights_round_trip_through_npz(tmp_path):
    w = synth.dgap_weights(7, K=8, hidden=32)
    path = tmp_path / "dgap_weights.npz"
    synth.save_weights(path, w)
    back = synth.load_weights(path)
    assert sorted(back) == sorted(w)
    for k in w:
        assert back[k].dtype == w[k].dtype and torch.equal(back[k], w[k])
    z = synth.logits(3, 1, 500)[0].numpy().astype(np.float64)
    a = dgap.restore_row(z, 8, -1.0, *synth.split_weights(w))
    b = dgap.restore_row(z, 8, -1.0, *synth.split_weights(back))
    assert np.array_equal(a["val"], b["val"]) and a["r"] == b["r"]
