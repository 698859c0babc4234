"""dgap_restore (CUDA, through the C ABI) against the float64 oracle.

Bit-exact: top-K indices, untouched logits, the gate (outside a 1e-4 band of
|f - logit(tau)|).  Within tolerance: corrected logits 1e-4 absolute, risk
1e-5, features.  The greedy token is compared where no near-tie makes it
depend on rounding."""

import numpy as np
import pytest
import torch

import _util
from oracle import dgap as odgap
from paper_2607_16248_gb300 import kvq, synth

pytestmark = pytest.mark.gpu


def _compare(z_in, out, z_after, K, tau, det, cor, require_gate=None):
    B, V = z_in.shape
    idx = out["topk_idx"].cpu().numpy()
    val = out["topk_val"].cpu().numpy()
    risk = out["risk"].cpu().numpy()
    gate = out["gate"].cpu().numpy()
    feats = out["features"].cpu().numpy()
    nxt = out["next_token"].cpu().numpy()
    lt = kvq.logit(tau)
    checked_gate = 0
    for b in range(B):
        ref = odgap.restore_row(z_in[b].astype(np.float64), K, tau, det, cor)
        assert idx[b].tolist() == ref["idx"].tolist(), f"row {b} top-K"
        assert abs(risk[b] - ref["r"]) <= _util.RISK_TOL
        np.testing.assert_allclose(feats[b], ref["phi"], rtol=2e-5, atol=2e-5)
        if abs(ref["f"] - lt) > _util.GATE_BAND or not np.isfinite(lt):
            assert bool(gate[b]) == ref["gate"], f"row {b} gate"
            checked_gate += 1
        if gate[b]:
            assert np.abs(val[b] - ref["val"]).max() <= _util.LOGIT_TOL
        else:
            assert np.array_equal(val[b], z_in[b][idx[b]])
        # every logit outside the gated window is bit-identical
        mask = np.ones(V, bool)
        if gate[b]:
            mask[idx[b]] = False
            assert np.abs(z_after[b][idx[b]] - ref["val"]).max() <= _util.LOGIT_TOL
        assert np.array_equal(z_after[b][mask].view(np.uint32), z_in[b][mask].view(np.uint32))
        # greedy token: the decision in float32 on the oracle's merged values
        zt = z_after[b].astype(np.float32)
        top = np.sort(np.concatenate([zt[idx[b]], [z_in[b][ref["idx_K"]]]]))[::-1]
        if top.size < 2 or top[0] - top[1] > 2 * _util.LOGIT_TOL:
            assert nxt[b] == ref["next_token"]
    if require_gate is not None:
        assert checked_gate >= require_gate


def _run(B, V, K, tau, seed, hidden=256, logits=None):
    w = synth.dgap_weights(seed, K=K, hidden=hidden)
    det, cor = synth.split_weights(w)
    m = kvq.DGAP(w, K=K, tau=tau)
    z = synth.logits(seed, B, V) if logits is None else logits
    zin = z.numpy().copy()
    zd = z.cuda()
    out = m.restore(zd)
    torch.cuda.synchronize()
    return zin, out, zd.cpu().numpy(), det, cor


@pytest.mark.parametrize("V", [33, 1000, 4096, 4097, 32000, 128256, 152064])
@pytest.mark.parametrize("tau", [-1.0, 1.0])
def test_vocab_sizes_forced_gate(kvq_lib, V, tau):
    K = 32
    zin, out, zout, det, cor = _run(3, V, K, tau, seed=V % 97)
    assert out["gate"].cpu().numpy().tolist() == [int(tau < 0)] * 3
    _compare(zin, out, zout, K, tau, det, cor)


@pytest.mark.parametrize("K", [2, 8, 33, 64])
def test_window_sizes(kvq_lib, K):
    zin, out, zout, det, cor = _run(4, 20000, K, -1.0, seed=K, hidden=64)
    _compare(zin, out, zout, K, -1.0, det, cor)


def test_paper_threshold_mixed_rows(kvq_lib):
    # tau = 0.60 (Sec. 5.5): the seeded rows must all lie outside the band
    # |f - logit(tau)| <= GATE_BAND, so the gate is compared on every row
    zin, out, zout, det, cor = _run(16, 32768, 32, 0.60, seed=4)
    _compare(zin, out, zout, 32, 0.60, det, cor, require_gate=16)


@pytest.mark.parametrize("offset", [-4e-4, -2e-4, 2e-4, 4e-4])
def test_gate_decided_just_outside_the_band(kvq_lib, offset):
    # tau placed so that one row's detector output f sits |offset| (2 to 4
    # band widths) from logit(tau): that row's gate must still match the
    # oracle exactly, on both sides of the threshold (Eq. 13: r > tau)
    B, V, K = 4, 32768, 32
    w = synth.dgap_weights(7, K=K)
    det, cor = synth.split_weights(w)
    z = synth.logits(71, B, V)
    f = [odgap.restore_row(r, K, 2.0, det, cor)["f"] for r in z.numpy().astype(np.float64)]
    lt = f[1] - offset  # row 1 is gated exactly when offset > 0
    tau = float(1.0 / (1.0 + np.exp(-lt)))
    assert abs(kvq.logit(tau) - lt) < 1e-9
    assert all(abs(x - kvq.logit(tau)) > _util.GATE_BAND for x in f)
    zin, out, zout, det, cor = _run(B, V, K, tau, seed=7, logits=z)
    assert bool(out["gate"][1].item()) == (offset > 0)
    _compare(zin, out, zout, K, tau, det, cor, require_gate=B)


def test_quantile_threshold_gates_about_thirty_percent(kvq_lib):
    B, V, K = 64, 32768, 32
    w = synth.dgap_weights(4, K=K)
    det, cor = synth.split_weights(w)
    z = synth.logits(41, B, V)
    f = np.array([odgap.restore_row(r, K, 2.0, det, cor)["f"] for r in z.numpy().astype(np.float64)])
    fs = np.sort(f)
    lo = int(0.62 * B)
    gaps = fs[lo + 1:int(0.78 * B)] - fs[lo:int(0.78 * B) - 1]
    i = lo + int(np.argmax(gaps))
    tau = float(1 / (1 + np.exp(-(fs[i] + fs[i + 1]) / 2)))
    zin, out, zout, det, cor = _run(B, V, K, tau, seed=4, logits=z)
    g = out["gate"].cpu().numpy()
    assert 0.2 <= g.mean() <= 0.4
    _compare(zin, out, zout, K, tau, det, cor, require_gate=B)


def test_ties_and_signed_zeros(kvq_lib):
    B, V, K = 4, 5000, 32
    g = synth.generator(9)
    z = torch.randint(0, 4, (B, V), generator=g).float()
    z[1] = 0.0
    z[2, ::2] = -0.0
    z[3] = torch.arange(V, dtype=torch.float32).flip(0) * 0 - 1.5
    zin, out, zout, det, cor = _run(B, V, K, -1.0, seed=9, logits=z)
    idx = out["topk_idx"].cpu().numpy()
    assert idx[1].tolist() == list(range(K))
    assert idx[3].tolist() == list(range(K))
    _compare(zin, out, zout, K, -1.0, det, cor)


def test_ties_across_chunk_lists(kvq_lib):
    # 32 chunk lists of a 128256-token row whose leaders tie: every list all
    # one key (more survivors than the exact ranking holds: the radix
    # fallback), a few lists tied at the bound, and keys rounded to a coarse
    # grid
    B, V, K = 3, 128256, 32
    g = synth.generator(19)
    z = torch.empty(B, V)
    z[0] = torch.randint(0, 40, (V,), generator=g).float()
    z[1] = torch.randint(0, 6000, (V,), generator=g).float() / 8.0
    z[2] = torch.round(torch.randn(V, generator=g) * 12.0) / 4.0
    zin, out, zout, det, cor = _run(B, V, K, -1.0, seed=19, logits=z)
    idx = out["topk_idx"].cpu().numpy()
    assert idx[0].tolist() == np.flatnonzero(z[0].numpy() == 39.0)[:K].tolist()
    _compare(zin, out, zout, K, -1.0, det, cor)


def test_shift_invariance_on_gpu(kvq_lib):
    B, V, K = 4, 10000, 32
    z = synth.logits(12, B, V)
    a = _run(B, V, K, 0.6, seed=12, logits=z.clone())
    b = _run(B, V, K, 0.6, seed=12, logits=z + 8.0)
    assert np.array_equal(a[1]["topk_idx"].cpu().numpy(), b[1]["topk_idx"].cpu().numpy())
    np.testing.assert_allclose(a[1]["risk"].cpu().numpy(), b[1]["risk"].cpu().numpy(),
                               atol=1e-5)
    np.testing.assert_allclose(a[1]["features"].cpu().numpy(),
                               b[1]["features"].cpu().numpy(), atol=1e-4)


def test_repeated_calls_reuse_workspace(kvq_lib):
    B, V, K = 2, 50000, 32
    w = synth.dgap_weights(3, K=K)
    det, cor = synth.split_weights(w)
    m = kvq.DGAP(w, K=K, tau=-1.0)
    ws = m.workspace(B, V)
    for seed in range(5):
        z = synth.logits(100 + seed, B, V)
        zin = z.numpy().copy()
        zd = z.cuda()
        out = m.restore(zd, workspace=ws)
        torch.cuda.synchronize()
        _compare(zin, out, zd.cpu().numpy(), K, -1.0, det, cor)
