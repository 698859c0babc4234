"""Seeded synthetic inputs for the decode step and the DGAP epilogue.

Shared by the tests (which feed the same tensors to the CUDA path and to the
CPU oracle), ``bench.py`` and the smoke check.  This module draws random
numbers only; it holds none of the method's arithmetic.

Recipe (one decode step of a Llama/Mistral/Qwen-shaped model; no datasets or
trained weights are available, so these stand in for real traces):
* queries, keys, values: fp16 N(0, 1); in the keys, 4 channels per
  (layer, kv-head), drawn without replacement, are multiplied by 10 for every
  token (channel outliers, the reason keys are grouped per channel);
* logits: fp32 N(0, 3^2) (standard deviation 3);
* detector / corrector: PyTorch-Linear-style U(-1/sqrt(fan_in), 1/sqrt(fan_in))
  for every weight and bias.
"""

import torch

HEAD_DIM = 128


def generator(seed, device="cpu"):
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def kv_heads(seed, n_kv_heads, L, device="cpu", outliers=4, outlier_scale=10.0):
    """Keys and values fp16 [n_kv_heads, L, 128] of one sequence / layer."""
    g = generator(seed, device)
    k = torch.randn(n_kv_heads, L, HEAD_DIM, generator=g, device=device)
    v = torch.randn(n_kv_heads, L, HEAD_DIM, generator=g, device=device)
    for h in range(n_kv_heads):
        ch = torch.randperm(HEAD_DIM, generator=g, device=device)[:outliers]
        k[h, :, ch] *= outlier_scale
    return k.half(), v.half()


def queries(seed, batch, n_q_heads, device="cpu"):
    g = generator(seed, device)
    return torch.randn(batch, n_q_heads, HEAD_DIM, generator=g, device=device).half()


def logits(seed, batch, vocab, sigma=3.0, device="cpu"):
    g = generator(seed, device)
    return torch.randn(batch, vocab, generator=g, device=device) * sigma


def paired_logits(seed, rows, vocab, sigma=3.0, noise=0.3, device="cpu"):
    """Synthetic paired traces: FP16-cache logits z_fp (Gaussian, std sigma)
    and low-bit-cache logits z_q = z_fp + Gaussian noise (std noise), fp32
    [rows, vocab] each."""
    g = generator(seed, device)
    z_fp = torch.randn(rows, vocab, generator=g, device=device) * sigma
    z_q = z_fp + torch.randn(rows, vocab, generator=g, device=device) * noise
    return z_fp, z_q


def ragged_lengths(seed, batch, lo=8192, hi=32768):
    """Per-sequence context lengths drawn uniformly from [lo, hi]."""
    g = generator(seed)
    return [int(x) for x in torch.randint(lo, hi + 1, (batch,), generator=g)]


def dgap_weights(seed, K=32, hidden=256):
    """Seeded random-init detector (8 -> hidden -> 1) and corrector
    (5K + 8 -> hidden -> K) weights, fp32 on the CPU, row-major [out][in]."""
    g = generator(seed)

    def u(shape, fan_in):
        b = 1.0 / fan_in ** 0.5
        return (torch.rand(*shape, generator=g, dtype=torch.float64) * 2 - 1).mul(b).float()

    nin = 5 * K + 8
    return {
        "det_w1": u((hidden, 8), 8), "det_b1": u((hidden,), 8),
        "det_w2": u((hidden,), hidden), "det_b2": u((1,), hidden),
        "cor_w1": u((hidden, nin), nin), "cor_b1": u((hidden,), nin),
        "cor_w2": u((K, hidden), hidden), "cor_b2": u((K,), hidden),
    }


def save_weights(path, w):
    """Write a weight dict (detector and corrector tensors) to an .npz file,
    so a run's seeded parameters can be kept and reloaded."""
    import numpy as np
    np.savez(path, **{k: v.cpu().numpy() for k, v in w.items()})


def load_weights(path):
    """The weight dict written by save_weights (fp32 CPU tensors)."""
    import numpy as np
    with np.load(path) as f:
        return {k: torch.from_numpy(f[k].copy()) for k in f.files}


def split_weights(w):
    """(detector, corrector) dicts of float64 numpy arrays, w2 as [out][in]."""
    def a(t):
        return t.detach().cpu().double().numpy()
    det = dict(w1=a(w["det_w1"]), b1=a(w["det_b1"]), w2=a(w["det_w2"]).reshape(1, -1),
               b2=a(w["det_b2"]))
    cor = dict(w1=a(w["cor_w1"]), b1=a(w["cor_b1"]), w2=a(w["cor_w2"]), b2=a(w["cor_b2"]))
    return det, cor


# The decode-step workloads: model attention shapes at the stated contexts.
WORKLOADS = {
    "tiny-k2v2-4k": dict(batch=1, n_q_heads=32, n_kv_heads=8, bits=2, context=4096, layers=1,
                         vocab=32000, seed=1),
    "llama8b-k1v1-32k": dict(batch=1, n_q_heads=32, n_kv_heads=8, bits=1, context=32768,
                             layers=32, vocab=128256, seed=2),
    "llama8b-sweep-128k": dict(batch=1, n_q_heads=32, n_kv_heads=8, bits=(1, 2, 4, 8),
                               context=131072, layers=32, vocab=128256, seed=3),
    "mistral7b-k2v2-ragged": dict(batch=16, n_q_heads=32, n_kv_heads=8, bits=2,
                                  context=(8192, 32768), layers=32, vocab=32768, seed=4,
                                  gated_fraction=0.3),
    "qwen14b-k1v1-64k": dict(batch=8, n_q_heads=40, n_kv_heads=8, bits=1, context=65536,
                             layers=48, vocab=152064, seed=5),
}
