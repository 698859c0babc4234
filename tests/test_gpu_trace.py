"""KVQ_TRACE=1 prints one line per launch (entry point, shapes, grid)."""

import os
import subprocess
import sys
from pathlib import Path

import pytest

pytestmark = pytest.mark.gpu
ROOT = Path(__file__).resolve().parents[1]

SCRIPT = r"""
import torch
from paper_2607_16248_gb300 import kvq, synth
cfg = kvq.CacheConfig(batch=1, n_q_heads=8, n_kv_heads=2, bits_k=1, bits_v=1, max_len=1024)
c = kvq.QuantKVCache(cfg)
k, v = synth.kv_heads(1, 2, 300, device="cuda")
kvq.kvq_pack(c, k[None], v[None])
q = synth.queries(1, 1, 8, device="cuda")
g = synth.generator(2, "cuda")
kn = torch.randn(1, 2, 128, generator=g, device="cuda").half()
kvq.kvq_decode_step(c, kn, kn, q, n_splits=3)
torch.cuda.synchronize()
"""


@pytest.mark.parametrize("value,expect", [("1", True), ("0", False)])
def test_trace_lines(kvq_lib, value, expect):
    env = dict(os.environ, KVQ_TRACE=value, PYTHONPATH=str(ROOT))
    r = subprocess.run([sys.executable, "-c", SCRIPT], env=env, cwd=ROOT, capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stderr.splitlines() if l.startswith("kvq: ")]
    if expect:
        assert any(l.startswith("kvq: kvq_pack ") for l in lines), r.stderr
        step = [l for l in lines if l.startswith("kvq: kvq_decode_step ")]
        assert step and "grid (6) x 512, splits 3" in step[0], lines
    else:
        assert not lines
