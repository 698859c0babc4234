"""The bench's algorithmic bytes (the numerator of every roofline fraction):
per (sequence, kv-head) Lq packed tokens at 16(b_k + b_v) + 32 bytes and the
fp16 window at 512 bytes per token, plus q in (fp16) and out (fp16) per
query head (fp16 both), worked out by hand for the small and Llama workloads."""

import sys
from pathlib import Path

sys.path.insert(0, str(Path(__file__).resolve().parents[1]))

import bench  # noqa: E402


def test_tiny_k2v2_4096():
    # L = 4096: Lq = 3968 packed tokens at 96 B, 128 window tokens at 512 B,
    # 8 kv-heads; 32 query heads x 128 x (2 + 2) B
    assert bench.attn_bytes(4096, 8, 32, 2, 2) == 8 * (3968 * 96 + 128 * 512) + 32 * 128 * 4
    assert bench.attn_bytes(4096, 8, 32, 2, 2) == 3588096


def test_llama_k1v1_32768():
    # 32640 packed tokens at 64 B: the ~17.26 MB per layer of the Llama line
    assert bench.attn_bytes(32768, 8, 32, 1, 1) == 17252352


def test_window_only_and_packing_edges():
    # below R + 32 tokens nothing is packed; at 160 one group is
    assert bench.attn_bytes(159, 1, 4, 1, 1) == 159 * 512 + 4 * 128 * 4
    assert bench.attn_bytes(160, 1, 4, 1, 1) == 32 * 64 + 128 * 512 + 4 * 128 * 4
    assert bench.attn_bytes(0, 2, 8, 4, 4) == 8 * 128 * 4
    # K8V8 packs 16 x 16 + 32 = 288 B per token
    assert bench.attn_bytes(131072, 8, 32, 8, 8) == 8 * (130944 * 288 + 128 * 512) + 32 * 128 * 4


def test_drift_step_bytes():
    w = dict(rows=256, vocab=128256, k_max=256)
    metrics, window = bench.drift_bytes(w)
    assert metrics == 2 * 256 * 128256 * 4 + 256 * 13 + 256 * 256 * 4
    assert window == 256 * 256 * 4 + 256 * 4 + 4

