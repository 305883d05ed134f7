"""The benchmark's algorithmic work model against the hand-counted figures of
the 7B shape: 202,375,168 parameters per layer (4 hidden^2 + 3 ffn hidden),
2 FLOPs per multiply-add, bf16 weights read once."""
import sys
import os

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import synth  # noqa: E402

PER_LAYER = 4 * 4096 * 4096 + 3 * 11008 * 4096


def test_parameters_per_layer():
    assert PER_LAYER == 202_375_168


@pytest.mark.parametrize("M", [283, 200, 30, 1])
def test_layer_work_counts(M):
    d = synth.dims_for("layer7b")
    pos = np.sort(np.random.default_rng(M).choice(d.pass_len, M, replace=False))
    f, b = bench.layer_work(d, pos)
    attn = 4 * 4096 * float(np.sum(pos + 1))
    assert f == pytest.approx(2 * M * PER_LAYER + attn, rel=1e-12)
    kv = 2 * d.cache_len * 4096 * 2
    assert b == pytest.approx(PER_LAYER * 2 + kv + M * 2 * 4096 * 2 + 2 * M * 4096 * 4, rel=1e-12)
    # every row uses each bf16 weight once (2 FLOPs per 2 bytes): about M FLOPs per byte,
    # so the whole sweep sits at or below the ~280 FLOP/B ridge of the measured peaks
    if M >= 30:
        assert abs(f / b - M) / M < 0.05
