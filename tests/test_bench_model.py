"""The benchmark's step work model (the roofline denominators it reports)
against hand counts for the OpenVLA-7B shape: 6,476,005,376 backbone
parameters (12.95 GB of bf16 weights per pass), seven passes per step (the
prefix pass and six single-token decode passes), 2 FLOPs per multiply-add."""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import synth  # noqa: E402

D = synth.dims_for("openvla7b")
PER_LAYER = 4 * 4096 * 4096 + 3 * 11008 * 4096
W_PASS = 32 * PER_LAYER * 2  # bytes of bf16 backbone weights read by one pass


def _full():
    S = D.pass_len
    return [S] * D.n_layers, np.arange(S)


def test_backbone_size():
    assert 32 * PER_LAYER == 6_476_005_376
    assert W_PASS == pytest.approx(12.95e9, rel=1e-3)


def test_full_step_counts():
    M, idx = _full()
    passes = bench.step_work(D, M, idx)
    assert len(passes) == D.n_action  # prefix + 6 decode passes
    # every pass reads the backbone once (plus the head rows; the prefix pass also the patch projection)
    for f, b, w in passes:
        assert W_PASS <= w < W_PASS * 1.01
    f0 = passes[0][0]
    gemm = D.pass_len * 2 * 32 * PER_LAYER
    assert gemm <= f0 < gemm * 1.05  # attention, patch embedding and head are a few per cent
    F, B, _ = bench.batch_work(D, [M], [idx])
    assert F == pytest.approx(sum(p[0] for p in passes))
    assert B == pytest.approx(sum(p[1] + p[2] for p in passes))
    # the step is HBM-bound at the measured peaks: about 13.6 ms of 91-92 GB
    t = max(F / 1891.6e12, B / 6754.1e9)
    assert B == pytest.approx(92.0e9, rel=0.01)
    assert t == pytest.approx(13.6e-3, rel=0.01)


def test_cached_rows_cut_only_the_prefix_flops():
    S = D.pass_len
    M_full, idx = _full()
    M_cached = [S - (int(p) * 230) // 1000 for p in synth.linear_schedule(D.n_layers)]
    full = bench.step_work(D, M_full, idx)
    cached = bench.step_work(D, M_cached, idx)
    assert cached[0][0] < full[0][0]
    # decode passes and weight bytes do not depend on the reuse
    for a, b in zip(full[1:], cached[1:]):
        assert a == b
    assert cached[0][2] == full[0][2]


class _FakeSmi:
    def __init__(self, text):
        self.text = text

    def terminate(self):
        pass

    def communicate(self, timeout=None):
        return self.text, ""


def test_clock_samples_are_parsed():
    """The clocks line of the bench: median SM clock under load, the maximum,
    and every throttle reason seen Active in any sample."""
    rows = ["0, 2070, 2070, 900.5, 0x0, Not Active, Not Active, Not Active, Not Active",
            "0, 1980, 2070, 1390.0, 0x4, Not Active, Not Active, Not Active, Active",
            "0, 2070, 2070, 1100.0, 0x0, Not Active, Not Active, Not Active, Not Active",
            "garbage line",
            "0, [N/A], 2070, 0, 0x0, Not Active, Not Active, Not Active, Not Active"]
    c = bench.Clocks.__new__(bench.Clocks)
    c.p = _FakeSmi("\n".join(rows))
    got = c.stop()
    assert got["sm_mhz"] == 2070.0 and got["sm_max_mhz"] == 2070.0 and got["samples"] == 3
    assert got["reasons"] == ["sw_power_cap"]
    c.p = None
    assert c.stop()["reasons"] == ["nvidia-smi unavailable"]


def test_full_step_matches_the_papers_table_one():
    """Table I counts one operation per multiply-add: 1.83-1.89 TFLOPs per full
    OpenVLA step (average 1.87).  The benchmark counts 2 FLOPs per
    multiply-add over the prefix pass and the six decode rows: half of it
    lands inside the table's range."""
    M, idx = _full()
    F, _, _ = bench.batch_work(D, [M], [idx])
    assert 1.83e12 <= F / 2 <= 1.89e12
    assert F / 2 == pytest.approx(1.87e12, rel=0.01)


def test_mean_flops_follow_the_mixture_law():
    """Over an episode whose gate fires on a fraction f of the steps, the mean
    counted work is f * F_full + (1 - f) * F_cached exactly; the paper's own
    Long-suite figures obey the same law (0.24 * 1.88 + 0.76 * 1.43 = 1.54)."""
    S = D.pass_len
    M_full, idx = _full()
    M_cached = [S - (int(p) * 230) // 1000 for p in synth.linear_schedule(D.n_layers)]
    F_full = bench.batch_work(D, [M_full], [idx])[0]
    F_cached = bench.batch_work(D, [M_cached], [idx])[0]
    fired = [1, 0, 0, 0, 1, 0, 0, 0, 0, 0, 0, 0, 1, 0, 0, 0, 0, 0, 0, 0, 1, 0, 0, 0, 0]
    total = sum(bench.batch_work(D, [M_full if b else M_cached], [idx])[0] for b in fired)
    f = sum(fired) / len(fired)
    assert total / len(fired) == pytest.approx(f * F_full + (1 - f) * F_cached, rel=1e-12)
    assert 0.24 * 1.88 + 0.76 * 1.43 == pytest.approx(1.54, abs=0.005)
