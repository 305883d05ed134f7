"""Pins of the oracle's Eq. (1) ingredients (top-1/top-2 softmax margin over
the action bins), its bf16 rounding and its RoPE table."""
import math

import numpy as np
import pytest

import oracle
import synth
from tests.restate import _bf16_fast, bf16_round


def test_equal_logits_give_zero_margin_and_lowest_bin():
    a, pm, gap = oracle.margin(np.full(256, 0.37))
    assert a == 0 and pm == 0.0 and gap == 0.0


@pytest.mark.parametrize("delta", [1e-6, 0.01, 0.5, 3.0, 20.0])
@pytest.mark.parametrize("where", [0, 17, 255])
def test_two_level_logits_closed_form(delta, where):
    lg = np.zeros(256)
    lg[where] = delta
    a, pm, gap = oracle.margin(lg)
    want = math.expm1(delta) / (math.exp(delta) + 255.0)
    assert a == where
    assert pm == pytest.approx(want, rel=1e-12, abs=1e-300)
    assert gap == pytest.approx(delta, rel=1e-15)


def test_tie_between_top_two_gives_zero_margin_and_lower_index():
    lg = np.linspace(-1, 1, 256)
    lg[200] = lg[100] = 5.0
    a, pm, gap = oracle.margin(lg)
    assert a == 100 and pm == 0.0 and gap == 0.0


def test_random_logits_against_softmax_definition():
    rng = np.random.default_rng(0)
    for _ in range(200):
        lg = rng.normal(0, rng.uniform(0.1, 5), 256)
        a, pm, gap = oracle.margin(lg)
        p = np.exp(lg - lg.max())
        p /= p.sum()
        srt = np.sort(p)[::-1]
        assert a == int(np.argmax(lg))
        assert pm == pytest.approx(srt[0] - srt[1], rel=1e-9, abs=1e-15)
        sl = np.sort(lg)[::-1]
        assert gap == pytest.approx(sl[0] - sl[1], rel=1e-12)


def test_round_bf16_matches_exact_nearest_even():
    rng = np.random.default_rng(1)
    vals = list(rng.normal(0, 1, 400)) + list(rng.normal(0, 1e-30, 50)) + list(rng.normal(0, 1e30, 50))
    # exact midpoints between neighbouring bf16 values (ties -> even)
    for m in range(128, 256, 7):
        for e in (-3, 0, 5):
            vals.append((m + 0.5) * 2.0 ** (e - 7))
            vals.append(-(m + 0.5) * 2.0 ** (e - 7))
    vals += [0.0, 1.0, -2.0, 3.0e38, 1e-40]
    vals = np.array(vals)
    want = bf16_round(vals)
    got = np.array([oracle.round_bf16(v) for v in vals])
    np.testing.assert_array_equal(got, want)
    np.testing.assert_array_equal(_bf16_fast(vals), want)


def test_rope_table_closed_form_and_rotation():
    d = synth.dims_for("tiny")
    cs, sn = oracle.rope_table(d, 50)
    half = d.head_dim // 2
    for p in (0, 1, 7, 49):
        for i in (0, 1, half - 1):
            ang = p * d.rope_theta ** (-2.0 * i / d.head_dim)
            assert cs[p, i] == np.float32(math.cos(ang))
            assert sn[p, i] == np.float32(math.sin(ang))
    assert np.all(cs[0] == 1.0) and np.all(sn[0] == 0.0)
    # each (cos, sin) pair is a rotation: cos^2 + sin^2 = 1 to fp32 accuracy
    np.testing.assert_allclose(cs.astype(np.float64) ** 2 + sn.astype(np.float64) ** 2, 1.0, atol=1e-6)
