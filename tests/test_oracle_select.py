"""Pins of the oracle's Stage 1 (patch similarity) and Stage 3 selection
(Sec. III-B) against exact brute force with Python integers and Fractions."""
import functools
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth

TINY = synth.dims_for("tiny")
TWO_VIEW = synth.dims_for("tiny", n_views=2, proprio_dim=8, n_action=8, parallel=1)


def _pv(d, frame, v):
    p = d.patch
    gw, gh = d.img_w // p, d.img_h // p
    view, r = divmod(v, gw * gh)
    py, px = divmod(r, gw)
    return [int(x) for x in frame[view, py * p:(py + 1) * p, px * p:(px + 1) * p, :].reshape(-1)]


def _cos_gt(a, b, thr: Fraction) -> bool:
    dd = sum(x * y for x, y in zip(a, b))
    na = sum(x * x for x in a)
    nb = sum(y * y for y in b)
    if na == 0 and nb == 0:
        return 1 > thr
    if na == 0 or nb == 0 or dd == 0:
        return 0 > thr
    return Fraction(dd * dd, na * nb) > thr * thr


def _cos2(a, b) -> Fraction:
    dd = sum(x * y for x, y in zip(a, b))
    na = sum(x * x for x in a)
    nb = sum(y * y for y in b)
    if na == 0 and nb == 0:
        return Fraction(1)
    if na == 0 or nb == 0:
        return Fraction(0)
    return Fraction(dd * dd, na * nb)


@pytest.mark.parametrize("d", [TINY, TWO_VIEW])
def test_patch_stats_match_integer_brute_force(d):
    rng = np.random.default_rng(1)
    f = rng.integers(0, 256, size=(d.n_views, d.img_h, d.img_w, 3), dtype=np.uint8)
    g = rng.integers(0, 256, size=(d.n_views, d.img_h, d.img_w, 3), dtype=np.uint8)
    for v in range(d.n_visual):
        a, b = _pv(d, f, v), _pv(d, g, v)
        got = oracle.patch_stats(d, f, g, v)
        assert got == (sum(x * y for x, y in zip(a, b)), sum(x * x for x in a), sum(y * y for y in b))


def test_is_static_closed_forms():
    a = np.array([3, 4] + [0] * 586, dtype=np.int64)
    b = np.array([4, 3] + [0] * 586, dtype=np.int64)
    dd, na, nb = int(a @ b), int(a @ a), int(b @ b)  # cos = 24/25 exactly
    assert not oracle.is_static(dd, na, nb, 24, 25)      # equal is not above
    assert oracle.is_static(dd, na, nb, 23, 25)
    assert not oracle.is_static(dd, na, nb, 96, 100)
    assert oracle.is_static(dd, na, nb, 959, 1000)
    # identical patch: cos = 1; strict '>' means tau = 1 marks nothing static
    assert oracle.is_static(na, na, na, 996, 1000)
    assert not oracle.is_static(na, na, na, 1, 1)
    # b = 2a: cos = 1
    assert oracle.is_static(2 * na, na, 4 * na, 999999, 1000000)
    # both all-zero: cos = 1; exactly one all-zero: cos = 0
    assert oracle.is_static(0, 0, 0, 996, 1000)
    assert not oracle.is_static(0, 0, 0, 1, 1)
    assert not oracle.is_static(0, na, 0, 0, 1)
    assert not oracle.is_static(0, 0, nb, 0, 1)
    # orthogonal: cos = 0 is not above tau = 0; any positive overlap is
    assert not oracle.is_static(0, 25, 25, 0, 1)
    assert oracle.is_static(1, 25, 25, 0, 1)
    # extreme magnitudes: 588 bytes of 255 (products near 2^104)
    big = 588 * 255 * 255
    assert oracle.is_static(big, big, big, 4294967294, 4294967295)
    assert not oracle.is_static(big - 1, big, big, 4294967294, 4294967295)


def test_is_static_random_vs_fraction():
    rng = np.random.default_rng(2)
    for _ in range(3000):
        n = int(rng.integers(1, 40))
        a = [int(x) for x in rng.integers(0, 256, n)]
        # b close to a so that cos lands near typical thresholds
        b = [min(255, max(0, x + int(rng.integers(-3, 4)))) for x in a]
        if rng.random() < 0.1:
            b = [0] * n
        num = int(rng.integers(0, 1001))
        den = 1000
        dd = sum(x * y for x, y in zip(a, b))
        na = sum(x * x for x in a)
        nb = sum(y * y for y in b)
        assert oracle.is_static(dd, na, nb, num, den) == _cos_gt(a, b, Fraction(num, den))


def test_reuse_order_is_a_strict_total_order_matching_fractions():
    rng = np.random.default_rng(3)
    pats = []
    for i in range(60):
        a = [int(x) for x in rng.integers(0, 4, 6)]
        b = [int(x) for x in rng.integers(0, 4, 6)]
        if i % 7 == 0:
            b = list(a)  # exact ties in similarity
        pats.append((a, b))
    keys = []
    for a, b in pats:
        keys.append((sum(x * y for x, y in zip(a, b)), sum(x * x for x in a), sum(y * y for y in b)))
    want = sorted(range(len(pats)), key=lambda i: (-_cos2(*pats[i]), i))

    def cmp(i, j):
        if i == j:
            return 0
        return -1 if oracle.more_similar(keys[i], i, keys[j], j) else 1

    got = sorted(range(len(pats)), key=functools.cmp_to_key(cmp))
    assert got == want
    for i in range(len(pats)):
        for j in range(len(pats)):
            if i != j:
                assert oracle.more_similar(keys[i], i, keys[j], j) != oracle.more_similar(keys[j], j, keys[i], i)


def _brute_select(d, frame, prev, tau, permille):
    thr = Fraction(*tau)
    S, L = d.pass_len, d.n_layers
    mask = [1 if _cos_gt(_pv(d, frame, v), _pv(d, prev, v), thr) else 0 for v in range(d.n_visual)]
    stat = [v for v in range(d.n_visual) if mask[v]]
    order = sorted(stat, key=lambda v: (-_cos2(_pv(d, frame, v), _pv(d, prev, v)), v))
    spos = {1 + v for v in stat}
    idx = [p for p in range(S) if p not in spos] + [1 + v for v in reversed(order)]
    M = [S - (int(permille[l]) * len(stat)) // 1000 for l in range(L)]
    return len(stat), mask, idx, M


@pytest.mark.parametrize("d", [TINY, TWO_VIEW])
def test_select_matches_brute_force(d):
    rng = np.random.default_rng(4)
    eps = synth.make_episode(d, 5, seed=3)
    for t in range(1, 5):
        for tau in [(95, 100), (996, 1000), (0, 1), (1, 1)]:
            for pm in [np.zeros(d.n_layers), np.full(d.n_layers, 1000),
                       rng.integers(0, 1001, d.n_layers)]:
                pm = pm.astype(np.uint16)
                n, mask, idx, M = oracle.select(d, eps[t, 0], eps[t - 1, 0], True, tau, pm, False)
                bn, bmask, bidx, bM = _brute_select(d, eps[t, 0], eps[t - 1, 0], tau, pm)
                assert n == bn
                assert list(mask) == bmask
                assert list(idx) == bidx
                assert list(M) == bM
                # R_l = idx[:M_l] always contains every non-static position
                for l in range(d.n_layers):
                    assert set(range(d.pass_len)) - {1 + v for v in range(d.n_visual) if mask[v]} <= set(idx[:M[l]])


def test_select_full_branch_and_missing_previous_frame():
    d = TINY
    eps = synth.make_episode(d, 2, seed=5)
    pm = synth.full_schedule(d.n_layers)
    n, mask, idx, M = oracle.select(d, eps[1, 0], eps[0, 0], True, (95, 100), pm, True)
    assert list(idx) == list(range(d.pass_len)) and list(M) == [d.pass_len] * d.n_layers
    assert n == int(mask.sum()) > 0
    n, mask, idx, M = oracle.select(d, eps[1, 0], eps[0, 0], False, (95, 100), pm, True)
    assert n == 0 and mask.sum() == 0


def test_select_identical_frames_everything_static():
    d = TINY
    f = synth.make_episode(d, 1, seed=6)[0, 0]
    n, mask, idx, M = oracle.select(d, f, f, True, (996, 1000), synth.full_schedule(d.n_layers), False)
    assert n == d.n_visual and mask.all()
    assert list(M) == [d.pass_len - d.n_visual] * d.n_layers
    assert sorted(idx[:d.pass_len - d.n_visual]) == [0] + list(range(d.n_visual + 1, d.pass_len))


def test_select_rejects_permille_above_1000():
    d = TINY
    f = synth.make_episode(d, 1, seed=6)[0, 0]
    pm = synth.full_schedule(d.n_layers)
    pm[0] = 1001
    with pytest.raises(ValueError):
        oracle.select(d, f, f, True, (996, 1000), pm, False)
