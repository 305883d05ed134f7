"""Pins of the oracle's entropy-adaptive Stage 3 (Sec. III-B, Stage 3).

The paper says only that each layer's normalized attention entropy sets its
reuse proportion -- low entropy, more reuse -- with weighted growth
smoothing against abrupt transitions.  No formula is given, so the mapping
below is this library's reading and its parity is unpinned against the
paper; what is pinned is that the oracle computes the reading it states:
  * the schedule: closed forms (entropy 0 -> hi, entropy 1 -> lo, no
    smoothing, full smoothing, the geometric step response) and exact
    rational arithmetic on random inputs;
  * the layer entropy: W_q = 0 makes every text row's softmax uniform over
    its keys, so every normalized entropy is exactly 1; on random models it
    equals an independent numpy restatement (tests/restate.py) to 1e-9;
  * timing: the first step and a step after a reset use the caller's
    schedule, every later step the one the previous step's entropies give;
    a replayed (forced) schedule decides the selection while the reported
    schedule stays the oracle's own; Stage 3 adaptive off leaves everything
    as the caller's schedule gives it.
"""
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth
from tests.restate import Restated

DIMS = {
    "tiny_f32": synth.dims_for("tiny"),
    "tiny_bf16": synth.dims_for("tiny", dtype="bf16"),
    "tiny_oft": synth.dims_for("tiny", n_views=2, proprio_dim=8, n_action=8, parallel=1),
}
S3 = (500, 900, 500)  # lo, hi, weight (per mille)


def _pp(prop, t):
    return None if prop is None else prop[t, 0]


# --------------------------------------------------------------------------
# the schedule
# --------------------------------------------------------------------------

def _exact(ent, lo, hi, w):
    out, r = [], None
    for l, e in enumerate(ent):
        t = Fraction(hi) - Fraction(hi - lo) * Fraction(e)
        r = t if l == 0 else r + Fraction(w, 1000) * (t - r)
        out.append(min(1000, max(0, r.numerator // r.denominator)))
    return out, r


@pytest.mark.parametrize("lo,hi,w", [(500, 900, 500), (0, 1000, 250), (300, 300, 700), (0, 1000, 1000)])
def test_constant_entropy(lo, hi, w):
    L = 9
    np.testing.assert_array_equal(oracle.entropy_schedule(np.zeros(L), lo, hi, w), [hi] * L)
    np.testing.assert_array_equal(oracle.entropy_schedule(np.ones(L), lo, hi, w), [lo] * L)


def test_no_smoothing_and_full_smoothing():
    ent = np.array([0.1, 0.9, 0.5, 0.25, 0.75])
    t = 900 - 400 * ent
    np.testing.assert_array_equal(oracle.entropy_schedule(ent, 500, 900, 1000), np.floor(t))
    np.testing.assert_array_equal(oracle.entropy_schedule(ent, 500, 900, 0), [int(np.floor(t[0]))] * 5)


@pytest.mark.parametrize("w", [125, 500, 875])
def test_step_response(w):
    """Entropy 0 up to layer k, 1 from there: r_l = lo + (hi - lo)(1 - w)^(l-k+1)."""
    L, k, lo, hi = 12, 4, 200, 1000
    ent = np.array([0.0] * k + [1.0] * (L - k))
    got = oracle.entropy_schedule(ent, lo, hi, w)
    a = 1 - Fraction(w, 1000)
    for l in range(L):
        r = Fraction(hi) if l < k else lo + (hi - lo) * a ** (l - k + 1)
        assert got[l] == r.numerator // r.denominator, (l, got[l], float(r))


def test_random_inputs_against_exact_rationals():
    rng = np.random.default_rng(3)
    for _ in range(200):
        L = int(rng.integers(1, 40))
        lo = int(rng.integers(0, 1001))
        hi = int(rng.integers(lo, 1001))
        w = int(rng.integers(0, 1001))
        ent = rng.random(L)
        want, _ = _exact(ent, lo, hi, w)
        got = oracle.entropy_schedule(ent, lo, hi, w)
        # fp64 agrees with exact arithmetic except within rounding of an integer
        for l in range(L):
            if got[l] != want[l]:
                r = _exact(ent[:l + 1], lo, hi, w)[1]
                assert abs(float(r) - round(float(r))) < 1e-9, (l, got[l], want[l])


def test_lower_entropy_reuses_more():
    rng = np.random.default_rng(4)
    ent = rng.random(16)
    base = oracle.entropy_schedule(ent, 400, 950, 600)
    for l in range(16):
        e2 = ent.copy()
        e2[l] = max(0.0, e2[l] - 0.3)
        assert (oracle.entropy_schedule(e2, 400, 950, 600) >= base).all()


# --------------------------------------------------------------------------
# the layer entropy
# --------------------------------------------------------------------------

@pytest.mark.parametrize("name", list(DIMS))
def test_uniform_attention_has_entropy_one(name):
    """W_q = 0 in every layer: each text row's softmax is uniform over its
    keys, so every normalized entropy is ln(n) / ln(n) = 1."""
    d = DIMS[name]
    w = synth.make_weights(d, seed=21)
    for lay in w["layers"]:
        lay["wq"] = lay["wq"] * 0
    orc = oracle.Oracle(d, w)
    frames = synth.make_episode(d, 2, seed=21)
    prompt = synth.make_prompt(d, seed=21)
    prop = synth.make_proprio(d, 2, seed=21)
    c = orc.new_cache(1)
    pm = synth.linear_schedule(d.n_layers)
    o0 = orc.step(c, frames[0], prompt, _pp(prop, 0), tau_sim=(95, 100), permille=pm, s3_adaptive=S3)
    np.testing.assert_allclose(o0["layer_entropy"][0], 1.0, rtol=0, atol=1e-12)
    np.testing.assert_array_equal(o0["schedule"][0], pm)  # nothing measured before the first step
    o1 = orc.step(c, frames[1], prompt, _pp(prop, 1), tau_sim=(95, 100), permille=pm, s3_adaptive=S3)
    np.testing.assert_array_equal(o1["schedule"][0], [S3[0]] * d.n_layers)
    assert o1["recomputed"][0] == 0
    nS = int(o1["static_mask"][0].sum())
    np.testing.assert_array_equal(o1["M"][0], d.pass_len - (S3[0] * nS) // 1000)


@pytest.mark.parametrize("name", list(DIMS))
def test_layer_entropy_matches_the_restatement(name):
    d = DIMS[name]
    w = synth.make_weights(d, seed=22)
    orc = oracle.Oracle(d, w)
    ref = Restated(d, w)
    frames = synth.make_episode(d, 3, seed=22)
    prompt = synth.make_prompt(d, seed=22)
    prop = synth.make_proprio(d, 3, seed=22)
    c = orc.new_cache(1)
    sched = synth.linear_schedule(d.n_layers)
    for t in range(3):
        o = orc.step(c, frames[t], prompt, _pp(prop, t), tau_sim=(95, 100), permille=sched, s3_adaptive=S3)
        r = ref.step(frames[t][0], prompt[0], _pp(prop, t), (95, 100), 0.0, o["schedule"][0])
        np.testing.assert_array_equal(o["M"][0], r["M"])
        np.testing.assert_allclose(o["layer_entropy"][0], r["layer_entropy"], rtol=1e-9, atol=0)
        assert ((o["layer_entropy"][0] > 0) & (o["layer_entropy"][0] <= 1)).all()
        # the next step's schedule is the reading applied to these entropies
        nxt = oracle.entropy_schedule(o["layer_entropy"][0], *S3)
        if t:
            np.testing.assert_array_equal(o["schedule"][0], prev_next)
        prev_next = nxt


def test_timing_reset_forced_and_off():
    d = DIMS["tiny_bf16"]
    w = synth.make_weights(d, seed=23)
    orc = oracle.Oracle(d, w)
    frames = synth.make_episode(d, 4, seed=23)
    prompt = synth.make_prompt(d, seed=23)
    pm = synth.linear_schedule(d.n_layers)
    kw = dict(tau_sim=(95, 100), permille=pm)
    # off: the caller's schedule, no entropy
    c = orc.new_cache(1)
    for t in range(2):
        o = orc.step(c, frames[t], prompt, **kw)
        np.testing.assert_array_equal(o["schedule"][0], pm)
        assert not o["layer_entropy"].any()
    # on: step 1 uses step 0's entropies; a reset forgets them
    c = orc.new_cache(1)
    o0 = orc.step(c, frames[0], prompt, s3_adaptive=S3, **kw)
    o1 = orc.step(c, frames[1], prompt, s3_adaptive=S3, **kw)
    np.testing.assert_array_equal(o1["schedule"][0], oracle.entropy_schedule(o0["layer_entropy"][0], *S3))
    c.reset(0)
    o2 = orc.step(c, frames[2], prompt, s3_adaptive=S3, **kw)
    np.testing.assert_array_equal(o2["schedule"][0], pm)
    # a forced schedule decides the selection; the reported one is still the own
    forced = np.full((1, d.n_layers), 1000, np.uint16)
    o3 = orc.step(c, frames[3], prompt, s3_adaptive=S3, s3_forced=forced, **kw)
    np.testing.assert_array_equal(o3["schedule"][0], oracle.entropy_schedule(o2["layer_entropy"][0], *S3))
    nS = int(o3["static_mask"][0].sum())
    assert o3["recomputed"][0] == 0 and nS > 0
    np.testing.assert_array_equal(o3["M"][0], d.pass_len - nS)


@pytest.mark.parametrize("s3", [(600, 500, 500), (0, 1001, 500), (0, 900, 1001), (-1, 900, 500)])
def test_bad_arguments_are_refused(s3):
    d = DIMS["tiny_f32"]
    orc = oracle.Oracle(d, synth.make_weights(d, seed=24))
    frames = synth.make_episode(d, 1, seed=24)
    with pytest.raises(ValueError):
        orc.step(orc.new_cache(1), frames[0], synth.make_prompt(d, seed=24), s3_adaptive=s3)
