"""Pins of the oracle's other per-token signals (Sec. IV-A and Sec. VI): the
probability margin of the softmax over the whole vocabulary, the entropy of
the action-bin distribution, and the action delta between consecutive steps.

  * entropy: equal logits give ln n; the two-level closed form; shift
    invariance; random logits against scipy's entropy of the softmax;
  * vocabulary margin: with vocab == n_bins it is the bin margin bit for bit;
    with zero LM-head rows outside the bins every other token has logit 0
    exactly, so the margin is the softmax top-2 gap of the bin logits plus
    those zeros; duplicated rows make the top two probabilities equal (0);
    margin kind 2 drives the gate;
  * action delta: the L1 distance in bins between consecutive steps' ids,
    0 on the first step and after a reset.
"""
import math

import numpy as np
import pytest

import oracle
import synth


# --------------------------------------------------------------------------
# entropy
# --------------------------------------------------------------------------

@pytest.mark.parametrize("n", [2, 7, 256, 32000])
def test_entropy_of_equal_logits_is_log_n(n):
    assert oracle.entropy(np.full(n, 0.37)) == pytest.approx(math.log(n), rel=1e-13, abs=1e-13)


@pytest.mark.parametrize("delta", [0.0, 0.5, 3.0, 20.0])
def test_entropy_two_level_closed_form(delta):
    n = 256
    lg = np.zeros(n)
    lg[17] = delta
    z = math.exp(delta) + n - 1
    p1, p = math.exp(delta) / z, 1.0 / z
    want = -p1 * math.log(p1) - (n - 1) * p * math.log(p)
    assert oracle.entropy(lg) == pytest.approx(want, rel=1e-12)


def test_entropy_against_scipy_and_shift_invariance():
    scipy_stats = pytest.importorskip("scipy.stats")
    rng = np.random.default_rng(3)
    for _ in range(20):
        lg = rng.normal(0, rng.uniform(0.1, 8.0), 256)
        p = np.exp(lg - lg.max())
        p /= p.sum()
        h = oracle.entropy(lg)
        assert h == pytest.approx(float(scipy_stats.entropy(p)), rel=1e-10, abs=1e-12)
        assert oracle.entropy(lg + 123.25) == pytest.approx(h, rel=1e-12, abs=1e-12)
    one_hot = np.full(256, -1e4)
    one_hot[3] = 0.0
    assert oracle.entropy(one_hot) == 0.0


def test_step_entropy_is_that_of_the_returned_logits():
    d = synth.dims_for("tiny")
    orc = oracle.Oracle(d, synth.make_weights(d, seed=5))
    f = synth.make_episode(d, 1, seed=5)[0]
    o = orc.step(orc.new_cache(1), f, synth.make_prompt(d, seed=5))
    for a in range(d.n_action):
        assert o["entropy"][0, a] == oracle.entropy(o["logits"][0, a])
        assert 0.0 < o["entropy"][0, a] < math.log(d.n_bins)


# --------------------------------------------------------------------------
# margin of the softmax over the whole vocabulary
# --------------------------------------------------------------------------

def _vocab_case(d, seed, rows=None, gain=1.0):
    w = synth.make_weights(d, seed=seed)
    if rows == "zero":
        w["lm_head"][: d.vocab - d.n_bins] = 0
    elif rows == "copy":
        nb = d.n_bins
        for r in range(d.vocab - nb):
            w["lm_head"][r] = w["lm_head"][d.vocab - nb + (r % nb)]
    w["final_norm"] = w["final_norm"] * gain
    orc = oracle.Oracle(d, w)
    frames = synth.make_episode(d, 2, seed=seed)
    if d.vocab > d.n_bins:
        prompt = synth.make_prompt(d, seed=seed)
    else:  # every token is an action bin: BOS then any ids
        prompt = np.random.default_rng(seed).integers(2, d.vocab, (1, d.n_text)).astype(np.int32)
        prompt[:, 0] = 1
    c = orc.new_cache(1)
    return [orc.step(c, frames[t], prompt, want_vocab_margin=True) for t in range(2)]


def test_vocab_margin_equals_bin_margin_when_the_vocabulary_is_the_bins():
    d = synth.dims_for("tiny", vocab=256)
    for o in _vocab_case(d, 6):
        np.testing.assert_array_equal(o["vocab_margin"], o["margins"])


@pytest.mark.parametrize("gain", [1.0, 30.0])
def test_vocab_margin_with_zero_rows_outside_the_bins(gain):
    d = synth.dims_for("tiny")  # vocab 512: 256 tokens whose LM-head rows are zero
    for o in _vocab_case(d, 7, rows="zero", gain=gain):
        for a in range(d.n_action):
            lg = np.concatenate([o["logits"][0, a], np.zeros(d.vocab - d.n_bins)])
            top = np.sort(lg)[::-1]
            want = (math.exp(top[0] - top[0]) - math.exp(top[1] - top[0])) / np.exp(lg - top[0]).sum()
            assert o["vocab_margin"][0, a] == pytest.approx(want, rel=1e-12, abs=1e-15)
            assert o["vocab_margin"][0, a] <= o["margins"][0, a] + 1e-15


def test_vocab_margin_is_zero_when_every_logit_appears_twice():
    d = synth.dims_for("tiny")
    for o in _vocab_case(d, 8, rows="copy"):
        assert np.all(o["vocab_margin"] == 0.0)
        assert np.all(o["margins"] > 0.0)


def test_vocab_margin_drives_the_gate_with_margin_kind_2():
    d = synth.dims_for("tiny")
    orc = oracle.Oracle(d, synth.make_weights(d, seed=9))
    frames = synth.make_episode(d, 3, seed=9)
    prompt = synth.make_prompt(d, seed=9)
    c = orc.new_cache(1)
    o = orc.step(c, frames[0], prompt, margin_kind=2, want_vocab_margin=True)
    assert o["step_margin"][0] == pytest.approx(np.mean(o["vocab_margin"][0]), rel=1e-15)
    m = o["step_margin"][0]
    # the gate compares m_{t-1} of this kind: just above it fires, just below it does not
    o1 = orc.step(c, frames[1], prompt, margin_kind=2, tau_margin=m * (1 + 1e-9), want_vocab_margin=True)
    assert o1["recomputed"][0] == 1
    m1 = o1["step_margin"][0]
    o2 = orc.step(c, frames[2], prompt, margin_kind=2, tau_margin=m1 * (1 - 1e-9), want_vocab_margin=True)
    assert o2["recomputed"][0] == 0


def test_margin_kind_out_of_range_is_rejected():
    d = synth.dims_for("tiny")
    orc = oracle.Oracle(d, synth.make_weights(d, seed=10))
    with pytest.raises(ValueError):
        orc.step(orc.new_cache(1), synth.make_episode(d, 1, seed=10)[0], synth.make_prompt(d, seed=10),
                 margin_kind=3)


# --------------------------------------------------------------------------
# action delta
# --------------------------------------------------------------------------

def test_action_delta_is_the_l1_distance_between_consecutive_steps():
    d = synth.dims_for("tiny")
    # weights seed 12: a model whose actions follow the instruction; a new
    # instruction every step, so that the actions change
    orc = oracle.Oracle(d, synth.make_weights(d, seed=12))
    frames = synth.make_episode(d, 5, seed=12, batch=2)
    prompts = [synth.make_prompt(d, seed=12 + t, batch=2) for t in range(5)]
    c = orc.new_cache(2)
    prev = None
    seen_nonzero = False
    for t in range(5):
        if t == 3:
            c.reset(1)
        o = orc.step(c, frames[t], prompts[t], tau_sim=(95, 100))
        for b in range(2):
            if prev is None or (t == 3 and b == 1):
                assert o["action_delta"][b] == 0
            else:
                assert o["action_delta"][b] == int(np.abs(o["action_ids"][b] - prev[b]).sum())
        prev = o["action_ids"].copy()
        seen_nonzero = seen_nonzero or bool(o["action_delta"].any())
    assert seen_nonzero, "no step changed an action: the case tests nothing"
