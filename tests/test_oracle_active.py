"""Sequences that sit a step out (a running batch that episodes join and
leave): the oracle steps only the active sequences of a cache.

  * a step sat out changes nothing of that sequence: its cache (K, V, layer
    inputs), gate state and previous frame are as before, so its next step
    equals the step it would have run without the pause, bit for bit;
  * the other sequences of the batch step exactly as they would alone;
  * the outputs of a sequence that sat out are zero.
"""
import numpy as np
import pytest

import oracle
import synth

DIMS = {"tiny_f32": synth.dims_for("tiny"), "tiny_oft": synth.dims_for("tiny", n_views=2, proprio_dim=8,
                                                                       n_action=8, parallel=1)}
KEYS = ("action_ids", "margins", "logit_gap", "logits", "recomputed", "gate_auto", "step_margin", "static_mask",
        "idx", "M", "entropy", "action_delta")


def _pp(prop, t):
    return None if prop is None else prop[t]


@pytest.mark.parametrize("name", list(DIMS))
def test_sitting_out_is_invisible_to_the_sequence(name):
    d = DIMS[name]
    orc = oracle.Oracle(d, synth.make_weights(d, seed=91))
    frames = synth.make_episode(d, 3, seed=91, batch=2)
    prompt = synth.make_prompt(d, seed=91, batch=2)
    prop = synth.make_proprio(d, 3, seed=91, batch=2)
    kw = dict(tau_sim=(95, 100), tau_margin=0.0, permille=synth.linear_schedule(d.n_layers))
    paused, plain = orc.new_cache(2), orc.new_cache(2)
    orc.step(paused, frames[0], prompt, _pp(prop, 0), **kw)
    orc.step(plain, frames[0], prompt, _pp(prop, 0), **kw)
    before = {kind: [paused.read(1, kind, l) for l in range(d.n_layers)] for kind in ("K", "V", "H")}
    state = paused.state(1)
    # step 1: sequence 1 sits out in `paused`; both sequences step in `plain`
    o1 = orc.step(paused, frames[1], prompt, _pp(prop, 1), active=np.array([1, 0], np.uint8), **kw)
    for k in KEYS:
        assert not np.any(o1[k][1]), k
    for kind in ("K", "V", "H"):
        for l in range(d.n_layers):
            np.testing.assert_array_equal(paused.read(1, kind, l), before[kind][l])
    assert paused.state(1) == state
    # sequence 0 stepped as it did in `plain` (sequences are independent)
    o1p = orc.step(plain, frames[1], prompt, _pp(prop, 1), **kw)
    for k in KEYS:
        np.testing.assert_array_equal(o1[k][0], o1p[k][0], err_msg=k)
    # sequence 1's next step, from frame 2, equals a cache that never saw frame 1 for it
    ref = orc.new_cache(1)
    orc.step(ref, frames[0][1:], prompt[1:], None if prop is None else prop[0][1:], **kw)
    o2 = orc.step(paused, frames[2], prompt, _pp(prop, 2), **kw)
    o2r = orc.step(ref, frames[2][1:], prompt[1:], None if prop is None else prop[2][1:], **kw)
    for k in KEYS:
        np.testing.assert_array_equal(o2[k][1], o2r[k][0], err_msg=k)


def test_a_new_episode_joins_through_reset_and_activation():
    """A slot that sat out and is reset runs its next step as a fresh episode."""
    d = DIMS["tiny_f32"]
    orc = oracle.Oracle(d, synth.make_weights(d, seed=92))
    frames = synth.make_episode(d, 3, seed=92, batch=2)
    prompt = synth.make_prompt(d, seed=92, batch=2)
    c = orc.new_cache(2)
    orc.step(c, frames[0], prompt, tau_sim=(95, 100))
    orc.step(c, frames[1], prompt, tau_sim=(95, 100), active=np.array([1, 0], np.uint8))
    c.reset(1)
    o = orc.step(c, frames[2], prompt, tau_sim=(95, 100))
    fresh = orc.new_cache(1)
    of = orc.step(fresh, frames[2][1:], prompt[1:], tau_sim=(95, 100))
    assert o["recomputed"][1] == 1
    for k in KEYS:
        np.testing.assert_array_equal(o[k][1], of[k][0], err_msg=k)
