"""Invariants the method fixes, checked bit for bit in the oracle.

I1  reuse-nothing (every per-mille 0) equals the full forward.
I2  identical frames after a full step on that frame, with any reuse
    schedule, equal the full forward (reused K/V and cached layer inputs are
    exactly what a full pass would recompute).
I3  a gated step (margin below theta_m) equals reset + step: invalidation
    runs "as if no cache existed" (Algorithm 1).
I4  theta_m = 0 never fires (margins are >= 0 and the test is strict);
    theta_m = +inf fires on every step (full inference every step).
Lag the gate of step t reads the margin of step t-1 (one-step reactive lag).
"""
import numpy as np
import pytest

import oracle
import synth

DIMS = {
    "tiny_f32": synth.dims_for("tiny"),
    "tiny_bf16": synth.dims_for("tiny", dtype="bf16"),
    "tiny_oft": synth.dims_for("tiny", n_views=2, proprio_dim=8, n_action=8, parallel=1),
}
KEYS = ("action_ids", "margins", "logit_gap", "logits", "step_margin")


def _setup(name, seed=21):
    d = DIMS[name]
    w = synth.make_weights(d, seed=seed)
    frames = synth.make_episode(d, 3, seed=seed)
    prompt = synth.make_prompt(d, seed=seed)
    prop = synth.make_proprio(d, 3, seed=seed)
    return d, oracle.Oracle(d, w), frames, prompt, prop


def _pp(prop, t):
    return None if prop is None else prop[t, 0]


def _same_outputs(a, b):
    for k in KEYS:
        np.testing.assert_array_equal(a[k], b[k], err_msg=k)


def _same_cache(d, ca, cb, kinds=("K", "V", "H")):
    for l in range(d.n_layers):
        for kind in kinds:
            np.testing.assert_array_equal(ca.read(0, kind, l), cb.read(0, kind, l), err_msg=f"{kind}{l}")


@pytest.mark.parametrize("name", list(DIMS))
def test_I1_reuse_nothing_equals_full(name):
    d, orc, frames, prompt, prop = _setup(name)
    zero = np.zeros(d.n_layers, np.uint16)
    ca, cb = orc.new_cache(1), orc.new_cache(1)
    for c in (ca, cb):
        orc.step(c, frames[0], prompt, _pp(prop, 0), tau_sim=(95, 100), tau_margin=0.0, permille=zero)
    a = orc.step(ca, frames[1], prompt, _pp(prop, 1), tau_sim=(95, 100), tau_margin=0.0, permille=zero,
                 gate_override=np.array([0], np.int8))
    b = orc.step(cb, frames[1], prompt, _pp(prop, 1), tau_sim=(95, 100), tau_margin=0.0, permille=zero,
                 gate_override=np.array([1], np.int8))
    assert a["recomputed"][0] == 0 and b["recomputed"][0] == 1
    assert a["static_mask"].sum() > 0  # the cached branch really ran with a non-identity order
    assert list(a["idx"][0]) != list(range(d.pass_len))
    _same_outputs(a, b)
    _same_cache(d, ca, cb)


@pytest.mark.parametrize("name", list(DIMS))
@pytest.mark.parametrize("sched", ["all", "linear"])
def test_I2_identical_frames_with_reuse_equal_full(name, sched):
    d, orc, frames, prompt, prop = _setup(name)
    pm = synth.full_schedule(d.n_layers) if sched == "all" else synth.linear_schedule(d.n_layers)
    ca, cb = orc.new_cache(1), orc.new_cache(1)
    for c in (ca, cb):
        orc.step(c, frames[0], prompt, _pp(prop, 0), tau_sim=(996, 1000), tau_margin=0.0, permille=pm)
    a = orc.step(ca, frames[0], prompt, _pp(prop, 0), tau_sim=(996, 1000), tau_margin=0.0, permille=pm,
                 gate_override=np.array([0], np.int8))
    b = orc.step(cb, frames[0], prompt, _pp(prop, 0), tau_sim=(996, 1000), tau_margin=0.0, permille=pm,
                 gate_override=np.array([1], np.int8))
    assert a["recomputed"][0] == 0 and a["static_mask"].all()
    assert a["M"][0].min() < d.pass_len
    _same_outputs(a, b)
    _same_cache(d, ca, cb, kinds=("K", "V"))


@pytest.mark.parametrize("name", list(DIMS))
def test_I3_gated_step_equals_reset_then_step(name):
    d, orc, frames, prompt, prop = _setup(name)
    pm = synth.linear_schedule(d.n_layers)
    ca, cb = orc.new_cache(1), orc.new_cache(1)
    for c in (ca, cb):
        orc.step(c, frames[0], prompt, _pp(prop, 0), tau_sim=(95, 100), tau_margin=0.0, permille=pm)
        orc.step(c, frames[1], prompt, _pp(prop, 1), tau_sim=(95, 100), tau_margin=0.0, permille=pm)
    a = orc.step(ca, frames[2], prompt, _pp(prop, 2), tau_sim=(95, 100), tau_margin=float("inf"), permille=pm)
    cb.reset(0)
    b = orc.step(cb, frames[2], prompt, _pp(prop, 2), tau_sim=(95, 100), tau_margin=0.0, permille=pm)
    assert a["recomputed"][0] == 1 and a["gate_auto"][0] == 1
    assert b["recomputed"][0] == 1 and b["gate_auto"][0] == 1
    _same_outputs(a, b)
    _same_cache(d, ca, cb)
    assert ca.state(0) == cb.state(0)


@pytest.mark.parametrize("name", ["tiny_f32", "tiny_oft"])
def test_I4_thresholds_zero_and_infinity_and_one_step_lag(name):
    d, orc, _, prompt, _ = _setup(name)
    frames = synth.make_episode(d, 6, seed=5)
    prop = synth.make_proprio(d, 6, seed=5)
    pm = synth.linear_schedule(d.n_layers)
    for tau_m, want in ((0.0, 0), (float("inf"), 1)):
        c = orc.new_cache(1)
        prev_m = None
        for t in range(6):
            o = orc.step(c, frames[t], prompt, _pp(prop, t), tau_sim=(95, 100), tau_margin=tau_m, permille=pm)
            assert o["step_margin"][0] >= 0.0
            if t == 0:
                assert o["recomputed"][0] == 1  # empty cache: as if no cache existed
            else:
                assert o["recomputed"][0] == want
                assert o["gate_auto"][0] == int(prev_m < tau_m)
            prev_m = o["step_margin"][0]
    # an intermediate threshold: the flag at step t is exactly m_{t-1} < tau
    c = orc.new_cache(1)
    ms, flags = [], []
    for t in range(6):
        tau_m = 6.0e-4 if d.parallel == 0 else 1e-4
        o = orc.step(c, frames[t], prompt, _pp(prop, t), tau_sim=(95, 100), tau_margin=tau_m, permille=pm)
        ms.append(o["step_margin"][0])
        flags.append(int(o["recomputed"][0]))
    for t in range(1, 6):
        assert flags[t] == int(ms[t - 1] < tau_m)


def test_batch_rows_are_independent_sequences():
    """A batch of two sequences equals the two sequences run alone."""
    d = DIMS["tiny_f32"]
    w = synth.make_weights(d, seed=3)
    orc = oracle.Oracle(d, w)
    fr = synth.make_episode(d, 2, seed=9, batch=2)
    pr = synth.make_prompt(d, seed=9, batch=2)
    cb = orc.new_cache(2)
    outs = [orc.step(cb, fr[t], pr, tau_sim=(95, 100), tau_margin=0.0) for t in range(2)]
    for b in range(2):
        c1 = orc.new_cache(1)
        for t in range(2):
            o1 = orc.step(c1, fr[t, b:b + 1], pr[b:b + 1], tau_sim=(95, 100), tau_margin=0.0)
            for k in KEYS + ("idx", "M", "static_mask", "recomputed"):
                np.testing.assert_array_equal(outs[t][k][b], o1[k][0], err_msg=k)


def test_gate_comparison_is_strict():
    """m_{t-1} equal to theta_m does not fire; the next representable value above does."""
    d, orc, frames, prompt, prop = _setup("tiny_f32")
    for tau_off, want in ((0.0, 0), (1.0, 1)):
        c = orc.new_cache(1)
        o = orc.step(c, frames[0], prompt, None, tau_sim=(95, 100), tau_margin=0.0)
        m = float(o["step_margin"][0])
        tau = m if tau_off == 0.0 else float(np.nextafter(m, np.inf))
        o2 = orc.step(c, frames[1], prompt, None, tau_sim=(95, 100), tau_margin=tau)
        assert o2["gate_auto"][0] == want and o2["recomputed"][0] == want
