"""GPU parity of the other per-token signals against the oracle, through the
C-ABI: the entropy of each action token's bin softmax, the margin of the
softmax over the whole vocabulary (also as the gate signal, margin kind 2),
and the action delta between consecutive steps (Sec. IV-A, Sec. VI)."""
import numpy as np
import pytest

import synth
from gpu_common import SMALL, Lockstep, episode

pytestmark = pytest.mark.gpu

CASES = [("small", 1), ("small_batch", 3), ("small_oft", 1), ("tiny", 1)]


def _pp(prop, t):
    return None if prop is None else prop[t]


@pytest.mark.parametrize("name,batch", CASES, ids=[c[0] for c in CASES])
def test_signals_lockstep(name, batch):
    d = SMALL[name]
    ls = Lockstep(d, synth.make_weights(d, seed=51), batch=batch)
    frames, _, prop = episode(d, 4, seed=51, batch=batch)
    tau = (95, 100) if name == "tiny" else (996, 1000)
    for t in range(4):
        # a new instruction every step, so that the actions (and the delta) change
        prompt = synth.make_prompt(d, seed=51 + t, batch=batch)
        ls.step(frames[t], prompt, _pp(prop, t), tau, 0.0, synth.linear_schedule(d.n_layers), want_vocab=True)
    print(name, [(r["entropy_diff"], r["delta_compared"], r["max_logit_diff"]) for r in ls.log])


@pytest.mark.parametrize("name", ["small", "tiny"])
def test_vocab_margin_as_the_gate_signal(name):
    """Margin kind 2 drives the gate; theta_m between the episode's margins
    makes both branches run."""
    d = SMALL[name]
    w = synth.make_weights(d, seed=52)
    frames, prompt, prop = episode(d, 6, seed=52)
    tau = (95, 100) if name == "tiny" else (996, 1000)
    import oracle
    orc = oracle.Oracle(d, w)
    c = orc.new_cache(1)
    ms = [orc.step(c, frames[t], prompt, _pp(prop, t), tau_sim=tau, margin_kind=2, want_vocab_margin=True)
          ["step_margin"][0] for t in range(6)]
    theta = float(np.median(ms))
    ls = Lockstep(d, w)
    for t in range(6):
        ls.step(frames[t], prompt, _pp(prop, t), tau, theta, synth.linear_schedule(d.n_layers), margin_kind=2)
    ran = [r["recomputed"][0] for r in ls.log]
    print(name, theta, ms, ran)


def test_vocab_margin_switching_recaptures_the_graph():
    """Asking for the whole-vocabulary margin changes the launch list: steps
    without, with, and without it again stay in parity."""
    d = SMALL["small"]
    ls = Lockstep(d, synth.make_weights(d, seed=53))
    frames, prompt, prop = episode(d, 9, seed=53)
    for t in range(9):
        ls.step(frames[t], prompt, _pp(prop, t), (996, 1000), 0.0, synth.linear_schedule(d.n_layers),
                want_vocab=3 <= t < 6)
