"""The optional parts of the step together, against the oracle in lock-step:
a running batch whose sequences sit steps out and rejoin (reading 21),
Stage 2 removal (Sec. III-B), the entropy-adaptive Stage 3 (reading 22) and
the whole-vocabulary margin driving the gate (margin kind 2, Sec. IV-A), with
the gate free to fire.  Every step compares selection, flags, ids, logits and
every signal as the single-feature tests do."""
import numpy as np
import pytest

import synth
from tests.gpu_common import SMALL, Lockstep, episode

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["small_batch", "tiny"])
def test_all_options_in_one_episode(cuda_device, name):
    d = SMALL[name].replace(max_batch=3)
    ls = Lockstep(d, synth.make_weights(d, seed=71), batch=3)
    frames, prompt, _ = episode(d, 6, seed=71, batch=3)
    pm = synth.linear_schedule(d.n_layers)
    plan = [[1, 1, 1], [1, 0, 1], [0, 1, 1], [1, 1, 0], [1, 1, 1], [1, 0, 1]]
    taus = [0.0, 0.0, 1e-3, 0.0, float("inf"), 0.0]
    for t, act in enumerate(plan):
        if t == 3:  # a new episode joins slot 0
            ls.oc.reset(0)
            ls.ctx.reset(ls.gc, 0)
        o, g, rep = ls.step(frames[t], prompt, None, (95, 100), taus[t], pm, margin_kind=2,
                            active=np.array(act, np.uint8), s2_top_k=4, s2_layer=d.n_layers - 1,
                            s3=(400, 950, 600))
        stepped = np.array(act, bool)
        assert not g["logits"][~stepped].any()
        if taus[t] == float("inf"):
            assert (g["recomputed"][stepped] == 1).all()
