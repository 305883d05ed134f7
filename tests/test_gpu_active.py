"""GPU parity of a running batch whose sequences sit steps out (episodes
joining and leaving), against the oracle: a paused sequence's outputs are
zero and its next step is the one it would have run without the pause; the
other sequences step as usual; a reset slot joins as a fresh episode."""
import numpy as np
import pytest

import synth
from tests.gpu_common import SMALL, Lockstep, episode

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["small_batch", "tiny"])
def test_running_batch_parity(cuda_device, name):
    d = SMALL[name].replace(max_batch=3)
    ls = Lockstep(d, synth.make_weights(d, seed=95), batch=3)
    frames, prompt, _ = episode(d, 7, seed=95, batch=3)
    pm = synth.linear_schedule(d.n_layers)
    plan = [[1, 1, 1], [1, 0, 1], [1, 0, 0], [0, 1, 1], [1, 1, 1], [0, 0, 0], [1, 1, 1]]
    for t, act in enumerate(plan):
        if t == 4:  # a new episode joins slot 2
            ls.oc.reset(2)
            ls.ctx.reset(ls.gc, 2)
        o, g, rep = ls.step(frames[t], prompt, None, (95, 100), 0.0, pm, active=np.array(act, np.uint8))
        for b in range(3):
            if not act[b]:
                assert not g["logits"][b].any() and g["recomputed"][b] == 0
        if t == 4:
            assert g["recomputed"][2] == 1
