"""The oracle's whole step against the independent numpy restatement
(tests/restate.py) on small models: full and cached branches, fp32 and bf16
storage, autoregressive and parallel action decoding; and the KV-cache
decode against a one-shot causal forward of the same sequence."""
import numpy as np
import pytest

import oracle
import synth
from tests.restate import Restated

CASES = {
    "tiny_f32": synth.dims_for("tiny"),
    "tiny_bf16": synth.dims_for("tiny", dtype="bf16"),
    "tiny_oft": synth.dims_for("tiny", n_views=2, proprio_dim=8, n_action=8, parallel=1),
}


def _episode(d, n, seed):
    frames = synth.make_episode(d, n, seed=seed)
    prompt = synth.make_prompt(d, seed=seed)
    prop = synth.make_proprio(d, n, seed=seed)
    return frames, prompt, prop


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("sched", ["all", "linear"])
def test_oracle_matches_restatement(name, sched):
    d = CASES[name]
    w = synth.make_weights(d, seed=11)
    orc = oracle.Oracle(d, w)
    cache = orc.new_cache(1)
    ref = Restated(d, w)
    frames, prompt, prop = _episode(d, 4, seed=2)
    pm = synth.full_schedule(d.n_layers) if sched == "all" else synth.linear_schedule(d.n_layers)
    tol = 2e-5 if d.dtype == "f32" else 2e-2
    n_cached = 0
    for t in range(4):
        # tau_m = 0 keeps the cached branch running; step 2 forces a full pass
        override = 1 if t == 2 else -1
        pp = None if prop is None else prop[t, 0]
        o = orc.step(cache, frames[t], prompt, pp, tau_sim=(95, 100), tau_margin=0.0, permille=pm,
                     gate_override=np.array([override], np.int8))
        r = ref.step(frames[t, 0], prompt[0], pp, (95, 100), 0.0, pm, override=override)
        n_cached += 1 - int(o["recomputed"][0])
        assert o["recomputed"][0] == r["recomputed"]
        assert o["gate_auto"][0] == r["gate_auto"]
        np.testing.assert_array_equal(o["static_mask"][0], r["static_mask"])
        np.testing.assert_array_equal(o["idx"][0], r["idx"])
        np.testing.assert_array_equal(o["M"][0], r["M"])
        np.testing.assert_allclose(o["logits"][0], r["logits"], atol=tol, rtol=0)
        np.testing.assert_allclose(o["margins"][0], r["margins"], atol=tol * 1e-2 + 1e-9, rtol=1e-3)
        # ids must agree wherever the top-2 logit gap is clearly larger than the tolerance
        clear = r["logit_gap"] > 4 * tol
        np.testing.assert_array_equal(o["action_ids"][0][clear], r["action_ids"][clear])
    assert n_cached == 2


@pytest.mark.parametrize("name", ["tiny_f32", "tiny_bf16"])
def test_kv_cache_decode_equals_one_shot_causal_forward(name):
    """The decode passes (one token, attending the cache) give the same
    logits as recomputing the whole sequence with a causal mask."""
    d = CASES[name]
    w = synth.make_weights(d, seed=12)
    orc = oracle.Oracle(d, w)
    cache = orc.new_cache(1)
    frames, prompt, _ = _episode(d, 1, seed=4)
    o = orc.step(cache, frames[0], prompt, None, tau_sim=(95, 100), tau_margin=0.0,
                 permille=synth.full_schedule(d.n_layers))
    ids = o["action_ids"][0]
    # one causal forward over the prefix followed by the fed action tokens
    ref = Restated(d, w)
    P, D = d.prefix_len, d.n_action
    rows = [ref.embed(p, frames[0, 0], prompt[0], None) for p in range(P)]
    rows += [ref.f32(ref.tok[d.vocab - d.n_bins + int(ids[a])]) for a in range(D - 1)]
    x = np.stack(rows)
    pos = list(range(P + D - 1))
    for l in range(d.n_layers):
        x = ref.layer(l, x, pos)
    tol = 2e-5 if d.dtype == "f32" else 2e-2
    for a in range(D):
        lg, *_ = ref.head_out(x[P - 1 + a])
        np.testing.assert_allclose(o["logits"][0, a], lg, atol=tol, rtol=0)
