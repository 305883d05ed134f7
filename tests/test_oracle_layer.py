"""The oracle's one-layer entry (orc_layer) and cache write, used by the
one-layer workload (a 7B-shaped layer over a pre-filled cache, sweeping the
number of recomputed rows).

  * a full step records every position's layer inputs (H): one layer over all
    positions from H[l] gives H[l+1] bit for bit and rewrites the same K/V;
  * causality: a row's output does not depend on the rows at later positions;
  * a cache write reads back unchanged; bad arguments are refused.
"""
import numpy as np
import pytest

import oracle
import synth

DIMS = {"tiny_f32": synth.dims_for("tiny"), "tiny_bf16": synth.dims_for("tiny", dtype="bf16")}


@pytest.mark.parametrize("name", list(DIMS))
def test_layer_over_every_position_reproduces_the_step(name):
    # H[l] (l >= 1) is the input the step gave layer l; four layers give two
    # inner layers with both their input and output recorded
    d = DIMS[name].replace(n_layers=4)
    orc = oracle.Oracle(d, synth.make_weights(d, seed=71))
    c = orc.new_cache(1)
    orc.step(c, synth.make_episode(d, 1, seed=71)[0], synth.make_prompt(d, seed=71))
    pos = np.arange(d.pass_len, dtype=np.int32)
    for l in range(1, d.n_layers - 1):
        h_in, h_out = c.read(0, "H", l), c.read(0, "H", l + 1)
        k0, v0 = c.read(0, "K", l), c.read(0, "V", l)
        out = orc.layer(c, 0, l, pos, h_in)
        np.testing.assert_array_equal(out, h_out)
        np.testing.assert_array_equal(c.read(0, "K", l), k0)
        np.testing.assert_array_equal(c.read(0, "V", l), v0)


@pytest.mark.parametrize("name", list(DIMS))
def test_a_row_does_not_see_later_rows(name):
    d = DIMS[name]
    orc = oracle.Oracle(d, synth.make_weights(d, seed=72))
    _, x, k, v = synth.make_layer_case(d, 3, seed=72)
    kv = [k, v]
    outs = []
    for pos in ([5, 30, 60], [5, 30], [5]):
        c = orc.new_cache(1)
        c.write(0, "K", 0, kv[0])
        c.write(0, "V", 0, kv[1])
        outs.append(orc.layer(c, 0, 0, pos, x[: len(pos)]))
    np.testing.assert_array_equal(outs[0][:2], outs[1])
    np.testing.assert_array_equal(outs[0][:1], outs[2])
    # and a row does see an earlier one: the fresh K/V at 5 replaced the cached one
    c = orc.new_cache(1)
    c.write(0, "K", 0, kv[0])
    c.write(0, "V", 0, kv[1])
    alone = orc.layer(c, 0, 0, [30], x[1:2])
    assert not np.array_equal(alone, outs[1][1:2])


def test_cache_write_reads_back_and_bad_arguments_are_refused():
    d = DIMS["tiny_f32"]
    orc = oracle.Oracle(d, synth.make_weights(d, seed=73))
    c = orc.new_cache(2)
    v = np.random.default_rng(3).normal(size=(d.cache_len, d.hidden)).astype(np.float32)
    c.write(1, "V", 1, v)
    np.testing.assert_array_equal(c.read(1, "V", 1), v)
    assert not c.read(0, "V", 1).any()
    x = np.zeros((2, d.hidden), np.float32)
    for seq, layer, pos in ((0, 0, [3, 3]), (0, 0, [d.pass_len]), (2, 0, [1, 2]), (0, d.n_layers, [1, 2]),
                            (0, 0, [-1, 2])):
        with pytest.raises(ValueError):
            orc.layer(c, seq, layer, pos, x)
