"""Pins of the oracle's Stage 2 (Sec. III-B, task-relevant filtering).

The relevance of visual patch v is the softmax probability that the text
queries put on its key (position 1 + v), summed over the text rows and the
heads, at one chosen layer of the previous step; the top_k patches by
relevance are never reused.  Pinned here by:
  * the ranking against a lexicographic sort (value descending, index
    ascending);
  * a closed form: with W_q = 0 at the chosen layer every score is 0, so a
    text row at position p puts exactly 1/(p+1) on each visual key;
  * a position pin: at layer 0, patches with all-zero pixels have zero keys
    and so identical relevance; the single non-zero patch is the only one
    that differs, at its own index;
  * invariants: top_k >= Nv recomputes everything (equals the full branch
    bit for bit), the removal set of step t is the top_k of step t-1's
    relevance, a reset forgets it, and the relevance is a probability mass.
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


def _text_positions(d):
    """Prompt positions that can see the visual keys (BOS at 0 cannot)."""
    lo, hi = synth.positions(d)["text"]
    return list(range(lo, hi))


def _pp(prop, t):
    return None if prop is None else prop[t, 0]


# --------------------------------------------------------------------------
# the removal set
# --------------------------------------------------------------------------

@pytest.mark.parametrize("n,k", [(64, 0), (64, 1), (64, 20), (64, 63), (64, 64), (64, 100), (512, 120)])
def test_top_k_matches_lexicographic_sort(n, k):
    rng = np.random.default_rng(n * 1000 + k)
    rel = rng.integers(0, 12, n).astype(np.float64) / 7.0  # many ties
    order = np.lexsort((np.arange(n), -rel))  # value descending, then index ascending
    want = np.zeros(n, np.uint8)
    want[order[:k]] = 1
    np.testing.assert_array_equal(oracle.top_k(rel, k), want)


def test_top_k_all_equal_takes_lowest_indices():
    got = oracle.top_k(np.full(10, 0.25), 3)
    assert list(got) == [1, 1, 1, 0, 0, 0, 0, 0, 0, 0]


@pytest.mark.parametrize("d", [DIMS["tiny_f32"], DIMS["tiny_oft"]])
def test_select2_removes_relevant_static_patches(d):
    """Reusable = Stage-1 static and not relevant; the order and counts follow
    from that set exactly as without Stage 2."""
    eps = synth.make_episode(d, 3, seed=3)
    rng = np.random.default_rng(5)
    pm = synth.linear_schedule(d.n_layers)
    for t in (1, 2):
        rel = rng.random(d.n_visual)
        for k in (0, 5, d.n_visual // 2, d.n_visual):
            n, mask, idx, M, relevant = oracle.select(d, eps[t, 0], eps[t - 1, 0], True, (95, 100), pm, False,
                                                      relevance=rel, top_k=k)
            np.testing.assert_array_equal(relevant, oracle.top_k(rel, k))
            reusable = mask.astype(bool) & ~relevant.astype(bool)
            assert n == int(reusable.sum())
            # without Stage 2, on a frame pair whose static set is exactly `reusable`,
            # Stage 3 gives the same counts; and every non-reusable position leads idx
            assert list(M) == [d.pass_len - (int(pm[l]) * n) // 1000 for l in range(d.n_layers)]
            lead = set(range(d.pass_len)) - {1 + v for v in np.flatnonzero(reusable)}
            assert set(idx[:len(lead)]) == lead
            assert sorted(idx[:len(lead)]) == list(idx[:len(lead)])
            assert set(idx[len(lead):]) == {1 + v for v in np.flatnonzero(reusable)}
            # the reusable tail keeps the Stage-3 order of the plain selection
            _, _, idx0, _ = oracle.select(d, eps[t, 0], eps[t - 1, 0], True, (95, 100), pm, False)
            tail0 = [p for p in idx0 if 1 <= p <= d.n_visual and reusable[p - 1]]
            assert list(idx[len(lead):]) == tail0


# --------------------------------------------------------------------------
# the relevance itself
# --------------------------------------------------------------------------

@pytest.mark.parametrize("name", list(DIMS))
@pytest.mark.parametrize("layer", [0, 1])
def test_uniform_attention_closed_form(name, layer):
    """W_q = 0 at the chosen layer: q = 0, every score 0, softmax uniform over
    the p + 1 keys of a text row at position p, for a full and a cached step."""
    d = DIMS[name]
    w = synth.make_weights(d, seed=8)
    w["layers"][layer]["wq"] = w["layers"][layer]["wq"] * 0
    orc = oracle.Oracle(d, w)
    frames = synth.make_episode(d, 2, seed=8)
    prompt = synth.make_prompt(d, seed=8)
    prop = synth.make_proprio(d, 2, seed=8)
    want = d.n_heads * sum(1.0 / (p + 1) for p in _text_positions(d))
    c = orc.new_cache(1)
    for t in range(2):
        o = orc.step(c, frames[t], prompt, _pp(prop, t), tau_sim=(95, 100), tau_margin=0.0,
                     permille=synth.linear_schedule(d.n_layers), s2_top_k=3, s2_layer=layer,
                     gate_override=np.array([-1 if t else 1], np.int8))
        assert o["recomputed"][0] == (1 if t == 0 else 0)
        np.testing.assert_allclose(o["relevance"][0], want, rtol=1e-12, atol=0)
        # uniform relevance: the removal set is the lowest indices
        np.testing.assert_array_equal(o["relevant"][0], [1] * 3 + [0] * (d.n_visual - 3) if t else 0)


@pytest.mark.parametrize("name", ["tiny_f32", "tiny_bf16"])
@pytest.mark.parametrize("vstar", [0, 5, 63])
def test_single_nonzero_patch_is_the_one_that_stands_out(name, vstar):
    """Layer 0: a patch of zero pixels embeds to 0, normalises to 0 and has key
    0, so every such patch draws the same probability; only patch v* differs,
    and it must appear at index v* (position 1 + v*)."""
    d = DIMS[name]
    orc = oracle.Oracle(d, synth.make_weights(d, seed=9))
    frame = np.zeros((d.n_views, d.img_h, d.img_w, 3), np.uint8)
    gw = d.img_w // d.patch
    py, px = divmod(vstar, gw)
    rng = np.random.default_rng(vstar)
    frame[0, py * d.patch:(py + 1) * d.patch, px * d.patch:(px + 1) * d.patch] = rng.integers(
        1, 256, (d.patch, d.patch, 3))
    c = orc.new_cache(1)
    o = orc.step(c, frame, synth.make_prompt(d, seed=9), None, s2_top_k=1, s2_layer=0)
    rel = o["relevance"][0]
    others = np.delete(rel, vstar)
    assert np.all(others == others[0])
    assert rel[vstar] != others[0]


@pytest.mark.parametrize("name", list(DIMS))
def test_relevance_is_a_probability_mass(name):
    d = DIMS[name]
    orc = oracle.Oracle(d, synth.make_weights(d, seed=10))
    frames = synth.make_episode(d, 2, seed=10)
    prop = synth.make_proprio(d, 2, seed=10)
    c = orc.new_cache(1)
    bound = d.n_heads * len(_text_positions(d))
    for t in range(2):
        o = orc.step(c, frames[t], synth.make_prompt(d, seed=10), _pp(prop, t), tau_sim=(95, 100),
                     s2_top_k=4, s2_layer=d.n_layers - 1)
        rel = o["relevance"][0]
        assert np.all(rel > 0)  # every text row sees every visual key; softmax is positive
        assert rel.sum() < bound
        assert np.all(rel < d.n_heads * len(_text_positions(d)))


# --------------------------------------------------------------------------
# Stage 2 inside the step
# --------------------------------------------------------------------------

@pytest.mark.parametrize("name", list(DIMS))
def test_every_patch_relevant_equals_full_branch(name):
    """top_k = Nv: nothing is reusable, so a cached step recomputes every row
    in position order, exactly as the full branch does."""
    d = DIMS[name]
    w = synth.make_weights(d, seed=11)
    orc = oracle.Oracle(d, w)
    frames = synth.make_episode(d, 2, seed=11)
    prompt = synth.make_prompt(d, seed=11)
    prop = synth.make_proprio(d, 2, seed=11)
    pm = synth.full_schedule(d.n_layers)
    ca, cb = orc.new_cache(1), orc.new_cache(1)
    for c in (ca, cb):
        orc.step(c, frames[0], prompt, _pp(prop, 0), tau_sim=(95, 100), permille=pm, s2_top_k=d.n_visual,
                 s2_layer=0)
    a = orc.step(ca, frames[1], prompt, _pp(prop, 1), tau_sim=(95, 100), permille=pm, s2_top_k=d.n_visual,
                 s2_layer=0, gate_override=np.array([0], np.int8))
    b = orc.step(cb, frames[1], prompt, _pp(prop, 1), tau_sim=(95, 100), permille=pm, s2_top_k=d.n_visual,
                 s2_layer=0, gate_override=np.array([1], np.int8))
    assert a["recomputed"][0] == 0 and b["recomputed"][0] == 1
    assert a["static_mask"].sum() > 0 and a["relevant"].all()
    assert list(a["M"][0]) == [d.pass_len] * d.n_layers
    for k in ("action_ids", "margins", "logit_gap", "logits", "step_margin", "relevance"):
        np.testing.assert_array_equal(a[k], b[k], err_msg=k)


def test_removal_uses_the_previous_steps_relevance_and_reset_forgets_it():
    d = DIMS["tiny_f32"]
    orc = oracle.Oracle(d, synth.make_weights(d, seed=12))
    frames = synth.make_episode(d, 5, seed=12)
    prompt = synth.make_prompt(d, seed=12)
    c = orc.new_cache(1)
    kw = dict(tau_sim=(95, 100), permille=synth.linear_schedule(d.n_layers), s2_layer=1)
    o0 = orc.step(c, frames[0], prompt, None, s2_top_k=6, **kw)
    assert o0["relevant"].sum() == 0  # no previous step
    o1 = orc.step(c, frames[1], prompt, None, s2_top_k=6, gate_override=np.array([0], np.int8), **kw)
    np.testing.assert_array_equal(o1["relevant"][0], oracle.top_k(o0["relevance"][0], 6))
    # a step with Stage 2 off measures nothing, so the next step removes nothing
    o2 = orc.step(c, frames[2], prompt, None, s2_top_k=0, gate_override=np.array([0], np.int8), **kw)
    assert o2["relevance"].sum() == 0 and o2["relevant"].sum() == 0
    o3 = orc.step(c, frames[3], prompt, None, s2_top_k=6, gate_override=np.array([0], np.int8), **kw)
    assert o3["relevant"].sum() == 0
    c.reset()
    o4 = orc.step(c, frames[4], prompt, None, s2_top_k=6, **kw)
    assert o4["recomputed"][0] == 1 and o4["relevant"].sum() == 0


def test_stage2_off_is_the_plain_step():
    d = DIMS["tiny_bf16"]
    w = synth.make_weights(d, seed=13)
    orc = oracle.Oracle(d, w)
    frames = synth.make_episode(d, 3, seed=13)
    prompt = synth.make_prompt(d, seed=13)
    ca, cb = orc.new_cache(1), orc.new_cache(1)
    for t in range(3):
        a = orc.step(ca, frames[t], prompt, None, tau_sim=(95, 100), s2_top_k=0, s2_layer=0)
        b = orc.step(cb, frames[t], prompt, None, tau_sim=(95, 100))
        for k in ("action_ids", "margins", "logits", "static_mask", "idx", "M", "relevance", "relevant"):
            np.testing.assert_array_equal(a[k], b[k], err_msg=k)


def test_stage2_rejects_bad_arguments():
    d = DIMS["tiny_f32"]
    orc = oracle.Oracle(d, synth.make_weights(d, seed=14))
    f = synth.make_episode(d, 1, seed=14)[0]
    c = orc.new_cache(1)
    for kw in (dict(s2_top_k=-1), dict(s2_top_k=2, s2_layer=d.n_layers), dict(s2_top_k=2, s2_layer=-1)):
        with pytest.raises(ValueError):
            orc.step(c, f, synth.make_prompt(d, seed=14), None, **kw)
