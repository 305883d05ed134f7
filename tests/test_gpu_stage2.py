"""GPU parity of Stage 2 (Sec. III-B, task-relevant filtering) against the
oracle, through the C-ABI.

Each step compares, besides everything the other parity tests compare, the
relevance the library measured at the chosen layer (within REL_TOL of the
oracle's) and the removal set it decided from the previous step's relevance
(equal to the oracle's outside the tie band).  In lock-step runs the library
applies the oracle's removal set, so a tie-band difference cannot make the
two trajectories part; the free-running run applies its own."""
import numpy as np
import pytest

import synth
from gpu_common import SMALL, Lockstep, episode

pytestmark = pytest.mark.gpu

CASES = [  # (workload, batch, top_k)
    ("small", 1, 8),
    ("small_batch", 3, 16),
    ("small_oft", 1, 120),
    ("small_wide", 2, 8),
    ("tiny", 1, 8),
]


def _pp(prop, t):
    return None if prop is None else prop[t]


@pytest.mark.parametrize("name,batch,top_k", CASES, ids=[c[0] for c in CASES])
@pytest.mark.parametrize("where", ["first", "last"])
def test_stage2_lockstep(name, batch, top_k, where):
    d = SMALL[name]
    layer = 0 if where == "first" else d.n_layers - 1
    ls = Lockstep(d, synth.make_weights(d, seed=41), batch=batch)
    frames, prompt, prop = episode(d, 5, seed=41, batch=batch)
    tau = (95, 100) if name == "tiny" else (996, 1000)
    removed = 0
    for t in range(5):
        o, g, rep = ls.step(frames[t], prompt, _pp(prop, t), tau, 0.0, synth.linear_schedule(d.n_layers),
                            s2_top_k=top_k, s2_layer=layer)
        assert o["relevance"].min() > 0
        removed += int((o["relevant"] & o["static_mask"]).sum())
    assert removed > 0, "Stage 2 never took a static patch out: the case tests nothing"
    print(name, where, [(r["rel_diff"], r["removal_diffs"], r["max_logit_diff"]) for r in ls.log])


def test_stage2_free_running_tiny():
    """fp32: the library decides its own removal sets and they equal the oracle's."""
    d = SMALL["tiny"]
    ls = Lockstep(d, synth.make_weights(d, seed=42))
    frames, prompt, prop = episode(d, 5, seed=42)
    for t in range(5):
        ls.step(frames[t], prompt, _pp(prop, t), (95, 100), 0.0, synth.linear_schedule(d.n_layers), s2_top_k=8,
                s2_layer=1, s2_lockstep=False)
    assert sum(r["removal_diffs"] for r in ls.log) == 0


def test_stage2_switching_on_off_and_layer():
    """Stage 2 off, on at layer 0, on at the last layer, off again: the step is
    captured into a new graph whenever the launch list changes."""
    d = SMALL["small"]
    ls = Lockstep(d, synth.make_weights(d, seed=43))
    frames, prompt, prop = episode(d, 12, seed=43)
    plan = [(0, 0)] * 3 + [(8, 0)] * 3 + [(8, d.n_layers - 1)] * 3 + [(0, 0)] * 3
    for t, (k, layer) in enumerate(plan):
        ls.step(frames[t], prompt, _pp(prop, t), (996, 1000), 0.0, synth.linear_schedule(d.n_layers), s2_top_k=k,
                s2_layer=layer)


def test_stage2_every_patch_relevant_equals_full_branch():
    """top_k = Nv keeps every patch out of the reusable set: the cached branch
    then recomputes every row in position order, as the full branch does, and
    gives the same bits."""
    import torch

    from paper_2608_10824_gb300 import Context
    d = SMALL["small"]
    w = synth.weights_to(synth.make_weights(d, seed=44), "cuda")
    frames, prompt, _ = episode(d, 2, seed=44)
    ctx = Context(d, w, max_batch=1)
    res = []
    for branch in (0, 1):
        c = ctx.new_cache(1)
        kw = dict(tau_sim=(996, 1000), tau_margin=0.0, permille=synth.full_schedule(d.n_layers),
                  s2_top_k=d.n_visual, s2_layer=0, want=("logits", "idx", "M", "relevance", "relevant"))
        ctx.step(c, torch.from_numpy(frames[0]).cuda(), torch.from_numpy(prompt).cuda(), **kw)
        g = ctx.step(c, torch.from_numpy(frames[1]).cuda(), torch.from_numpy(prompt).cuda(),
                     gate_override=torch.tensor([branch], dtype=torch.int8, device="cuda"), **kw)
        torch.cuda.synchronize()
        res.append({k: v.cpu().numpy() for k, v in g.items()})
    a, b = res
    assert a["recomputed"][0] == 0 and b["recomputed"][0] == 1
    assert a["relevant"].all() and list(a["M"][0]) == [d.pass_len] * d.n_layers
    for k in ("action_ids", "margins", "logit_gap", "logits", "step_margin", "relevance", "idx"):
        np.testing.assert_array_equal(a[k], b[k], err_msg=k)


def test_stage2_argument_errors():
    import torch

    from paper_2608_10824_gb300 import Context, VlacError
    d = SMALL["tiny"]
    ctx = Context(d, synth.weights_to(synth.make_weights(d, seed=45), "cuda"), max_batch=1)
    c = ctx.new_cache(1)
    frames, prompt, _ = episode(d, 1, seed=45)
    f, p = torch.from_numpy(frames[0]).cuda(), torch.from_numpy(prompt).cuda()
    for kw in (dict(s2_top_k=-1), dict(s2_top_k=4, s2_layer=d.n_layers), dict(s2_top_k=4, s2_layer=-1)):
        with pytest.raises(VlacError):
            ctx.step(c, f, p, **kw)
    ctx.step(c, f, p, s2_top_k=4, s2_layer=0)  # the context stays usable
    torch.cuda.synchronize()
    assert ctx.sync_error() == 0
