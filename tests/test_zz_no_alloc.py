"""The allocation-free selection call (vlac_select_noalloc) is for callers
that cannot allocate device memory while they run: a real-time control loop
whose memory is fixed before it starts, or a host framework that owns every
device allocation and forbids a library from making its own.  It must give
exactly the static mask, recompute order, per-layer row counts and recompute
flags that vlac_step computes, on calls made one after another (its fixed
scratch is reused by every call).  This file is collected last on purpose."""
import numpy as np
import pytest
import torch

import synth
from tests.gpu_common import SMALL, episode

pytestmark = pytest.mark.gpu

VLAC_ERR_UNSUPPORTED = -7


def _step_selection(d, B, frames, prompt, prop, tau_sim, pm, seed_w):
    """vlac_step over frame 0 (empty cache), frame 1 (cached) and frame 2 (gate
    forced to fire); returns the selection outputs of each step."""
    from paper_2608_10824_gb300 import Context
    w = synth.weights_to(synth.make_weights(d, seed=seed_w), "cuda")
    ctx = Context(d, w, max_batch=B)
    cache = ctx.new_cache(B)
    want = ("static_mask", "idx", "M", "gate_auto")
    steps = []
    for t, tau_m in ((0, 0.0), (1, 0.0), (2, float("inf"))):
        o = ctx.step(cache, frames[t], prompt, prop[t], tau_sim=tau_sim, tau_margin=tau_m, permille=pm, want=want)
        steps.append({k: v.clone() for k, v in o.items()})
    torch.cuda.synchronize()
    assert ctx.sync_error() == 0
    return steps


def _check_noalloc_against(d, B, frames, steps, tau_sim, pm):
    from paper_2608_10824_gb300.vlac import select_noalloc
    valid = torch.ones(B, dtype=torch.uint8, device="cuda")
    # the allocation-free call on the same inputs, twice in a row
    for t, tau_m in ((1, 0.0), (2, float("inf"))):
        m_prev = steps[t - 1]["step_margin"]
        got = select_noalloc(d, frames[t], frames[t - 1], valid, m_prev, tau_sim=tau_sim, tau_margin=tau_m,
                             permille=pm, max_batch=B)
        torch.cuda.synchronize()
        for k in ("static_mask", "idx", "M", "recomputed"):
            assert torch.equal(got[k], steps[t][k]), (t, k)
    assert steps[1]["recomputed"].sum().item() == 0 and steps[2]["recomputed"].sum().item() == B


@pytest.mark.parametrize("name", ["small", "small_oft"])
def test_noalloc_selection_matches_step_on_consecutive_calls(name, cuda_device):
    d = SMALL[name]
    B = 2
    frames, prompt, prop = episode(d, 3, seed=41, batch=B)
    fr = [torch.from_numpy(np.ascontiguousarray(f)).cuda() for f in frames]
    pr = torch.from_numpy(prompt).cuda()
    pp = [None] * len(fr) if prop is None else [torch.from_numpy(np.ascontiguousarray(p)).cuda() for p in prop]
    pm = synth.linear_schedule(d.n_layers)
    tau_sim = (95, 100) if d.img_h < 224 else (996, 1000)
    steps = _step_selection(d, B, fr, pr, pp, tau_sim, pm, seed_w=41)
    _check_noalloc_against(d, B, fr, steps, tau_sim, pm)


# 64 x 64 = 4096 patches of 14 x 14: the most visual patches the dims accept
BIG = synth.Dims(n_layers=2, hidden=256, n_heads=4, head_dim=64, ffn=688, vocab=512, n_bins=256,
                 img_h=896, img_w=896, patch=14, n_views=1, n_text=8, proprio_dim=0, n_action=7, parallel=0,
                 dtype="f32", max_batch=1)


def test_noalloc_accepts_the_largest_patch_grid(cuda_device):
    """4096 patches of one sequence fit the fixed scratch; the selection
    kernel then needs more than 48 KB of shared memory, in both entry points."""
    d = BIG
    frames, prompt, _ = episode(d, 3, seed=43, batch=1, kind="redraw")
    fr = [torch.from_numpy(np.ascontiguousarray(f)).cuda() for f in frames]
    pr = torch.from_numpy(prompt).cuda()
    pm = synth.linear_schedule(d.n_layers)
    steps = _step_selection(d, 1, fr, pr, [None] * 3, (95, 100), pm, seed_w=43)
    assert 0 < steps[1]["static_mask"].sum().item() < d.n_visual
    _check_noalloc_against(d, 1, fr, steps, (95, 100), pm)


def test_noalloc_rejects_work_beyond_its_scratch(cuda_device):
    from paper_2608_10824_gb300 import VlacError
    from paper_2608_10824_gb300.vlac import select_noalloc
    # the same 4096-patch grid: one sequence fits, eight do not
    d = BIG.replace(max_batch=8)
    small = torch.zeros((8, 16), dtype=torch.uint8, device="cuda")
    m = torch.zeros(8, device="cuda")
    with pytest.raises(VlacError) as e:
        select_noalloc(d, small, small, small[:, 0].contiguous(), m, out={
            "static_mask": small, "idx": small, "M": small, "recomputed": small[:, 0].contiguous()})
    assert e.value.code == VLAC_ERR_UNSUPPORTED
