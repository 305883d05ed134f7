"""The allocation-free selection call (vlac_select_noalloc) is for callers
that cannot allocate device memory while they run -- inside a stream capture,
in a real-time loop with memory fixed up front, or in a host framework that
owns every allocation.  It must give exactly the static mask, recompute order,
per-layer row counts and recompute flags that vlac_step computes, on calls
made one after another (its fixed scratch is reused by every call).  This file
is collected last on purpose."""
import numpy as np
import pytest
import torch

import synth
from tests.gpu_common import SMALL, episode

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["small", "small_oft"])
def test_noalloc_selection_matches_step_on_consecutive_calls(name, cuda_device):
    from paper_2608_10824_gb300 import Context
    from paper_2608_10824_gb300.vlac import select_noalloc
    d = SMALL[name]
    B = 2
    w = synth.weights_to(synth.make_weights(d, seed=41), "cuda")
    ctx = Context(d, w, max_batch=B)
    cache = ctx.new_cache(B)
    frames, prompt, prop = episode(d, 3, seed=41, batch=B)
    fr = [torch.from_numpy(np.ascontiguousarray(f)).cuda() for f in frames]
    pr = torch.from_numpy(prompt).cuda()
    pp = [None] * len(fr) if prop is None else [torch.from_numpy(np.ascontiguousarray(p)).cuda() for p in prop]
    pm = synth.linear_schedule(d.n_layers)
    tau_sim = (95, 100) if d.img_h < 224 else (996, 1000)
    want = ("static_mask", "idx", "M", "gate_auto")
    # the step path: frame 0 (empty cache), frame 1 (cached), frame 2 (gate forced to fire)
    steps = []
    for t, tau_m in ((0, 0.0), (1, 0.0), (2, float("inf"))):
        o = ctx.step(cache, fr[t], pr, pp[t], tau_sim=tau_sim, tau_margin=tau_m, permille=pm, want=want)
        steps.append({k: v.clone() for k, v in o.items()})
    torch.cuda.synchronize()
    assert ctx.sync_error() == 0
    # the allocation-free call on the same inputs, twice in a row
    valid = torch.ones(B, dtype=torch.uint8, device="cuda")
    for t, tau_m in ((1, 0.0), (2, float("inf"))):
        m_prev = steps[t - 1]["step_margin"]
        got = select_noalloc(d, fr[t], fr[t - 1], valid, m_prev, tau_sim=tau_sim, tau_margin=tau_m, permille=pm,
                             max_batch=B)
        torch.cuda.synchronize()
        for k in ("static_mask", "idx", "M", "recomputed"):
            assert torch.equal(got[k], steps[t][k]), (t, k)
    assert steps[1]["recomputed"].sum().item() == 0 and steps[2]["recomputed"].sum().item() == B


def test_noalloc_rejects_work_beyond_its_scratch(cuda_device):
    from paper_2608_10824_gb300 import VlacError
    from paper_2608_10824_gb300.vlac import select_noalloc
    # 8 sequences x 4096 patches of statistics do not fit the fixed scratch
    d = synth.Dims(n_layers=2, hidden=256, n_heads=2, head_dim=128, ffn=768, vocab=1024, n_bins=256,
                   img_h=896, img_w=896, patch=14, n_views=1, n_text=8, proprio_dim=0, n_action=7, parallel=0,
                   dtype="bf16", max_batch=8)
    small = torch.zeros((8, 16), dtype=torch.uint8, device="cuda")
    m = torch.zeros(8, device="cuda")
    with pytest.raises(VlacError) as e:
        select_noalloc(d, small, small, small[:, 0].contiguous(), m, out={
            "static_mask": small, "idx": small, "M": small, "recomputed": small[:, 0].contiguous()})
    assert e.value.code == -1
