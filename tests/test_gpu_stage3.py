"""GPU parity of the entropy-adaptive Stage 3 (Sec. III-B, Stage 3; this
library's reading of it, see vlac_step_opts.s3_adaptive) against the oracle.

Lock-step episodes apply the oracle's schedule on both sides (the library's
own schedule is still compared: exact except at a layer whose smoothed value
sits within the entropy bar of an integer), the layer entropies within
ENT_TOL; a free-running fp32 episode; off reports the caller's schedule; an
adaptive schedule with lo = hi equals that constant schedule bit for bit;
switching on and off; argument errors."""
import numpy as np
import pytest
import torch

import synth
from tests.gpu_common import SMALL, Lockstep, episode

pytestmark = pytest.mark.gpu

S3 = (500, 900, 500)


def _pp(prop, t):
    return None if prop is None else prop[t]


@pytest.mark.parametrize("name", ["small", "small_oft", "small_batch", "tiny"])
def test_stage3_lockstep(name, cuda_device):
    d = SMALL[name]
    B = d.max_batch
    ls = Lockstep(d, synth.make_weights(d, seed=61), batch=B)
    frames, prompt, prop = episode(d, 4, seed=61, batch=B)
    pm = synth.linear_schedule(d.n_layers)
    tau = (95, 100) if d.img_h < 224 else (996, 1000)
    for t in range(4):
        o, g, rep = ls.step(frames[t], prompt, _pp(prop, t), tau, 0.0, pm, s3=S3)
        if t:
            assert (o["schedule"] != pm).any()  # the derived schedule is in use
            assert (o["recomputed"] == 0).all()


def test_stage3_free_running_fp32(cuda_device):
    d = SMALL["tiny"]
    ls = Lockstep(d, synth.make_weights(d, seed=62))
    frames, prompt, _ = episode(d, 4, seed=62)
    for t in range(4):
        ls.step(frames[t], prompt, None, (95, 100), 0.0, synth.linear_schedule(d.n_layers), s3=S3,
                s3_lockstep=False)


def test_stage3_switching_on_and_off(cuda_device):
    d = SMALL["small"]
    ls = Lockstep(d, synth.make_weights(d, seed=63))
    frames, prompt, _ = episode(d, 6, seed=63)
    pm = synth.linear_schedule(d.n_layers)
    for t, s3 in enumerate([None, S3, S3, None, S3, (300, 950, 250)]):
        ls.step(frames[t], prompt, None, (95, 100), 0.0, pm, s3=s3)


def test_constant_adaptive_schedule_equals_the_fixed_one(cuda_device):
    """lo = hi = x gives x at every layer whatever the entropies: the steps
    equal those of the fixed schedule x, outputs and cache bit for bit."""
    from paper_2608_10824_gb300 import Context
    d = SMALL["small"]
    w = synth.weights_to(synth.make_weights(d, seed=64), "cuda")
    frames, prompt, _ = episode(d, 3, seed=64)
    fr = [torch.from_numpy(np.ascontiguousarray(f)).cuda() for f in frames]
    pr = torch.from_numpy(prompt).cuda()
    x = 700
    ctx = Context(d, w, max_batch=1)
    ca, cb = ctx.new_cache(1), ctx.new_cache(1)
    fixed = np.full(d.n_layers, x, np.uint16)
    for t in range(3):
        a = ctx.step(ca, fr[t], pr, tau_sim=(95, 100), permille=fixed, want=("logits", "M", "schedule"))
        b = ctx.step(cb, fr[t], pr, tau_sim=(95, 100), permille=fixed, s3_adaptive=(x, x, 300),
                     want=("logits", "M", "schedule"))
        torch.cuda.synchronize()
        assert ctx.sync_error() == 0
        for k in ("action_ids", "margins", "logits", "M", "step_margin", "schedule"):
            assert torch.equal(a[k], b[k]), (t, k)
    assert torch.equal(ca.mem[:ca.mem.numel() // 2], cb.mem[:cb.mem.numel() // 2])


def test_stage3_bad_arguments(cuda_device):
    from paper_2608_10824_gb300 import Context, VlacError
    d = SMALL["small"]
    ctx = Context(d, synth.weights_to(synth.make_weights(d, seed=65), "cuda"), max_batch=1)
    frames, prompt, _ = episode(d, 1, seed=65)
    f, p = torch.from_numpy(frames[0]).cuda(), torch.from_numpy(prompt).cuda()
    c = ctx.new_cache(1)
    for s3 in [(600, 500, 500), (0, 1001, 500), (0, 900, 1001), (-1, 900, 500)]:
        with pytest.raises(VlacError) as e:
            ctx.step(c, f, p, s3_adaptive=s3)
        assert e.value.code == -1
