"""Bitwise invariants of the CUDA path (GPU against itself), the same ones
the oracle satisfies: reuse-nothing equals the full pass, identical frames
with reuse equal the full pass, a gated step equals reset + step, and two
runs of the same episode are identical.  Whole cache memory is compared."""
import numpy as np
import pytest
import torch

import synth
from tests.gpu_common import SMALL, episode

pytestmark = pytest.mark.gpu

WANT = ("gate_auto", "logits", "static_mask", "idx", "M")
KEYS = ("action_ids", "margins", "logit_gap", "logits", "step_margin")


def _setup(name, seed=31):
    from paper_2608_10824_gb300 import Context
    d = SMALL[name]
    w = synth.weights_to(synth.make_weights(d, seed=seed), "cuda")
    frames, prompt, prop = episode(d, 3, seed=seed)
    ctx = Context(d, w, max_batch=1)
    dev = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a)).cuda()
    return d, ctx, [dev(f) for f in frames], dev(prompt), (None if prop is None else [dev(p) for p in prop])


def _pp(prop, t):
    return None if prop is None else prop[t]


def _step(ctx, cache, f, prompt, prop, pm, tau_m=0.0, override=None, tau_sim=(95, 100)):
    ovr = None if override is None else torch.tensor([override], dtype=torch.int8, device="cuda")
    out = ctx.step(cache, f, prompt, prop, tau_sim=tau_sim, tau_margin=tau_m, permille=pm, gate_override=ovr,
                   want=WANT)
    torch.cuda.synchronize()
    assert ctx.sync_error() == 0
    return {k: v.cpu() for k, v in out.items()}


def _same(a, b):
    for k in KEYS:
        assert torch.equal(a[k], b[k]), k


@pytest.mark.parametrize("name", ["small", "small_oft", "tiny"])
def test_reuse_nothing_equals_full(name, cuda_device):
    d, ctx, frames, prompt, prop = _setup(name)
    zero = np.zeros(d.n_layers, np.uint16)
    ca, cb = ctx.new_cache(1), ctx.new_cache(1)
    for c in (ca, cb):
        _step(ctx, c, frames[0], prompt, _pp(prop, 0), zero)
    a = _step(ctx, ca, frames[1], prompt, _pp(prop, 1), zero, override=0)
    b = _step(ctx, cb, frames[1], prompt, _pp(prop, 1), zero, override=1)
    assert a["recomputed"].item() == 0 and b["recomputed"].item() == 1
    assert a["idx"].tolist()[0] != list(range(d.pass_len))
    _same(a, b)
    assert torch.equal(ca.mem, cb.mem)


@pytest.mark.parametrize("name", ["tiny", "small", "small_oft"])
def test_identical_frames_with_reuse_equal_full(name, cuda_device):
    """Bitwise on both paths: the tensor-core GEMM sums every row in the same
    fp32 order (two accumulator chains, at most 256 rows per pass) whatever
    number of rows the pass recomputes, so a cached pass with few rows gives
    the full pass's values for the rows it recomputes."""
    d, ctx, frames, prompt, prop = _setup(name)
    pm = synth.linear_schedule(d.n_layers)
    ca, cb = ctx.new_cache(1), ctx.new_cache(1)
    for c in (ca, cb):
        _step(ctx, c, frames[0], prompt, _pp(prop, 0), pm, tau_sim=(996, 1000))
    a = _step(ctx, ca, frames[0], prompt, _pp(prop, 0), pm, override=0, tau_sim=(996, 1000))
    b = _step(ctx, cb, frames[0], prompt, _pp(prop, 0), pm, override=1, tau_sim=(996, 1000))
    assert a["recomputed"].item() == 0 and bool(a["static_mask"].all())
    _same(a, b)
    assert torch.equal(ca.mem, cb.mem)


@pytest.mark.parametrize("name", ["small", "small_oft"])
def test_gated_step_equals_reset_then_step(name, cuda_device):
    d, ctx, frames, prompt, prop = _setup(name)
    pm = synth.linear_schedule(d.n_layers)
    ca, cb = ctx.new_cache(1), ctx.new_cache(1)
    for c in (ca, cb):
        _step(ctx, c, frames[0], prompt, _pp(prop, 0), pm)
        _step(ctx, c, frames[1], prompt, _pp(prop, 1), pm)
    a = _step(ctx, ca, frames[2], prompt, _pp(prop, 2), pm, tau_m=float("inf"))
    ctx.reset(cb, 0)
    b = _step(ctx, cb, frames[2], prompt, _pp(prop, 2), pm, tau_m=0.0)
    assert a["recomputed"].item() == 1 and a["gate_auto"].item() == 1
    assert b["recomputed"].item() == 1
    _same(a, b)
    assert torch.equal(ca.mem, cb.mem)


def test_runs_are_deterministic(cuda_device):
    d, ctx, frames, prompt, prop = _setup("small_oft")
    pm = synth.linear_schedule(d.n_layers)
    outs = []
    for _ in range(2):
        c = ctx.new_cache(1)
        outs.append([_step(ctx, c, frames[t], prompt, _pp(prop, t), pm) for t in range(3)] + [c.mem.clone()])
    for t in range(3):
        _same(outs[0][t], outs[1][t])
    assert torch.equal(outs[0][3], outs[1][3])


def test_theta_zero_never_fires_and_infinity_always_fires(cuda_device):
    d, ctx, frames, prompt, prop = _setup("small")
    pm = synth.linear_schedule(d.n_layers)
    for tau_m, want in ((0.0, 0), (float("inf"), 1)):
        c = ctx.new_cache(1)
        for t in range(3):
            o = _step(ctx, c, frames[t], prompt, None, pm, tau_m=tau_m)
            assert o["recomputed"].item() == (1 if t == 0 else want)
            assert o["step_margin"].item() >= 0.0
