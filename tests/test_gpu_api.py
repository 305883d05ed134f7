"""Error behaviour of the C-ABI on a GPU: documented status codes for bad
arguments and bounded device waits (a wait that nothing completes gives up,
records VLAC_ERR_TIMEOUT and leaves the context usable)."""
import numpy as np
import pytest
import torch

import synth
from tests.gpu_common import SMALL, episode

pytestmark = pytest.mark.gpu


def _ctx(name="small"):
    from paper_2608_10824_gb300 import Context
    d = SMALL[name]
    return d, Context(d, synth.weights_to(synth.make_weights(d, seed=1), "cuda"), max_batch=2)


def test_bounded_wait_gives_up_and_context_stays_usable(cuda_device):
    from paper_2608_10824_gb300.vlac import ERRORS
    d, ctx = _ctx()
    rc = ctx.selftest_wait(1000)
    assert ERRORS[rc] == "VLAC_ERR_TIMEOUT"
    frames, prompt, _ = episode(d, 1, seed=2)
    c = ctx.new_cache(1)
    out = ctx.step(c, torch.from_numpy(frames[0]).cuda(), torch.from_numpy(prompt).cuda())
    torch.cuda.synchronize()
    assert ctx.sync_error() == 0
    assert out["recomputed"].item() == 1


def test_invalid_arguments(cuda_device):
    from paper_2608_10824_gb300 import VlacError
    d, ctx = _ctx()
    frames, prompt, _ = episode(d, 1, seed=2)
    f, p = torch.from_numpy(frames[0]).cuda(), torch.from_numpy(prompt).cuda()
    c = ctx.new_cache(1)
    with pytest.raises(VlacError) as e:
        ctx.step(c, f, p, permille=np.full(d.n_layers, 1001, np.uint16))
    assert e.value.code == -1
    with pytest.raises(VlacError) as e:
        ctx.step(c, f, p, tau_sim=(1, 0))
    assert e.value.code == -1
    with pytest.raises(VlacError) as e:
        ctx.new_cache(3)  # above max_batch
    assert e.value.code == -1
    with pytest.raises(VlacError) as e:
        ctx.reset(c, 1)  # out-of-range sequence
    assert e.value.code == -1
    # a cache of another context is a state error
    d2, ctx2 = _ctx()
    with pytest.raises(VlacError) as e:
        ctx2.step(c, f, p)
    assert e.value.code == -6


def test_bad_prompt_id_is_a_device_check(cuda_device):
    d, ctx = _ctx()
    frames, prompt, _ = episode(d, 1, seed=2)
    bad = prompt.copy()
    bad[0, 3] = d.vocab + 5
    c = ctx.new_cache(1)
    ctx.step(c, torch.from_numpy(frames[0]).cuda(), torch.from_numpy(bad).cuda())
    torch.cuda.synchronize()
    assert ctx.sync_error() == -5
    assert ctx.sync_error() == 0  # cleared once reported


def test_unsupported_dims():
    from paper_2608_10824_gb300 import VlacError
    from paper_2608_10824_gb300.vlac import Context
    d = SMALL["small"].replace(head_dim=96, n_heads=2, hidden=192)
    with pytest.raises(VlacError) as e:
        Context(d, synth.weights_to(synth.make_weights(d, seed=1), "cuda"))
    assert e.value.code in (-7, -1)


@pytest.mark.parametrize("path", ["dpass", "chain"])
@pytest.mark.parametrize("polls", [0, 1])
def test_step_kernels_give_up_and_the_context_stays_usable(cuda_device, monkeypatch, polls, path):
    """The prefix GEMM's, the prefix attention's and the decode path's bounded
    waits (the persistent pass's ring, K/V staging and grid-barrier waits, or
    the chain's GEMV ring waits), run out on purpose (0 polls: every wait
    gives up at once; 1 poll: wherever a copy has not landed by the first
    poll): the step latches VLAC_ERR_TIMEOUT (or, with 1 poll, may happen to
    finish), nothing hangs or faults, and a normal step on a new cache of the
    same context then matches the oracle."""
    from paper_2608_10824_gb300.vlac import ERRORS
    from tests.gpu_common import Lockstep
    monkeypatch.setenv("VLAC_DPASS", "1" if path == "dpass" else "0")
    d = SMALL["small"]
    w = synth.make_weights(d, seed=5)
    ls = Lockstep(d, w)
    frames, prompt, _ = episode(d, 2, seed=5)
    f, p = torch.from_numpy(frames[0]).cuda(), torch.from_numpy(prompt).cuda()
    ls.ctx.set_wait_limit(polls)
    c = ls.ctx.new_cache(1)
    ls.ctx.step(c, f, p)
    torch.cuda.synchronize()
    rc = ls.ctx.sync_error()
    assert ERRORS.get(rc) == "VLAC_ERR_TIMEOUT" or (polls > 0 and rc == 0), rc
    ls.ctx.set_wait_limit(1 << 24)
    # the lock-step cache is a fresh one of the same context
    for t in range(2):
        ls.step(frames[t], prompt, None, (95, 100), 0.0, synth.linear_schedule(d.n_layers))


@pytest.mark.parametrize("n", [1, 2, 3, 4])
def test_allocation_failure_is_reported_and_leaks_nothing(cuda_device, monkeypatch, n):
    """Host-side fault injection: the n-th allocation of vlac_create fails as
    cudaMalloc would (VLAC_FAIL_ALLOC, no GPU fault involved).  The call
    returns VLAC_ERR_OOM, frees what it had allocated, and the next create on
    the same device works."""
    from paper_2608_10824_gb300 import Context, VlacError
    d = SMALL["small"]
    w = synth.weights_to(synth.make_weights(d, seed=7), "cuda")
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    monkeypatch.setenv("VLAC_FAIL_ALLOC", str(n))
    with pytest.raises(VlacError) as e:
        Context(d, w, max_batch=1)
    assert e.value.code == -3
    torch.cuda.synchronize()
    assert abs(torch.cuda.mem_get_info()[0] - free0) < (32 << 20)
    monkeypatch.delenv("VLAC_FAIL_ALLOC")
    ctx = Context(d, w, max_batch=1)
    frames, prompt, _ = episode(d, 1, seed=7)
    out = ctx.step(ctx.new_cache(1), torch.from_numpy(frames[0]).cuda(), torch.from_numpy(prompt).cuda())
    torch.cuda.synchronize()
    assert ctx.sync_error() == 0 and out["recomputed"].item() == 1


def test_a_copied_cache_resumes_the_episode(cuda_device):
    """The cache is the step's whole resumable state and lives in caller
    memory: copying its bytes into a new cache of the same context (a
    checkpoint) and stepping both gives the same outputs bit for bit."""
    from paper_2608_10824_gb300 import Context
    d = SMALL["small_oft"]
    ctx = Context(d, synth.weights_to(synth.make_weights(d, seed=8), "cuda"), max_batch=1)
    frames, prompt, prop = episode(d, 5, seed=8)
    f = [torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in frames]
    p = torch.from_numpy(prompt).cuda()
    pp = [torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in prop]
    pm = synth.linear_schedule(d.n_layers)
    a = ctx.new_cache(1)
    for t in range(3):
        ctx.step(a, f[t], p, pp[t], permille=pm)
    torch.cuda.synchronize()
    b = ctx.new_cache(1)
    b.mem.copy_(a.mem)
    for t in (3, 4):
        oa = ctx.step(a, f[t], p, pp[t], permille=pm, want=("logits", "idx"))
        ob = ctx.step(b, f[t], p, pp[t], permille=pm, want=("logits", "idx"))
        torch.cuda.synchronize()
        for k in ("action_ids", "margins", "logits", "idx", "step_margin", "recomputed"):
            assert torch.equal(oa[k], ob[k]), (t, k)
    assert ctx.sync_error() == 0
    assert torch.equal(a.mem, b.mem)
