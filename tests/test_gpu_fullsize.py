"""Parity at the full workload sizes: the OpenVLA-7B shape (32 layers, hidden
4096, 283-token prefix, 7 autoregressive action tokens), the OpenVLA-OFT shape
(two views, proprio, 56 parallel action positions: 596 rows, three GEMM passes)
and the batch of 8 sequences, against the fp64 oracle on the host.

The steps run in the launch configuration the benchmark times.  Selection,
recompute flags and action ids (outside the exemption) must match exactly;
the logits within LOGIT_TOL_DEEP, twice the spread measured between two runs
of the GPU path that differ only in the fp32 summation order of their GEMM
partial sums (test_summation_order_floor).  The oracle
takes several seconds per 7B step, so each episode is short and covers both
branches: a full pass (empty cache) and a cached step (theta_m = 0); the
OpenVLA-7B episode then lets the gate fire (theta_m = +inf) and runs one more
cached step.  Every step prints its largest logit difference.  For the
batch, the oracle runs two of the eight sequences (the sequences of a batch
are independent), and their outputs are compared with those rows of the batch.
"""
import gc

import numpy as np
import pytest

import synth
from tests.gpu_common import FLAG_TIE_DEEP, LOGIT_TOL_DEEP, Lockstep, compare

pytestmark = [pytest.mark.gpu, pytest.mark.timeout(1800)]


def _weights(d, seed):
    w_gpu = synth.make_weights(d, seed=seed, device="cuda")
    return synth.weights_to(w_gpu, "cpu"), w_gpu


def _run_lockstep(name, taus, seed):
    """One lock-step episode, theta_m per frame from `taus`; returns the
    branch each step ran."""
    d = synth.dims_for(name)
    n_frames = len(taus)
    w_cpu, w_gpu = _weights(d, seed)
    ls = Lockstep(d, w_cpu, w_gpu, logit_tol=LOGIT_TOL_DEEP)
    del w_gpu
    frames = synth.make_episode(d, n_frames, seed=seed, kind="scene")
    prompt = synth.make_prompt(d, seed=seed)
    prop = synth.make_proprio(d, n_frames, seed=seed)
    pm = synth.linear_schedule(d.n_layers)
    branches = []
    for t in range(n_frames):
        o, g, rep = ls.step(frames[t], prompt, None if prop is None else prop[t], (996, 1000), taus[t], pm)
        branches.append(int(o["recomputed"][0]))
        print(f"{name} frame {t}: recomputed {branches[-1]}, max logit diff {rep['max_logit_diff']:.4e}, "
              f"median {rep['median_logit_diff']:.4e}, id mismatches {rep['id_mismatch']}")
        if not branches[-1]:  # a cached step reused static patches at every layer
            assert g["M"][0].max() < d.pass_len
    del ls
    gc.collect()
    return branches


def test_openvla7b_parity(cuda_device):
    """Full pass (empty cache), cached step (theta_m = 0 never fires), the
    gate firing after a cached step (theta_m = +inf, Algorithm 1), and a
    cached step after the gated one."""
    inf = float("inf")
    assert _run_lockstep("openvla7b", [0.0, 0.0, inf, 0.0], seed=11) == [1, 0, 1, 0]


def test_oft7b_parity(cuda_device):
    assert _run_lockstep("oft7b", [0.0, 0.0], seed=12) == [1, 0]


@pytest.mark.parametrize("tau_m", [0.0, 0.02, 0.05, 0.1, 0.2])
def test_batch7b_sampled_parity(cuda_device, tau_m):
    """The batch of 8 at every theta_m of its sweep: the oracle runs two of the
    eight sequences over the first frames (the parity window), the library
    the whole batch.  The sampled sequences take the oracle's branch on both
    sides; their gate's own decision must match the oracle's wherever the
    oracle's m_{t-1} lies outside FLAG_TIE_DEEP of theta_m."""
    import torch

    import oracle
    from paper_2608_10824_gb300 import Context
    d = synth.dims_for("batch7b")
    B, pick = d.max_batch, [0, 5]
    w_cpu, w_gpu = _weights(d, 13)
    n = 3 if tau_m == 0.0 else 2
    frames = synth.make_episode(d, n, seed=13, batch=B, kind="scene", speeds=synth.batch_speeds(B, seed=13))
    prompt = synth.make_prompt(d, seed=13, batch=B)
    pm = synth.linear_schedule(d.n_layers)
    ctx = Context(d, w_gpu, max_batch=B)
    del w_gpu
    cache, probe = ctx.new_cache(B), ctx.new_cache(B)
    orc = oracle.Oracle(d, w_cpu)
    oc = orc.new_cache(len(pick))
    fr = [torch.from_numpy(np.ascontiguousarray(f)).cuda() for f in frames]
    pr = torch.from_numpy(np.ascontiguousarray(prompt)).cuda()
    want = ("gate_auto", "logits", "static_mask", "idx", "M")
    prev_m = None
    branches = []
    for t in range(n):
        o = orc.step(oc, frames[t][pick], prompt[pick], tau_sim=(996, 1000), tau_margin=tau_m, permille=pm)
        # the sampled sequences take the oracle's branch (their own gate
        # decision is still compared, outside the deep tie band); the others
        # follow their own gate
        ovr = torch.full((B,), -1, dtype=torch.int8)
        for i, b in enumerate(pick):
            ovr[b] = int(o["recomputed"][i])
        ovr = ovr.cuda()
        # the decoded bins are fed back, so the sampled rows take the oracle's
        # bins and the others their own: a copy of the cache runs the step
        # first to find those
        probe.mem.copy_(cache.mem)
        own = ctx.step(probe, fr[t], pr, tau_sim=(996, 1000), tau_margin=tau_m, permille=pm,
                       gate_override=ovr)["action_ids"]
        forced = own.clone()
        forced[pick] = torch.from_numpy(o["action_ids"].astype(np.int32)).cuda()
        g = ctx.step(cache, fr[t], pr, tau_sim=(996, 1000), tau_margin=tau_m, permille=pm, forced_ids=forced,
                     gate_override=ovr, want=want)
        torch.cuda.synchronize()
        assert ctx.sync_error() == 0
        g = {k: v.cpu().numpy()[pick] for k, v in g.items()}
        rep = compare(d, o, g, prev_m, tau_m, LOGIT_TOL_DEEP, FLAG_TIE_DEEP)
        branches.append(o["recomputed"].tolist())
        print(f"batch7b tau {tau_m} frame {t}: recomputed {branches[-1]}, max logit diff "
              f"{rep['max_logit_diff']:.4e}, median {rep['median_logit_diff']:.4e}, "
              f"id mismatches {rep['id_mismatch']}")
        prev_m = o["step_margin"].copy()
    assert branches[0] == [1, 1]
    if tau_m == 0.0:
        assert all(b == [0, 0] for b in branches[1:])
    del ctx, cache, probe, orc
    gc.collect()


def test_summation_order_floor(cuda_device):
    """The bar of the deep tests: two GPU runs of one full 7B step that differ
    only in the split-K summation order already differ by a few 1e-2 in the
    logits; the oracle's distance is of the same size and within the bar."""
    import os

    import torch

    import oracle
    from paper_2608_10824_gb300 import Context
    d = synth.dims_for("openvla7b")
    w_cpu, w_gpu = _weights(d, 11)
    frames = synth.make_episode(d, 1, seed=11, kind="scene")
    prompt = synth.make_prompt(d, seed=11)
    pm = synth.linear_schedule(d.n_layers)
    orc = oracle.Oracle(d, w_cpu)
    o = orc.step(orc.new_cache(1), frames[0], prompt, tau_sim=(996, 1000), tau_margin=0.0, permille=pm)
    forced = torch.from_numpy(o["action_ids"].astype(np.int32)).cuda()
    logits = []
    old = os.environ.get("VLAC_SPLITS")
    try:
        for sp in ("1,4,1,4", "8,8,8,8"):
            os.environ["VLAC_SPLITS"] = sp
            ctx = Context(d, w_gpu, max_batch=1)
            g = ctx.step(ctx.new_cache(1), torch.from_numpy(frames[0]).cuda(), torch.from_numpy(prompt).cuda(),
                         tau_sim=(996, 1000), tau_margin=0.0, permille=pm, forced_ids=forced, want=("logits",))
            torch.cuda.synchronize()
            logits.append(g["logits"].cpu().numpy().astype(np.float64))
            del ctx
    finally:
        if old is None:
            os.environ.pop("VLAC_SPLITS", None)
        else:
            os.environ["VLAC_SPLITS"] = old
    floor = np.abs(logits[0] - logits[1]).max()
    dist = max(np.abs(lg - o["logits"]).max() for lg in logits)
    print(f"summation-order floor {floor:.4e}, oracle distance {dist:.4e}")
    assert 2e-3 < floor <= LOGIT_TOL_DEEP / 2, floor
    assert dist <= LOGIT_TOL_DEEP, (dist, floor)
    del w_gpu
    gc.collect()
