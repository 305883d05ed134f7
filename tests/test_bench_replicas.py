"""bench.py with N > 1: one replica per rank, each on its own seeded episode,
no collective on the data path; the timed region's duration is the slowest
rank's, and the rate counts every rank's sequence-steps.  Run here as two
gloo ranks on the CPU (the GPU run uses NCCL with the same helpers)."""
import json
import os
import socket
import sys
import types

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist

    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r "took" 10 * (r + 1) ms; every rank must see the slowest
        ms = bench.reduce_max(10.0 * (rank + 1), dist, torch.device("cpu"))
        q.put((rank, ms, bench.replica_seed(7, rank), bench.aggregate_rate(world, 2, 5, ms / 1e3)))
    finally:
        dist.destroy_process_group()


def test_two_replicas_reduce_to_the_slowest_rank():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    try:
        res = sorted(q.get(timeout=120) for _ in procs)
    finally:
        for p in procs:
            p.join(timeout=60)
    assert [p.exitcode for p in procs] == [0, 0]
    (r0, ms0, s0, v0), (r1, ms1, s1, v1) = res
    assert (r0, r1) == (0, 1)
    assert ms0 == ms1 == 20.0            # MAX over ranks
    assert s0 != s1                      # each replica replays its own episode
    assert v0 == v1 == pytest.approx(2 * 2 * 5 / 0.020)  # whole-job sequence-steps per second


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max(3.5, None, None) == 3.5
    assert bench.replica_seed(7, 0) == 7
    assert bench.aggregate_rate(1, 8, 10, 2.0) == 40.0


def test_reference_arm_runs_on_rank_zero_only(capsys):
    """Under torchrun the reference arm's other ranks exit without work."""
    sys.path.insert(0, ROOT)
    import bench
    import synth
    d = synth.dims_for("tiny")
    args = types.SimpleNamespace(tau_margin=0.0, warmup=3, steps=1, gpus=2, config="tiny", seed=0)
    bench.run_reference(args, d, None, None, None, None, rank=1)
    assert capsys.readouterr().out == ""


def test_bench_line_fields_are_json_serialisable():
    """The config block a rank prints is plain JSON."""
    sys.path.insert(0, ROOT)
    import bench
    import synth
    d = synth.dims_for("openvla7b")
    args = types.SimpleNamespace(tau_margin=0.05, gpus=1, config="openvla7b")
    block = bench.config_block(d, args)
    assert json.loads(json.dumps(block)) == block
    assert "workload" in block
