#!/usr/bin/env python
"""Throughput of the gated cached VLA step at the OpenVLA-7B shape.

One step = Algorithm 1 for one frame: gate, Stage-1 patch similarity,
Stage-3 selection, the partial (or full) 32-layer prefix pass, 6 decode
passes and the Eq. (1) margin.  Workload: a seeded 50-frame synthetic scene
episode (224x224 frames, 256 patches, 27 text tokens, 7 action tokens),
tau_sim = 0.996, reuse 0.9 -> 0.5 over the layers, tau_margin = 0.05;
random-init bf16 weights.  Episodes restart (cache reset) every 50 steps.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line (rank 0).  With N > 1 (torchrun), every rank runs an
independent replica on its own GPU with its own episode; there is no
collective on the data path.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "cached VLA steps/sec at OpenVLA-7B shape (1 GB300) and % of step roofline"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
EPISODE = 50
# frames per synthetic episode: the batched serving workload runs 200-frame episodes
EPISODE_LEN = {"batch7b": 200}
TAU_SWEEP = (0.0, 0.02, 0.05, 0.1, 0.2)
TAU_SIM = (996, 1000)
CPU_LAYERS = 2  # the CPU oracle sample runs this many of the 32 layers
# dram__bytes_read.sum + dram__bytes_write.sum of one dgemv_kernel launch,
# averaged over the four projections of a decode layer, from one ncu capture
# of the current kernel (profiles/dgemv_openvla7b_decode_layer.txt); the
# weights and launch shapes are the same in both single-sequence workloads.
# Reported only while the kernel is the one the counters were taken on.
DGEMV_TRAFFIC_PER_LAUNCH: dict = {c: 102.06e6 for c in ("openvla7b", "layer7b")}
DGEMV_TRAFFIC_NOTE = "ncu capture only for the 7B-shaped decode layer"
# The same counters for one persistent decode pass (dpass_kernel), per decoder
# layer it streams (profiles/dpass_openvla7b_decode.md): a launch of the
# one-layer 7B model; a launch over L layers moves L times as much.
DPASS_TRAFFIC_PER_LAYER: dict = {"7b": 409.85e6}


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return {k: float(j[k]) for k in FALLBACK_PEAKS}, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# ---------------------------------------------------------------------------
# Algorithmic work of one step (2 FLOPs per multiply-add)
# ---------------------------------------------------------------------------

def step_work(d, M_seq, idx_seq):
    """FLOPs and bytes one sequence's step must move, from its per-layer row
    counts M[l] and recompute order idx (what the method computes), per pass:
    a list of (flops, bytes other than weights, weight bytes)."""
    Hd, F, L, nb = d.hidden, d.ffn, d.n_layers, d.n_bins
    P, D = d.prefix_len, d.n_action
    M_seq = [int(m) for m in M_seq]
    idx_seq = np.asarray(idx_seq, dtype=np.int64)
    per_row = 2 * (4 * Hd * Hd + 3 * F * Hd)            # QKV + O + gate/up + down
    w_bytes = L * (4 * Hd * Hd + 3 * F * Hd) * 2        # bf16 weights of one pass
    head_bytes = nb * Hd * 2
    passes = []
    # prefix pass
    fp = 0.0
    bp = 0.0
    for l in range(L):
        rows = idx_seq[:M_seq[l]]
        fp += M_seq[l] * per_row + 4 * Hd * float(np.sum(rows + 1))   # QK^T and PV over j <= pos
        bp += 2 * d.pass_len * Hd * 2                                   # read K and V of the layer
        bp += M_seq[l] * 2 * Hd * 2                                     # write fresh K/V
        if l > 0:
            bp += max(M_seq[l - 1], M_seq[l]) * Hd * 4                  # record / reload layer inputs
    n_vis0 = int(np.sum((idx_seq[:M_seq[0]] >= 1) & (idx_seq[:M_seq[0]] <= d.n_visual)))
    fp += 2 * n_vis0 * d.patch_dim * Hd + 2 * nb * Hd * (D if d.parallel else 1)
    bp += 2 * d.n_views * d.img_h * d.img_w * 3
    passes.append((fp, bp, float(w_bytes + head_bytes + Hd * d.patch_dim * 2)))
    # autoregressive decode passes
    if not d.parallel:
        for a in range(1, D):
            pos = P + a - 1
            fd = L * (per_row + 4 * Hd * (pos + 1)) + 2 * nb * Hd
            bd = L * (2 * (pos + 1) * Hd * 2 + 2 * Hd * 2) + Hd * 2
            passes.append((fd, bd, float(w_bytes + head_bytes)))
    return passes


def layer_work(d, pos):
    """FLOPs and bytes of one decoder layer for rows at positions `pos` over
    a cache of d.cache_len positions (the one-layer workload): the layer's
    weights, the cache's K and V read, the rows' fresh K/V written and their
    fp32 inputs read and outputs written."""
    Hd, F = d.hidden, d.ffn
    pos = np.asarray(pos, dtype=np.int64)
    M = int(pos.size)
    flops = M * 2 * (4 * Hd * Hd + 3 * F * Hd) + 4 * Hd * float(np.sum(pos + 1))
    nbytes = (4 * Hd * Hd + 3 * F * Hd) * 2 + 2 * d.cache_len * Hd * 2 + M * 2 * Hd * 2 + 2 * M * Hd * 4
    return flops, nbytes


def run_layer_sweep(args, d):
    """The one-layer workload: per recomputed-row count M, the device time of
    one decoder layer (vlac_layer_bench) over a cache pre-filled with N(0, 1)
    values, averaged over --steps calls after --warmup, against the layer's
    roofline.  Prints one JSON line."""
    import torch

    from paper_2608_10824_gb300 import Context
    dev = torch.device("cuda", 0)
    w = synth.make_weights(d, seed=args.seed, device=dev, lm_head_rows=d.n_bins)
    ctx = Context(d, w, max_batch=1)
    del w
    torch.cuda.empty_cache()
    cache = ctx.new_cache(1)
    dt = torch.bfloat16 if d.dtype == "bf16" else torch.float32
    pk, src = peaks()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)   # 256 MB > L2, written between calls
    results = []
    for M in [m for m in (d.pass_len, 200, 120, 60, 30) if m <= d.pass_len]:
        pos, x, k0, v0 = synth.make_layer_case(d, M, seed=args.seed)
        ctx.cache_load(cache, 0, 0, torch.from_numpy(k0).to(dt).to(dev), torch.from_numpy(v0).to(dt).to(dev))
        pos_d = torch.from_numpy(pos).to(dev)
        x0 = torch.from_numpy(x).to(dev)
        xb = torch.empty_like(x0)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
        for i in range(args.warmup + args.steps):
            xb.copy_(x0)
            flush.fill_(i & 255)
            if i >= args.warmup:
                ev[i - args.warmup][0].record()
            ctx.layer_bench(cache, 0, 0, pos_d, xb)
            if i >= args.warmup:
                ev[i - args.warmup][1].record()
        torch.cuda.synchronize()
        assert ctx.sync_error() == 0
        ms = float(np.mean([a.elapsed_time(b) for a, b in ev]))
        f, b = layer_work(d, pos)
        t_roof = max(f / (pk["bf16_tflops"] * 1e12), b / (pk["hbm_gbs"] * 1e9))
        results.append({"M": M, "ms": ms, "roofline_ms": t_roof * 1e3, "frac": t_roof * 1e3 / ms,
                        "tflops": f / (ms / 1e3) / 1e12, "gbs": b / (ms / 1e3) / 1e9})
    print(json.dumps({"metric": "one decoder layer (7B shape) per recomputed-row count", "unit": "ms",
                      "workload": f"{args.config}: 1 layer, hidden {d.hidden}, {d.n_heads}x{d.head_dim} heads, "
                                  f"SwiGLU {d.ffn}, {d.pass_len}-position prefix pass, cache of {d.cache_len} "
                                  f"positions pre-filled N(0, 1), seeded sorted positions, inputs N(0, 1)",
                      "steps": args.steps, "warmup": args.warmup, "peaks": src, "l2": "256 MB written between calls",
                      "results": results}))


def batch_work(d, Ms, idxs):
    """(flops, bytes, per-pass [(flops, bytes)]) of one step of a batch: the
    sequences' own work adds up, the weights are read once per pass."""
    per_seq = [step_work(d, Ms[b], idxs[b]) for b in range(len(Ms))]
    passes = []
    for i in range(len(per_seq[0])):
        f = sum(ps[i][0] for ps in per_seq)
        b = sum(ps[i][1] for ps in per_seq) + per_seq[0][i][2]
        passes.append((f, b))
    return sum(p[0] for p in passes), sum(p[1] for p in passes), passes


# ---------------------------------------------------------------------------
# Clocks during the timed region
# ---------------------------------------------------------------------------

class Clocks:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, dev_index: int):
        self.p = None
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                                       "-lms", "200", "-i", str(dev_index)], stdout=subprocess.PIPE,
                                      stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        try:
            out, _ = self.p.communicate(timeout=5)
        except Exception:
            self.p.kill()
            out = ""
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() in ("active", "0x1", "1"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# CPU oracle sample (the cpu_baseline leg and the reference arm)
# ---------------------------------------------------------------------------

def oracle_sample(d, frames, prompt, prop, pm, tau_m, n_steps, seed, budget_s=None):
    """Times the CPU oracle on the first CPU_LAYERS layers of each step of the
    same episode and scales the step time by n_layers / CPU_LAYERS."""
    import torch

    import oracle
    ds = d.replace(n_layers=CPU_LAYERS, max_batch=1)
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    w = synth.make_weights(ds, seed=seed, device=dev, lm_head_rows=d.n_bins)
    w = synth.weights_to(w, "cpu")
    orc = oracle.Oracle(ds, w)
    cache = orc.new_cache(1)
    times = []
    t_begin = time.perf_counter()
    for t in range(n_steps):
        if t % EPISODE == 0:
            cache.reset()
        t0 = time.perf_counter()
        orc.step(cache, frames[t % EPISODE][:1], prompt[:1], None if prop is None else prop[t % EPISODE][:1],
                 tau_sim=TAU_SIM, tau_margin=tau_m, permille=pm[:CPU_LAYERS], want_logits=False)
        times.append((time.perf_counter() - t0) * d.n_layers / CPU_LAYERS)
        if budget_s is not None and time.perf_counter() - t_begin > budget_s:
            break
    return times


def cores_used():
    n = os.environ.get("OMP_NUM_THREADS")
    return int(n) if n else (os.cpu_count() or 1)


def run_reference(args, d, frames, prompt, prop, pm, rank):
    if rank != 0:
        return
    times = oracle_sample(d, frames, prompt, prop, pm, args.tau_margin, args.warmup + args.steps, seed=args.seed)
    timed = times[args.warmup:]
    total = sum(timed)
    v = len(timed) / total
    sample = (f"each step: the CPU oracle (fp64, plain C + OpenMP) runs the first {CPU_LAYERS} of "
              f"{d.n_layers} layers of the step (prefix pass and every decode pass), time scaled by "
              f"{d.n_layers}/{CPU_LAYERS}")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": "steps/s", "n_gpus": args.gpus,
        "steps": len(timed), "warmup": args.warmup, "ms_per_step": 1e3 * total / len(timed),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_block(d, args),
        "cpu_baseline": {"value": v, "unit": "steps/s", "cores": cores_used(), "kind": "oracle", "sample": sample},
        "e2e": {"value": v, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


# ---------------------------------------------------------------------------
# Replicas (N > 1): one process per GPU, each with its own episode; no
# collective on the data path, only the timing reduction
# ---------------------------------------------------------------------------

def replica_seed(seed: int, rank: int) -> int:
    """Each rank replays its own seeded episode."""
    return seed + rank


def reduce_max(value: float, dist, device) -> float:
    """The slowest rank's time (MAX over ranks); `dist` None means one rank."""
    if dist is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate_rate(world: int, B: int, K: int, seconds: float) -> float:
    """Whole-job sequence-steps per second: every rank ran K steps of B sequences."""
    return world * B * K / seconds


def config_block(d, args):
    vis = f"{d.n_views}x{d.img_h}x{d.img_w} frame(s) -> {d.n_visual} patches"
    act = (f"{d.n_action} parallel action positions" if d.parallel else f"{d.n_action} autoregressive action tokens")
    extra = f", {d.proprio_dim}-d proprio token" if d.proprio_dim else ""
    batch = (f", batch of {d.max_batch} episodes with blob speeds U[0, 8] px/frame" if d.max_batch > 1 else "")
    return {"workload": f"{args.config}: OpenVLA-7B-shaped Llama-2 backbone ({d.n_layers} layers, hidden {d.hidden}, "
                        f"{d.n_heads}x{d.head_dim} heads, SwiGLU {d.ffn}, vocab {d.vocab}, {d.n_bins} action bins), "
                        f"{vis}{extra}, {d.n_text} text tokens, {act}, {EPISODE}-frame scene episode{batch}",
            "global_batch": d.max_batch * args.gpus, "seq_len": d.pass_len, "parallelism": f"replicas x{args.gpus}",
            "tau_sim": f"{TAU_SIM[0]}/{TAU_SIM[1]}", "tau_margin": args.tau_margin,
            "reuse_permille": "linear 900 -> 500", "l2": "inputs larger than L2 (13 GB of weights per pass)",
            "stage2": (f"top_k {args.stage2_top_k} by the text-to-vision relevance of layer {stage2_layer(d, args)}"
                       if getattr(args, "stage2_top_k", 0) > 0 else "off")}


def stage2_layer(d, args) -> int:
    layer = getattr(args, "stage2_layer", None)
    return d.n_layers // 2 if layer is None else layer


# ---------------------------------------------------------------------------
# Our arm
# ---------------------------------------------------------------------------

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default="openvla7b")
    ap.add_argument("--tau-margin", type=float, default=0.05)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--cpu-budget", type=float, default=25.0, help="seconds of oracle work for cpu_baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--tau-sweep", action="store_true",
                    help="time K steps at every theta_m of the batched workload's sweep (0, .02, .05, .1, .2)")
    ap.add_argument("--layer-sweep", action="store_true",
                    help="time one decoder layer per recomputed-row count (the one-layer workload) instead")
    ap.add_argument("--stage2-top-k", type=int, default=0,
                    help="Stage 2 (task-relevant filtering): patches kept out of the reuse set; 0 = off")
    ap.add_argument("--stage2-layer", type=int, default=None, help="layer whose attention gives the relevance")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    global EPISODE
    EPISODE = EPISODE_LEN.get(args.config, EPISODE)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    d = synth.dims_for(args.config)
    if args.layer_sweep:
        run_layer_sweep(args, synth.dims_for("layer7b") if args.config == "openvla7b" else d)
        return
    seed = replica_seed(args.seed, rank)
    B = d.max_batch
    frames = synth.make_episode(d, EPISODE, seed=seed, batch=B, kind="scene",
                                speeds=synth.batch_speeds(B, seed=seed) if B > 1 else None)
    prompt = synth.make_prompt(d, seed=seed, batch=B)
    prop = synth.make_proprio(d, EPISODE, seed=seed, batch=B)   # None without a proprio token
    pm = synth.linear_schedule(d.n_layers)

    if args.impl == "reference":
        run_reference(args, d, frames, prompt, prop, pm, rank)
        return

    import torch
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    from paper_2608_10824_gb300 import Context

    dev = torch.device("cuda", local)
    w = synth.make_weights(d, seed=args.seed, device=dev)
    ctx = Context(d, w, max_batch=B)
    del w
    torch.cuda.empty_cache()
    cache = ctx.new_cache(B)
    fr_dev = torch.from_numpy(frames).to(dev)          # [T][B][views][H][W][3]
    pr_dev = torch.from_numpy(prompt).to(dev)
    pp_dev = None if prop is None else torch.from_numpy(np.ascontiguousarray(prop, np.float32)).to(dev)
    K, W = args.steps, args.warmup
    outs = ctx.alloc_outputs(B, want=("M", "idx", "gate_auto"))
    hist = {k: torch.zeros((K,) + tuple(v.shape), dtype=v.dtype, device=dev) for k, v in outs.items()}

    def one_step(t, out, tau=None):
        if t % EPISODE == 0:
            ctx.reset(cache)
        ctx.step(cache, fr_dev[t % EPISODE], pr_dev, None if pp_dev is None else pp_dev[t % EPISODE],
                 tau_sim=TAU_SIM, tau_margin=args.tau_margin if tau is None else tau, permille=pm, out=out,
                 s2_top_k=args.stage2_top_k, s2_layer=stage2_layer(d, args))

    def barrier():
        torch.cuda.synchronize()
        if dist is not None:
            dist.barrier()
            torch.cuda.synchronize()

    pk, src = peaks()
    stream = torch.cuda.current_stream()

    def timed_pass(t0, tau):
        """K steps from frame t0 at theta_m = tau, bracketed by barriers and
        CUDA events on the launching stream; returns (ms over ranks, launches,
        clocks, work)."""
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        clk = Clocks(local)
        time.sleep(0.3)
        n0 = ctx.launch_count()
        e0.record(stream)
        for k in range(K):
            one_step(t0 + k, {n: hist[n][k] for n in hist}, tau)
        e1.record(stream)
        barrier()
        clocks = clk.stop()
        launches = ctx.launch_count() - n0
        ms = reduce_max(e0.elapsed_time(e1), dist, dev)
        assert ctx.sync_error() == 0
        # algorithmic work of the timed steps
        Ms = hist["M"].cpu().numpy()           # [K][B][L]
        idxs = hist["idx"].cpu().numpy()       # [K][B][S]
        rec = hist["recomputed"].cpu().numpy()  # [K][B]
        F_tot = B_tot = gemm_flops = 0.0
        t_roof_step = t_roof_pass = 0.0
        per_row = 2 * (4 * d.hidden * d.hidden + 3 * d.ffn * d.hidden)
        for k in range(K):
            f_, b_, passes = batch_work(d, Ms[k], idxs[k])
            F_tot += f_
            B_tot += b_
            gemm_flops += float(Ms[k].sum()) * per_row
            t_roof_step += max(f_ / (pk["bf16_tflops"] * 1e12), b_ / (pk["hbm_gbs"] * 1e9))
            t_roof_pass += sum(max(fp / (pk["bf16_tflops"] * 1e12), bp / (pk["hbm_gbs"] * 1e9))
                               for fp, bp in passes)
        t_meas = ms / 1e3 / K
        roof = {"frac": t_roof_step / K / t_meas, "frac_per_pass": t_roof_pass / K / t_meas,
                "t_roof_ms": 1e3 * t_roof_step / K, "t_meas_ms": 1e3 * t_meas,
                "alg_tflop_per_step": F_tot / K / 1e12, "alg_gb_per_step": B_tot / K / 1e9,
                "peaks": src, "fire_rate": float(rec.mean())}
        return ms, launches, clocks, roof, gemm_flops

    for t in range(W):
        one_step(t, outs)
    barrier()
    assert ctx.sync_error() == 0
    # ---- timed region: device-resident inputs ----
    ms, launches, clocks, step_roof, gemm_flops = timed_pass(W, None)
    value = aggregate_rate(world, B, K, ms / 1e3)   # sequence-steps per second
    # ---- optionally: K more steps at every theta_m of the sweep ----
    sweep = None
    if args.tau_sweep:
        sweep = []
        for i, tau in enumerate(TAU_SWEEP):
            s_ms, _, s_clocks, s_roof, _ = timed_pass(W + K * (1 + i), tau)
            sweep.append({"tau_margin": tau, "value": aggregate_rate(world, B, K, s_ms / 1e3), "unit": "steps/s",
                          "ms_per_step": s_ms / K, "fire_rate": s_roof["fire_rate"], "step_roofline": s_roof,
                          "clocks": s_clocks})
    # ---- the same K frames once more at theta_m = 0: the gate never fires,
    # every step after the first of an episode takes the cached branch ----
    cached = None
    if args.tau_margin != 0.0 and not args.tau_sweep:
        c_ms, _, c_clocks, c_roof, _ = timed_pass(W + K, 0.0)
        cached = {"tau_margin": 0.0, "value": aggregate_rate(world, B, K, c_ms / 1e3), "unit": "steps/s",
                  "ms_per_step": c_ms / K, "step_roofline": c_roof, "clocks": c_clocks}

    # ---- per-kind device time, second pass with per-launch events ----
    ctx.prof_enable(True)
    for k in range(K):
        one_step(W + 2 * K + k, outs)
    barrier()
    ctx.prof_enable(False)
    g_ms, g_n, g_bytes = ctx.prof_read(0)
    p_ms, p_n, p_bytes = ctx.prof_read(1)
    kinds = ["decode_gemv", "prefix_gemm", "prefix_attn", "decode_attn", "prefix_rows", "head", "other"]
    breakdown = {"decode_gemv": g_ms / K, "prefix_gemm": p_ms / K}
    for i in range(2, len(kinds)):
        breakdown[kinds[i]] = ctx.prof_read(i)[0] / K
    gemv_gbs = g_bytes / (g_ms / 1e3) / 1e9 if g_ms > 0 else None
    gemm_gbs = p_bytes / (p_ms / 1e3) / 1e9 if p_ms > 0 else None
    gemm_tfs = gemm_flops / (p_ms / 1e3) / 1e12 if p_ms > 0 else None
    # one launch per decode token: the persistent decode pass ran (bf16,
    # head_dim 128, one or two sequences); else one per projection
    persistent = 0 < g_n <= K * max(1, d.n_action - 1)
    if g_n and persistent:
        # the persistent pass (weights of every layer + attention) dominates
        per_layer = DPASS_TRAFFIC_PER_LAYER.get("7b") if d.hidden == 4096 and d.ffn == 11008 else None
        roof = {"bound": "hbm", "achieved": gemv_gbs, "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": gemv_gbs / pk["hbm_gbs"], "traffic": None if per_layer is None else per_layer * d.n_layers,
                "kernel": "dpass_kernel (persistent decode pass: every layer's weight stream and attention)",
                "launches": g_n, "avg_launch_us": 1e3 * g_ms / g_n, "peak_source": f"{src} hbm_gbs",
                **({} if per_layer is not None else {"traffic_note": "no ncu capture of this kernel at this shape"})}
    elif g_n:
        # weight streaming of the decode passes dominates the step
        roof = {"bound": "hbm", "achieved": gemv_gbs, "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": gemv_gbs / pk["hbm_gbs"], "traffic": DGEMV_TRAFFIC_PER_LAUNCH.get(args.config),
                "kernel": "dgemv_kernel (decode weight streaming)", "launches": g_n,
                **({} if args.config in DGEMV_TRAFFIC_PER_LAUNCH else {"traffic_note": DGEMV_TRAFFIC_NOTE}),
                "avg_launch_us": 1e3 * g_ms / g_n, "peak_source": f"{src} hbm_gbs"}
    else:
        # no decode passes: the prefix GEMMs (tensor cores) dominate
        roof = {"bound": "tensor", "achieved": gemm_tfs, "peak": pk["bf16_tflops_sustained"], "unit": "TFLOP/s",
                "frac": gemm_tfs / pk["bf16_tflops_sustained"], "traffic": None,
                "kernel": "gemm_tc_kernel (tcgen05 prefix projections)", "launches": p_n,
                "avg_launch_us": 1e3 * p_ms / max(p_n, 1), "peak_source": f"{src} bf16_tflops_sustained"}

    # ---- end to end through the public API with host buffers ----
    fr_host = torch.from_numpy(frames).pin_memory()
    pr_host = torch.from_numpy(prompt).pin_memory()
    pp_host = None if pp_dev is None else pp_dev.cpu().pin_memory()
    f_buf = torch.empty_like(fr_dev[0])
    p_buf = torch.empty_like(pr_dev)
    q_buf = None if pp_dev is None else torch.empty_like(pp_dev[0])
    res_host = {n: torch.empty(outs[n].shape, dtype=outs[n].dtype).pin_memory()
                for n in ("action_ids", "margins", "recomputed", "step_margin")}
    h2d = f_buf.numel() * f_buf.element_size() + p_buf.numel() * p_buf.element_size()
    if q_buf is not None:
        h2d += q_buf.numel() * q_buf.element_size()
    d2h = sum(v.numel() * v.element_size() for v in res_host.values())
    barrier()
    t0 = time.perf_counter()
    for k in range(K):
        t = W + 3 * K + k
        f_buf.copy_(fr_host[t % EPISODE], non_blocking=True)
        p_buf.copy_(pr_host, non_blocking=True)
        if q_buf is not None:
            q_buf.copy_(pp_host[t % EPISODE], non_blocking=True)
        if t % EPISODE == 0:
            ctx.reset(cache)
        ctx.step(cache, f_buf, p_buf, q_buf, tau_sim=TAU_SIM, tau_margin=args.tau_margin, permille=pm, out=outs,
                 s2_top_k=args.stage2_top_k, s2_layer=stage2_layer(d, args))
        for n, hbuf in res_host.items():
            hbuf.copy_(outs[n], non_blocking=True)
        torch.cuda.current_stream().synchronize()  # the action is needed before the next frame
    e2e_s = reduce_max(time.perf_counter() - t0, dist, dev)
    e2e = aggregate_rate(world, B, K, e2e_s)

    # ---- CPU oracle baseline (rank 0, N = 1 only) ----
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        times = oracle_sample(d, frames, prompt, prop, pm, args.tau_margin, 10 ** 6, seed=args.seed,
                              budget_s=args.cpu_budget)
        cpu = {"value": len(times) / sum(times), "unit": "steps/s", "cores": cores_used(), "kind": "oracle",
               "sample": f"{len(times)} steps of the first sequence's episode; the oracle runs the first "
                         f"{CPU_LAYERS} of {d.n_layers} layers of each step, time scaled by "
                         f"{d.n_layers}/{CPU_LAYERS}"}

    if rank != 0:
        return
    line = {
        "metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": ms / K, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic (seeded scene frames, random-init N(0,0.02) bf16 weights)",
        "config": config_block(d, args),
        "step_roofline": step_roof,
        "cached_branch": cached,
        "tau_sweep": sweep,
        "roofline": roof,
        "prefix_gemm": {"weight_gbs": gemm_gbs, "tflops": gemm_tfs, "launches": p_n,
                        "avg_launch_us": 1e3 * p_ms / max(p_n, 1)},
        "device_ms_per_step_by_kind": {k: round(v, 4) for k, v in breakdown.items()},
        "by_kind_note": (f"per-launch CUDA events in a second, non-graph pass of the same K steps serialise the "
                         f"launches: the kinds sum to {sum(breakdown.values()):.2f} ms per step against "
                         f"{ms / K:.2f} ms of graph replay in the timed pass"
                         + ("; decode_gemv is the persistent decode pass, which also runs the decode attention"
                            if persistent else "")),
        "clocks": clocks,
        "e2e": {"value": e2e, "unit": "steps/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "note": "frames + prompt (+ proprio) H2D from pinned memory, action ids/margins/flags D2H, "
                        "synchronised every step (closed loop)"},
        "gpu_launches": int(launches),
        "cpu_baseline": cpu,
    }
    if B > 1:
        line["unit_note"] = f"steps/s counts sequence-steps: {B} sequences per batched step"
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
