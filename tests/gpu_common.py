"""Shared pieces of the GPU parity tests: small workloads the oracle finishes
in seconds, and a lock-step driver that runs the oracle and the CUDA library
on the same seeded inputs and compares every step."""
from __future__ import annotations

import numpy as np

import synth

# Tolerances.  Logits: the stated bar for bf16 weights is abs 2e-2; the fp32
# model is held to 1e-3.  Action ids may differ only where the oracle's
# probability margin p1 - p2 is below 1e-3.  Flags may differ only where the
# oracle's m_{t-1} is within 1e-4 of theta_m (the step is then re-synced by
# forcing the oracle's branch).
LOGIT_TOL = {"bf16": 2e-2, "f32": 1e-3}
# Full 32-layer 7B shapes: two runs of the GPU path that differ only in the
# fp32 summation order of the GEMM partial sums differ by up to 4.2e-2 in the
# logits (the bf16 re-rounding of every layer's GEMM inputs amplifies any
# fp32-level difference; the figure moves with every change of summation
# order, 3.4e-2 to 4.2e-2 so far), so the bar there is about twice the
# largest measured floor.
LOGIT_TOL_DEEP = 1e-1
ID_EXEMPT_MARGIN = 1e-3
# At that depth an argmax flips wherever the oracle's two candidate logits
# are closer than the logit error can move them apart: with every logit
# within LOGIT_TOL_DEEP, a differing id is only possible where the oracle's
# logit for its own bin exceeds its logit for the GPU's bin by less than
# twice the bar.  The deep tests exempt exactly those ids, and require the
# GPU's id to be the first maximum of the GPU's own logits.
FLAG_TIE = 1e-4
# At 32 layers the margins are held to 0.05 x LOGIT_TOL_DEEP (see compare), so
# the library's m_{t-1} may sit on the other side of theta_m wherever the
# oracle's lies within that band of it.
FLAG_TIE_DEEP = 0.05 * LOGIT_TOL_DEEP
# Stage 2 relevance, relative to the sequence's largest relevance.  At layer
# 0 the kernel sums fp32 probabilities of the same bf16 (or fp32) Q and K the
# oracle sums in fp64 (REL_TOL).  At a deeper layer of a bf16 model Q and K
# also carry the earlier layers' GEMM-input roundings (a bf16 flip moves a
# score by up to 2^-8 of one of its terms), so the probabilities move by the
# score error rather than by fp32 rounding: REL_TOL_DEEP, about three times
# the largest distance measured on the small models (6.1e-4 at layer 1).
# A removal-set difference is allowed only for patches whose oracle relevance
# lies within twice the bar of the oracle's k-th / (k+1)-th midpoint.
REL_TOL = {"bf16": 1e-4, "f32": 1e-5}
REL_TOL_DEEP = {"bf16": 2e-3, "f32": 1e-5}
# Stage 3 adaptive: a layer's normalized attention entropy is a mean of
# functions of the same softmax probabilities the relevance sums, so it is held
# to the deep relevance bar (absolute: the entropy is already normalized to 1).
ENT_TOL = {"bf16": 2e-3, "f32": 1e-5}
# Entropy of the bin softmax: H moves by at most max_j |l_j - E_p[l]| per unit
# of logit error, about 5 for these models' logit spread, so the bar is five
# times the logit bar; the library's entropy must also match the entropy of
# its own logits to fp32 rounding.
ENTROPY_FACTOR = 5.0

SMALL = {
    # bf16 path (tcgen05 GEMMs), head_dim 128, autoregressive decode
    "small": synth.Dims(n_layers=2, hidden=256, n_heads=2, head_dim=128, ffn=768, vocab=1024, n_bins=256,
                        img_h=112, img_w=112, patch=14, n_views=1, n_text=8, proprio_dim=0, n_action=7,
                        parallel=0, dtype="bf16"),
    # bf16, two 224x224 views + proprio + 56-position parallel block: 596 rows (> 384: three GEMM passes)
    "small_oft": synth.Dims(n_layers=2, hidden=256, n_heads=4, head_dim=64, ffn=512, vocab=512, n_bins=256,
                            img_h=224, img_w=224, patch=14, n_views=2, n_text=27, proprio_dim=8, n_action=56,
                            parallel=1, dtype="bf16"),
    # bf16, batch of three sequences with ragged recompute sets
    "small_batch": synth.Dims(n_layers=2, hidden=256, n_heads=2, head_dim=128, ffn=768, vocab=1024, n_bins=256,
                              img_h=112, img_w=112, patch=14, n_views=1, n_text=8, proprio_dim=0, n_action=7,
                              parallel=0, dtype="bf16", max_batch=3),
    # bf16, MLP width 4160: the down-projection's K (4160) spans three
    # 2048-element decode-GEMV chunks (the last one 64 elements); two sequences
    "small_wide": synth.Dims(n_layers=2, hidden=256, n_heads=2, head_dim=128, ffn=4160, vocab=1024, n_bins=256,
                             img_h=112, img_w=112, patch=14, n_views=1, n_text=8, proprio_dim=0, n_action=7,
                             parallel=0, dtype="bf16", max_batch=2),
    # bf16, hidden 2304 (18 x 128 heads), MLP width 4608: every decode GEMV's K
    # spans two or three 2048-element chunks (the last one partial), and the
    # decode projections have more row groups than a GB300 has SMs
    "wide": synth.Dims(n_layers=2, hidden=2304, n_heads=18, head_dim=128, ffn=4608, vocab=1024, n_bins=256,
                       img_h=112, img_w=112, patch=14, n_views=1, n_text=8, proprio_dim=0, n_action=7,
                       parallel=0, dtype="bf16", max_batch=2),
    # fp32 tiny model (SIMT path)
    "tiny": synth.dims_for("tiny"),
}


def episode(d, n_frames: int, seed: int, batch: int = 1, kind=None):
    frames = synth.make_episode(d, n_frames, seed=seed, batch=batch, kind=kind)
    prompt = synth.make_prompt(d, seed=seed, batch=batch)
    prop = synth.make_proprio(d, n_frames, seed=seed, batch=batch)
    return frames, prompt, prop


class Lockstep:
    """Runs the oracle and the library side by side, one step at a time."""

    def __init__(self, d, w_cpu, w_gpu=None, batch: int = 1, logit_tol=None):
        import torch

        import oracle
        from paper_2608_10824_gb300 import Context
        self.d, self.B = d, batch
        if w_gpu is None:
            w_gpu = synth.weights_to(w_cpu, "cuda")
        self.orc = oracle.Oracle(d, w_cpu)
        self.oc = self.orc.new_cache(batch)
        self.ctx = Context(d, w_gpu, max_batch=batch)
        self.gc = self.ctx.new_cache(batch)
        self.torch = torch
        self.prev_m = None
        self.prev_rel = None
        self.prev_ids = None
        self.prev_ent = None
        self.log = []
        self.logit_tol = logit_tol

    def step(self, frames, prompt, proprio, tau_sim, tau_m, permille, margin_kind=0, force_branch=None,
             active=None, s2_top_k=0, s2_layer=None, s2_lockstep=True, want_vocab=False, s3=None,
             s3_lockstep=True):
        """active: uint8 [B], 0 = the sequence sits the step out (both sides).
        s2_top_k > 0: Stage 2 on both sides; with s2_lockstep the library
        applies the oracle's removal set (its own is still compared).
        want_vocab: also the whole-vocabulary margin (always with margin kind 2).
        s3 = (lo, hi, weight): the entropy-adaptive Stage 3 on both sides; with
        s3_lockstep the library applies the oracle's schedule (its own is
        still compared)."""
        torch = self.torch
        d, B = self.d, self.B
        act = None if active is None else np.ascontiguousarray(active, np.uint8)
        vocab = want_vocab or margin_kind == 2
        if s2_layer is None:
            s2_layer = d.n_layers // 2
        o = self.orc.step(self.oc, frames, prompt, proprio, tau_sim=tau_sim, tau_margin=tau_m,
                          permille=permille, margin_kind=margin_kind,
                          gate_override=None if force_branch is None else np.full(B, force_branch, np.int8),
                          active=act, s2_top_k=s2_top_k, s2_layer=s2_layer, want_vocab_margin=vocab,
                          s3_adaptive=s3)
        # branch: free-running, except where the oracle's m_{t-1} sits in the tie zone
        ovr = np.full(B, -1, np.int8) if force_branch is None else np.full(B, force_branch, np.int8)
        if self.prev_m is not None and force_branch is None:
            tie = np.abs(self.prev_m - tau_m) < FLAG_TIE
            ovr[tie] = o["recomputed"][tie]
        g = self.ctx.step(
            self.gc, torch.from_numpy(np.ascontiguousarray(frames)).cuda(),
            torch.from_numpy(np.ascontiguousarray(prompt)).cuda(),
            None if proprio is None else torch.from_numpy(np.ascontiguousarray(proprio, np.float32)).cuda(),
            tau_sim=tau_sim, tau_margin=tau_m, permille=permille, margin_kind=margin_kind,
            gate_override=torch.from_numpy(ovr).cuda(),
            forced_ids=torch.from_numpy(o["action_ids"].astype(np.int32)).cuda(),
            want=("gate_auto", "logits", "static_mask", "idx", "M", "relevance", "relevant", "entropy", "action_delta",
                  "layer_entropy", "schedule")
            + (("vocab_margin",) if vocab else ()),
            active=None if act is None else torch.from_numpy(act).cuda(),
            s2_top_k=s2_top_k, s2_layer=s2_layer,
            s2_forced=(torch.from_numpy(np.ascontiguousarray(o["relevant"])).cuda()
                       if s2_top_k > 0 and s2_lockstep else None),
            s3_adaptive=s3,
            s3_forced=(torch.from_numpy(np.ascontiguousarray(o["schedule"]).view(np.int16)).cuda()
                       if s3 is not None and s3_lockstep else None))
        torch.cuda.synchronize()
        g = {k: v.cpu().numpy() for k, v in g.items()}
        err = self.ctx.sync_error()
        assert err == 0, f"device error {err}"
        rep = compare(d, o, g, self.prev_m, tau_m, self.logit_tol)
        stepped = np.ones(B, bool) if act is None else act != 0
        rep.update(compare_stage2(d, o, g, s2_top_k, self.prev_rel, stepped, s2_layer))
        rep.update(compare_signals(d, o, g, self.prev_ids, self.logit_tol, stepped))
        rep.update(compare_stage3(d, o, g, s3, self.prev_ent, stepped))
        if s3 is not None:
            pe = o["layer_entropy"].copy()
            if act is not None and self.prev_ent is not None:
                pe[~stepped] = self.prev_ent[~stepped]
            self.prev_ent = pe
        # the ids a sequence's next action delta is measured against: a sequence
        # that sat the step out keeps those of the last step it ran
        po, pg = o["action_ids"].copy(), g["action_ids"].copy()
        if act is not None and self.prev_ids is not None:
            po[~stepped], pg[~stepped] = self.prev_ids[0][~stepped], self.prev_ids[1][~stepped]
        self.prev_ids = (po, pg)
        rel = o["relevance"].copy() if s2_top_k > 0 else None
        m = o["step_margin"].copy()
        if act is not None and self.prev_m is not None:  # a paused sequence keeps its m_{t-1}
            m = np.where(act != 0, m, self.prev_m)
            if rel is not None and self.prev_rel is not None:  # and its relevance
                rel = np.where(act[:, None] != 0, rel, self.prev_rel)
        self.prev_m = m
        self.prev_rel = rel
        self.log.append(rep)
        return o, g, rep


def compare(d, o, g, prev_m, tau_m, logit_tol=None, flag_tie=FLAG_TIE):
    """Checks one step; returns a small report of the numeric gaps.  The
    gate's own decision (gate_auto) must match outside `flag_tie` of theta_m."""
    B = o["action_ids"].shape[0]
    for k in ("static_mask", "idx", "M", "recomputed"):
        np.testing.assert_array_equal(g[k], o[k], err_msg=k)
    for b in range(B):
        tie = prev_m is not None and abs(prev_m[b] - tau_m) < flag_tie
        if not tie:
            assert g["gate_auto"][b] == o["gate_auto"][b], f"gate_auto[{b}]"
    tol = LOGIT_TOL[d.dtype] if logit_tol is None else logit_tol
    diff = np.abs(g["logits"].astype(np.float64) - o["logits"])
    assert diff.max() <= tol, f"logits differ by {diff.max():.3e} > {tol}"
    # at depth the largest difference is held to the floor-derived bar; the
    # stated bar still holds for the typical (median) logit
    assert np.median(diff) <= LOGIT_TOL[d.dtype], f"median logit difference {np.median(diff):.3e}"
    mism = g["action_ids"] != o["action_ids"]
    exempt = o["margins"] < ID_EXEMPT_MARGIN
    if logit_tol is not None:
        gl = g["logits"].astype(np.float64)
        np.testing.assert_array_equal(np.argmax(gl, axis=-1), g["action_ids"], err_msg="GPU id vs GPU logits")
        o_own = np.take_along_axis(o["logits"], o["action_ids"][..., None].astype(np.int64), -1)[..., 0]
        o_gpu = np.take_along_axis(o["logits"], g["action_ids"][..., None].astype(np.int64), -1)[..., 0]
        exempt = exempt | (o_own - o_gpu < 2 * logit_tol)
    bad = mism & ~exempt
    assert not bad.any(), (f"action ids differ outside the exemption: {np.argwhere(bad)}, "
                           f"oracle margins {o['margins'][bad]}")
    np.testing.assert_allclose(g["margins"], o["margins"], atol=max(tol * 0.05, 1e-6), rtol=0.05)
    return {"max_logit_diff": float(diff.max()), "median_logit_diff": float(np.median(diff)),
            "id_mismatch": int(mism.sum()),
            "id_exempt": int(exempt.sum()), "recomputed": o["recomputed"].tolist()}


def compare_stage2(d, o, g, top_k, prev_rel, stepped=None, s2_layer=0):
    """Stage 2: this step's relevance within REL_TOL of the oracle's (relative
    to the sequence's largest), and the removal set the library decided from
    its previous relevance equal to the oracle's except inside the tie band
    around the oracle's k-th / (k+1)-th midpoint."""
    if top_k == 0:
        assert not g["relevance"].any() and not g["relevant"].any(), "Stage 2 off: nothing measured or removed"
        return {"rel_diff": 0.0, "removal_diffs": 0}
    tol = (REL_TOL if s2_layer == 0 else REL_TOL_DEEP)[d.dtype]
    worst, diffs = 0.0, 0
    for b in range(o["relevance"].shape[0]):
        if stepped is not None and not stepped[b]:  # sat the step out: both sides return zeros
            assert not g["relevance"][b].any() and not g["relevant"][b].any()
            continue
        scale = float(np.max(o["relevance"][b]))
        err = float(np.max(np.abs(g["relevance"][b].astype(np.float64) - o["relevance"][b]))) / scale
        assert err <= tol, f"relevance of sequence {b} differs by {err:.3e} (relative) > {tol}"
        worst = max(worst, err)
        bad = g["relevant"][b] != o["relevant"][b]
        if bad.any():
            assert prev_rel is not None, "a removal set without a previous relevance"
            r = np.sort(prev_rel[b])[::-1]
            mid = 0.5 * (r[top_k - 1] + r[top_k]) if top_k < r.size else -np.inf
            band = 2 * tol * float(np.max(prev_rel[b]))
            outside = bad & (np.abs(prev_rel[b] - mid) > band)
            assert not outside.any(), f"removal set differs outside the tie band: {np.flatnonzero(outside)}"
            diffs += int(bad.sum())
    return {"rel_diff": worst, "removal_diffs": diffs}
def compare_stage3(d, o, g, s3, prev_ent, stepped=None):
    """Stage 3 adaptive: the layer entropies within ENT_TOL of the oracle's;
    the library's own schedule equal to the oracle's except for a layer whose
    smoothed per-mille value, computed exactly from the oracle's previous
    entropies, lies within (hi - lo) x ENT_TOL of an integer.  Off: the
    caller's schedule is reported and nothing is measured."""
    g_sched = g["schedule"].astype(np.int64) & 0xFFFF
    if s3 is None:
        assert not g["layer_entropy"].any()
        np.testing.assert_array_equal(g_sched, o["schedule"])
        return {"ent_diff": 0.0, "sched_diffs": 0}
    lo, hi, w = s3
    tol = ENT_TOL[d.dtype]
    worst, diffs = 0.0, 0
    for b in range(o["schedule"].shape[0]):
        if stepped is not None and not stepped[b]:
            assert not g["layer_entropy"][b].any() and not g_sched[b].any()
            continue
        err = float(np.max(np.abs(g["layer_entropy"][b].astype(np.float64) - o["layer_entropy"][b])))
        assert err <= tol, f"layer entropy of sequence {b} differs by {err:.3e} > {tol}"
        worst = max(worst, err)
        bad = g_sched[b] != o["schedule"][b]
        if bad.any():
            assert prev_ent is not None, "a derived schedule without a previous step"
            r, near = 0.0, []
            for l, e in enumerate(prev_ent[b]):
                t = hi - (hi - lo) * float(e)
                r = t if l == 0 else r + (w / 1000.0) * (t - r)
                near.append(abs(r - round(r)) <= (hi - lo) * tol + 1e-9)
            outside = bad & ~np.array(near)
            assert not outside.any(), f"schedule differs away from a rounding boundary at layers {np.flatnonzero(outside)}"
            diffs += int(bad.sum())
    return {"ent_diff": worst, "sched_diffs": diffs}


def compare_signals(d, o, g, prev_ids, logit_tol=None, stepped=None):
    """Entropy within ENTROPY_FACTOR x the logit bar of the oracle's (and
    within fp32 rounding of the entropy of the library's own logits); the
    whole-vocabulary margin like the bin margin; the action delta exact for
    every sequence whose ids agree with the oracle's on this and the
    previous step."""
    tol = LOGIT_TOL[d.dtype] if logit_tol is None else logit_tol
    if stepped is not None and not stepped.all():  # sequences that sat the step out return zeros
        assert not g["entropy"][~stepped].any() and not g["action_delta"][~stepped].any()
        if not stepped.any():
            return {"entropy_diff": 0.0, "delta_compared": 0}
        o = {k: (v[stepped] if isinstance(v, np.ndarray) and v.shape[:1] == stepped.shape else v) for k, v in o.items()}
        g = {k: (v[stepped] if isinstance(v, np.ndarray) and v.shape[:1] == stepped.shape else v) for k, v in g.items()}
        if prev_ids is not None:
            prev_ids = (prev_ids[0][stepped], prev_ids[1][stepped])
    gl = g["logits"].astype(np.float64)
    p = np.exp(gl - gl.max(-1, keepdims=True))
    z = p.sum(-1, keepdims=True)
    own = np.log(z[..., 0]) - (p * (gl - gl.max(-1, keepdims=True))).sum(-1) / z[..., 0]
    np.testing.assert_allclose(g["entropy"], own, atol=1e-4, rtol=1e-5, err_msg="entropy vs own logits")
    ediff = float(np.max(np.abs(g["entropy"] - o["entropy"])))
    assert ediff <= ENTROPY_FACTOR * tol, f"entropy differs by {ediff:.3e}"
    if "vocab_margin" in g and "vocab_margin" in o:
        np.testing.assert_allclose(g["vocab_margin"], o["vocab_margin"], atol=max(tol * 0.05, 1e-6), rtol=0.05,
                                   err_msg="vocabulary margin")
    same = (g["action_ids"] == o["action_ids"]).all(-1)
    if prev_ids is not None:
        same &= (prev_ids[0] == prev_ids[1]).all(-1)
    np.testing.assert_array_equal(g["action_delta"][same], o["action_delta"][same], err_msg="action delta")
    return {"entropy_diff": ediff, "delta_compared": int(same.sum())}
