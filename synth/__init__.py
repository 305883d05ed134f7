"""Seeded synthetic workloads for the Gated VLA-Cache step.

This module only draws inputs: model weights, camera frames, prompts,
proprioception and per-layer reuse schedules.  It holds none of the method's
arithmetic, so the CPU oracle and the CUDA path can both be fed from it.

Shapes and distributions follow the workloads of the paper's experiments
(Sec. V, "Experimental Setup"): OpenVLA's Llama-2-7B backbone with 224x224
frames cut into 14x14 patches (N = 256, Sec. III-A), OpenVLA-OFT with two
views, a proprio token and an 8x7 action chunk decoded in parallel, and
50-step episodes.  Trained weights and LIBERO frames are not available, so
weights are N(0, 0.02) with unit RMSNorm gains and frames are procedurally
generated scenes (a static texture with moving blobs).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional

import numpy as np
import torch

__all__ = [
    "Dims", "CONFIGS", "dims_for", "make_weights", "make_prompt",
    "make_episode", "make_proprio", "linear_schedule", "positions",
]


@dataclasses.dataclass(frozen=True)
class Dims:
    """Backbone and input geometry of one workload."""
    n_layers: int
    hidden: int
    n_heads: int
    head_dim: int
    ffn: int
    vocab: int
    n_bins: int
    img_h: int
    img_w: int
    patch: int
    n_views: int
    n_text: int          # prompt length including BOS
    proprio_dim: int     # 0 = no proprio token
    n_action: int        # D action tokens (AR) or chunk positions (parallel)
    parallel: int        # 0 = autoregressive decode, 1 = parallel action block
    dtype: str           # "f32" or "bf16"
    rope_theta: float = 10000.0
    rms_eps: float = 1e-5
    max_batch: int = 1

    @property
    def n_patches(self) -> int:          # per view
        return (self.img_h // self.patch) * (self.img_w // self.patch)

    @property
    def n_visual(self) -> int:
        return self.n_views * self.n_patches

    @property
    def patch_dim(self) -> int:
        return self.patch * self.patch * 3

    @property
    def prefix_len(self) -> int:         # P: BOS + visual + proprio + rest of text
        return self.n_text + self.n_visual + (1 if self.proprio_dim > 0 else 0)

    @property
    def pass_len(self) -> int:           # S: positions computed in the prefix pass
        return self.prefix_len + (self.n_action if self.parallel else 0)

    @property
    def cache_len(self) -> int:          # K/V positions held per sequence
        return self.pass_len + (0 if self.parallel else self.n_action - 1)

    def replace(self, **kw) -> "Dims":
        return dataclasses.replace(self, **kw)


_LLAMA7B = dict(n_layers=32, hidden=4096, n_heads=32, head_dim=128, ffn=11008,
                vocab=32000, n_bins=256, patch=14, img_h=224, img_w=224,
                n_text=27, dtype="bf16")

CONFIGS: Dict[str, Dims] = {
    # Tiny fp32 decoder: 2 layers, 64 patches from a 112x112 frame, 8 text tokens.
    "tiny": Dims(n_layers=2, hidden=256, n_heads=4, head_dim=64, ffn=688, vocab=512,
                 n_bins=256, img_h=112, img_w=112, patch=14, n_views=1, n_text=8,
                 proprio_dim=0, n_action=7, parallel=0, dtype="f32"),
    # One Llama-2-7B layer over a 290-token prefix (256 visual + 27 text + 7 action).
    "layer7b": Dims(**{**_LLAMA7B, "n_layers": 1}, n_views=1, proprio_dim=0,
                    n_action=7, parallel=0),
    # OpenVLA-7B shape: 32 layers, 256 visual + 27 text, 7 autoregressive action tokens.
    "openvla7b": Dims(**_LLAMA7B, n_views=1, proprio_dim=0, n_action=7, parallel=0),
    # OpenVLA-OFT shape: 2 views, proprio token, 8x7 action chunk decoded in one pass.
    "oft7b": Dims(**_LLAMA7B, n_views=2, proprio_dim=8, n_action=56, parallel=1),
    # Batched serving: OpenVLA-7B shape, 8 sequences per step.
    "batch7b": Dims(**_LLAMA7B, n_views=1, proprio_dim=0, n_action=7, parallel=0,
                    max_batch=8),
}


def dims_for(name: str, **overrides) -> Dims:
    d = CONFIGS[name]
    return d.replace(**overrides) if overrides else d


def positions(d: Dims) -> Dict[str, object]:
    """Token layout of one sequence: BOS, visual (view-major, row-major
    patches), proprio, the remaining text, then the parallel action block."""
    nv = d.n_visual
    has_p = 1 if d.proprio_dim > 0 else 0
    return {
        "bos": 0,
        "visual": (1, 1 + nv),
        "proprio": (1 + nv) if has_p else None,
        "text": (1 + nv + has_p, d.prefix_len),
        "action": (d.prefix_len, d.prefix_len + d.n_action) if d.parallel else None,
    }


# ----------------------------------------------------------------------------
# Weights
# ----------------------------------------------------------------------------

def _torch_dtype(d: Dims):
    return torch.float32 if d.dtype == "f32" else torch.bfloat16


def _normal(shape, seed: int, key: int, device, dtype, std: float = 0.02):
    g = torch.Generator(device=device)
    g.manual_seed((seed * 1_000_003 + key * 7919 + 17) % (2 ** 62))
    t = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    t.mul_(std)
    return t.to(dtype)


def make_weights(d: Dims, seed: int = 0, device="cpu", lm_head_rows: Optional[int] = None):
    """All matrices and embeddings N(0, 0.02) drawn from `seed`, rounded to the
    storage dtype (bf16 by round-to-nearest-even); RMSNorm gains are 1.

    Matrices are row-major [out][in].  `lm_head_rows` limits the drawn LM head
    to its last rows (only the action-bin rows are ever read)."""
    dt = _torch_dtype(d)
    hd, f = d.hidden, d.ffn
    qd = d.n_heads * d.head_dim
    w: Dict[str, object] = {}
    w["tok_emb"] = _normal((d.vocab, hd), seed, 1, device, dt)
    w["patch_w"] = _normal((hd, d.patch_dim), seed, 2, device, dt)
    w["proprio_w"] = _normal((hd, d.proprio_dim), seed, 3, device, dt) if d.proprio_dim else None
    w["action_emb"] = _normal((d.n_action, hd), seed, 4, device, dt) if d.parallel else None
    layers: List[Dict[str, torch.Tensor]] = []
    for l in range(d.n_layers):
        k = 100 + 16 * l
        layers.append({
            "attn_norm": torch.ones(hd, device=device, dtype=dt),
            "wq": _normal((qd, hd), seed, k + 0, device, dt),
            "wk": _normal((qd, hd), seed, k + 1, device, dt),
            "wv": _normal((qd, hd), seed, k + 2, device, dt),
            "wo": _normal((hd, qd), seed, k + 3, device, dt),
            "ffn_norm": torch.ones(hd, device=device, dtype=dt),
            "w_gate": _normal((f, hd), seed, k + 4, device, dt),
            "w_up": _normal((f, hd), seed, k + 5, device, dt),
            "w_down": _normal((hd, f), seed, k + 6, device, dt),
        })
    w["layers"] = layers
    w["final_norm"] = torch.ones(hd, device=device, dtype=dt)
    rows = d.vocab if lm_head_rows is None else lm_head_rows
    head = _normal((rows, hd), seed, 5, device, dt)
    if rows < d.vocab:
        full = torch.zeros((d.vocab, hd), device=device, dtype=dt)
        full[d.vocab - rows:] = head
        head = full
    w["lm_head"] = head
    return w


def weights_to(w, device):
    out = {}
    for k, v in w.items():
        if k == "layers":
            out[k] = [{kk: vv.to(device) for kk, vv in lay.items()} for lay in v]
        else:
            out[k] = None if v is None else v.to(device)
    return out


# ----------------------------------------------------------------------------
# Prompts, proprio and schedules
# ----------------------------------------------------------------------------

def make_prompt(d: Dims, seed: int = 0, batch: int = 1) -> np.ndarray:
    """[batch][n_text] int32: BOS (=1) then ids uniform in [3, vocab - n_bins)."""
    rng = np.random.default_rng(seed * 31 + 7)
    ids = rng.integers(3, d.vocab - d.n_bins, size=(batch, d.n_text), dtype=np.int64)
    ids[:, 0] = 1
    return ids.astype(np.int32)


def make_proprio(d: Dims, n_frames: int, seed: int = 0, batch: int = 1) -> Optional[np.ndarray]:
    """[n_frames][batch][proprio_dim] float32 random walk (step N(0, 0.05))."""
    if d.proprio_dim == 0:
        return None
    rng = np.random.default_rng(seed * 131 + 3)
    steps = rng.normal(0.0, 0.05, size=(n_frames, batch, d.proprio_dim))
    return np.cumsum(steps, axis=0).astype(np.float32)


def make_layer_case(d: Dims, M: int, seed: int = 0):
    """The one-layer workload: a seeded sample of M distinct prefix positions
    (sorted), the rows' layer inputs N(0, 1) in float32 [M][hidden], and the
    layer's cache K and V, each [cache_len][hidden] N(0, 1) stored in the
    model's dtype (returned as float32 arrays holding those values)."""
    rng = np.random.default_rng(seed * 7919 + M)
    pos = np.sort(rng.choice(d.pass_len, size=M, replace=False)).astype(np.int32)
    x = rng.normal(size=(M, d.hidden)).astype(np.float32)
    kv = []
    for key in (11, 12):
        t = _normal((d.cache_len, d.hidden), seed, key, "cpu", _torch_dtype(d), std=1.0)
        kv.append(t.float().numpy())
    return pos, x, kv[0], kv[1]


def linear_schedule(n_layers: int, first: int = 900, last: int = 500) -> np.ndarray:
    """Per-layer reuse proportion in per-mille, linear from `first` to `last`."""
    if n_layers == 1:
        return np.array([first], dtype=np.uint16)
    l = np.arange(n_layers)
    s = (first * (n_layers - 1 - l) + last * l) // (n_layers - 1)
    return s.astype(np.uint16)


def full_schedule(n_layers: int, permille: int = 1000) -> np.ndarray:
    return np.full(n_layers, permille, dtype=np.uint16)


# ----------------------------------------------------------------------------
# Frames
# ----------------------------------------------------------------------------

def _redraw_episode(d: Dims, n_frames: int, rng, p_redraw: float) -> np.ndarray:
    """Frame 0 is uniform random bytes; each later frame redraws every patch
    with probability `p_redraw` as fresh uniform bytes and copies it otherwise."""
    h, w, p = d.img_h, d.img_w, d.patch
    frames = np.empty((n_frames, d.n_views, h, w, 3), dtype=np.uint8)
    frames[0] = rng.integers(0, 256, size=(d.n_views, h, w, 3), dtype=np.uint8)
    for t in range(1, n_frames):
        frames[t] = frames[t - 1]
        for v in range(d.n_views):
            redraw = rng.random((h // p, w // p)) < p_redraw
            for py, px in zip(*np.nonzero(redraw)):
                frames[t, v, py * p:(py + 1) * p, px * p:(px + 1) * p] = rng.integers(
                    0, 256, size=(p, p, 3), dtype=np.uint8)
    return frames


def _texture(h, w, rng) -> np.ndarray:
    y, x = np.mgrid[0:h, 0:w].astype(np.float64)
    tex = np.empty((h, w, 3), dtype=np.float64)
    for c in range(3):
        ph1, ph2 = rng.uniform(0, 2 * math.pi, size=2)
        noise = rng.uniform(-20, 20, size=(h, w))
        tex[..., c] = 128 + 60 * np.sin(x / 7 + ph1) * np.cos(y / 11 + ph2) + noise
    return np.clip(np.rint(tex), 0, 255).astype(np.uint8)


def _bounce(start: float, vel: float, t: int, lo: float, hi: float) -> float:
    span = hi - lo
    if span <= 0:
        return lo
    z = (start - lo + vel * t) % (2 * span)
    return lo + (z if z <= span else 2 * span - z)


def _scene_view(n_frames, h, w, rng, speed: float, jitter_frames=(20, 26)) -> np.ndarray:
    """Static texture + a 40x40 blob moving `speed` px/frame along a seeded
    direction (bouncing off the borders) + a 24x24 gripper blob that is
    displaced by integer jitter in [-4, 4] px on frames 20..25 only."""
    tex = _texture(h, w, rng)
    colour = rng.integers(0, 256, size=3, dtype=np.uint8)
    gcolour = rng.integers(0, 256, size=3, dtype=np.uint8)
    ang = rng.uniform(0, 2 * math.pi)
    vx, vy = speed * math.cos(ang), speed * math.sin(ang)
    bx0, by0 = rng.uniform(0, w - 40), rng.uniform(0, h - 40)
    gx, gy = int(rng.integers(8, w - 32)), int(rng.integers(8, h - 32))
    jit = rng.integers(-4, 5, size=(n_frames, 2))
    out = np.empty((n_frames, h, w, 3), dtype=np.uint8)
    for t in range(n_frames):
        f = tex.copy()
        bx = int(round(_bounce(bx0, vx, t, 0, w - 40)))
        by = int(round(_bounce(by0, vy, t, 0, h - 40)))
        f[by:by + 40, bx:bx + 40] = colour
        ox, oy = (jit[t] if jitter_frames[0] <= t < jitter_frames[1] else (0, 0))
        x0 = min(max(gx + int(ox), 0), w - 24)
        y0 = min(max(gy + int(oy), 0), h - 24)
        f[y0:y0 + 24, x0:x0 + 24] = gcolour
        out[t] = f
    return out


def make_episode(d: Dims, n_frames: int, seed: int = 0, batch: int = 1,
                 kind: Optional[str] = None, speeds=None) -> np.ndarray:
    """[n_frames][batch][n_views][H][W][3] uint8 frames.

    kind "redraw": uniform-random first frame, patches redrawn with p = 0.3.
    kind "scene":  textured scene with a moving blob (3 px/frame unless
                   `speeds` gives one speed per sequence) and a jittering
                   gripper blob; every view has its own motion seed."""
    if kind is None:
        kind = "redraw" if d.img_h < 224 else "scene"
    out = np.empty((n_frames, batch, d.n_views, d.img_h, d.img_w, 3), dtype=np.uint8)
    for b in range(batch):
        if kind == "redraw":
            rng = np.random.default_rng(seed * 1009 + b)
            out[:, b] = _redraw_episode(d, n_frames, rng, 0.3)
        else:
            sp = 3.0 if speeds is None else float(speeds[b])
            for v in range(d.n_views):
                rng = np.random.default_rng(seed * 1009 + b * 17 + v * 101 + 5)
                out[:, b, v] = _scene_view(n_frames, d.img_h, d.img_w, rng, sp)
    return out


def batch_speeds(batch: int, seed: int = 0) -> np.ndarray:
    """Per-sequence blob speeds for the batched workload, U[0, 8] px/frame."""
    return np.random.default_rng(seed * 7 + 1).uniform(0.0, 8.0, size=batch)
