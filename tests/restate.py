"""Independent numpy restatement of the Gated VLA-Cache step, used to pin the
C oracle.  It is written separately from ``oracle/orc.c`` (vectorised numpy,
Python integers and ``fractions.Fraction`` for the exact parts) and imports
nothing from ``oracle``.  Agreement is checked within tolerances, not bit for
bit, because the summation orders differ.

Follows: Sec. III-A (patches -> token embeddings, concatenated with text),
Sec. III-B Stage 1 (patch cosine vs tau) and Stage 3 (per-layer reuse
proportion), Eq. (1) (top-1/top-2 probability margin) and Algorithm 1
(gate -> full pass or partial pass -> decode).
"""
from __future__ import annotations

from fractions import Fraction

import numpy as np


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Nearest bf16 value (ties to even) of float64 values, via the two
    neighbouring bf16 candidates of the truncated bit pattern."""
    x = np.asarray(x, dtype=np.float64)
    f32 = x.astype(np.float32)  # only used to find the candidate neighbourhood
    bits = f32.view(np.uint32) & np.uint32(0xFFFF0000)
    lo = bits.view(np.float32).astype(np.float64)
    step_bits = (bits + np.uint32(0x10000)).view(np.float32).astype(np.float64)
    down_bits = (bits - np.uint32(0x10000)).view(np.float32).astype(np.float64)
    out = np.empty_like(x)
    for i, (v, a, b, c) in enumerate(zip(x.ravel(), lo.ravel(), step_bits.ravel(), down_bits.ravel())):
        cands = [a, b, c]
        best = None
        for cnd in cands:
            if not np.isfinite(cnd):
                continue
            dist = abs(Fraction(v) - Fraction(cnd))
            if best is None or dist < best[0] or (dist == best[0] and _even(cnd) and not _even(best[1])):
                best = (dist, cnd)
        out.ravel()[i] = best[1]
    return out


def _even(v: float) -> bool:
    b = np.array([v], dtype=np.float32).view(np.uint32)[0]
    return ((int(b) >> 16) & 1) == 0


class Restated:
    """Alg. 1 on host numpy arrays for one sequence (small models only)."""

    def __init__(self, d, w):
        import torch
        self.d = d
        self.bf16 = d.dtype == "bf16"

        def a(t):
            return None if t is None else t.detach().to(torch.float64).cpu().numpy()

        self.tok = a(w["tok_emb"])
        self.pw = a(w["patch_w"])
        self.prw = a(w.get("proprio_w"))
        self.act = a(w.get("action_emb"))
        self.layers = [{k: a(v) for k, v in lay.items()} for lay in w["layers"]]
        self.fnorm = a(w["final_norm"])
        self.head = a(w["lm_head"])[d.vocab - d.n_bins:]
        nv = d.n_visual
        self.Nv = nv
        self.P = d.prefix_len
        self.S = d.pass_len
        self.T = d.cache_len
        half = d.head_dim // 2
        inv = np.array([d.rope_theta ** (-2.0 * i / d.head_dim) for i in range(half)])
        ang = np.arange(self.T)[:, None] * inv[None, :]
        self.cos = np.cos(ang).astype(np.float32).astype(np.float64)
        self.sin = np.sin(ang).astype(np.float32).astype(np.float64)
        L = d.n_layers
        self.K = np.zeros((L, self.T, d.hidden))
        self.V = np.zeros((L, self.T, d.hidden))
        self.H = np.zeros((L, self.S, d.hidden))
        self.prev = None
        self.m_prev = 0.0
        self.valid = False
        self.ent_sum = None  # per layer: [sum of normalized entropies, count] while a prefix pass runs

    # -- storage roundings --------------------------------------------------
    def act_r(self, x):
        x = np.asarray(x, dtype=np.float64)
        if self.bf16:
            return _bf16_fast(x)
        return x.astype(np.float32).astype(np.float64)

    @staticmethod
    def f32(x):
        return np.asarray(x, dtype=np.float64).astype(np.float32).astype(np.float64)

    # -- pieces --------------------------------------------------------------
    def patch_vec(self, frame, v):
        d = self.d
        p = d.patch
        gw, gh = d.img_w // p, d.img_h // p
        view, r = divmod(v, gw * gh)
        py, px = divmod(r, gw)
        return frame[view, py * p:(py + 1) * p, px * p:(px + 1) * p, :].reshape(-1).astype(np.int64)

    @staticmethod
    def cos2_key(a, b) -> Fraction:
        """cos^2 as an exact fraction; both patches all-zero -> 1, one all-zero -> 0."""
        dd, na, nb = int(a @ b), int(a @ a), int(b @ b)
        if na == 0 and nb == 0:
            return Fraction(1)
        if na == 0 or nb == 0:
            return Fraction(0)
        return Fraction(dd * dd, na * nb)

    @staticmethod
    def cos_above(a, b, thr: Fraction) -> bool:
        """Exact test cos(a, b) > thr for thr >= 0."""
        dd, na, nb = int(a @ b), int(a @ a), int(b @ b)
        if na == 0 and nb == 0:
            return Fraction(1) > thr
        if na == 0 or nb == 0 or dd <= 0:
            return Fraction(0) > thr
        return Fraction(dd * dd, na * nb) > thr * thr

    def rmsnorm(self, x, g):
        ms = np.mean(x * x, axis=-1, keepdims=True)
        return self.act_r(x / np.sqrt(ms + self.d.rms_eps) * g)

    def rope(self, x, pos):
        d = self.d
        half = d.head_dim // 2
        x = x.reshape(len(pos), d.n_heads, d.head_dim).copy()
        c = self.cos[pos][:, None, :]
        s = self.sin[pos][:, None, :]
        a, b = x[..., :half].copy(), x[..., half:].copy()
        x[..., :half] = a * c - b * s
        x[..., half:] = b * c + a * s
        return x.reshape(len(pos), -1)

    def embed(self, pos, frame, prompt, proprio):
        d = self.d
        hp = 1 if d.proprio_dim else 0
        if pos == 0:
            return self.f32(self.tok[prompt[0]])
        if 1 <= pos <= self.Nv:
            pv = self.patch_vec(frame, pos - 1).astype(np.float64)
            return self.f32(self.pw @ pv / 255.0)
        if hp and pos == self.Nv + 1:
            return self.f32(self.prw @ proprio.astype(np.float64))
        if pos < self.P:
            return self.f32(self.tok[prompt[pos - self.Nv - hp]])
        return self.f32(self.act[pos - self.P])

    def key_limit(self, pos):
        if self.d.parallel and pos >= self.P:
            return self.P + self.d.n_action
        return pos + 1

    def layer(self, l, x, pos):
        d = self.d
        W = self.layers[l]
        pos = np.asarray(pos)
        h = self.rmsnorm(x, W["attn_norm"])
        q = self.rope(h @ W["wq"].T, pos)
        k = self.rope(h @ W["wk"].T, pos)
        v = h @ W["wv"].T
        q = self.act_r(q)
        self.K[l, pos] = self.act_r(k)
        self.V[l, pos] = self.act_r(v)
        hd, nh = d.head_dim, d.n_heads
        out = np.zeros_like(q)
        hp = 1 if d.proprio_dim else 0
        for i, p in enumerate(pos):
            nk = self.key_limit(int(p))
            text = int(p) == 0 or self.Nv + hp < int(p) < self.P
            for hh in range(nh):
                sl = slice(hh * hd, (hh + 1) * hd)
                sc = self.K[l, :nk, sl] @ q[i, sl] / np.sqrt(hd)
                e = np.exp(sc - sc.max())
                prob = e / e.sum()
                out[i, sl] = prob @ self.V[l, :nk, sl]
                if self.ent_sum is not None and text and nk >= 2:
                    nz = prob[prob > 0]
                    self.ent_sum[l][0] += float(-(nz * np.log(nz)).sum() / np.log(nk))
                    self.ent_sum[l][1] += 1
        x = self.f32(x + self.act_r(out) @ W["wo"].T)
        h2 = self.rmsnorm(x, W["ffn_norm"])
        g = h2 @ W["w_gate"].T
        u = h2 @ W["w_up"].T
        a = self.act_r(g / (1.0 + np.exp(-g)) * u)
        return self.f32(x + a @ W["w_down"].T)

    def head_out(self, x):
        h = self.rmsnorm(x, self.fnorm)
        lg = self.head @ h
        b1 = int(np.argmax(lg))
        l1 = lg[b1]
        l2 = np.max(np.delete(lg, b1))
        p = np.exp(lg - l1) / np.exp(lg - l1).sum()
        return lg, b1, p[b1] - np.max(np.delete(p, b1)), l1 - l2

    # -- Algorithm 1 ---------------------------------------------------------
    def step(self, frame, prompt, proprio, tau, tau_m, permille, margin_kind=0, reduction=None,
             override=-1, forced=None):
        d = self.d
        L, S, P, D = d.n_layers, self.S, self.P, d.n_action
        if reduction is None:
            reduction = 1 if d.parallel else 0
        gate = (not self.valid) or self.m_prev < tau_m
        full = gate if override < 0 else bool(override)
        if not self.valid:
            full = True
        thr = Fraction(tau[0], tau[1])
        mask = np.zeros(self.Nv, np.uint8)
        keys = {}
        if self.valid:
            for v in range(self.Nv):
                a, b = self.patch_vec(frame, v), self.patch_vec(self.prev, v)
                mask[v] = 1 if self.cos_above(a, b, thr) else 0
                keys[v] = self.cos2_key(a, b)
        if full:
            idx = list(range(S))
            M = [S] * L
        else:
            stat = [v for v in range(self.Nv) if mask[v]]
            order = sorted(stat, key=lambda v: (-keys[v], v))  # most similar first
            stat_pos = {1 + v for v in stat}
            idx = [p for p in range(S) if p not in stat_pos] + [1 + v for v in reversed(order)]
            M = [S - (int(permille[l]) * len(stat)) // 1000 for l in range(L)]
        x = np.stack([self.embed(idx[i], frame, prompt, proprio) for i in range(M[0])])
        self.ent_sum = [[0.0, 0] for _ in range(L)]
        for l in range(L):
            if l > 0:
                for i in range(M[l - 1]):
                    self.H[l, idx[i]] = x[i]
                if M[l] > M[l - 1]:
                    x = np.concatenate([x, self.H[l, idx[M[l - 1]:M[l]]]], axis=0)
                else:
                    x = x[:M[l]]
            x = self.layer(l, x, idx[:M[l]])
        layer_entropy = np.array([e / n if n else 0.0 for e, n in self.ent_sum])
        self.ent_sum = None
        ids, margins, gaps, logits = [], [], [], []
        for a in range(D):
            if d.parallel:
                xr = x[idx.index(P + a)]
            elif a == 0:
                xr = x[idx.index(P - 1)]
            else:
                fed = forced[a - 1] if forced is not None else ids[a - 1]
                xr = self.f32(self.tok[d.vocab - d.n_bins + fed])[None, :]
                p = P + a - 1
                for l in range(L):
                    xr = self.layer(l, xr, [p])
                xr = xr[0]
            lg, b1, pm, gap = self.head_out(xr)
            ids.append(b1)
            margins.append(pm)
            gaps.append(gap)
            logits.append(lg)
        sig = np.array(gaps if margin_kind == 1 else margins)
        m_t = float(sig.min() if reduction == 1 else sig.mean())
        self.m_prev, self.valid, self.prev = m_t, True, frame.copy()
        return dict(action_ids=np.array(ids), margins=np.array(margins), logit_gap=np.array(gaps),
                    logits=np.stack(logits), recomputed=int(full), gate_auto=int(gate),
                    step_margin=m_t, static_mask=mask, idx=np.array(idx), M=np.array(M),
                    layer_entropy=layer_entropy)


def _bf16_fast(x: np.ndarray) -> np.ndarray:
    """Vectorised nearest-bf16 (ties to even) of float64 values: scale each
    value so that its bf16 grid becomes the integers, then round half to even
    with numpy's rint."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)
    r = np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)
    sub = np.ldexp(np.rint(np.ldexp(x, 133)), -133)  # bf16 subnormals: spacing 2^-133
    r = np.where(e - 8 < -133, sub, r)
    return np.where(np.isfinite(x), r, x)
