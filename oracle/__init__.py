"""CPU oracle for the Gated VLA-Cache step (ctypes binding of liboracle.so).

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and
the benchmark's CPU-baseline / reference leg may import this package.  It
shares no code with the CUDA library: its arithmetic lives in ``orc.c``.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "liboracle.so")
_SRC = [os.path.join(_HERE, "orc.c")]
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile liboracle.so in place (gcc, OpenMP, strict IEEE fp64)."""
    newest = max(os.path.getmtime(p) for p in _SRC + [os.path.join(_HERE, "orc.h")])
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= newest:
        return _SO
    tmp = _SO + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O3", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
           "-fno-fast-math", "-Wall", "-o", tmp] + _SRC + ["-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _SO)
    return _SO


class _Dims(C.Structure):
    _fields_ = [(n, C.c_int32) for n in (
        "n_layers", "hidden", "n_heads", "head_dim", "ffn", "vocab", "n_bins",
        "img_h", "img_w", "patch", "n_views", "n_text", "proprio_dim", "n_action",
        "parallel", "bf16")] + [("rope_theta", C.c_double), ("rms_eps", C.c_double)]


_PP = C.POINTER(C.c_void_p)


class _Weights(C.Structure):
    _fields_ = [("tok_emb", C.c_void_p), ("patch_w", C.c_void_p), ("proprio_w", C.c_void_p),
                ("action_emb", C.c_void_p)] + [(n, _PP) for n in (
                    "attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down")] + [
                ("final_norm", C.c_void_p), ("lm_head", C.c_void_p)]


class _Opts(C.Structure):
    _fields_ = [("margin_kind", C.c_int32), ("reduction", C.c_int32),
                ("gate_override", C.c_void_p), ("forced_ids", C.c_void_p),
                ("s2_top_k", C.c_int32), ("s2_layer", C.c_int32), ("active", C.c_void_p),
                ("s3_adaptive", C.c_int32), ("s3_lo", C.c_int32), ("s3_hi", C.c_int32), ("s3_weight", C.c_int32),
                ("s3_forced", C.c_void_p)]


class _Out(C.Structure):
    _fields_ = [("action_ids", C.c_void_p), ("margins", C.c_void_p), ("logit_gap", C.c_void_p),
                ("logits", C.c_void_p), ("recomputed", C.c_void_p), ("gate_auto", C.c_void_p),
                ("step_margin", C.c_void_p), ("static_mask", C.c_void_p), ("idx", C.c_void_p),
                ("M", C.c_void_p), ("relevance", C.c_void_p), ("relevant", C.c_void_p),
                ("entropy", C.c_void_p), ("vocab_margin", C.c_void_p), ("action_delta", C.c_void_p),
                ("layer_entropy", C.c_void_p), ("schedule", C.c_void_p)]


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = C.CDLL(_SO)
            vp, i32, u32 = C.c_void_p, C.c_int32, C.c_uint32
            L.orc_create.argtypes = [C.POINTER(_Dims), C.POINTER(_Weights), C.POINTER(vp)]
            L.orc_destroy.argtypes = [vp]
            L.orc_cache_new.argtypes = [vp, C.c_int, C.POINTER(vp)]
            L.orc_cache_free.argtypes = [vp]
            L.orc_reset.argtypes = [vp, C.c_int]
            L.orc_entropy_schedule.argtypes = [vp, C.c_int, C.c_int, C.c_int, C.c_int, vp]
            L.orc_step.argtypes = [vp, vp, vp, vp, vp, u32, u32, C.c_double, vp,
                                   C.POINTER(_Opts), C.POINTER(_Out)]
            L.orc_cache_read.argtypes = [vp, C.c_int, C.c_int, C.c_int, vp]
            L.orc_cache_write.argtypes = [vp, C.c_int, C.c_int, C.c_int, vp]
            L.orc_layer.argtypes = [vp, vp, C.c_int, C.c_int, C.c_int, vp, vp]
            L.orc_cache_state.argtypes = [vp, C.c_int, C.POINTER(C.c_double), C.POINTER(C.c_int)]
            L.orc_patch_stats.argtypes = [C.POINTER(_Dims), vp, vp, C.c_int, C.POINTER(C.c_int64),
                                          C.POINTER(C.c_int64), C.POINTER(C.c_int64)]
            L.orc_is_static.argtypes = [C.c_int64, C.c_int64, C.c_int64, u32, u32]
            L.orc_more_similar.argtypes = [C.c_int64, C.c_int64, C.c_int64, C.c_int,
                                           C.c_int64, C.c_int64, C.c_int64, C.c_int]
            L.orc_select.argtypes = [C.POINTER(_Dims), vp, vp, C.c_int, u32, u32, vp, C.c_int,
                                     vp, vp, vp]
            L.orc_select2.argtypes = [C.POINTER(_Dims), vp, vp, C.c_int, u32, u32, vp, C.c_int,
                                      vp, C.c_int, vp, vp, vp, vp]
            L.orc_top_k.argtypes = [vp, C.c_int, C.c_int, vp]
            L.orc_margin.argtypes = [vp, C.c_int, C.POINTER(i32), C.POINTER(C.c_double),
                                     C.POINTER(C.c_double)]
            L.orc_entropy.argtypes = [vp, C.c_int]
            L.orc_entropy.restype = C.c_double
            L.orc_round_bf16.argtypes = [C.c_double]
            L.orc_round_bf16.restype = C.c_double
            L.orc_rope_table.argtypes = [C.POINTER(_Dims), C.c_int, vp, vp]
            _lib = L
    return _lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data


def c_dims(d) -> _Dims:
    return _Dims(d.n_layers, d.hidden, d.n_heads, d.head_dim, d.ffn, d.vocab, d.n_bins,
                 d.img_h, d.img_w, d.patch, d.n_views, d.n_text, d.proprio_dim, d.n_action,
                 d.parallel, 1 if d.dtype == "bf16" else 0, float(d.rope_theta), float(d.rms_eps))


# ---------------------------------------------------------------------------
# Pieces, for pin tests
# ---------------------------------------------------------------------------

def patch_stats(d, frame: np.ndarray, prev: np.ndarray, v: int):
    frame = np.ascontiguousarray(frame, dtype=np.uint8)
    prev = np.ascontiguousarray(prev, dtype=np.uint8)
    a, b, c = C.c_int64(), C.c_int64(), C.c_int64()
    dd = c_dims(d)
    lib().orc_patch_stats(C.byref(dd), _ptr(frame), _ptr(prev), v, C.byref(a), C.byref(b), C.byref(c))
    return a.value, b.value, c.value


def is_static(dot: int, na: int, nb: int, num: int, den: int) -> bool:
    return bool(lib().orc_is_static(dot, na, nb, num, den))


def more_similar(ki, i, kj, j) -> bool:
    return bool(lib().orc_more_similar(ki[0], ki[1], ki[2], i, kj[0], kj[1], kj[2], j))


def select(d, frame, prev, have_prev: bool, tau, permille, full: bool, relevance=None, top_k: int = 0):
    """Stages 1-3; with `relevance` and top_k > 0 also Stage 2.  Returns
    (|reusable|, Stage-1 mask, idx, M) and, with Stage 2, the relevant set."""
    frame = np.ascontiguousarray(frame, dtype=np.uint8)
    prev = np.ascontiguousarray(prev, dtype=np.uint8)
    permille = np.ascontiguousarray(permille, dtype=np.uint16)
    mask = np.zeros(d.n_visual, dtype=np.uint8)
    idx = np.zeros(d.pass_len, dtype=np.int32)
    M = np.zeros(d.n_layers, dtype=np.int32)
    dd = c_dims(d)
    if relevance is None and top_k == 0:
        n = lib().orc_select(C.byref(dd), _ptr(frame), _ptr(prev), int(have_prev), tau[0], tau[1],
                             _ptr(permille), int(full), _ptr(mask), _ptr(idx), _ptr(M))
        if n < 0:
            raise ValueError("orc_select rejected its arguments")
        return n, mask, idx, M
    rel = None if relevance is None else np.ascontiguousarray(relevance, dtype=np.float64)
    relevant = np.zeros(d.n_visual, dtype=np.uint8)
    n = lib().orc_select2(C.byref(dd), _ptr(frame), _ptr(prev), int(have_prev), tau[0], tau[1],
                          _ptr(permille), int(full), _ptr(rel), int(top_k), _ptr(mask), _ptr(relevant),
                          _ptr(idx), _ptr(M))
    if n < 0:
        raise ValueError("orc_select2 rejected its arguments")
    return n, mask, idx, M, relevant


def top_k(rel: np.ndarray, k: int) -> np.ndarray:
    """Stage 2's removal set of a relevance vector (1 = among the top k)."""
    r = np.ascontiguousarray(rel, dtype=np.float64)
    out = np.zeros(r.size, dtype=np.uint8)
    lib().orc_top_k(_ptr(r), r.size, int(k), _ptr(out))
    return out


def entropy_schedule(ent, lo: int, hi: int, weight: int) -> np.ndarray:
    """Stage 3's per-mille schedule from per-layer normalized entropies."""
    e = np.ascontiguousarray(ent, dtype=np.float64)
    out = np.zeros(e.size, dtype=np.uint16)
    lib().orc_entropy_schedule(_ptr(e), e.size, int(lo), int(hi), int(weight), _ptr(out))
    return out


def margin(logits: np.ndarray):
    lg = np.ascontiguousarray(logits, dtype=np.float64)
    a, pm, gap = C.c_int32(), C.c_double(), C.c_double()
    lib().orc_margin(_ptr(lg), lg.size, C.byref(a), C.byref(pm), C.byref(gap))
    return a.value, pm.value, gap.value


def entropy(logits: np.ndarray) -> float:
    lg = np.ascontiguousarray(logits, dtype=np.float64)
    return lib().orc_entropy(_ptr(lg), lg.size)


def round_bf16(v: float) -> float:
    return lib().orc_round_bf16(float(v))


def rope_table(d, n_pos: int):
    half = d.head_dim // 2
    cs = np.zeros((n_pos, half), dtype=np.float32)
    sn = np.zeros((n_pos, half), dtype=np.float32)
    dd = c_dims(d)
    lib().orc_rope_table(C.byref(dd), n_pos, _ptr(cs), _ptr(sn))
    return cs, sn


# ---------------------------------------------------------------------------
# Whole step
# ---------------------------------------------------------------------------

class Oracle:
    """Host-memory oracle of one model; weights are CPU torch tensors (kept alive)."""

    def __init__(self, d, weights):
        import torch
        self.d = d
        self._keep = []

        def p(t):
            if t is None:
                return None
            t = t.detach().to("cpu").contiguous()
            assert t.dtype == (torch.bfloat16 if d.dtype == "bf16" else torch.float32)
            self._keep.append(t)
            return t.data_ptr()

        def arr(name):
            a = (C.c_void_p * d.n_layers)(*[p(lay[name]) for lay in weights["layers"]])
            self._keep.append(a)
            return C.cast(a, _PP)

        self._w = _Weights(p(weights["tok_emb"]), p(weights["patch_w"]), p(weights.get("proprio_w")),
                           p(weights.get("action_emb")), arr("attn_norm"), arr("wq"), arr("wk"),
                           arr("wv"), arr("wo"), arr("ffn_norm"), arr("w_gate"), arr("w_up"),
                           arr("w_down"), p(weights["final_norm"]), p(weights["lm_head"]))
        self._dims = c_dims(d)
        h = C.c_void_p()
        r = lib().orc_create(C.byref(self._dims), C.byref(self._w), C.byref(h))
        if r != 0:
            raise ValueError(f"orc_create failed ({r})")
        self._h = h

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and h.value:
            lib().orc_destroy(h)
            self._h = None

    def new_cache(self, batch: int = 1) -> "OracleCache":
        return OracleCache(self, batch)

    def layer(self, cache: "OracleCache", seq: int, layer: int, pos, x) -> np.ndarray:
        """One decoder layer for the rows at positions `pos` with inputs x
        [n][hidden]; returns their outputs (the cache's K/V at those positions
        are written)."""
        pos = np.ascontiguousarray(pos, dtype=np.int32)
        out = np.array(x, dtype=np.float32, copy=True, order="C")
        r = lib().orc_layer(self._h, cache._h, seq, layer, pos.size, _ptr(pos), _ptr(out))
        if r != 0:
            raise ValueError(f"orc_layer failed ({r})")
        return out

    def step(self, cache: "OracleCache", frames, prompt, proprio=None, tau_sim=(996, 1000),
             tau_margin: float = 0.0, permille=None, margin_kind: int = 0, reduction: Optional[int] = None,
             gate_override=None, forced_ids=None, want_logits: bool = True, s2_top_k: int = 0,
             s2_layer: Optional[int] = None, want_vocab_margin: bool = False, active=None,
             s3_adaptive=None, s3_forced=None):
        """s3_adaptive: None (the caller's schedule) or (lo, hi, weight) per mille
        for the entropy-adaptive Stage 3; s3_forced [B][L] replays a schedule."""
        d, B = self.d, cache.batch
        D, S, L = d.n_action, d.pass_len, d.n_layers
        frames = np.ascontiguousarray(frames, dtype=np.uint8).reshape(B, d.n_views, d.img_h, d.img_w, 3)
        prompt = np.ascontiguousarray(prompt, dtype=np.int32).reshape(B, d.n_text)
        if proprio is not None:
            proprio = np.ascontiguousarray(proprio, dtype=np.float32).reshape(B, d.proprio_dim)
        if permille is None:
            permille = np.full(L, 1000, dtype=np.uint16)
        permille = np.ascontiguousarray(permille, dtype=np.uint16)
        if reduction is None:
            reduction = 1 if d.parallel else 0
        go = None if gate_override is None else np.ascontiguousarray(gate_override, dtype=np.int8).reshape(B)
        fi = None if forced_ids is None else np.ascontiguousarray(forced_ids, dtype=np.int32).reshape(B, D)
        out = {
            "action_ids": np.zeros((B, D), np.int32), "margins": np.zeros((B, D), np.float64),
            "logit_gap": np.zeros((B, D), np.float64),
            "logits": np.zeros((B, D, d.n_bins), np.float64) if want_logits else None,
            "recomputed": np.zeros(B, np.uint8), "gate_auto": np.zeros(B, np.uint8),
            "step_margin": np.zeros(B, np.float64), "static_mask": np.zeros((B, d.n_visual), np.uint8),
            "idx": np.zeros((B, S), np.int32), "M": np.zeros((B, L), np.int32),
            "relevance": np.zeros((B, d.n_visual), np.float64), "relevant": np.zeros((B, d.n_visual), np.uint8),
            "entropy": np.zeros((B, D), np.float64),
            "vocab_margin": np.zeros((B, D), np.float64) if want_vocab_margin else None,
            "action_delta": np.zeros(B, np.int32),
            "layer_entropy": np.zeros((B, L), np.float64), "schedule": np.zeros((B, L), np.uint16),
        }
        co = _Out(*[_ptr(out[k]) for k in ("action_ids", "margins", "logit_gap", "logits", "recomputed",
                                           "gate_auto", "step_margin", "static_mask", "idx", "M",
                                           "relevance", "relevant", "entropy", "vocab_margin", "action_delta",
                                           "layer_entropy", "schedule")])
        if s2_layer is None:
            s2_layer = L // 2
        act = None if active is None else np.ascontiguousarray(active, dtype=np.uint8).reshape(B)
        s3 = (0, 0, 0) if s3_adaptive is None else tuple(int(v) for v in s3_adaptive)
        sf = None if s3_forced is None else np.ascontiguousarray(s3_forced, dtype=np.uint16).reshape(B, L)
        opts = _Opts(margin_kind, reduction, _ptr(go), _ptr(fi), int(s2_top_k), int(s2_layer), _ptr(act),
                     int(s3_adaptive is not None), s3[0], s3[1], s3[2], _ptr(sf))
        r = lib().orc_step(self._h, cache._h, _ptr(frames), _ptr(prompt), _ptr(proprio), tau_sim[0],
                           tau_sim[1], float(tau_margin), _ptr(permille), C.byref(opts), C.byref(co))
        if r != 0:
            raise ValueError(f"orc_step failed ({r})")
        if not want_logits:
            del out["logits"]
        if not want_vocab_margin:
            del out["vocab_margin"]
        return out


class OracleCache:
    def __init__(self, orc: Oracle, batch: int):
        self.orc, self.batch = orc, batch
        h = C.c_void_p()
        r = lib().orc_cache_new(orc._h, batch, C.byref(h))
        if r != 0:
            raise MemoryError(f"orc_cache_new failed ({r})")
        self._h = h

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and h.value:
            lib().orc_cache_free(h)
            self._h = None

    def reset(self, seq: int = -1):
        if lib().orc_reset(self._h, seq) != 0:
            raise ValueError("bad sequence index")

    def read(self, seq: int, kind: str, layer: int) -> np.ndarray:
        d = self.orc.d
        n = d.pass_len if kind == "H" else d.cache_len
        dst = np.zeros((n, d.hidden), np.float32)
        k = {"K": 0, "V": 1, "H": 2}[kind]
        if lib().orc_cache_read(self._h, seq, k, layer, _ptr(dst)) != 0:
            raise ValueError("bad cache read")
        return dst

    def write(self, seq: int, kind: str, layer: int, values: np.ndarray):
        d = self.orc.d
        src = np.ascontiguousarray(values, dtype=np.float32).reshape(d.cache_len, d.hidden)
        if lib().orc_cache_write(self._h, seq, {"K": 0, "V": 1}[kind], layer, _ptr(src)) != 0:
            raise ValueError("bad cache write")

    def state(self, seq: int):
        m, v = C.c_double(), C.c_int()
        lib().orc_cache_state(self._h, seq, C.byref(m), C.byref(v))
        return m.value, v.value
