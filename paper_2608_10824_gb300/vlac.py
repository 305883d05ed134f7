"""ctypes binding of libvlac (include/vlac.h).

Argument marshalling only: every step of the method runs in the library's
CUDA kernels.  PyTorch supplies device memory and streams.  Importing this
module does not load the library; the first call does, and raises
``RuntimeError`` if ``libvlac.so`` is missing or fails to load.
"""
from __future__ import annotations

import ctypes as C
import os
import threading
from typing import Dict, Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libvlac.so")
_lock = threading.Lock()
_lib = None

VLAC_OK = 0
ERRORS = {-1: "VLAC_ERR_INVALID_ARG", -2: "VLAC_ERR_CUDA", -3: "VLAC_ERR_OOM", -4: "VLAC_ERR_TIMEOUT",
          -5: "VLAC_ERR_DEVICE_CHECK", -6: "VLAC_ERR_STATE", -7: "VLAC_ERR_UNSUPPORTED"}
F32, BF16 = 0, 1
MARGIN_PROB, MARGIN_LOGIT, MARGIN_VOCAB = 0, 1, 2
REDUCE_DEFAULT, REDUCE_MEAN, REDUCE_MIN = -1, 0, 1


class VlacError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {ERRORS.get(code, code)} ({code})")


class Dims(C.Structure):
    _fields_ = [(n, C.c_int32) for n in (
        "n_layers", "hidden", "n_heads", "head_dim", "ffn", "vocab", "n_bins", "img_h", "img_w", "patch",
        "n_views", "n_text", "proprio_dim", "n_action", "parallel", "dtype")] + [
        ("rope_theta", C.c_float), ("rms_eps", C.c_float), ("max_batch", C.c_int32)]


_PP = C.POINTER(C.c_void_p)


class Weights(C.Structure):
    _fields_ = [("tok_emb", C.c_void_p), ("patch_w", C.c_void_p), ("proprio_w", C.c_void_p),
                ("action_emb", C.c_void_p)] + [(n, _PP) for n in (
                    "attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down")] + [
                ("final_norm", C.c_void_p), ("lm_head", C.c_void_p)]


class Rational(C.Structure):
    _fields_ = [("num", C.c_uint32), ("den", C.c_uint32)]


class StepOpts(C.Structure):
    _fields_ = [("margin_kind", C.c_int32), ("reduction", C.c_int32), ("gate_override", C.c_void_p),
                ("forced_ids", C.c_void_p), ("active", C.c_void_p), ("s2_top_k", C.c_int32), ("s2_layer", C.c_int32),
                ("s2_forced", C.c_void_p), ("s3_adaptive", C.c_int32), ("s3_lo", C.c_int32),
                ("s3_hi", C.c_int32), ("s3_weight", C.c_int32), ("s3_forced", C.c_void_p)]


class StepOut(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in (
        "action_ids", "margins", "logit_gap", "recomputed", "step_margin", "gate_auto", "logits",
        "static_mask", "idx", "M", "relevance", "relevant", "entropy", "vocab_margin", "action_delta",
        "layer_entropy", "schedule")]


EXPORTS = ["vlac_create", "vlac_destroy", "vlac_cache_bytes", "vlac_cache_init", "vlac_cache_destroy",
           "vlac_step", "vlac_reset", "vlac_sync_error", "vlac_launch_count", "vlac_selftest_wait",
           "vlac_set_wait_limit",
           "vlac_prof_enable", "vlac_prof_read", "vlac_select_noalloc", "vlac_strerror", "vlac_layer_bench",
           "vlac_cache_load", "vlac_cache_store"]


def lib():
    """Loads libvlac.so (once) and declares its signatures."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(f"libvlac.so is not built ({LIB_PATH}); run paper_2608_10824_gb300.build()")
            L = C.CDLL(LIB_PATH)
            vp, i32 = C.c_void_p, C.c_int
            L.vlac_create.argtypes = [C.POINTER(Dims), C.POINTER(Weights), C.POINTER(vp)]
            L.vlac_destroy.argtypes = [vp]
            L.vlac_cache_bytes.argtypes = [vp, i32, C.POINTER(C.c_size_t)]
            L.vlac_cache_init.argtypes = [vp, vp, C.c_size_t, i32, C.POINTER(vp)]
            L.vlac_cache_destroy.argtypes = [vp]
            L.vlac_step.argtypes = [vp, vp, vp, vp, vp, Rational, C.c_float, vp, C.POINTER(StepOpts),
                                    C.POINTER(StepOut), vp]
            L.vlac_reset.argtypes = [vp, i32, vp]
            L.vlac_sync_error.argtypes = [vp]
            L.vlac_launch_count.argtypes = [vp]
            L.vlac_launch_count.restype = C.c_uint64
            L.vlac_selftest_wait.argtypes = [vp, C.c_uint32]
            L.vlac_set_wait_limit.argtypes = [vp, C.c_uint32]
            L.vlac_prof_enable.argtypes = [vp, i32]
            L.vlac_prof_read.argtypes = [vp, i32, C.POINTER(C.c_double), C.POINTER(C.c_uint64),
                                         C.POINTER(C.c_double)]
            L.vlac_select_noalloc.argtypes = [C.POINTER(Dims), i32, vp, vp, vp, vp, Rational, C.c_float, vp, vp,
                                              vp, vp, vp, vp, vp]
            L.vlac_layer_bench.argtypes = [vp, vp, i32, i32, vp, i32, vp, vp]
            L.vlac_cache_load.argtypes = [vp, i32, i32, vp, vp, vp]
            L.vlac_cache_store.argtypes = [vp, i32, i32, vp, vp, vp]
            L.vlac_strerror.argtypes = [i32]
            L.vlac_strerror.restype = C.c_char_p
            for name in EXPORTS:
                if name not in ("vlac_launch_count", "vlac_strerror"):
                    getattr(L, name).restype = C.c_int
            _lib = L
    return _lib


def _check(rc: int, where: str):
    if rc != VLAC_OK:
        raise VlacError(rc, where)


def c_dims(d, max_batch: Optional[int] = None) -> Dims:
    return Dims(d.n_layers, d.hidden, d.n_heads, d.head_dim, d.ffn, d.vocab, d.n_bins, d.img_h, d.img_w,
                d.patch, d.n_views, d.n_text, d.proprio_dim, d.n_action, d.parallel,
                BF16 if d.dtype == "bf16" else F32, float(d.rope_theta), float(d.rms_eps),
                int(max_batch if max_batch is not None else d.max_batch))


def _ptr(t) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream_ptr(stream) -> Optional[int]:
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


class Context:
    """A model on the current CUDA device: repacked weights and workspace."""

    def __init__(self, d, weights: Dict, max_batch: Optional[int] = None):
        self.d = d
        self.max_batch = int(max_batch if max_batch is not None else d.max_batch)
        keep = []

        def arr(name):
            a = (C.c_void_p * d.n_layers)(*[lay[name].data_ptr() for lay in weights["layers"]])
            keep.append(a)
            return C.cast(a, _PP)

        w = Weights(_ptr(weights["tok_emb"]), _ptr(weights["patch_w"]), _ptr(weights.get("proprio_w")),
                    _ptr(weights.get("action_emb")), arr("attn_norm"), arr("wq"), arr("wk"), arr("wv"),
                    arr("wo"), arr("ffn_norm"), arr("w_gate"), arr("w_up"), arr("w_down"),
                    _ptr(weights["final_norm"]), _ptr(weights["lm_head"]))
        self._dims = c_dims(d, self.max_batch)
        h = C.c_void_p()
        _check(lib().vlac_create(C.byref(self._dims), C.byref(w), C.byref(h)), "vlac_create")
        self._h = h

    def close(self):
        h = getattr(self, "_h", None)
        if h is not None and h.value:
            lib().vlac_destroy(h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def cache_bytes(self, batch: int) -> int:
        n = C.c_size_t()
        _check(lib().vlac_cache_bytes(self._h, batch, C.byref(n)), "vlac_cache_bytes")
        return n.value

    def new_cache(self, batch: int = 1) -> "Cache":
        return Cache(self, batch)

    def alloc_outputs(self, batch: int, want: Sequence[str] = ()) -> Dict:
        import torch
        d, dev = self.d, torch.device("cuda")
        D = d.n_action
        out = {
            "action_ids": torch.zeros((batch, D), dtype=torch.int32, device=dev),
            "margins": torch.zeros((batch, D), dtype=torch.float32, device=dev),
            "logit_gap": torch.zeros((batch, D), dtype=torch.float32, device=dev),
            "recomputed": torch.zeros((batch,), dtype=torch.uint8, device=dev),
            "step_margin": torch.zeros((batch,), dtype=torch.float32, device=dev),
        }
        shapes = {"gate_auto": ((batch,), torch.uint8), "logits": ((batch, D, d.n_bins), torch.float32),
                  "static_mask": ((batch, d.n_visual), torch.uint8), "idx": ((batch, d.pass_len), torch.int32),
                  "M": ((batch, d.n_layers), torch.int32),
                  "relevance": ((batch, d.n_visual), torch.float32),
                  "relevant": ((batch, d.n_visual), torch.uint8),
                  "entropy": ((batch, D), torch.float32), "vocab_margin": ((batch, D), torch.float32),
                  "action_delta": ((batch,), torch.int32),
                  "layer_entropy": ((batch, d.n_layers), torch.float32),
                  "schedule": ((batch, d.n_layers), torch.int16)}
        for k in want:
            shp, dt = shapes[k]
            out[k] = torch.zeros(shp, dtype=dt, device=dev)
        return out

    def step(self, cache: "Cache", frames, prompt, proprio=None, tau_sim=(996, 1000), tau_margin: float = 0.0,
             permille=None, margin_kind: int = MARGIN_PROB, reduction: int = REDUCE_DEFAULT, gate_override=None,
             forced_ids=None, out: Optional[Dict] = None, want: Sequence[str] = (), stream=None,
             active=None, s2_top_k: int = 0, s2_layer: Optional[int] = None, s2_forced=None,
             s3_adaptive=None, s3_forced=None) -> Dict:
        """One step for every sequence of `cache`; inputs are CUDA tensors.
        Returns the dict of device output tensors (allocated unless given).
        s2_top_k > 0 turns on Stage 2 with the relevance of layer s2_layer
        (default: the middle layer); s2_forced (CUDA uint8 [B][Nv]) replaces
        its removal set (lock-step replay).  s3_adaptive = (lo, hi, weight)
        per mille turns on the entropy-adaptive Stage 3; s3_forced (CUDA
        uint16 [B][L]) replaces its schedule (lock-step replay)."""
        d = self.d
        if permille is None:
            permille = np.full(d.n_layers, 1000, dtype=np.uint16)
        permille = np.ascontiguousarray(permille, dtype=np.uint16)
        if out is None:
            out = self.alloc_outputs(cache.batch, want)
        so = StepOut(*[_ptr(out.get(k)) for k in (
            "action_ids", "margins", "logit_gap", "recomputed", "step_margin", "gate_auto", "logits",
            "static_mask", "idx", "M", "relevance", "relevant", "entropy", "vocab_margin", "action_delta",
            "layer_entropy", "schedule")])
        if s2_layer is None:
            s2_layer = d.n_layers // 2
        s3 = (0, 0, 0) if s3_adaptive is None else tuple(int(v) for v in s3_adaptive)
        opts = StepOpts(margin_kind, reduction, _ptr(gate_override), _ptr(forced_ids), _ptr(active), int(s2_top_k),
                        int(s2_layer), _ptr(s2_forced), int(s3_adaptive is not None), s3[0], s3[1], s3[2],
                        _ptr(s3_forced))
        rc = lib().vlac_step(self._h, cache._h, frames.data_ptr(), prompt.data_ptr(), _ptr(proprio),
                             Rational(int(tau_sim[0]), int(tau_sim[1])), float(tau_margin),
                             permille.ctypes.data, C.byref(opts), C.byref(so), _stream_ptr(stream))
        _check(rc, "vlac_step")
        return out

    def layer_bench(self, cache: "Cache", seq: int, layer: int, pos, x, stream=None):
        """One decoder layer for the rows at positions `pos` (CUDA int32 [M]);
        x (CUDA fp32 [M][hidden]) holds their inputs and receives their outputs."""
        assert pos.dtype.itemsize == 4 and x.is_contiguous() and x.shape[0] == pos.shape[0]
        _check(lib().vlac_layer_bench(self._h, cache._h, seq, layer, pos.data_ptr(), int(pos.shape[0]),
                                      x.data_ptr(), _stream_ptr(stream)), "vlac_layer_bench")

    def cache_load(self, cache: "Cache", seq: int, layer: int, K, V, stream=None):
        """K, V: CUDA [cache_len][hidden] in the model's dtype, into the cache."""
        _check(lib().vlac_cache_load(cache._h, seq, layer, K.data_ptr(), V.data_ptr(), _stream_ptr(stream)),
               "vlac_cache_load")

    def cache_store(self, cache: "Cache", seq: int, layer: int, K, V, stream=None):
        """K, V: CUDA [cache_len][hidden] in the model's dtype, filled from the cache."""
        _check(lib().vlac_cache_store(cache._h, seq, layer, K.data_ptr(), V.data_ptr(), _stream_ptr(stream)),
               "vlac_cache_store")

    def reset(self, cache: "Cache", seq: int = -1, stream=None):
        _check(lib().vlac_reset(cache._h, seq, _stream_ptr(stream)), "vlac_reset")

    def sync_error(self) -> int:
        return lib().vlac_sync_error(self._h)

    def launch_count(self) -> int:
        return int(lib().vlac_launch_count(self._h))

    def prof_enable(self, on: bool = True):
        _check(lib().vlac_prof_enable(self._h, int(on)), "vlac_prof_enable")

    def prof_read(self, kind: int):
        """(total device ms, launches, algorithmic bytes) of the timed launches of `kind`."""
        ms, n, by = C.c_double(), C.c_uint64(), C.c_double()
        _check(lib().vlac_prof_read(self._h, kind, C.byref(ms), C.byref(n), C.byref(by)), "vlac_prof_read")
        return ms.value, n.value, by.value

    def selftest_wait(self, spin_limit: int) -> int:
        return lib().vlac_selftest_wait(self._h, spin_limit)

    def set_wait_limit(self, polls: int):
        """Test hook: polls after which the step kernels' bounded waits give up."""
        _check(lib().vlac_set_wait_limit(self._h, int(polls)), "vlac_set_wait_limit")


def select_noalloc(d, frames, prev_frames, valid, m_prev, tau_sim=(996, 1000), tau_margin: float = 0.0,
                   permille=None, gate_override=None, out: Optional[Dict] = None, max_batch: Optional[int] = None,
                   stream=None) -> Dict:
    """Selection step without allocating device memory (see vlac_select_noalloc
    in include/vlac.h).  Inputs are CUDA tensors; `out` may hold preallocated
    outputs (static_mask, idx, M, recomputed), which this call then fills."""
    import torch
    B = frames.shape[0]
    if permille is None:
        permille = np.full(d.n_layers, 1000, dtype=np.uint16)
    permille = np.ascontiguousarray(permille, dtype=np.uint16)
    if out is None:
        dev = frames.device
        out = {"static_mask": torch.zeros((B, d.n_visual), dtype=torch.uint8, device=dev),
               "idx": torch.zeros((B, d.pass_len), dtype=torch.int32, device=dev),
               "M": torch.zeros((B, d.n_layers), dtype=torch.int32, device=dev),
               "recomputed": torch.zeros((B,), dtype=torch.uint8, device=dev)}
    dims = c_dims(d, max_batch if max_batch is not None else max(B, d.max_batch))
    rc = lib().vlac_select_noalloc(C.byref(dims), B, frames.data_ptr(), prev_frames.data_ptr(), valid.data_ptr(),
                                   m_prev.data_ptr(), Rational(int(tau_sim[0]), int(tau_sim[1])),
                                   float(tau_margin), permille.ctypes.data, _ptr(gate_override),
                                   out["static_mask"].data_ptr(), out["idx"].data_ptr(), out["M"].data_ptr(),
                                   out["recomputed"].data_ptr(), _stream_ptr(stream))
    _check(rc, "vlac_select_noalloc")
    return out


class Cache:
    """Device memory (a torch uint8 tensor) formatted by the library as a cache."""

    def __init__(self, ctx: Context, batch: int):
        import torch
        self.ctx, self.batch = ctx, batch
        nbytes = ctx.cache_bytes(batch)
        self._buf = torch.zeros(nbytes + 256, dtype=torch.uint8, device="cuda")
        base = self._buf.data_ptr()
        off = (-base) % 256
        self.mem = self._buf[off:off + nbytes]  # the formatted cache region
        h = C.c_void_p()
        _check(lib().vlac_cache_init(ctx._h, base + off, nbytes, batch, C.byref(h)), "vlac_cache_init")
        self._h = h

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and h.value:
            try:
                lib().vlac_cache_destroy(h)
            except Exception:
                pass
            self._h = None
