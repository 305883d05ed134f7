"""The C-ABI library loads on a host without a GPU, exports every entry
point include/vlac.h declares, and rejects invalid dims before touching the
device."""
import ctypes as C
import os
import re

import pytest

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "vlac.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(vlac_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    import paper_2608_10824_gb300 as pkg
    pkg.build()
    return pkg.lib()


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("vlac_create", "vlac_step", "vlac_reset", "vlac_destroy", "vlac_cache_bytes", "vlac_cache_init",
              "vlac_strerror"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    missing = [n for n in _declared() if not hasattr(lib, n)]
    assert not missing, missing


def test_strerror_names_every_code(lib):
    for code in (0, -1, -2, -3, -4, -5, -6, -7):
        s = lib.vlac_strerror(code)
        assert s and s != b"unknown error"
    assert lib.vlac_strerror(-99) == b"unknown error"


def test_invalid_dims_rejected_without_a_device(lib):
    from paper_2608_10824_gb300.vlac import Weights, c_dims
    h = C.c_void_p()
    w = Weights()
    bad = [
        synth.dims_for("tiny", n_heads=3),                     # heads * head_dim != hidden
        synth.dims_for("tiny", img_h=100),                     # image not a multiple of the patch
        synth.dims_for("tiny", n_text=1),                      # autoregressive decode needs a text token
        synth.dims_for("tiny", max_batch=9),
        synth.dims_for("tiny", n_bins=1),
    ]
    for d in bad:
        dd = c_dims(d)
        assert lib.vlac_create(C.byref(dd), C.byref(w), C.byref(h)) == -1
    dd = c_dims(synth.dims_for("tiny", head_dim=32, n_heads=8))  # valid, not implemented
    assert lib.vlac_create(C.byref(dd), C.byref(w), C.byref(h)) == -7
    dd = c_dims(synth.dims_for("tiny", dtype="bf16"))         # ffn 688 is not a multiple of 64 for bf16
    assert lib.vlac_create(C.byref(dd), C.byref(w), C.byref(h)) == -7
    assert lib.vlac_create(None, C.byref(w), C.byref(h)) == -1


def test_null_handles_are_invalid_arguments(lib):
    assert lib.vlac_destroy(None) == -1
    assert lib.vlac_cache_destroy(None) == -1
    assert lib.vlac_reset(None, 0, None) == -1
    n = C.c_size_t()
    assert lib.vlac_cache_bytes(None, 1, C.byref(n)) == -1
    assert lib.vlac_launch_count(None) == 0
    # the one-layer entry and the cache K/V copies refuse NULL handles before any device call
    assert lib.vlac_layer_bench(None, None, 0, 0, None, 1, None, None) == -1
    assert lib.vlac_cache_load(None, 0, 0, None, None, None) == -1
    assert lib.vlac_cache_store(None, 0, 0, None, None, None) == -1
