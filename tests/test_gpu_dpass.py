"""The persistent decode pass (one cooperative launch per decode token,
VLAC_DPASS=1) against the oracle, on the shapes it supports (bf16,
head_dim 128, one or two sequences): the same bars as the per-projection
chain."""
import os

import pytest

import synth
from tests.gpu_common import SMALL, Lockstep, episode

pytestmark = pytest.mark.gpu


@pytest.fixture
def dpass_on():
    old = os.environ.get("VLAC_DPASS")
    os.environ["VLAC_DPASS"] = "1"
    yield
    if old is None:
        os.environ.pop("VLAC_DPASS", None)
    else:
        os.environ["VLAC_DPASS"] = old


@pytest.mark.parametrize("chunks", ["auto", "1", "3"])
@pytest.mark.parametrize("name,batch", [("small", 1), ("small_wide", 1), ("small_wide", 2), ("wide", 1), ("wide", 2)])
def test_dpass_parity(name, batch, chunks, dpass_on, cuda_device, monkeypatch):
    """chunks: key ranges per (sequence, head) in the attention phase (1: one
    CTA per head; otherwise the ranges' partials are combined by the last)."""
    if chunks != "auto":
        monkeypatch.setenv("VLAC_DPASS_ATTN_CHUNKS", chunks)
    d = SMALL[name]
    w = synth.make_weights(d, seed=21)
    ls = Lockstep(d, w, batch=batch)
    frames, prompt, _ = episode(d, 3, seed=22, batch=batch)
    pm = synth.linear_schedule(d.n_layers)
    for t in range(3):
        ls.step(frames[t], prompt, None, (95, 100), 0.0, pm)
