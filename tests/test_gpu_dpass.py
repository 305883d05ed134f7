"""The two decode paths against the oracle: the persistent decode pass (one
cooperative launch per decode token; the default where it applies: bf16,
head_dim 128, one or two sequences) and the per-projection chain
(VLAC_DPASS=0; every other shape).  Both are held to the same bars, on the
shapes the persistent pass supports, so that the chain stays covered there."""
import pytest

import synth
from tests.gpu_common import SMALL, Lockstep, episode

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("path", ["dpass", "chain"])
@pytest.mark.parametrize("chunks", ["auto", "1", "3"])
@pytest.mark.parametrize("name,batch", [("small", 1), ("small_wide", 1), ("small_wide", 2), ("wide", 1), ("wide", 2)])
def test_decode_path_parity(name, batch, chunks, path, cuda_device, monkeypatch):
    """chunks: key ranges per (sequence, head) in the persistent pass's
    attention phase (1: one CTA per head; otherwise the ranges' partials are
    combined by the last to finish)."""
    if path == "chain" and chunks != "auto":
        pytest.skip("the key ranges are the persistent pass's")
    monkeypatch.setenv("VLAC_DPASS", "1" if path == "dpass" else "0")
    if chunks != "auto":
        monkeypatch.setenv("VLAC_DPASS_ATTN_CHUNKS", chunks)
    d = SMALL[name]
    w = synth.make_weights(d, seed=21)
    ls = Lockstep(d, w, batch=batch)
    frames, prompt, _ = episode(d, 3, seed=22, batch=batch)
    pm = synth.linear_schedule(d.n_layers)
    for t in range(3):
        ls.step(frames[t], prompt, None, (95, 100), 0.0, pm)


@pytest.mark.parametrize("name", ["small", "wide"])
def test_decode_paths_without_staging(name, cuda_device, monkeypatch):
    """The persistent pass with its attention reading every K/V row from
    global memory (VLAC_DPASS_KV=0), as it does where the staging buffer
    does not fit."""
    monkeypatch.setenv("VLAC_DPASS", "1")
    monkeypatch.setenv("VLAC_DPASS_KV", "0")
    d = SMALL[name]
    ls = Lockstep(d, synth.make_weights(d, seed=23))
    frames, prompt, _ = episode(d, 3, seed=24)
    pm = synth.linear_schedule(d.n_layers)
    for t in range(3):
        ls.step(frames[t], prompt, None, (95, 100), 0.0, pm)
