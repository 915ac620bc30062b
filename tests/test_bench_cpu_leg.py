"""The CPU-oracle leg of bench.py without a GPU: host copies of a workload's rows (here drawn
by torch on the CPU) go through the float64 oracle on a spawn pool, and the fused head's oracle
runs on a small host sample."""
import os
import sys
import types

import numpy as np
import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2608_16798_gb300 import workloads as W  # noqa: E402


@pytest.mark.parametrize("name,n,starts", [("tiny", 512, (0,)), ("edge", 96, (0,)), ("longhorizon", 40, (0, 32768))])
def test_oracle_slice_timing(name, n, starts):
    w = W.WORKLOADS[name]
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    pieces = []
    for lo in starts:
        lg = torch.empty((n, w.vocab), dtype=dt)
        W.logits_rows_torch(w, 0, lo, n, lg)
        pieces.append((lo, lg, W.sample_tokens_torch(lg, 0, lo, w)))
    sl = bench.OracleSlice(w, pieces, bench.ORACLE_PARAMS[name])
    try:
        # the host copy holds the device rows bit for bit
        got = sl.raw[:n].view(np.int16 if w.dtype == "bf16" else np.int32)
        want = pieces[0][1].view(torch.int16 if w.dtype == "bf16" else torch.int32).numpy()
        assert np.array_equal(got, want)
        inp = sl.oracle_inputs()
        assert (inp["ref"] is not None) == bool(w.ref_noise_std)
        assert np.all(np.isfinite(inp["old"]))
        r = bench.time_oracle_slice(sl)
    finally:
        sl.close()
    assert r["rows"] == n * len(starts) and r["tokens_per_s"] > 0 and r["cores"] >= 1


def test_oracle_head_timing():
    hb = types.SimpleNamespace()
    V, D, T = 1000, 128, 16
    g = torch.Generator().manual_seed(0)
    hb.hidden = torch.randn(T, D, generator=g).to(torch.bfloat16)
    hb.weight = (torch.randn(V, D, generator=g) * 0.02).to(torch.bfloat16)
    hb.ids = torch.randint(0, V, (T,), dtype=torch.int32, generator=g)
    hb.old = torch.randn(T, generator=g) - 7.0
    hs = bench.HeadSample(torch, hb, 8)
    assert hs.hidden.shape == (8, D) and hs.weight.shape == (V, D)
    r = bench.time_oracle_head(hs)
    assert r["rows"] == 8 and r["flops"] == 6.0 * 8 * D * V and r["tokens_per_s"] > 0


def test_oracle_slice_failure_is_reported_not_raised(monkeypatch):
    """A slice that cannot be made (shared memory short) is reported as unavailable."""
    def no_room(*a, **k):
        raise OSError(28, "No space left on device")

    monkeypatch.setattr(bench, "OracleSlice", no_room)
    sl = bench.make_oracle_slice(W.WORKLOADS["tiny"], [], {})
    assert isinstance(sl, str) and "OSError" in sl
    assert bench.time_oracle_slice(sl) == {"unavailable": sl}


def test_oracle_slice_falls_back_to_fewer_rows(monkeypatch):
    """A span too large for shared memory is retried as its first rows; only when that fails
    too is the slice reported as unavailable."""
    made = []

    class Tight:
        def __init__(self, w, pieces, params):
            n = sum(int(lg.shape[0]) for _, lg, _ in pieces)
            if n > 8:
                raise OSError(28, "No space left on device")
            made.append(n)

    monkeypatch.setattr(bench, "OracleSlice", Tight)
    lg, ids = torch.zeros((20, 4)), torch.zeros(20, dtype=torch.int32)
    sl = bench.make_oracle_slice(W.WORKLOADS["tiny"], [(0, lg, ids)], {}, fallback_rows=8)
    assert isinstance(sl, Tight) and made == [8]
    sl = bench.make_oracle_slice(W.WORKLOADS["tiny"], [(0, lg, ids)], {}, fallback_rows=12)
    assert isinstance(sl, str) and "OSError" in sl
