"""The benchmark's roofline arithmetic on CPU: the algorithmic bytes and flops
a step of each workload moves (the method's own work, each term written out
here from the workload's shape), the choice of the bound, and the DRAM
traffic read from profiles/dram_traffic.md, which goes null as soon as the
captured kernel's sources change."""

import math

import pytest

import bench
from paper_2607_13205_gb300 import inputs as I


def test_long_workload_counts():
    w = I.WORKLOADS["long"]                      # L=32, b=4, Hkv=8, G=4, W=64, N=32768, d=128
    c = bench.path_counts(w, 0.10)
    units = 32 * 4 * 8
    k_bytes = units * 32768 * 128 * 2            # bf16 K, read once
    q_bytes = units * (4 * 64) * 128 * 2         # the window rows of every unit
    s_bytes = units * 32768 * 4                  # fp32 pre-pool scores written
    assert c["score"]["bytes"] == k_bytes + q_bytes + s_bytes
    assert c["score"]["flops"] == 2.0 * units * 256 * 32768 * 128          # one Q K^T
    assert c["score"]["hw_flops"] == 2.0 * c["score"]["flops"]            # the exact two passes
    kept = math.ceil(0.10 * 32768)
    assert c["kept"] == kept == 3277
    # kept index written, then K and V rows read and written
    assert c["compact"]["bytes"] == units * kept * 4 + 2 * 2 * units * kept * 128 * 2
    assert c["compact"]["bytes"] / 1e9 == pytest.approx(3.449, abs=1e-3)
    # scores and roles read, index written
    assert c["select"]["bytes"] == units * 32768 * 4 + 4 * 32768 + units * kept * 4
    assert c["path_bytes"] / 1e9 == pytest.approx(12.39, abs=0.01)


def test_h2o_counts_are_causal():
    w = I.WORKLOADS["h2o"]                       # every position a query row, causal
    c = bench.path_counts(w, 0.05)
    units = w.L * w.b * w.Hkv
    pairs = w.n * (w.n + 1) / 2
    assert c["score"]["flops"] == pytest.approx(2.0 * units * w.G * pairs * w.d)
    assert c["score"]["bytes"] == units * w.n * w.d * 2 + units * w.G * w.n * w.d * 2 + units * w.n * 4


def test_varlen_counts_use_each_sequence():
    w = I.WORKLOADS["ragged"]
    c = bench.path_counts(w, 0.10)
    n_mean = sum(w.seqlens) / w.b
    units = w.L * w.b * w.Hkv
    assert c["score"]["bytes"] == pytest.approx(units * n_mean * w.d * 2 + units * w.G * w.W * w.d * 2
                                                + units * n_mean * 4)
    assert c["kept"] == pytest.approx(sum(math.ceil(0.10 * x) for x in w.seqlens) / w.b)


def _peaks():
    return {"hbm_gbs": 6000.0, "bf16_tflops": 2000.0, "source": "test"}


def test_roofline_takes_the_slower_bound():
    counts = {"a": {"bytes": 6e9, "flops": 1e12}, "b": {"bytes": 1e6, "flops": 0.0}}
    # 6e9 B at 6 TB/s is 1 ms, 1e12 flop at 2 PF/s is 0.5 ms: HBM-bound
    r = bench.roofline(counts, {"a": 2.0, "b": 0.1}, _peaks(), ["a", "b"], "x", "snapkv", 0, 1.0)
    assert r["kernel"] == "a" and r["bound"] == "hbm"
    assert r["achieved"] == pytest.approx(6e9 / 2e-3 / 1e9) and r["frac"] == pytest.approx(0.5)
    assert r["traffic"] == 1.0
    counts["a"]["flops"] = 4e12                  # now 2 ms of tensor work
    r = bench.roofline(counts, {"a": 4.0, "b": 0.1}, _peaks(), ["a", "b"], "x", "snapkv", 0, None)
    assert r["bound"] == "tensor" and r["frac"] == pytest.approx(0.5)


def test_traffic_row_is_scaled_by_units_and_goes_stale(monkeypatch):
    got, note = bench.measured_traffic("long", "snapkv", "score")
    if got is None:
        pytest.skip(f"the score capture does not match the current sources ({note})")
    # the 2-layer capture of 64 units, scaled to the 1024-unit launch
    assert 10e9 < got < 20e9 and "scaled by units" in note
    monkeypatch.setattr(bench, "source_hash", lambda files: "0" * 16)
    got, note = bench.measured_traffic("long", "snapkv", "score")
    assert got is None and note.startswith("stale")
