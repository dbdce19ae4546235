"""Host-side pieces of bench.py that feed the JSON line (no GPU): the measured
peaks, and the DRAM traffic record that roofline.traffic reports only while the
profiled kernel sources are unchanged."""
import json
import os

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_peaks_are_the_measured_ones():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    pk = bench.load_peaks()
    if not os.path.exists(path):  # written per machine, not committed
        assert pk["source"] == "fallback"
        return
    with open(path) as f:
        m = json.load(f)
    assert pk["source"] == "measured"
    assert pk["hbm_gbs"] == m["hbm_gbs"] and pk["bf16_tflops"] == m["bf16_tflops"]


def test_traffic_record_shape_and_scaling():
    """Each entry: captured read + write bytes at `captured_batch` sequences,
    scaled to the workload's batch (traffic grows with the sequences processed)."""
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        rec = json.load(f)
    from paper_2608_02625_gb300 import workloads
    n = 0
    for kfile, kernels in rec.items():
        if not kfile.endswith(".cu"):
            continue
        for kname, per_w in kernels.items():
            for wname, e in per_w.items():
                w = workloads.get(wname)
                cap = e["dram_read_bytes_captured"] + e["dram_write_bytes_captured"]
                assert e["dram_bytes_per_launch"] == cap * w.B / e["captured_batch"]
                assert len(e["source_sha"]) == 16
                n += 1
    assert n >= 2


def test_traffic_is_dropped_when_the_kernel_changed(monkeypatch):
    key = ("vocab.cu", "vocab_rows_kernel", "c3_batch32_512")
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        e = json.load(f)["vocab.cu"]["vocab_rows_kernel"]["c3_batch32_512"]
    monkeypatch.setattr(bench, "kernel_source_sha", lambda fname: e["source_sha"])
    assert bench.recorded_traffic(*key) == e["dram_bytes_per_launch"]
    monkeypatch.setattr(bench, "kernel_source_sha", lambda fname: "0" * 16)
    assert bench.recorded_traffic(*key) is None
    assert bench.recorded_traffic("vocab.cu", "no_such_kernel", "c3_batch32_512") is None


def test_source_sha_covers_the_shared_headers(monkeypatch):
    """The hash changes with the kernel file and with the headers it includes."""
    real_open = open
    seen = []

    def spy(path, *a, **k):
        seen.append(os.path.basename(path))
        return real_open(path, *a, **k)

    monkeypatch.setattr("builtins.open", spy)
    bench.kernel_source_sha("attn_tc.cu")
    assert {"attn_tc.cu", "dlm_common.cuh", "update_impl.cuh"} <= set(seen)
