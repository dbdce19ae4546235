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


def test_reference_arm_json_line():
    """bench.py --impl reference on the tiny workload: one JSON line with the
    contract's keys; the oracle's workers never outnumber the sequences."""
    import subprocess
    import sys
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--config",
                        "c1_tiny_f32", "--steps", "1", "--warmup", "3"], capture_output=True, text=True, timeout=300,
                       cwd=ROOT)
    assert r.returncode == 0, r.stderr
    d = json.loads(r.stdout.strip().splitlines()[-1])
    assert d["impl"] == "reference" and d["metric"] == "refine_steps_per_sec" and d["unit"] == "steps/s"
    assert d["higher_is_better"] is True and d["value"] > 0
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] == 1  # c1 has one sequence
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert d["config"]["workload"] == "c1_tiny_f32"
    # A step is the whole batch and its time is time that passed.
    assert abs(d["ms_per_step"] * d["steps"] - d["timed_region_s"] * 1e3) <= 1e-6 * d["timed_region_s"] * 1e3
    assert "whole batch" in cb["sample"]


def test_clock_summary_window_and_reasons():
    """The clock record keeps the samples inside the timed region (all samples
    when none fell inside), the median SM clock and every active reason."""
    c = bench.ClockSampler(0)
    c.samples = [(1.0, 1500.0, 2070.0, set()), (2.0, 2070.0, 2070.0, {"sw_power_cap"}),
                 (2.5, 2060.0, 2070.0, set()), (3.0, 2070.0, 2070.0, {"hw_slowdown"}), (9.0, 900.0, 2070.0, set())]
    s = c.summary(1.9, 3.1)
    assert s["samples"] == 3 and s["sm_mhz"] == 2070.0 and s["sm_mhz_min"] == 2060.0
    assert s["reasons"] == ["hw_slowdown", "sw_power_cap"] and s["window"] == "timed region"
    s = c.summary(4.0, 5.0)
    assert s["samples"] == 5 and s["window"].startswith("whole run")
