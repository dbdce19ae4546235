"""Throughput of one bidirectional refine step (attention -> vocabulary
reduction -> update) on GB300, as refine steps/s over a whole batch.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME] [--impl ours|reference]

Default workload: the batched 32 x 512 refine (128 prompt + 384 response
tokens per sequence, prompts U{64..256}, 32/4 heads, head_dim 128,
V = 151552, bf16). Inputs are synthetic (seeded generator) and resident in HBM
before timing; every input is larger than L2, so no flush is needed.

Prints one JSON line (rank 0). For N > 1 (torchrun) every rank runs its own
replica on its own seeded batch (weak scaling, no collective on the data
path); the step time is the max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import multiprocessing as mp
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "refine_steps_per_sec"
# The paper's own headline numbers (Table 1, Table 4): end-to-end seconds per
# example of whole-model decoding on hardware it does not name. Context only:
# they are speedups of a decoding scheme, not a refine-step throughput.
PAPER_CONTEXT = {
    "speedups": {"flash_flash_vs_selected_block_ar_gsm8k_384": 1.20, "mini_flash_vs_flash_math_384": 2.17},
    "seconds_per_example": {"gsm8k_384": [19.38, 16.09], "math_384": [40.90, 18.82]},
    "hardware": "not stated by the paper",
    "comparable": False,
}
UNIT = "steps/s"
DEFAULT_CONFIG = "c3_batch32_512"


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        return {"hbm_gbs": pk["hbm_gbs"], "bf16_tflops": pk["bf16_tflops"],
                "bf16_tflops_sustained": pk.get("bf16_tflops_sustained"), "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


# ---------------------------------------------------------------- clocks

class ClockSampler:
    """Samples the SM clock and the throttle reasons during the timed region.

    Read-only queries only. Through NVML (the driver's libnvidia-ml, via
    ctypes) every 2 ms when it loads, so that even a region of ~20 ms carries
    several samples; otherwise nvidia-smi's own loop every 5 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    # NVML clock event reason bits
    REASON_BITS = {"sw_power_cap": 0x4, "hw_slowdown": 0x8, "sw_thermal_slowdown": 0x20,
                   "hw_thermal_slowdown": 0x40}

    def __init__(self, gpu_index: int, pci_bus_id: str | None = None):
        self.gpu = gpu_index
        self.pci = pci_bus_id
        self.proc = None
        self.samples = []     # (host time, sm_mhz, sm_max_mhz, set of active reason names)
        self.source = None
        self._stop = threading.Event()

    def _nvml(self):
        import ctypes
        lib = ctypes.CDLL("libnvidia-ml.so.1")
        if lib.nvmlInit_v2() != 0:
            return None
        h = ctypes.c_void_p()
        if not (self.pci and lib.nvmlDeviceGetHandleByPciBusId_v2(self.pci.encode(), ctypes.byref(h)) == 0):
            if lib.nvmlDeviceGetHandleByIndex_v2(self.gpu, ctypes.byref(h)) != 0:
                return None
        reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            lib.nvmlDeviceGetCurrentClocksThrottleReasons
        mhz, mx, rs = ctypes.c_uint(), ctypes.c_uint(), ctypes.c_ulonglong()

        def poll():
            if lib.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(mhz)) != 0:   # NVML_CLOCK_SM
                return None
            lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx))
            reasons_fn(h, ctypes.byref(rs))
            return (float(mhz.value), float(mx.value),
                    {n for n, bit in self.REASON_BITS.items() if rs.value & bit})
        return poll if poll() is not None else None

    def __enter__(self):
        poll = None
        try:
            poll = self._nvml()
        except Exception:
            poll = None
        if poll is not None:
            self.source = "nvml every 2 ms"

            def run():
                while not self._stop.is_set():
                    r = poll()
                    if r is not None:
                        self.samples.append((time.time(),) + r)
                    time.sleep(0.002)
            self.thread = threading.Thread(target=run, daemon=True)
            self.thread.start()
            return self
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "5"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.source = "nvidia-smi -lms 5"
            self.thread = threading.Thread(target=self._read_smi, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None
        return self

    def _read_smi(self):
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.strip().split(",")]
            if len(parts) < 9:
                continue
            try:
                sm, mx = float(parts[1]), float(parts[2])
            except ValueError:
                continue
            active = {nm for nm, val in zip(names, parts[5:9]) if val.lower().startswith("active")}
            self.samples.append((time.time(), sm, mx, active))

    def __exit__(self, *exc):
        self._stop.set()
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self, t0=None, t1=None):
        """Median SM clock and active throttle reasons of the samples taken in
        [t0, t1] (host time); all samples if the window caught none."""
        win = [x for x in self.samples if t0 is None or t0 <= x[0] <= t1]
        window = "timed region"
        if not win:
            win = list(self.samples)
            window = "whole run (no sample inside the timed region)"
        if not win:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "source": self.source}
        reasons = set()
        for x in win:
            reasons |= x[3]
        return {"sm_mhz": statistics.median(x[1] for x in win), "sm_max_mhz": max(x[2] for x in win),
                "sm_mhz_min": min(x[1] for x in win), "reasons": sorted(reasons), "samples": len(win),
                "window": window, "source": self.source}


# ---------------------------------------------------------------- traffic record

def kernel_source_sha(fname: str) -> str:
    h = hashlib.sha256()
    for f in (fname, "dlm_common.cuh", "update_impl.cuh"):
        with open(os.path.join(ROOT, "paper_2608_02625_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel_file: str, kernel: str, workload: str):
    """DRAM bytes per launch of `kernel` from the committed ncu summary, if the
    kernel source still matches the one profiled (else None)."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            rec = json.load(f)
        e = rec[kernel_file][kernel][workload]
        if e["source_sha"] != kernel_source_sha(kernel_file):
            return None
        return e["dram_bytes_per_launch"]
    except Exception:
        return None


# ---------------------------------------------------------------- CPU oracle timing

def _oracle_worker(conn, name, seqs):
    """A host core running the oracle on whole sequences `seqs` of the
    workload: fp64 attention over every head, the vocabulary reduction of
    every row, and the update of the sequence from those predictions. Inputs
    are generated once, before any timing."""
    import numpy as np
    import oracle
    from paper_2608_02625_gb300 import synth, workloads
    w = workloads.get(name)
    tok, msk = w.initial_state()
    n_all, p_all = w.seq_lens(), w.prompt_lens()

    def host(b, which, H):
        per = w.L * H * w.D
        x = synth.qkv_host(w.seed, which, (w.B, w.L, H, w.D), w.qkv_sigma, w.dtype, b * per, per)
        x = synth.bf16_bits_to_f32(x) if w.dtype == "bf16" else x
        return x.reshape(1, w.L, H, w.D)

    inputs = []
    for b in seqs:
        rows = np.arange(b * w.L, (b + 1) * w.L)
        x = w.logit_spec(0).rows_f32(rows, tok.reshape(-1)[rows], msk.reshape(-1)[rows])
        if w.dtype == "bf16":
            x = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(x))
        inputs.append((b, host(b, synth.S_Q, w.Hq), host(b, synth.S_K, w.Hkv), host(b, synth.S_V, w.Hkv), x))
    conn.send("ready")
    while conn.recv() == "run":
        t = [0.0, 0.0, 0.0]
        for b, q, k, v, x in inputs:
            t0 = time.perf_counter()
            oracle.bidir_attn(q, k, v, n_all[b:b + 1])
            t1 = time.perf_counter()
            am, cf, _ = oracle.vocab_confidence(x)
            t2 = time.perf_counter()
            oracle.refine_update(tok[b:b + 1], msk[b:b + 1], am[None, :], cf[None, :],
                                 edit_threshold=w.edit_threshold[0], remask_k=w.remask_k, remask_frac=w.remask_frac,
                                 mask_id=w.mask_id, prompt_lens=p_all[b:b + 1], seq_lens=n_all[b:b + 1])
            t3 = time.perf_counter()
            t = [t[0] + t1 - t0, t[1] + t2 - t1, t[2] + t3 - t2]
        conn.send(tuple(t))


class OracleTimer:
    """The oracle on the whole batch of a workload, spread over the host cores:
    single-threaded processes (spawned; at most one per sequence), each owning
    whole sequences (sequence b goes to process b mod P). One round is one
    refine step of the whole batch, and its time is the wall time until the
    last process is done."""

    def __init__(self, name: str, workers: int):
        from paper_2608_02625_gb300 import workloads
        self.w = workloads.get(name)
        self.name = name
        workers = max(1, min(workers, self.w.B))
        os.environ["OPENBLAS_NUM_THREADS"] = "1"
        os.environ["OMP_NUM_THREADS"] = "1"
        ctx = mp.get_context("spawn")
        self.conns, self.procs = [], []
        for i in range(workers):
            a, bconn = ctx.Pipe()
            seqs = list(range(i, self.w.B, workers))
            pr = ctx.Process(target=_oracle_worker, args=(bconn, name, seqs), daemon=True)
            pr.start()
            self.conns.append(a)
            self.procs.append(pr)
        self.ready = False

    def wait_ready(self):
        """Block until every worker has generated its inputs (they use the host
        cores and memory bandwidth until then)."""
        if not self.ready:
            for c in self.conns:
                assert c.recv() == "ready"
            self.ready = True

    def run(self):
        """One refine step of the whole batch on the oracle. Returns cpu_baseline."""
        self.wait_ready()
        t0 = time.perf_counter()
        for c in self.conns:
            c.send("run")
        parts = [c.recv() for c in self.conns]
        wall = time.perf_counter() - t0
        w = self.w
        cores = len(self.conns)
        return {"value": 1.0 / wall, "unit": UNIT, "cores": cores, "kind": "oracle", "ms_per_step": wall * 1e3,
                "sample": (f"the whole batch of {self.name} ({w.B} sequences, all {w.Hq} heads, all {w.L} "
                           f"vocabulary rows of {w.V}), one step, on {cores} single-threaded processes owning "
                           f"whole sequences; steps/s = 1 / wall time of the step"),
                "oracle_cpu_s_per_step": {"attn": sum(x[0] for x in parts), "vocab": sum(x[1] for x in parts),
                                          "update": sum(x[2] for x in parts)}}

    def close(self):
        for c in self.conns:
            try:
                c.send("stop")
            except Exception:
                pass
        for pr in self.procs:
            pr.join(timeout=10)


def host_workers():
    return max(1, min(64, os.cpu_count() or 1))


# ---------------------------------------------------------------- multi-GPU (replicas)

def replica_workload(base, rank: int):
    """Weak scaling: rank r refines its own seeded batch of the base workload's
    shape; ranks never exchange data."""
    from paper_2608_02625_gb300 import workloads
    return workloads.scaled(base, seed=base.seed + rank)


def max_over_ranks(value_ms: float, world: int, device) -> float:
    """The slowest rank's time: the job is done when its last replica is."""
    if world == 1:
        return value_ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([value_ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_steps_per_s(ms_per_step: float, world: int) -> float:
    """Whole-job refine steps/s: each of the `world` replicas finishes one
    step of its own batch every ms_per_step."""
    return world * 1000.0 / ms_per_step


# ---------------------------------------------------------------- GPU arm

def measure_loop(args, w, Bn, q, k, v, out, logits, tok0, msk0, params, seqlen, stream):
    """Refine passes on one resident batch with tokens / mask updated in place,
    until no confident edit remains or --loop-steps passes have run: (a) as one
    launch of a recorded loop, (b) pass by pass with n_edits read back by the
    host after each pass. Both run the same passes on the same buffers."""
    import torch
    d = tok0.device
    tok, msk = tok0.clone(), msk0.clone()
    am = torch.empty((w.B, w.L), dtype=torch.int32, device=d)
    cf = torch.empty((w.B, w.L), dtype=torch.float32, device=d)
    ls = torch.empty((w.B, w.L), dtype=torch.float32, device=d)
    ne = torch.zeros(w.B, dtype=torch.int32, device=d)
    ws = torch.zeros(w.B, dtype=torch.int32, device=d)
    steps = torch.zeros(1, dtype=torch.int32, device=d)

    def one_pass():
        Bn.dlm_bidir_attn(q, k, v, seqlen, out)
        if args.path == "fused":
            Bn.dlm_refine_step(logits, tok, msk, params, am, cf, ls, tok, msk, ne, ws)
        else:
            Bn.dlm_vocab_confidence(logits, am.view(-1), cf.view(-1), ls.view(-1))
            Bn.dlm_refine_update(tok, msk, am, cf, params, tok, msk, ne)

    def host_driven():
        n = 0
        for s in range(args.loop_steps):
            one_pass()
            n = s + 1
            if not bool((ne > 0).any()):   # host round trip after every pass
                break
        return n

    side = torch.cuda.Stream(d)
    side.wait_stream(stream)
    with torch.cuda.stream(side):
        Bn.dlm_loop_begin(steps)
        try:
            one_pass()
        except BaseException:
            Bn.dlm_loop_cancel()
            raise
        loop = Bn.dlm_loop_end(ne, args.loop_steps, steps)
    torch.cuda.synchronize()
    reps = 10
    try:
        with torch.cuda.stream(side):
            for _ in range(3):
                tok.copy_(tok0)
                msk.copy_(msk0)
                loop.launch()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            t_graph = 0.0
            for _ in range(reps):
                tok.copy_(tok0)
                msk.copy_(msk0)
                e0.record(side)
                loop.launch()
                e1.record(side)
                torch.cuda.synchronize()
                t_graph += e0.elapsed_time(e1)
            passes = int(steps.item())
            graph_state = (tok.clone(), msk.clone())
            t_host = 0.0
            for r in range(reps + 1):
                tok.copy_(tok0)
                msk.copy_(msk0)
                torch.cuda.synchronize()
                t0 = time.perf_counter()
                n_host = host_driven()
                torch.cuda.synchronize()
                if r > 0:   # the first run warms up
                    t_host += (time.perf_counter() - t0) * 1e3
            same = bool(torch.equal(tok, graph_state[0]) and torch.equal(msk, graph_state[1]))
    finally:
        loop.close()
    if Bn.device_error(clear=True):
        raise RuntimeError("device error word set during the loop measurement")
    return {"workload": w.name, "max_passes": args.loop_steps, "passes": passes, "passes_host_driven": n_host,
            "same_result": same, "ms_graph_launch": t_graph / reps, "ms_host_driven": t_host / reps,
            "note": "pass = attention + vocabulary reduction + in-place update on resident q/k/v and logits; "
                    "graph: CUDA events around one launch; host-driven: wall clock, one n_edits read-back per pass"}


def measure_fused_step(Bn, w, logits, tok, msk, params, stream, per_kernel, reps=20):
    """The vocabulary reduction and the update in one launch (dlm_refine_step)
    on the step's own resident buffers, against the two separate launches
    timed in the step (CUDA events around `reps` back-to-back launches)."""
    import torch
    d = logits.device
    am = torch.empty((w.B, w.L), dtype=torch.int32, device=d)
    cf = torch.empty((w.B, w.L), dtype=torch.float32, device=d)
    ls = torch.empty((w.B, w.L), dtype=torch.float32, device=d)
    nt, nm = torch.empty_like(tok), torch.empty_like(msk)
    ne = torch.empty(w.B, dtype=torch.int32, device=d)
    ws = torch.zeros(Bn.dlm_refine_step_workspace_bytes(w.B) // 4, dtype=torch.int32, device=d)

    def run():
        Bn.dlm_refine_step(logits, tok, msk, params, am, cf, ls, nt, nm, ne, ws)

    for _ in range(3):
        run()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        run()
    e1.record(stream)
    torch.cuda.synchronize()
    if Bn.device_error(clear=True):
        raise RuntimeError("device error word set during the fused-step measurement")
    ms = e0.elapsed_time(e1) / reps
    sep = per_kernel["vocab"] + per_kernel["update"]
    return {"ms": ms, "ms_separate_vocab_plus_update": sep, "ratio_fused_over_separate": ms / sep,
            "note": "dlm_refine_step (one launch: the CTA finishing a sequence's last row runs its update) on the "
                    "step's buffers; the step itself uses the separate launches, the faster of the two here"}


def measure_lmhead(args, w, Bn, peaks, reps=10):
    """The vocabulary projection fused with the reduction (dlm_lmhead_confidence)
    on the workload's N rows and V tokens at width d = --lmhead-d, against the
    unfused pair: a cuBLAS bf16 GEMM writing the bf16 logits (torch.matmul)
    followed by dlm_vocab_confidence. Inputs: seeded normals on the device."""
    import torch
    from paper_2608_02625_gb300 import synth, synth_gpu
    d = torch.device("cuda", torch.cuda.current_device())
    dm = args.lmhead_d
    hidden = torch.empty((w.N, dm), dtype=torch.bfloat16, device=d)
    weight = torch.empty((w.V, dm), dtype=torch.bfloat16, device=d)
    synth_gpu.fill_normal_(hidden, synth.stream_key(w.seed + 101, synth.S_Q), 1.0)
    synth_gpu.fill_normal_(weight, synth.stream_key(w.seed + 101, synth.S_K), 1.0 / dm ** 0.5)
    am = torch.empty(w.N, dtype=torch.int32, device=d)
    cf = torch.empty(w.N, dtype=torch.float32, device=d)
    ls = torch.empty(w.N, dtype=torch.float32, device=d)
    ws = torch.empty(Bn.dlm_lmhead_workspace_bytes(w.N), dtype=torch.uint8, device=d)
    stream = torch.cuda.current_stream(d)

    def timed(fn):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps

    t_fused = timed(lambda: Bn.dlm_lmhead_confidence(hidden, weight, am, cf, ls, ws))
    am_f = am.clone()
    logits = torch.empty((w.N, w.V), dtype=torch.bfloat16, device=d)

    def unfused():
        torch.matmul(hidden, weight.t(), out=logits)
        Bn.dlm_vocab_confidence(logits, am, cf, ls)

    t_unfused = timed(unfused)
    t_gemm = timed(lambda: torch.matmul(hidden, weight.t(), out=logits))
    agree = float((am == am_f).float().mean().item())
    del logits
    torch.cuda.empty_cache()
    if Bn.device_error(clear=True):
        raise RuntimeError("device error word set during the projection measurement")
    flops = 2.0 * w.N * w.V * dm
    return {"rows": w.N, "vocab": w.V, "d": dm, "flops": flops, "ms_fused": t_fused,
            "tflops_fused": flops / (t_fused * 1e-3) / 1e12,
            "frac_of_measured_bf16": flops / (t_fused * 1e-3) / 1e12 / peaks["bf16_tflops"],
            "ms_unfused_gemm_plus_vocab": t_unfused, "ms_cublas_gemm_alone": t_gemm,
            "argmax_agreement_fused_vs_unfused": agree,
            "note": "unfused = torch.matmul (cuBLAS, bf16 logits written) + dlm_vocab_confidence; "
                    "the fused kernel keeps fp32 logits, so argmax agreement below 1 is near-ties and bf16 rounding"}


def build_step(Bn, w, bufs, args, stream, mask_mode):
    """One refine step on the device buffers in `bufs` (q, k, v, logits, tok,
    msk, prompt, seqlen); adds its outputs and scratch to `bufs`. step(ev)
    records ev[0..3] around attention, the vocabulary reduction and the update."""
    import torch
    d = bufs["q"].device
    q, k, v, logits, tok, msk = (bufs[n] for n in ("q", "k", "v", "logits", "tok", "msk"))
    prompt, seqlen = bufs["prompt"], bufs["seqlen"]
    out = torch.empty_like(q)
    am = torch.empty(w.N, dtype=torch.int32, device=d)
    cf = torch.empty(w.N, dtype=torch.float32, device=d)
    ls = torch.empty(w.N, dtype=torch.float32, device=d)
    nt, nm = torch.empty_like(tok), torch.empty_like(msk)
    ne = torch.empty(w.B, dtype=torch.int32, device=d)
    params = Bn.RefineParams(w.edit_threshold[0], w.remask_k, w.remask_frac, w.mask_id, prompt, seqlen)
    workspace = torch.zeros(Bn.dlm_refine_step_workspace_bytes(w.B) // 4, dtype=torch.int32, device=d)
    tprob = torch.empty(w.N, dtype=torch.float32, device=d) if args.rank == "result" else None
    bufs.update(out=out, am=am, cf=cf, ls=ls, nt=nt, nm=nm, ne=ne, params=params)

    def rec(ev, i):
        if ev:
            ev[i].record(stream)

    def step(ev=None):
        rec(ev, 0)
        if mask_mode:
            Bn.dlm_attn_masked(q, k, v, seqlen, prompt, mask_mode, args.block, out)
        else:
            Bn.dlm_bidir_attn(q, k, v, seqlen, out)
        rec(ev, 1)
        if args.path == "fused":
            Bn.dlm_refine_step(logits, tok, msk, params, am.view(w.B, w.L), cf.view(w.B, w.L), ls.view(w.B, w.L),
                               nt, nm, ne, workspace)
            rec(ev, 2)
            rec(ev, 3)
            return
        Bn.dlm_vocab_confidence(logits, am, cf, ls)
        rec(ev, 2)
        if tprob is not None:
            Bn.dlm_token_prob(logits, tok.view(-1), ls, tprob)
            Bn.dlm_refine_update_ranked(tok, msk, am.view(w.B, w.L), cf.view(w.B, w.L), tprob.view(w.B, w.L),
                                        params, nt, nm, ne)
        else:
            Bn.dlm_refine_update(tok, msk, am.view(w.B, w.L), cf.view(w.B, w.L), params, nt, nm, ne)
        rec(ev, 3)

    return step


def measure_e2e(args, Bn, w, bufs, stream, mask_mode, world, d, copy_streams=4):
    """The same step end to end with HOST inputs: every step copies its inputs
    from pinned host memory and reads its outputs back, inside the timed
    region. Two device input sets alternate, so the copies of step s + 1
    (split over several copy streams, one DMA engine each) overlap the compute
    of step s; the compute of a step waits for its own copies."""
    import torch
    names = ("q", "k", "v", "logits", "tok", "msk", "prompt", "seqlen")
    host = {}
    for n in names:
        t = torch.empty(bufs[n].shape, dtype=bufs[n].dtype, pin_memory=True)
        t.copy_(bufs[n])
        host[n] = t
    sets = [bufs, {n: torch.empty_like(bufs[n]) for n in names}]
    steps = [None, None]
    steps[0] = build_step(Bn, w, sets[0], args, stream, mask_mode)   # new outputs for the e2e leg
    steps[1] = build_step(Bn, w, sets[1], args, stream, mask_mode)
    outs = ("nt", "nm", "ne")
    h_out = [{n: torch.empty(sets[i][n].shape, dtype=sets[i][n].dtype, pin_memory=True) for n in outs}
             for i in range(2)]
    h2d = sum(host[n].numel() * host[n].element_size() for n in names)
    d2h = sum(h_out[0][n].numel() * h_out[0][n].element_size() for n in outs)
    cstreams = [torch.cuda.Stream(d) for _ in range(copy_streams)]
    free = [torch.cuda.Event(), torch.cuda.Event()]
    free_recorded = [False, False]

    def copy_in(i):
        """Issue the host -> device copies of set i; returns the events the compute must wait for."""
        evs = []
        for c, cs in enumerate(cstreams):
            if free_recorded[i]:
                cs.wait_event(free[i])   # the set's previous step has consumed it
            with torch.cuda.stream(cs):
                for n in names:
                    src, dst = host[n], sets[i][n]
                    rows = src.shape[0]
                    if src.numel() * src.element_size() < (64 << 20):
                        if c == 0:
                            dst.copy_(src, non_blocking=True)
                        continue
                    lo, hi = rows * c // len(cstreams), rows * (c + 1) // len(cstreams)
                    dst[lo:hi].copy_(src[lo:hi], non_blocking=True)
            e = torch.cuda.Event()
            e.record(cs)
            evs.append(e)
        return evs

    def run(nsteps):
        pending = copy_in(0)
        for s in range(nsteps):
            i = s & 1
            for e in pending:
                stream.wait_event(e)
            if s + 1 < nsteps:
                nxt = copy_in(1 - i)          # overlaps this step's compute
            steps[i]()
            free[i].record(stream)
            free_recorded[i] = True
            for n in outs:
                h_out[i][n].copy_(sets[i][n], non_blocking=True)
            if s + 1 < nsteps:
                pending = nxt

    # Warm-up: after the host link has idled, host -> device copies start slow
    # and reach their full rate only after ~0.3 s of traffic (measured on this
    # GPU: 18, 57, then 212 GB/s over the first three 4 GB copies after 2 s of
    # idling), so the leg runs 20 untimed steps (~0.5 s of copies) first.
    run(20)
    torch.cuda.synchronize()
    k_e2e = max(4, min(args.steps, 20))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    e0.record(stream)
    run(k_e2e)
    e1.record(stream)
    torch.cuda.synchronize()
    te = max_over_ranks(e0.elapsed_time(e1) / k_e2e, world, d)
    if Bn.device_error(clear=True):
        raise RuntimeError("device error word set during the end-to-end measurement")
    return {"value": job_steps_per_s(te, world), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": te, "steps": k_e2e,
            "copies": f"{copy_streams} copy streams, two device input sets (copies of step s+1 overlap step s)"}


L2_BYTES = 129 * 1024 * 1024


def pci_bus_id(d):
    """NVML's PCI bus id of torch device d, or None if torch does not expose it."""
    try:
        import torch
        pr = torch.cuda.get_device_properties(d)
        return f"{pr.pci_domain_id:08x}:{pr.pci_bus_id:02x}:{pr.pci_device_id:02x}.0"
    except Exception:
        return None


def timed_launches(fn_of_set, nsets: int, reps: int, stream, warm: int = 3):
    """Mean device time (ms) per launch of fn_of_set(i % nsets), i < reps.

    The launches are captured once into a CUDA graph and the graph is replayed
    between two CUDA events: a short kernel timed eagerly would include the
    host's time to issue it (the binding takes ~10 us per call), while the
    graph hands the launches to the GPU back to back."""
    import torch
    for i in range(warm):
        fn_of_set(i % nsets)
    torch.cuda.synchronize()
    side = torch.cuda.Stream(stream.device)
    side.wait_stream(stream)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side, capture_error_mode="thread_local"):
        for i in range(reps):
            fn_of_set(i % nsets)
    torch.cuda.synchronize()
    with torch.cuda.stream(side):   # the graph runs on the current stream
        g.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(side)
        g.replay()
        e1.record(side)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps


def measure_workload_kernels(Bn, name: str, d, peaks, reps: int = 20):
    """The three kernels of one refine step of workload `name`, each timed on its
    own (CUDA events around each of `reps` launches). Inputs come from the seeded
    generator, resident in HBM; when one set of inputs fits in L2, enough copies
    rotate (at least three times the L2 together) that every launch reads HBM."""
    import torch
    from paper_2608_02625_gb300 import synth_gpu, workloads
    w = workloads.get(name)
    stream = torch.cuda.current_stream(d)
    qkv_bytes = 2 * w.B * w.L * (w.Hq + 2 * w.Hkv) * w.D
    per_set = w.logit_bytes() + qkv_bytes
    nsets = max(1, min(4, -(-3 * L2_BYTES // per_set)))
    tok_np, msk_np = w.initial_state()
    tok = torch.from_numpy(tok_np).to(d)
    msk = torch.from_numpy(msk_np).to(d)
    q, k, v = synth_gpu.qkv(w, 0, d)
    logits = synth_gpu.logits(w, 0, d, tok.view(-1), msk.view(-1))
    sets = [(q, k, v, logits)] + [tuple(t.clone() for t in (q, k, v, logits)) for _ in range(nsets - 1)]
    prompt = torch.from_numpy(w.prompt_lens()).to(d)
    seqlen = torch.from_numpy(w.seq_lens()).to(d)
    out = torch.empty_like(q)
    am = torch.empty(w.N, dtype=torch.int32, device=d)
    cf = torch.empty(w.N, dtype=torch.float32, device=d)
    ls = torch.empty(w.N, dtype=torch.float32, device=d)
    nt, nm = torch.empty_like(tok), torch.empty_like(msk)
    ne = torch.empty(w.B, dtype=torch.int32, device=d)
    params = Bn.RefineParams(w.edit_threshold[0], w.remask_k, w.remask_frac, w.mask_id, prompt, seqlen)
    clk = ClockSampler(d.index or 0, pci_bus_id(d)).__enter__()
    t0 = time.time()
    t_attn = timed_launches(lambda i: Bn.dlm_bidir_attn(sets[i][0], sets[i][1], sets[i][2], seqlen, out),
                            nsets, reps, stream)
    t_vocab = timed_launches(lambda i: Bn.dlm_vocab_confidence(sets[i][3], am, cf, ls), nsets, reps, stream)
    t_upd = timed_launches(lambda i: Bn.dlm_refine_update(tok, msk, am.view(w.B, w.L), cf.view(w.B, w.L), params,
                                                          nt, nm, ne), 1, reps, stream)
    t1 = time.time()
    clk.__exit__(None, None, None)
    if Bn.device_error(clear=True):
        raise RuntimeError(f"device error word set while timing {name}")
    flops = w.attn_flops()
    vb = w.vocab_bytes()
    step = t_attn + t_vocab + t_upd
    res = {"batch": w.B, "seq_len": w.L, "q_heads": w.Hq, "kv_heads": w.Hkv, "vocab": w.V,
           "attn": {"ms": t_attn, "tflops": flops / (t_attn * 1e-3) / 1e12,
                    "frac_of_measured_bf16": flops / (t_attn * 1e-3) / 1e12 / peaks["bf16_tflops"]},
           "vocab": {"ms": t_vocab, "gbs": vb / (t_vocab * 1e-3) / 1e9,
                     "frac_of_measured_hbm": vb / (t_vocab * 1e-3) / 1e9 / peaks["hbm_gbs"]},
           "update": {"ms": t_upd},
           "step_ms": step, "steps_per_s": 1000.0 / step,
           "refined_tokens_per_s": 1000.0 / step * w.refined_tokens(),
           "note": (f"kernels timed one by one, {reps} launches each replayed from a CUDA graph after 3 warm-ups; "
                    f"{nsets} rotating input "
                    f"set(s) ({'L2 flushed by rotation' if nsets > 1 else 'inputs larger than L2'}); step = "
                    f"attention + vocabulary reduction + update" + (" (step 0 of 4)" if w.steps > 1 else "")),
           "clocks": clk.summary(t0, t1)}
    del sets, logits, q, k, v
    torch.cuda.empty_cache()
    return res


def measure_e2e_lmhead(args, Bn, w, world, d, reps: int = 20):
    """One refine step end to end through the public API starting from the
    refiner's last hidden states instead of materialised logits: every step
    copies q, k, v, the hidden states [N, d] and the token state from pinned
    host memory, runs attention, the fused vocabulary projection + reduction
    (output weights resident, as a model's parameters are) and the update, and
    reads the new tokens, mask and edit counts back."""
    import torch
    from paper_2608_02625_gb300 import synth, synth_gpu
    stream = torch.cuda.current_stream(d)
    dm = args.lmhead_d
    q, k, v = synth_gpu.qkv(w, 0, d)
    hidden = torch.empty((w.N, dm), dtype=torch.bfloat16, device=d)
    weight = torch.empty((w.V, dm), dtype=torch.bfloat16, device=d)
    synth_gpu.fill_normal_(hidden, synth.stream_key(w.seed + 101, synth.S_Q), 1.0)
    synth_gpu.fill_normal_(weight, synth.stream_key(w.seed + 101, synth.S_K), 1.0 / dm ** 0.5)
    tok_np, msk_np = w.initial_state()
    dev_in = {"q": q, "k": k, "v": v, "hidden": hidden, "tok": torch.from_numpy(tok_np).to(d),
              "msk": torch.from_numpy(msk_np).to(d), "prompt": torch.from_numpy(w.prompt_lens()).to(d),
              "seqlen": torch.from_numpy(w.seq_lens()).to(d)}
    names = list(dev_in)
    host = {}
    for n in names:
        host[n] = torch.empty(dev_in[n].shape, dtype=dev_in[n].dtype, pin_memory=True)
        host[n].copy_(dev_in[n])
    sets = [dev_in, {n: torch.empty_like(dev_in[n]) for n in names}]
    out = torch.empty_like(q)
    am = torch.empty(w.N, dtype=torch.int32, device=d)
    cf = torch.empty(w.N, dtype=torch.float32, device=d)
    ls = torch.empty(w.N, dtype=torch.float32, device=d)
    lws = torch.empty(Bn.dlm_lmhead_workspace_bytes(w.N), dtype=torch.uint8, device=d)
    outs = [{"nt": torch.empty_like(dev_in["tok"]), "nm": torch.empty_like(dev_in["msk"]),
             "ne": torch.empty(w.B, dtype=torch.int32, device=d)} for _ in range(2)]
    h_out = [{n: torch.empty(o[n].shape, dtype=o[n].dtype, pin_memory=True) for n in o} for o in outs]
    h2d = sum(host[n].numel() * host[n].element_size() for n in names)
    d2h = sum(t.numel() * t.element_size() for t in h_out[0].values())
    cstream = torch.cuda.Stream(d)
    free = [torch.cuda.Event(), torch.cuda.Event()]
    used = [False, False]

    def copy_in(i):
        if used[i]:
            cstream.wait_event(free[i])
        with torch.cuda.stream(cstream):
            for n in names:
                sets[i][n].copy_(host[n], non_blocking=True)
        e = torch.cuda.Event()
        e.record(cstream)
        return e

    def step(i):
        st = sets[i]
        params = Bn.RefineParams(w.edit_threshold[0], w.remask_k, w.remask_frac, w.mask_id, st["prompt"],
                                 st["seqlen"])
        Bn.dlm_bidir_attn(st["q"], st["k"], st["v"], st["seqlen"], out)
        Bn.dlm_lmhead_confidence(st["hidden"], weight, am, cf, ls, lws)
        Bn.dlm_refine_update(st["tok"], st["msk"], am.view(w.B, w.L), cf.view(w.B, w.L), params, outs[i]["nt"],
                             outs[i]["nm"], outs[i]["ne"])

    def run(nsteps):
        pending = copy_in(0)
        for s_ in range(nsteps):
            i = s_ & 1
            stream.wait_event(pending)
            if s_ + 1 < nsteps:
                nxt = copy_in(1 - i)
            step(i)
            free[i].record(stream)
            used[i] = True
            for n in outs[i]:
                h_out[i][n].copy_(outs[i][n], non_blocking=True)
            if s_ + 1 < nsteps:
                pending = nxt

    run(10)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    e0.record(stream)
    run(reps)
    e1.record(stream)
    torch.cuda.synchronize()
    te = max_over_ranks(e0.elapsed_time(e1) / reps, world, d)
    if Bn.device_error(clear=True):
        raise RuntimeError("device error word set during the hidden-state end-to-end measurement")
    del sets, dev_in, host, weight, hidden
    torch.cuda.empty_cache()
    return {"value": job_steps_per_s(te, world), "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": te, "steps": reps, "d_model": dm,
            "path": "host q/k/v + hidden states -> dlm_bidir_attn -> dlm_lmhead_confidence -> dlm_refine_update "
                    "-> host tokens/mask/edit counts (output weights resident); copies of step s+1 overlap step s"}


def run_ours(args, rank, world):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2608_02625_gb300 import binding as Bn
    from paper_2608_02625_gb300 import synth_gpu, workloads

    base = workloads.get(args.config)
    if args.batch:
        base = workloads.scaled(base, B=args.batch, name=f"{base.name}_b{args.batch}")
    # Weak scaling: each rank refines its own seeded batch of the same shape.
    w = replica_workload(base, rank)
    d = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(d)
    peaks = load_peaks()

    timer = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline and not args.batch:
        timer = OracleTimer(base.name, host_workers())   # spawned before any GPU work

    # Inputs resident in HBM.
    q, k, v = synth_gpu.qkv(w, 0, d)
    tok_np, msk_np = w.initial_state()
    tok = torch.from_numpy(tok_np).to(d)
    msk = torch.from_numpy(msk_np).to(d)
    logits = synth_gpu.logits(w, 0, d, tok.view(-1), msk.view(-1))
    prompt = torch.from_numpy(w.prompt_lens()).to(d)
    seqlen = torch.from_numpy(w.seq_lens()).to(d)
    stream = torch.cuda.current_stream(d)
    fused = args.path == "fused"
    ranked = args.rank == "result"
    mask_mode = {"full": 0, "block_causal": 1, "block_local": 2}[args.attn_mask]
    bufs = dict(q=q, k=k, v=v, logits=logits, tok=tok, msk=msk, prompt=prompt, seqlen=seqlen)
    step = build_step(Bn, w, bufs, args, stream, mask_mode)
    out, params = bufs["out"], bufs["params"]

    if timer is not None:
        # The workers' input generation would compete with the host-link copies
        # of the end-to-end leg: let it finish before anything is timed.
        timer.wait_ready()
    clk = ClockSampler(d.index if d.index is not None else 0, pci_bus_id(d)).__enter__()
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if Bn.device_error(clear=True):
        raise RuntimeError("device error word set during warm-up")

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    host_t0 = time.time()
    t_start.record(stream)
    for i in range(args.steps):
        step(evs[i])
    t_end.record(stream)
    torch.cuda.synchronize()
    host_t1 = time.time()
    clk.__exit__(None, None, None)
    if world > 1:
        dist.barrier()
    total_ms = t_start.elapsed_time(t_end)
    per_kernel = {
        "attn": statistics.mean(e[0].elapsed_time(e[1]) for e in evs),
        "vocab": statistics.mean(e[1].elapsed_time(e[2]) for e in evs),
        "update": statistics.mean(e[2].elapsed_time(e[3]) for e in evs),
    }
    if Bn.device_error(clear=True):
        raise RuntimeError("device error word set during the timed region")
    total_ms = max_over_ranks(total_ms, world, d)
    ms_per_step = total_ms / args.steps

    # ---- end to end through the public API with host buffers
    e2e = None if args.no_e2e else measure_e2e(args, Bn, w, bufs, stream, mask_mode, world, d,
                                                  copy_streams=args.copy_streams)

    if rank != 0:
        return None

    # ---- multi-pass refinement: the recorded pass repeated by one graph launch
    # (device-side early stop) against the same passes driven from the host
    # The other workloads first: the projection GEMM below draws enough power
    # to leave the clocks under the power cap for a while after it.
    by_workload = {}
    for name in [x for x in args.workloads.split(",") if x and x != "none" and not args.batch]:
        by_workload[name] = measure_workload_kernels(Bn, name, d, peaks)
    lmhead_info = measure_lmhead(args, w, Bn, peaks) if args.lmhead_d > 0 else None
    e2e_lm = None if (args.no_e2e or args.lmhead_d <= 0) else measure_e2e_lmhead(args, Bn, w, world, d)
    loop_info = None
    if args.loop_steps > 0:
        loop_info = measure_loop(args, w, Bn, q, k, v, out, logits, tok, msk, params, seqlen, stream)
    fused_info = None if fused else measure_fused_step(Bn, w, logits, tok, msk, params, stream, per_kernel)

    attn_flops = w.attn_flops(mask_mode, args.block)
    vocab_bytes = w.vocab_bytes()
    kern = {
        "attn": {"achieved_tflops": attn_flops / (per_kernel["attn"] * 1e-3) / 1e12, "ms": per_kernel["attn"],
                 "flops": attn_flops},
        "vocab": {"achieved_gbs": vocab_bytes / (per_kernel["vocab"] * 1e-3) / 1e9, "ms": per_kernel["vocab"],
                  "bytes": vocab_bytes},
        "update": {"ms": per_kernel["update"]},
    }
    kern["attn"]["frac_of_measured_bf16"] = kern["attn"]["achieved_tflops"] / peaks["bf16_tflops"]
    if peaks.get("bf16_tflops_sustained"):
        # The kernel runs inside a long loop of steps: the sustained figure is the other bound.
        kern["attn"]["frac_of_measured_bf16_sustained"] = kern["attn"]["achieved_tflops"] / peaks["bf16_tflops_sustained"]
    kern["vocab"]["frac_of_measured_hbm"] = kern["vocab"]["achieved_gbs"] / peaks["hbm_gbs"]
    if ranked:
        kern["update"]["kernels"] = "token_prob_kernel + refine_update_kernel (ranking by the resulting token)"
    if fused:   # the vocabulary stream and the update share one launch
        kern["vocab"]["kernel"] = "vocab_step (vocabulary reduction + update)"
        kern["update"] = {"ms": 0.0, "fused_into": "vocab"}
    dominant = max(("attn", "vocab"), key=lambda kk: per_kernel[kk])
    if dominant == "vocab":
        roof = {"kernel": "vocab_step" if fused else "vocab_confidence", "bound": "hbm",
                "achieved": kern["vocab"]["achieved_gbs"],
                "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": kern["vocab"]["frac_of_measured_hbm"],
                "traffic": recorded_traffic("vocab.cu", "vocab_step_kernel" if fused else "vocab_rows_kernel",
                                            base.name),
                "algorithmic_bytes": vocab_bytes,
                "peak_source": peaks["source"]}
    else:
        roof = {"kernel": "bidir_attn", "bound": "tensor", "achieved": kern["attn"]["achieved_tflops"],
                "peak": peaks["bf16_tflops"], "unit": "TFLOP/s", "frac": kern["attn"]["frac_of_measured_bf16"],
                "traffic": recorded_traffic("attn_tc.cu", "attn_tc_kernel", base.name), "algorithmic_flops": attn_flops,
                "peak_source": peaks["source"]}

    steps_per_s = job_steps_per_s(ms_per_step, world)
    res = {
        "metric": METRIC, "value": steps_per_s, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": w.dtype, "data": "synthetic (seeded counter-based generator, resident in HBM)",
        "config": {"workload": base.name, "batch": w.B, "seq_len": w.L, "q_heads": w.Hq, "kv_heads": w.Hkv,
                   "head_dim": w.D, "vocab": w.V, "refined_tokens_per_step": w.refined_tokens(),
                   "l2": "no flush: logits and q/k/v are larger than L2 (129 MB)",
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU"},
        "refined_tokens_per_sec": steps_per_s * w.refined_tokens(),
        "kernels": kern,
        "roofline": roof,
        "gpu_launches": (2 if fused else 4 if ranked else 3) * args.steps,
        "path": args.path,
        "rank": args.rank,
        "attn_mask": args.attn_mask if not mask_mode else f"{args.attn_mask} (block {args.block})",
        "e2e": e2e,
        "loop": loop_info,
        "fused_step": fused_info,
        "lmhead": lmhead_info,
        "e2e_lmhead": e2e_lm,
        "kernels_by_workload": by_workload,
        "paper_context": PAPER_CONTEXT,
    }
    if timer is not None:
        res["cpu_baseline"] = timer.run()
        timer.close()
    res["clocks"] = clk.summary(host_t0, host_t1)
    res["peaks"] = peaks
    return res


def run_reference(args, rank, world):
    """The oracle as the reference arm: each step is one refine step of the
    whole batch of the workload on the host cores (see OracleTimer); the
    step time is the wall time that passed."""
    if rank != 0:
        return None
    from paper_2608_02625_gb300 import workloads
    w = workloads.get(args.config)
    timer = OracleTimer(args.config, host_workers())
    timer.wait_ready()
    for _ in range(args.warmup):
        timer.run()
    t0 = time.perf_counter()
    vals = [timer.run() for _ in range(args.steps)]
    wall = time.perf_counter() - t0
    timer.close()
    ms_per_step = wall * 1e3 / args.steps
    value = 1000.0 / ms_per_step
    cb = dict(vals[-1])
    cb["value"] = value
    cb["ms_per_step"] = ms_per_step
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": w.name, "batch": w.B, "seq_len": w.L, "q_heads": w.Hq, "kv_heads": w.Hkv,
                       "head_dim": w.D, "vocab": w.V},
            "refined_tokens_per_sec": value * w.refined_tokens(),
            "timed_region_s": wall,
            "cpu_baseline": cb, "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                                        "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--batch", type=int, default=None, help="override the workload's batch (profiling runs)")
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--copy-streams", type=int, default=4, help="host -> device copy streams of the end-to-end leg")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--loop-steps", type=int, default=4,
                    help="also time a recorded multi-pass loop with device-side early stop (0: skip)")
    ap.add_argument("--path", default="separate", choices=["fused", "separate"],
                    help="separate: dlm_vocab_confidence then dlm_refine_update (the faster of the two on "
                         "the 32 x 512 workload); fused: both in one launch (dlm_refine_step)")
    ap.add_argument("--workloads", default="c2_single_512,c4_long_2048,c5_heavy_4step",
                    help="other workloads whose three kernels are also timed one by one (comma list; none to skip)")
    ap.add_argument("--lmhead-d", type=int, default=2048,
                    help="also time the vocabulary projection fused with the reduction at this width (0: skip)")
    ap.add_argument("--attn-mask", default="full", choices=["full", "block_causal", "block_local"],
                    help="attention mask of the step (full: the refiner's bidirectional pass)")
    ap.add_argument("--block", type=int, default=64, help="block size of the block masks")
    ap.add_argument("--rank", default="conf", choices=["conf", "result"],
                    help="remask ranking: conf (maximum probability) or result (probability of the token each "
                         "position ends with: dlm_token_prob + dlm_refine_update_ranked)")
    args = ap.parse_args()
    if args.rank == "result" and args.path == "fused":
        ap.error("--rank result runs the separate path")
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if world > 1 and args.impl == "ours":
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", 0)))
        dist.init_process_group("nccl")
    res = run_reference(args, rank, world) if args.impl == "reference" else run_ours(args, rank, world)
    if rank == 0 and res is not None:
        print(json.dumps(res), flush=True)
    if world > 1 and args.impl == "ours":
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
