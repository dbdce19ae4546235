"""Builds libdlmrefine.so and libdlmsynth.so in-tree for sm_103a (GB300).

    python -m paper_2608_02625_gb300.build [--force] [--verbose] [--check-bounds --out DIR]

Each .cu is compiled to an object in parallel (nvcc, one -gencode), then the
objects are linked into position-independent shared libraries with the CUDA
runtime linked statically, so loading the library needs no libcudart on the
library path. The driver API entry used for TMA descriptors is resolved at
run time through the runtime (no -lcuda).

--check-bounds compiles with DLM_CHECK_BOUNDS, which makes the kernels check
their inputs' value contracts and report violations in the device error word
(DLM_DEVERR_INPUT); such a build goes to its own object directory and, with
--out, to another directory than the package's.
"""
from __future__ import annotations

import argparse
import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]

LIBS = {
    "libdlmrefine.so": ["dlm_api.cu", "attn_tc.cu", "attn_f32.cu", "vocab.cu", "update.cu", "loop.cu", "lmhead.cu",
                        "selftest.cu"],
    "libdlmsynth.so": ["synth.cu"],
}
HEADERS = ["dlm_common.cuh", "dlm_internal.h", "update_impl.cuh"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _flags(verbose: bool, check_bounds: bool = False):
    f = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-O2", "-I", INCLUDE,
                "--expt-relaxed-constexpr"]
    if check_bounds:
        f += ["-DDLM_CHECK_BOUNDS"]
    if verbose:
        f += ["-Xptxas", "-v"]
    return f


def _newest_input(srcs):
    paths = [os.path.join(CSRC, s) for s in srcs] + [os.path.join(CSRC, h) for h in HEADERS]
    paths += [os.path.join(INCLUDE, h) for h in os.listdir(INCLUDE)]
    return max(os.path.getmtime(p) for p in paths)


def _compile(src: str, verbose: bool, check_bounds: bool = False) -> tuple[str, str]:
    obj = os.path.join(BUILD + ("_checked" if check_bounds else ""), src.replace(".cu", ".o"))
    cmd = [nvcc()] + _flags(verbose, check_bounds) + ["-c", os.path.join(CSRC, src), "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
    return obj, r.stdout + r.stderr


def build(force: bool = False, verbose: bool = False, check_bounds: bool = False, out_dir: str | None = None) -> dict:
    out_dir = out_dir or PKG
    if check_bounds and os.path.abspath(out_dir) == PKG:
        raise ValueError("a --check-bounds build goes to its own directory (--out)")
    os.makedirs(BUILD + ("_checked" if check_bounds else ""), exist_ok=True)
    os.makedirs(out_dir, exist_ok=True)
    todo = {}
    for lib, srcs in LIBS.items():
        out = os.path.join(out_dir, lib)
        if force or not os.path.exists(out) or os.path.getmtime(out) < _newest_input(srcs):
            todo[lib] = srcs
    logs = {}
    if not todo:
        return logs
    srcs = sorted({s for v in todo.values() for s in v})
    with cf.ThreadPoolExecutor(max_workers=min(8, len(srcs))) as ex:
        futs = {s: ex.submit(_compile, s, verbose, check_bounds) for s in srcs}
        objs = {s: f.result() for s, f in futs.items()}
    for s, (_, log) in objs.items():
        logs[s] = log
    for lib, lsrcs in todo.items():
        out = os.path.join(out_dir, lib)
        tmp = out + ".tmp"
        cmd = [nvcc()] + ARCH + ["-shared", "-cudart", "static", "-o", tmp] + [objs[s][0] for s in lsrcs]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed for {lib}:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, out)
    return logs


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--force", action="store_true")
    ap.add_argument("--verbose", action="store_true", help="print ptxas register/smem usage")
    ap.add_argument("--check-bounds", action="store_true", help="compile the input-contract checks in")
    ap.add_argument("--out", default=None, help="directory of the libraries (required with --check-bounds)")
    args = ap.parse_args(argv)
    logs = build(force=args.force, verbose=args.verbose, check_bounds=args.check_bounds, out_dir=args.out)
    if args.verbose:
        for s, log in sorted(logs.items()):
            print(f"==== {s}\n{log}")
    print("built:", ", ".join(sorted(LIBS)) if logs or args.force else "up to date")


if __name__ == "__main__":
    sys.exit(main())
