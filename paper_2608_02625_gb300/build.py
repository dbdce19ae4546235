"""Builds libdlmrefine.so and libdlmsynth.so in-tree for sm_103a (GB300).

    python -m paper_2608_02625_gb300.build [--force] [--verbose]

Each .cu is compiled to an object in parallel (nvcc, one -gencode), then the
objects are linked into position-independent shared libraries with the CUDA
runtime linked statically, so loading the library needs no libcudart on the
library path. The driver API entry used for TMA descriptors is resolved at
run time through the runtime (no -lcuda).
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
    "libdlmrefine.so": ["dlm_api.cu", "attn_tc.cu", "attn_f32.cu", "vocab.cu", "update.cu", "loop.cu", "lmhead.cu"],
    "libdlmsynth.so": ["synth.cu"],
}
HEADERS = ["dlm_common.cuh", "dlm_internal.h", "update_impl.cuh"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _flags(verbose: bool):
    f = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-O2", "-I", INCLUDE,
                "--expt-relaxed-constexpr"]
    if verbose:
        f += ["-Xptxas", "-v"]
    return f


def _newest_input(srcs):
    paths = [os.path.join(CSRC, s) for s in srcs] + [os.path.join(CSRC, h) for h in HEADERS]
    paths += [os.path.join(INCLUDE, h) for h in os.listdir(INCLUDE)]
    return max(os.path.getmtime(p) for p in paths)


def _compile(src: str, verbose: bool) -> tuple[str, str]:
    obj = os.path.join(BUILD, src.replace(".cu", ".o"))
    cmd = [nvcc()] + _flags(verbose) + ["-c", os.path.join(CSRC, src), "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
    return obj, r.stdout + r.stderr


def build(force: bool = False, verbose: bool = False) -> dict:
    os.makedirs(BUILD, exist_ok=True)
    todo = {}
    for lib, srcs in LIBS.items():
        out = os.path.join(PKG, lib)
        if force or not os.path.exists(out) or os.path.getmtime(out) < _newest_input(srcs):
            todo[lib] = srcs
    logs = {}
    if not todo:
        return logs
    srcs = sorted({s for v in todo.values() for s in v})
    with cf.ThreadPoolExecutor(max_workers=min(8, len(srcs))) as ex:
        futs = {s: ex.submit(_compile, s, verbose) for s in srcs}
        objs = {s: f.result() for s, f in futs.items()}
    for s, (_, log) in objs.items():
        logs[s] = log
    for lib, lsrcs in todo.items():
        out = os.path.join(PKG, lib)
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
    args = ap.parse_args(argv)
    logs = build(force=args.force, verbose=args.verbose)
    if args.verbose:
        for s, log in sorted(logs.items()):
            print(f"==== {s}\n{log}")
    print("built:", ", ".join(sorted(LIBS)) if logs or args.force else "up to date")


if __name__ == "__main__":
    sys.exit(main())
