"""Device side of the seeded input generator (binding of libdlmsynth.so).

Fills CUDA tensors with exactly the bits ``synth.py`` produces on the host for
the same keys and element indices. Input generation only.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

from . import synth
from .workloads import Workload

_PKG = os.path.dirname(os.path.abspath(__file__))
library_path = os.path.join(_PKG, "libdlmsynth.so")


def _load():
    if not os.path.exists(library_path):
        raise ImportError(f"{library_path} is missing: build it with `python -m paper_2608_02625_gb300.build`")
    lib = ctypes.CDLL(library_path)
    lib.dlm_synth_normal.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_uint64,
                                     ctypes.c_int64, ctypes.c_float, ctypes.c_void_p]
    lib.dlm_synth_normal.restype = ctypes.c_int
    lib.dlm_synth_logits.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_int64,
                                     ctypes.c_int64, ctypes.c_int64, ctypes.c_uint64, ctypes.c_float,
                                     ctypes.c_void_p, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64,
                                     ctypes.c_uint64, ctypes.c_float, ctypes.c_float, ctypes.c_void_p,
                                     ctypes.c_void_p, ctypes.c_void_p]
    lib.dlm_synth_logits.restype = ctypes.c_int
    return lib


lib = _load()
_DT = {torch.bfloat16: 1, torch.float32: 2}


def _stream(t):
    return ctypes.c_void_p(torch.cuda.current_stream(t.device).cuda_stream)


def fill_normal_(t: torch.Tensor, key: int, sigma: float, e0: int = 0) -> torch.Tensor:
    assert t.is_cuda and t.is_contiguous() and t.dtype in _DT
    torch.cuda.set_device(t.device)
    st = lib.dlm_synth_normal(t.data_ptr(), _DT[t.dtype], t.numel(), key, e0,
                              float(synth.normal_scale(sigma)), _stream(t))
    if st != 0:
        raise RuntimeError(f"dlm_synth_normal failed ({st})")
    return t


_ZIPF_CACHE: dict = {}


def fill_logits_(t: torch.Tensor, spec: synth.LogitSpec, first_row: int = 0, tokens: torch.Tensor | None = None,
                 mask: torch.Tensor | None = None) -> torch.Tensor:
    """t: [rows, V] (row stride >= V, innermost contiguous) bf16/fp32 CUDA tensor."""
    assert t.is_cuda and t.dim() == 2 and t.stride(1) == 1 and t.dtype in _DT
    torch.cuda.set_device(t.device)
    rows, V = t.shape
    assert V == spec.V
    zt = None
    if spec.zipf_s is not None:
        key = (t.device, spec.V, spec.zipf_s)
        if key not in _ZIPF_CACHE:
            _ZIPF_CACHE[key] = torch.from_numpy(spec.zipf_table()).to(t.device)
        zt = _ZIPF_CACHE[key]
    cur = synth.peak_threshold(spec.peak_current) if spec.peak_current > 0 else 0
    if tokens is not None:
        assert tokens.dtype == torch.int32 and tokens.is_contiguous() and tokens.numel() == rows
        assert mask is not None and mask.dtype == torch.uint8 and mask.is_contiguous()
    st = lib.dlm_synth_logits(
        t.data_ptr(), _DT[t.dtype], first_row, rows, V, t.stride(0),
        synth.stream_key(spec.seed, synth.S_LOGIT), float(synth.normal_scale(spec.sigma)),
        zt.data_ptr() if zt is not None else None, synth.stream_key(spec.seed, synth.S_SHIFT),
        synth.stream_key(spec.seed, synth.S_PEAK), synth.peak_threshold(spec.peak_frac), cur,
        float(np.float32(spec.peak_base)), float(np.float32(spec.peak_width)),
        tokens.data_ptr() if tokens is not None else None, mask.data_ptr() if mask is not None else None,
        _stream(t))
    if st != 0:
        raise RuntimeError(f"dlm_synth_logits failed ({st})")
    return t


def qkv(w: Workload, step: int, device) -> tuple:
    """q [B,L,Hq,D], k, v [B,L,Hkv,D] of refine step ``step`` on ``device``."""
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    seed = w.step_seed(step)
    q = torch.empty((w.B, w.L, w.Hq, w.D), dtype=dt, device=device)
    k = torch.empty((w.B, w.L, w.Hkv, w.D), dtype=dt, device=device)
    v = torch.empty((w.B, w.L, w.Hkv, w.D), dtype=dt, device=device)
    fill_normal_(q, synth.stream_key(seed, synth.S_Q), w.qkv_sigma)
    fill_normal_(k, synth.stream_key(seed, synth.S_K), w.qkv_sigma)
    fill_normal_(v, synth.stream_key(seed, synth.S_V), w.qkv_sigma)
    return q, k, v


def logits(w: Workload, step: int, device, tokens=None, mask=None, out=None) -> torch.Tensor:
    """Logits [B*L, V] of refine step ``step``; ``tokens``/``mask`` are the current
    state (flattened [B*L]) when the workload plants peaks on current tokens."""
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    if out is None:
        out = torch.empty((w.N, w.V), dtype=dt, device=device)
    spec = w.logit_spec(step)
    if spec.peak_current > 0:
        assert tokens is not None and mask is not None
        fill_logits_(out, spec, 0, tokens.reshape(-1), mask.reshape(-1))
    else:
        fill_logits_(out, spec)
    return out
