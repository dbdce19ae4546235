"""Thin Python binding of libdlmrefine (argument marshalling only).

Each function has the name and argument order of its C entry point
(include/dlmrefine.h), takes torch CUDA tensors, builds the dlm_tensor
descriptors, sets the library's stream to torch's current stream of the
tensors' device and calls the library. All computation runs in the CUDA
kernels; a nonzero status raises DlmError. The shared library must have been
built (``python -m paper_2608_02625_gb300.build``): there is no fallback.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
library_path = os.path.join(_PKG, "libdlmrefine.so")

DLM_BF16, DLM_F32, DLM_I32, DLM_U8 = 1, 2, 3, 4
_DTYPES = {torch.bfloat16: DLM_BF16, torch.float32: DLM_F32, torch.int32: DLM_I32, torch.uint8: DLM_U8}


class DlmTensor(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("dtype", ctypes.c_int32), ("ndim", ctypes.c_int32),
                ("shape", ctypes.c_int64 * 4), ("stride", ctypes.c_int64 * 4)]


class DlmRefineParams(ctypes.Structure):
    _fields_ = [("edit_threshold", ctypes.c_float), ("remask_k", ctypes.c_int32),
                ("remask_frac", ctypes.c_float), ("mask_id", ctypes.c_int32),
                ("prompt_lens", ctypes.c_void_p), ("seq_lens", ctypes.c_void_p)]


class DlmError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"libdlmrefine status {status}: {message}")
        self.status = status


def _load():
    if not os.path.exists(library_path):
        raise ImportError(f"{library_path} is missing: build it with "
                          "`python -m paper_2608_02625_gb300.build` (no CPU fallback exists)")
    lib = ctypes.CDLL(library_path)
    P = ctypes.POINTER(DlmTensor)
    lib.dlm_bidir_attn.argtypes = [P, P, P, P, P]
    lib.dlm_attn_masked.argtypes = [P, P, P, P, P, ctypes.c_int32, ctypes.c_int32, P]
    lib.dlm_vocab_confidence.argtypes = [P, P, P, P]
    lib.dlm_refine_update.argtypes = [P, P, P, P, ctypes.POINTER(DlmRefineParams), P, P, P]
    lib.dlm_refine_step.argtypes = [P, P, P, ctypes.POINTER(DlmRefineParams), P, P, P, P, P, P,
                                    ctypes.c_void_p, ctypes.c_size_t]
    lib.dlm_token_prob.argtypes = [P, P, P, P]
    lib.dlm_lmhead_confidence.argtypes = [P, P, P, P, P, ctypes.c_void_p, ctypes.c_size_t]
    lib.dlm_lmhead_workspace_bytes.argtypes = [ctypes.c_int64]
    lib.dlm_lmhead_workspace_bytes.restype = ctypes.c_size_t
    lib.dlm_refine_update_ranked.argtypes = [P, P, P, P, P, ctypes.POINTER(DlmRefineParams), P, P, P]
    lib.dlm_refine_step_static.argtypes = [P, P, P, ctypes.POINTER(DlmRefineParams), P, P, P, P, P, P]
    lib.dlm_refine_step_workspace_bytes.argtypes = [ctypes.c_int64]
    lib.dlm_refine_step_workspace_bytes.restype = ctypes.c_size_t
    for f in ("dlm_bidir_attn", "dlm_attn_masked", "dlm_vocab_confidence", "dlm_refine_update", "dlm_refine_step",
              "dlm_refine_step_static", "dlm_token_prob", "dlm_refine_update_ranked", "dlm_lmhead_confidence",
              "dlm_set_stream", "dlm_set_attn_tiles_per_unit",
              "dlm_version", "dlm_get_device_error"):
        getattr(lib, f).restype = ctypes.c_int
    lib.dlm_loop_begin.argtypes = [ctypes.c_void_p]
    lib.dlm_loop_end.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.POINTER(ctypes.c_void_p)]
    lib.dlm_loop_cancel.argtypes = []
    lib.dlm_loop_launch.argtypes = [ctypes.c_void_p]
    lib.dlm_loop_destroy.argtypes = [ctypes.c_void_p]
    for f in ("dlm_loop_begin", "dlm_loop_end", "dlm_loop_cancel", "dlm_loop_launch", "dlm_loop_destroy"):
        getattr(lib, f).restype = ctypes.c_int
    lib.dlm_selftest_wait_timeout.argtypes = [ctypes.c_int64]
    lib.dlm_selftest_wait_timeout.restype = ctypes.c_int
    lib.dlm_set_stream.argtypes = [ctypes.c_void_p]
    lib.dlm_set_attn_tiles_per_unit.argtypes = [ctypes.c_int]
    lib.dlm_get_stream.restype = ctypes.c_void_p
    lib.dlm_status_string.restype = ctypes.c_char_p
    lib.dlm_status_string.argtypes = [ctypes.c_int]
    lib.dlm_last_error.restype = ctypes.c_char_p
    lib.dlm_get_device_error.argtypes = [ctypes.POINTER(ctypes.c_int32), ctypes.c_int]
    return lib


lib = _load()


def describe(t: torch.Tensor | None) -> DlmTensor | None:
    """dlm_tensor descriptor of a tensor (no copy)."""
    if t is None:
        return None
    if t.dtype not in _DTYPES:
        raise TypeError(f"unsupported dtype {t.dtype}")
    if t.dim() < 1 or t.dim() > 4:
        raise ValueError("tensors of rank 1..4 only")
    d = DlmTensor()
    n = t.dim()
    d.data = t.data_ptr() if t.numel() else None
    d.dtype = _DTYPES[t.dtype]
    d.ndim = n
    d.shape[:n] = t.shape
    d.stride[:n] = t.stride()
    return d


def _ref(d):
    return ctypes.byref(d) if d is not None else None


def _check(status: int):
    if status != 0:
        msg = lib.dlm_last_error().decode() or lib.dlm_status_string(status).decode()
        raise DlmError(status, msg)


def _prepare(*tensors):
    dev = -1
    for t in tensors:
        if t is None:
            continue
        idx = t.get_device()
        if idx < 0:
            raise ValueError("libdlmrefine takes CUDA tensors")
        if dev < 0:
            dev = idx
        elif idx != dev:
            raise ValueError("all tensors must be on one device")
    if dev < 0:
        raise ValueError("no tensor given")
    if torch.cuda.current_device() != dev:
        torch.cuda.set_device(dev)
    _check(lib.dlm_set_stream(ctypes.c_void_p(torch.cuda.current_stream(dev).cuda_stream)))


def dlm_version() -> int:
    return lib.dlm_version()


def dlm_status_string(status: int) -> str:
    return lib.dlm_status_string(status).decode()


def dlm_bidir_attn(q, k, v, seq_lens, out):
    """Non-causal GQA attention: out[b,i,h] = softmax(q k^T / sqrt(D)) v over keys j < n_b."""
    _prepare(q, k, v, seq_lens, out)
    dq, dk, dv, ds, do = (describe(t) for t in (q, k, v, seq_lens, out))
    _check(lib.dlm_bidir_attn(_ref(dq), _ref(dk), _ref(dv), _ref(ds), _ref(do)))
    return out


ATTN_FULL, ATTN_BLOCK_CAUSAL, ATTN_BLOCK_LOCAL = 0, 1, 2


def dlm_attn_masked(q, k, v, seq_lens, prompt_lens, mode: int, block: int, out):
    """Attention restricted by a block mask (ATTN_BLOCK_CAUSAL: prompt, earlier
    blocks and the own block; ATTN_BLOCK_LOCAL: prompt and the own block)."""
    _prepare(q, k, v, seq_lens, prompt_lens, out)
    ds = [describe(t) for t in (q, k, v, seq_lens, prompt_lens)]
    do = describe(out)
    _check(lib.dlm_attn_masked(*[_ref(d) for d in ds], int(mode), int(block), _ref(do)))
    return out


def dlm_vocab_confidence(logits, argmax, conf, lse):
    """Per row: argmax (lowest index), max softmax probability, log-sum-exp."""
    _prepare(logits, argmax, conf, lse)
    ds = [describe(t) for t in (logits, argmax, conf, lse)]
    _check(lib.dlm_vocab_confidence(*[_ref(d) for d in ds]))
    return argmax, conf, lse


@dataclasses.dataclass
class RefineParams:
    edit_threshold: float
    remask_k: int
    remask_frac: float
    mask_id: int
    prompt_lens: torch.Tensor  # int32 [B] on the device
    seq_lens: torch.Tensor     # int32 [B] on the device

    def to_c(self) -> DlmRefineParams:
        for t in (self.prompt_lens, self.seq_lens):
            if t.dtype != torch.int32 or not t.is_cuda or not t.is_contiguous():
                raise ValueError("prompt_lens / seq_lens must be contiguous int32 CUDA tensors")
        return DlmRefineParams(float(self.edit_threshold), int(self.remask_k), float(self.remask_frac),
                               int(self.mask_id), self.prompt_lens.data_ptr(), self.seq_lens.data_ptr())


def dlm_refine_update(tokens, mask, argmax, conf, params: RefineParams, new_tokens, new_mask, n_edits):
    """Commit masked positions, edit confident changes, remask the k least confident."""
    _prepare(tokens, mask, argmax, conf, new_tokens, new_mask, n_edits, params.prompt_lens, params.seq_lens)
    ds = [describe(t) for t in (tokens, mask, argmax, conf)]
    outs = [describe(t) for t in (new_tokens, new_mask, n_edits)]
    cp = params.to_c()
    _check(lib.dlm_refine_update(*[_ref(d) for d in ds], ctypes.byref(cp), *[_ref(d) for d in outs]))
    return new_tokens, new_mask, n_edits


def dlm_lmhead_workspace_bytes(rows: int) -> int:
    return lib.dlm_lmhead_workspace_bytes(int(rows))


def dlm_lmhead_confidence(hidden, weight, argmax, conf, lse, workspace):
    """argmax / conf / lse of hidden @ weight^T per row, without materialising the logits."""
    _prepare(hidden, weight, argmax, conf, lse, workspace)
    if not workspace.is_contiguous():
        raise ValueError("workspace must be contiguous")
    ds = [describe(t) for t in (hidden, weight, argmax, conf, lse)]
    nbytes = workspace.numel() * workspace.element_size()
    _check(lib.dlm_lmhead_confidence(*[_ref(d) for d in ds], ctypes.c_void_p(workspace.data_ptr() if nbytes else None),
                                     ctypes.c_size_t(nbytes)))
    return argmax, conf, lse


def dlm_token_prob(logits, tokens, lse, prob):
    """prob[r] = exp(logits[r, tokens[r]] - lse[r]) (0 for a token outside [0, V))."""
    _prepare(logits, tokens, lse, prob)
    ds = [describe(t) for t in (logits, tokens, lse, prob)]
    _check(lib.dlm_token_prob(*[_ref(d) for d in ds]))
    return prob


def dlm_refine_update_ranked(tokens, mask, argmax, conf, tok_prob, params: RefineParams, new_tokens, new_mask,
                             n_edits):
    """dlm_refine_update remasking by the probability of each position's resulting token."""
    _prepare(tokens, mask, argmax, conf, tok_prob, new_tokens, new_mask, n_edits, params.prompt_lens,
             params.seq_lens)
    ds = [describe(t) for t in (tokens, mask, argmax, conf, tok_prob)]
    outs = [describe(t) for t in (new_tokens, new_mask, n_edits)]
    cp = params.to_c()
    _check(lib.dlm_refine_update_ranked(*[_ref(d) for d in ds], ctypes.byref(cp), *[_ref(d) for d in outs]))
    return new_tokens, new_mask, n_edits


def dlm_refine_step_workspace_bytes(batch: int) -> int:
    return lib.dlm_refine_step_workspace_bytes(int(batch))


def dlm_refine_step(logits, tokens, mask, params: RefineParams, argmax, conf, lse, new_tokens, new_mask, n_edits,
                    workspace):
    """Vocabulary reduction and refine update in one launch.

    workspace: a CUDA tensor of at least dlm_refine_step_workspace_bytes(B) bytes,
    zero before its first use; each completed call leaves it zero again."""
    _prepare(logits, tokens, mask, argmax, conf, lse, new_tokens, new_mask, n_edits, workspace,
             params.prompt_lens, params.seq_lens)
    if not workspace.is_contiguous():
        raise ValueError("workspace must be contiguous")
    ins = [describe(t) for t in (logits, tokens, mask)]
    outs = [describe(t) for t in (argmax, conf, lse, new_tokens, new_mask, n_edits)]
    cp = params.to_c()
    nbytes = workspace.numel() * workspace.element_size()
    _check(lib.dlm_refine_step(*[_ref(d) for d in ins], ctypes.byref(cp), *[_ref(d) for d in outs],
                               ctypes.c_void_p(workspace.data_ptr() if nbytes else None), ctypes.c_size_t(nbytes)))
    return argmax, conf, lse, new_tokens, new_mask, n_edits


def dlm_refine_step_static(logits, tokens, mask, params: RefineParams, argmax, conf, lse, new_tokens, new_mask,
                           n_edits):
    """dlm_refine_step with the library's static scratch instead of a workspace,
    for callers that cannot allocate device memory. The first call on a device
    sets that device up (make it before any stream capture); calls that overlap
    on the GPU race on the shared scratch."""
    _prepare(logits, tokens, mask, argmax, conf, lse, new_tokens, new_mask, n_edits, params.prompt_lens,
             params.seq_lens)
    ins = [describe(t) for t in (logits, tokens, mask)]
    outs = [describe(t) for t in (argmax, conf, lse, new_tokens, new_mask, n_edits)]
    cp = params.to_c()
    _check(lib.dlm_refine_step_static(*[_ref(d) for d in ins], ctypes.byref(cp), *[_ref(d) for d in outs]))
    return argmax, conf, lse, new_tokens, new_mask, n_edits


class RefineLoop:
    """A recorded refine pass that the GPU repeats until no confident edit
    remains or max_steps passes have run (one graph launch)."""

    def __init__(self, handle: int, device: torch.device, steps_out: torch.Tensor):
        self._h = handle
        self.device = device
        self.steps_out = steps_out

    def launch(self):
        """Runs the loop on the current stream of its device; steps_out then
        holds the number of passes once the stream reaches that point."""
        if not self._h:
            raise ValueError("the loop has been destroyed")
        torch.cuda.set_device(self.device)
        _check(lib.dlm_set_stream(ctypes.c_void_p(torch.cuda.current_stream(self.device).cuda_stream)))
        _check(lib.dlm_loop_launch(ctypes.c_void_p(self._h)))

    def close(self):
        if self._h:
            _check(lib.dlm_loop_destroy(ctypes.c_void_p(self._h)))
            self._h = None


def dlm_loop_begin(steps_out: torch.Tensor):
    """Starts recording one refine pass on the current (non-default) stream."""
    if steps_out.dtype != torch.int32 or steps_out.numel() != 1:
        raise ValueError("steps_out must be a one-element int32 CUDA tensor")
    _prepare(steps_out)
    _check(lib.dlm_loop_begin(ctypes.c_void_p(steps_out.data_ptr())))


def dlm_loop_end(n_edits: torch.Tensor, max_steps: int, steps_out: torch.Tensor) -> RefineLoop:
    """Ends the recording: the pass repeats while passes < max_steps and some
    n_edits[b] > 0."""
    if n_edits.dtype != torch.int32 or not n_edits.is_contiguous() or n_edits.dim() != 1:
        lib.dlm_loop_cancel()
        raise ValueError("n_edits must be a contiguous int32 [B] CUDA tensor")
    h = ctypes.c_void_p()
    _check(lib.dlm_loop_end(ctypes.c_void_p(n_edits.data_ptr() if n_edits.numel() else None), n_edits.numel(),
                            int(max_steps), ctypes.byref(h)))
    return RefineLoop(h.value, n_edits.device, steps_out)


def dlm_loop_cancel():
    """Ends an unfinished recording on this thread, keeping nothing."""
    _check(lib.dlm_loop_cancel())


def dlm_set_attn_tiles_per_unit(tiles: int):
    """Query tiles per attention work unit on this thread: 0 automatic, 1 or 2."""
    _check(lib.dlm_set_attn_tiles_per_unit(int(tiles)))


def dlm_selftest_wait_timeout(budget_ns: int, device: int | None = None):
    """Runs a kernel whose bounded wait on a barrier nothing arrives on gives
    up after budget_ns; afterwards device_error() holds DLM_DEVERR_TIMEOUT."""
    dev = torch.cuda.current_device() if device is None else device
    torch.cuda.set_device(dev)
    _check(lib.dlm_set_stream(ctypes.c_void_p(torch.cuda.current_stream(dev).cuda_stream)))
    _check(lib.dlm_selftest_wait_timeout(int(budget_ns)))


def device_error(clear: bool = True) -> int:
    """The device error word (DLM_DEVERR_* bits) of the current device; synchronises."""
    bits = ctypes.c_int32(0)
    _check(lib.dlm_get_device_error(ctypes.byref(bits), 1 if clear else 0))
    return bits.value
