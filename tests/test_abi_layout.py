"""The binding's ctypes structures against the C header: a C program compiled
against include/dlmrefine.h prints the sizes and field offsets of dlm_tensor
and dlm_refine_params, and the ctypes layouts must equal them (no GPU)."""
import ctypes
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SRC = r"""
#include <stddef.h>
#include <stdio.h>
#include "dlmrefine.h"
int main(void) {
  printf("%zu %zu %zu %zu %zu %zu\n", sizeof(dlm_tensor), offsetof(dlm_tensor, data),
         offsetof(dlm_tensor, dtype), offsetof(dlm_tensor, ndim), offsetof(dlm_tensor, shape),
         offsetof(dlm_tensor, stride));
  printf("%zu %zu %zu %zu %zu %zu %zu\n", sizeof(dlm_refine_params),
         offsetof(dlm_refine_params, edit_threshold), offsetof(dlm_refine_params, remask_k),
         offsetof(dlm_refine_params, remask_frac), offsetof(dlm_refine_params, mask_id),
         offsetof(dlm_refine_params, prompt_lens), offsetof(dlm_refine_params, seq_lens));
  printf("%d %d %d %d\n", (int)DLM_BF16, (int)DLM_F32, (int)DLM_I32, (int)DLM_U8);
  return 0;
}
"""


def test_ctypes_layout_matches_the_header(tmp_path):
    cc = shutil.which("gcc") or shutil.which("cc")
    if not cc:
        pytest.skip("no C compiler")
    src = tmp_path / "layout.c"
    src.write_text(SRC)
    exe = tmp_path / "layout"
    r = subprocess.run([cc, "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    t = [int(x) for x in out[0].split()]
    p = [int(x) for x in out[1].split()]
    e = [int(x) for x in out[2].split()]
    from paper_2608_02625_gb300 import binding as B
    T, P = B.DlmTensor, B.DlmRefineParams
    assert t == [ctypes.sizeof(T), T.data.offset, T.dtype.offset, T.ndim.offset, T.shape.offset, T.stride.offset]
    assert p == [ctypes.sizeof(P), P.edit_threshold.offset, P.remask_k.offset, P.remask_frac.offset,
                 P.mask_id.offset, P.prompt_lens.offset, P.seq_lens.offset]
    assert e == [B.DLM_BF16, B.DLM_F32, B.DLM_I32, B.DLM_U8]
