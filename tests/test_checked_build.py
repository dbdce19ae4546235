"""The DLM_CHECK_BOUNDS build: it compiles (here, without a GPU), and on the GPU
its kernels report inputs outside their contracts (NaN or all -inf logit rows,
token ids outside [0, V)) as DLM_DEVERR_INPUT, which the default build never
sets."""
import ctypes
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
DLM_DEVERR_INPUT = 0x8


def test_checked_vocab_compiles(tmp_path):
    from paper_2608_02625_gb300 import build
    if not shutil.which("nvcc") and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    cmd = [build.nvcc()] + build._flags(False, check_bounds=True) + [
        "-c", os.path.join(build.CSRC, "vocab.cu"), "-o", str(tmp_path / "vocab.o")]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_header_documents_the_input_bit():
    text = open(os.path.join(ROOT, "include", "dlmrefine.h")).read()
    assert "#define DLM_DEVERR_INPUT 0x8" in text


@pytest.mark.gpu
def test_checked_build_reports_contract_violations(tmp_path):
    import torch
    from paper_2608_02625_gb300 import binding as Bn
    from paper_2608_02625_gb300 import build
    build.build(check_bounds=True, out_dir=str(tmp_path))
    checked = ctypes.CDLL(str(tmp_path / "libdlmrefine.so"))
    d = torch.device("cuda", 0)
    torch.cuda.set_device(d)

    def err_bits(lib):
        bits = ctypes.c_int32(0)
        assert lib.dlm_get_device_error(ctypes.byref(bits), 1) == 0
        return bits.value

    def vocab(lib, logits):
        n = logits.shape[0]
        outs = [torch.empty(n, dtype=t, device=d) for t in (torch.int32, torch.float32, torch.float32)]
        ds = [Bn.describe(t) for t in (logits, *outs)]
        assert lib.dlm_vocab_confidence(*[ctypes.byref(x) for x in ds]) == 0
        torch.cuda.synchronize()
        return outs

    g = torch.Generator().manual_seed(3)
    for lib in (checked, Bn.lib):
        err_bits(lib)  # start clean
    clean = torch.randn(64, 5000, generator=g).to(torch.bfloat16).to(d)
    for lib in (checked, Bn.lib):
        vocab(lib, clean)
        assert err_bits(lib) == 0
    for poison in ("nan", "neg_inf_row"):
        bad = clean.clone()
        if poison == "nan":
            bad[17, 1234] = float("nan")
        else:
            bad[40, :] = float("-inf")
        vocab(checked, bad)
        assert err_bits(checked) & DLM_DEVERR_INPUT, poison
        vocab(Bn.lib, bad)
        assert not err_bits(Bn.lib) & DLM_DEVERR_INPUT, poison
    # A token id outside [0, V) in the gather of dlm_token_prob.
    am, cf, ls = vocab(checked, clean)
    tokens = torch.randint(0, 5000, (64,), generator=g, dtype=torch.int32).to(d)
    tokens[5] = 5000
    prob = torch.empty(64, dtype=torch.float32, device=d)
    ds = [Bn.describe(t) for t in (clean, tokens, ls, prob)]
    assert checked.dlm_token_prob(*[ctypes.byref(x) for x in ds]) == 0
    torch.cuda.synchronize()
    assert err_bits(checked) & DLM_DEVERR_INPUT
    assert float(prob[5]) == 0.0
