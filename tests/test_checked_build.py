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


@pytest.mark.gpu
def test_static_step_clears_poisoned_scratch(tmp_path):
    """dlm_refine_step_static clears the counters it uses before it counts: with
    its static scratch filled with a nonzero pattern, a call still matches the
    workspace call (same library) bit for bit, twice in a row."""
    import numpy as np
    import torch
    from paper_2608_02625_gb300 import binding as Bn
    from paper_2608_02625_gb300 import build
    build.build(check_bounds=True, out_dir=str(tmp_path))
    checked = ctypes.CDLL(str(tmp_path / "libdlmrefine.so"))
    d = torch.device("cuda", 0)
    torch.cuda.set_device(d)
    stream = torch.cuda.current_stream(d)
    assert checked.dlm_set_stream(ctypes.c_void_p(stream.cuda_stream)) == 0
    B, L, V = 6, 96, 3000
    g = torch.Generator().manual_seed(17)
    logits = (torch.randn(B * L, V, generator=g) * 3).to(torch.bfloat16).to(d)
    tok = torch.randint(0, V, (B, L), generator=g, dtype=torch.int32).to(d)
    msk = (torch.rand(B, L, generator=g) < 0.25).to(torch.uint8).to(d)
    prompt = torch.randint(0, 40, (B,), generator=g, dtype=torch.int32).to(d)
    seqlen = torch.full((B,), L, dtype=torch.int32, device=d)
    params = Bn.RefineParams(0.8, 9, 0.0, V, prompt, seqlen).to_c()

    def outs():
        return [torch.empty((B, L), dtype=t, device=d) for t in (torch.int32, torch.float32, torch.float32,
                                                                 torch.int32, torch.uint8)] + \
               [torch.empty(B, dtype=torch.int32, device=d)]

    def descs(ts):
        return [ctypes.byref(Bn.describe(t)) for t in ts]

    ref = outs()
    ws = torch.zeros(B, dtype=torch.int32, device=d)
    st = checked.dlm_refine_step(*descs((logits, tok, msk)), ctypes.byref(params), *descs(ref),
                                 ctypes.c_void_p(ws.data_ptr()), ctypes.c_size_t(4 * B))
    assert st == 0
    for call in range(2):
        assert checked.dlm_checked_fill_static_scratch(0x55) == 0
        got = outs()
        assert checked.dlm_refine_step_static(*descs((logits, tok, msk)), ctypes.byref(params), *descs(got)) == 0
        torch.cuda.synchronize()
        for name, x, y in zip(("argmax", "conf", "lse", "tokens", "mask", "n_edits"), got, ref):
            assert torch.equal(x, y), f"call {call + 1}: {name} differs from the workspace call"
    bits = ctypes.c_int32(0)
    assert checked.dlm_get_device_error(ctypes.byref(bits), 1) == 0 and bits.value == 0


@pytest.mark.gpu
def test_real_pipelines_time_out_and_recover(tmp_path):
    """With a wait budget of 300 ns (checked build) the pipelined kernels' waits
    on their TMA loads and MMAs run out: attention and the fused projection
    return, record DLM_DEVERR_TIMEOUT and tear down (in-flight copies and MMAs
    drained, tensor memory freed). With the budget back at 2 s the same calls
    are correct and leave the error word clean."""
    import time

    import numpy as np
    import torch

    import oracle
    from paper_2608_02625_gb300 import binding as Bn
    from paper_2608_02625_gb300 import build
    build.build(check_bounds=True, out_dir=str(tmp_path))
    lib = ctypes.CDLL(str(tmp_path / "libdlmrefine.so"))
    lib.dlm_checked_set_wait_budget.argtypes = [ctypes.c_int64]
    lib.dlm_lmhead_workspace_bytes.argtypes = [ctypes.c_int64]
    lib.dlm_lmhead_workspace_bytes.restype = ctypes.c_size_t
    d = torch.device("cuda", 0)
    torch.cuda.set_device(d)
    assert lib.dlm_set_stream(ctypes.c_void_p(torch.cuda.current_stream(d).cuda_stream)) == 0

    def bits():
        b = ctypes.c_int32(0)
        assert lib.dlm_get_device_error(ctypes.byref(b), 1) == 0
        return b.value

    def descs(ts):
        return [ctypes.byref(Bn.describe(t)) for t in ts]

    g = torch.Generator().manual_seed(12)
    q = torch.randn(1, 256, 4, 128, generator=g).to(torch.bfloat16)
    k = torch.randn(1, 256, 2, 128, generator=g).to(torch.bfloat16)
    v = torch.randn(1, 256, 2, 128, generator=g).to(torch.bfloat16)
    sl = torch.tensor([250], dtype=torch.int32)
    # d = 2048: the projection's epilogue waits for 32 k-blocks of MMAs per
    # tile (microseconds), longer than the resolution of the GPU's global
    # timer, which the waits read.
    hid = torch.randn(256, 2048, generator=g).to(torch.bfloat16)
    wt = (torch.randn(4096, 2048, generator=g) / 45).to(torch.bfloat16)
    qd, kd, vd, sld, hd, wd = (t.to(d) for t in (q, k, v, sl, hid, wt))
    out = torch.empty_like(qd)
    am = torch.empty(256, dtype=torch.int32, device=d)
    cf = torch.empty(256, dtype=torch.float32, device=d)
    ls = torch.empty(256, dtype=torch.float32, device=d)
    nws = lib.dlm_lmhead_workspace_bytes(256)
    ws = torch.empty(nws, dtype=torch.uint8, device=d)

    def attn():
        return lib.dlm_bidir_attn(*descs((qd, kd, vd, sld, out)))

    def lmhead():
        return lib.dlm_lmhead_confidence(*descs((hd, wd, am, cf, ls)), ctypes.c_void_p(ws.data_ptr()),
                                         ctypes.c_size_t(nws))

    assert bits() == 0
    # Two query tiles per attention unit: the second slot's start waits for
    # the first slot's first hand-off, a wait of microseconds, longer than the
    # resolution of the global timer the waits read. With one tile per unit
    # (the automatic choice at this size) every wait can end within one tick.
    assert lib.dlm_set_attn_tiles_per_unit(2) == 0
    assert lib.dlm_checked_set_wait_budget(300) == 0
    try:
        for name, call in (("attention", attn), ("projection", lmhead)):
            t0 = time.perf_counter()
            assert call() == 0
            torch.cuda.synchronize()
            assert time.perf_counter() - t0 < 5.0, name
            assert bits() & 0x2, f"{name}: no DLM_DEVERR_TIMEOUT with a 300 ns budget"
    finally:
        assert lib.dlm_checked_set_wait_budget(2000000000) == 0
        assert lib.dlm_set_attn_tiles_per_unit(0) == 0
    assert attn() == 0 and lmhead() == 0
    torch.cuda.synchronize()
    assert bits() == 0
    ref = oracle.bidir_attn(q.float().numpy(), k.float().numpy(), v.float().numpy(), [250])
    assert np.abs(out.float().cpu().numpy() - ref).max() <= 2e-2
    lg = oracle.lm_head_logits(hid.float().numpy(), wt.float().numpy())
    r_am, _, r_ls = oracle.vocab_confidence(lg)
    top2 = np.sort(lg, axis=1)[:, -2:]
    clear = top2[:, 1] - top2[:, 0] > 1e-3
    assert np.array_equal(am.cpu().numpy()[clear], r_am[clear])
    assert np.abs(ls.cpu().numpy() - r_ls).max() <= 1e-3
