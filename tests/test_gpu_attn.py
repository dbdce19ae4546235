"""Step A1 (non-causal GQA attention) on the GPU against the oracle.

bf16: max abs error <= 2e-2 on every case, plus three bounds on the output's
own scale that a small systematic error would break (gpu_util:
max |err| <= 2^-7 max|ref|, mean |err| <= 2^-8 mean|ref|, signed bias
<= 2^-10 mean|ref|); fp32: 1e-5.
Output rows i >= n_b must be exactly zero. Every comparison reports its
error statistics (max abs, max abs / max|ref|, mean abs, signed bias) in the
test session's summary."""
import math

import numpy as np
import pytest
import torch

import oracle
from gpu_util import (ATTN_BIAS_REL_BF16, ATTN_MAX_REL_BF16, ATTN_MEAN_REL_BF16, ATTN_TOL_BF16, ATTN_TOL_F32, dev,
                      host_qkv_seq, report)
from paper_2608_02625_gb300 import synth, workloads

pytestmark = pytest.mark.gpu


def gpu_attn(q, k, v, seq_lens, out=None):
    from paper_2608_02625_gb300 import binding as Bn
    if out is None:
        out = torch.full(q.shape, float("nan"), dtype=q.dtype, device=q.device)
    sl = torch.tensor(np.asarray(seq_lens, dtype=np.int32), device=q.device) if seq_lens is not None else None
    Bn.dlm_bidir_attn(q, k, v, sl, out)
    torch.cuda.synchronize()
    assert Bn.device_error(clear=True) == 0
    return out


def compare(out_gpu: torch.Tensor, ref: np.ndarray, seq_lens, tol_abs, where=""):
    """Element-wise comparison with the oracle; returns the error statistics
    (also reported). bf16 results (tol_abs == ATTN_TOL_BF16) must also meet
    the output-scaled bounds."""
    g = out_gpu.float().cpu().numpy()
    B, L = g.shape[0], g.shape[1]
    valid = np.zeros(g.shape, dtype=bool)
    for b in range(B):
        n = min(max(int(seq_lens[b]), 0), L) if seq_lens is not None else L
        assert np.all(g[b, n:] == 0.0), f"{where}: padded rows of sequence {b} are not zero"
        valid[b, :n] = True
    assert np.all(np.isfinite(g)), f"{where}: non-finite output"
    err = np.abs(g - ref)
    worst = np.unravel_index(np.argmax(err), err.shape)
    assert np.all(err <= tol_abs), (f"{where}: max abs err {err.max():.3g} at {worst} "
                                    f"(gpu {g[worst]:.5g} ref {ref[worst]:.5g})")
    st = {"where": where, "dtype": "bf16" if tol_abs == ATTN_TOL_BF16 else "f32",
          "max_abs": 0.0, "max_rel": 0.0, "mean_abs": 0.0, "mean_rel": 0.0, "bias_rel": 0.0, "max_ref": 0.0}
    if valid.any():
        e, r, d = err[valid], np.abs(ref[valid]), (g - ref)[valid]
        st.update(max_abs=float(e.max()), mean_abs=float(e.mean()), max_ref=float(r.max()))
        if r.max() > 0:
            st["max_rel"] = float(e.max() / r.max())
            st["mean_rel"] = float(e.mean() / r.mean())
            st["bias_rel"] = float(np.mean(d * np.sign(ref[valid])) / r.mean())
    report("attention_errors", **st)
    if st["dtype"] == "bf16" and st["max_ref"] > 0:
        assert st["max_rel"] <= ATTN_MAX_REL_BF16, f"{where}: max |err| / max|ref| = {st['max_rel']:.3g}"
        assert st["mean_rel"] <= ATTN_MEAN_REL_BF16, f"{where}: mean |err| / mean|ref| = {st['mean_rel']:.3g}"
        assert abs(st["bias_rel"]) <= ATTN_BIAS_REL_BF16, f"{where}: signed bias / mean|ref| = {st['bias_rel']:.3g}"
    return st


def rand_qkv(B, L, Hq, Hkv, D, sigma, dtype, seed):
    g = torch.Generator().manual_seed(seed)
    dt = torch.bfloat16 if dtype == "bf16" else torch.float32
    q = (torch.randn(B, L, Hq, D, generator=g) * sigma).to(dt)
    k = (torch.randn(B, L, Hkv, D, generator=g) * sigma).to(dt)
    v = torch.randn(B, L, Hkv, D, generator=g).to(dt)
    return q, k, v


def run_case(B, L, Hq, Hkv, D, seq_lens, sigma, dtype="bf16", seed=0):
    q, k, v = rand_qkv(B, L, Hq, Hkv, D, sigma, dtype, seed)
    ref = oracle.bidir_attn(q.float().numpy(), k.float().numpy(), v.float().numpy(),
                            seq_lens if seq_lens is not None else [L] * B)
    out = gpu_attn(q.to(dev()), k.to(dev()), v.to(dev()), seq_lens)
    where = f"B{B} L{L} {Hq}/{Hkv} D{D} sl {list(seq_lens)} sigma {sigma:.3g}"
    return compare(out, ref, seq_lens, ATTN_TOL_F32 if dtype == "f32" else ATTN_TOL_BF16, where=where)


@pytest.mark.parametrize("sigma", [1 / math.sqrt(128), 1.0, 2.0])
@pytest.mark.parametrize("B,L,Hq,Hkv,D,sl", [
    (2, 300, 8, 2, 128, [300, 130]),          # several tiles + ragged tail, varlen
    (1, 128, 4, 4, 128, [128]),               # MHA: tiles paired across row blocks
    (2, 384, 6, 2, 128, [384, 257]),          # odd group size: pairs cross heads and rows
    (1, 50, 2, 1, 128, [50]),                 # L below one tile
    (3, 256, 4, 2, 64, [256, 1, 129]),        # head_dim 64
    (6, 260, 2, 1, 128, [0, 1, 127, 128, 129, 260]),  # edge lengths
])
@pytest.mark.parametrize("tiles", [0, 1, 2])
def test_bf16_cases(B, L, Hq, Hkv, D, sl, sigma, tiles):
    from paper_2608_02625_gb300 import binding as Bn
    Bn.dlm_set_attn_tiles_per_unit(tiles)
    try:
        run_case(B, L, Hq, Hkv, D, sl, sigma, "bf16", seed=B * L + Hq)
    finally:
        Bn.dlm_set_attn_tiles_per_unit(0)


@pytest.mark.parametrize("B,L,Hq,Hkv,D,sl", [(1, 128, 4, 2, 64, [128]), (2, 200, 4, 1, 128, [200, 77])])
def test_f32_cases(B, L, Hq, Hkv, D, sl):
    run_case(B, L, Hq, Hkv, D, sl, 1.0, "f32", seed=3)


def test_padding_garbage_never_read():
    """Key/value rows >= n_b full of NaN/Inf must not reach any output."""
    B, L, Hq, Hkv, D = 2, 256, 4, 2, 128
    q, k, v = rand_qkv(B, L, Hq, Hkv, D, 1.0, "bf16", 21)
    sl = [200, 131]
    ref = oracle.bidir_attn(q.float().numpy(), k.float().numpy(), v.float().numpy(), sl)
    for b, n in enumerate(sl):
        k[b, n:] = float("inf")
        v[b, n:] = float("nan")
        q[b, n:] = float("nan")
    out = gpu_attn(q.to(dev()), k.to(dev()), v.to(dev()), sl)
    compare(out, ref, sl, ATTN_TOL_BF16, "garbage padding")


@pytest.mark.parametrize("L,n", [(300, 300), (256, 250), (128, 128), (200, 129)])
def test_running_max_rises_every_tile(L, n):
    """Scores that grow along the keys (k_j = 2 j e_0, q = e_0) raise the
    running maximum by far more than the rescale threshold in every key
    sub-tile, the last one included, so the output-rescale path runs each time."""
    B, Hq, Hkv, D = 1, 4, 2, 128
    q = torch.zeros(B, L, Hq, D)
    q[..., 0] = 1.0
    k = torch.zeros(B, L, Hkv, D)
    k[0, :, :, 0] = (2.0 * torch.arange(L, dtype=torch.float32))[:, None]
    g = torch.Generator().manual_seed(9)
    v = torch.randn(B, L, Hkv, D, generator=g)
    q, k, v = q.to(torch.bfloat16), k.to(torch.bfloat16), v.to(torch.bfloat16)
    ref = oracle.bidir_attn(q.float().numpy(), k.float().numpy(), v.float().numpy(), [n])
    out = gpu_attn(q.to(dev()), k.to(dev()), v.to(dev()), [n])
    compare(out, ref, [n], ATTN_TOL_BF16, f"rising max L{L} n{n}")


def test_strided_views_of_packed_qkv():
    B, L, Hq, Hkv, D = 2, 256, 8, 2, 128
    packed = (torch.randn(B, L, Hq + 2 * Hkv, D) * 0.5).to(torch.bfloat16)
    q, k, v = packed[:, :, :Hq], packed[:, :, Hq:Hq + Hkv], packed[:, :, Hq + Hkv:]
    sl = [256, 100]
    ref = oracle.bidir_attn(q.float().numpy(), k.float().numpy(), v.float().numpy(), sl)
    pd = packed.to(dev())
    out = gpu_attn(pd[:, :, :Hq], pd[:, :, Hq:Hq + Hkv], pd[:, :, Hq + Hkv:], sl)
    compare(out, ref, sl, ATTN_TOL_BF16, "packed qkv")


def test_no_seq_lens_means_full_length():
    B, L, Hq, Hkv, D = 1, 200, 2, 1, 128
    q, k, v = rand_qkv(B, L, Hq, Hkv, D, 1.0, "bf16", 5)
    ref = oracle.bidir_attn(q.float().numpy(), k.float().numpy(), v.float().numpy(), [L])
    out = gpu_attn(q.to(dev()), k.to(dev()), v.to(dev()), None)
    compare(out, ref, None, ATTN_TOL_BF16, "no seq_lens")


C3_PAIRS = [(0, 0), (5, 13), (17, 31), (31, 7), (1, 8), (2, 17), (3, 30), (8, 1), (11, 22), (14, 9), (20, 4),
            (23, 27), (26, 15), (28, 2), (29, 19), (30, 24)]


@pytest.mark.parametrize("sigma", [1.0, 2.0])
@pytest.mark.parametrize("name,pairs", [("c2_single_512", "all"), ("c3_batch32_512", C3_PAIRS)])
def test_workload_shape_peaked(name, pairs, sigma):
    """The bench's shapes and lengths with peaked attention: q, k ~ N(0, sigma^2)
    (scores of standard deviation sigma^2), v ~ N(0, 1); the whole batch in
    one launch, the oracle on the listed (sequence, query head) pairs."""
    w = workloads.get(name)
    n = w.seq_lens()
    q, k, v = rand_qkv(w.B, w.L, w.Hq, w.Hkv, w.D, sigma, "bf16", seed=int(sigma * 100) + w.B)
    out = gpu_attn(q.to(dev()), k.to(dev()), v.to(dev()), n)
    if pairs == "all":
        pairs = [(b, h) for b in range(w.B) for h in range(w.Hq)]
    qf, kf, vf = q.float().numpy(), k.float().numpy(), v.float().numpy()
    g_out = out.float()
    for b, h in pairs:
        g = (h * w.Hkv) // w.Hq
        ref = oracle.bidir_attn(qf[b:b + 1, :, h:h + 1], kf[b:b + 1, :, g:g + 1], vf[b:b + 1, :, g:g + 1], [n[b]])
        compare(g_out[b:b + 1, :, h:h + 1], ref, [n[b]], ATTN_TOL_BF16,
                where=f"{name} peaked sigma {sigma:g} b={b} h={h}")


@pytest.mark.parametrize("name,pairs", [
    ("c1_tiny_f32", "all"),
    ("c2_single_512", "all"),
    ("c3_batch32_512", C3_PAIRS),
    ("c4_long_2048", [(0, 0), (3, 17), (7, 31)]),
    ("c5_heavy_4step", [(0, 0), (64, 9), (127, 15)]),
])
def test_workload_full_size(name, pairs):
    """The bench's launch (all sequences, all heads); the oracle recomputes the
    listed (sequence, query head) pairs from host-generated inputs."""
    from paper_2608_02625_gb300 import synth_gpu
    w = workloads.get(name)
    q, k, v = synth_gpu.qkv(w, 0, dev())
    n = w.seq_lens()
    out = gpu_attn(q, k, v, n)
    if pairs == "all":
        pairs = [(b, h) for b in range(w.B) for h in range(w.Hq)]
    tol = ATTN_TOL_F32 if w.dtype == "f32" else ATTN_TOL_BF16
    by_b = {}
    for b, h in pairs:
        by_b.setdefault(b, []).append(h)
    g_out = out.float()
    for b, heads in by_b.items():
        hq = host_qkv_seq(w, 0, synth.S_Q, b, w.Hq)
        hk = host_qkv_seq(w, 0, synth.S_K, b, w.Hkv)
        hv = host_qkv_seq(w, 0, synth.S_V, b, w.Hkv)
        for h in heads:
            g = (h * w.Hkv) // w.Hq
            ref = oracle.bidir_attn(hq[None, :, h:h + 1], hk[None, :, g:g + 1], hv[None, :, g:g + 1], [n[b]])
            compare(g_out[b:b + 1, :, h:h + 1], ref, [n[b]], tol, where=f"{name} b={b} h={h}")


@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("B,L,Hq,Hkv,D,sl,pl", [
    (2, 384, 6, 2, 128, [384, 257], [64, 100]),   # odd group size: pairs cross heads and rows
    (1, 512, 32, 4, 128, [512], [160]),           # one sequence of the paper's length
    (3, 256, 4, 2, 64, [256, 1, 129], [0, 0, 64]),  # head_dim 64, edge lengths
])
def test_tiles_per_unit_bit_identical(B, L, Hq, Hkv, D, sl, pl, mode):
    """One or two query tiles per work unit changes only which CTA slot runs a
    tile: every tile's arithmetic is the same, so the outputs are bit-identical."""
    from paper_2608_02625_gb300 import binding as Bn
    q, k, v = (t.to(dev()) for t in rand_qkv(B, L, Hq, Hkv, D, 1.0, "bf16", 17 + mode))
    n = torch.tensor(sl, dtype=torch.int32, device=dev())
    p = torch.tensor(pl, dtype=torch.int32, device=dev())
    outs = []
    for tiles in (1, 2):
        out = torch.full(q.shape, float("nan"), dtype=q.dtype, device=dev())
        Bn.dlm_set_attn_tiles_per_unit(tiles)
        try:
            if mode == 0:
                Bn.dlm_bidir_attn(q, k, v, n, out)
            else:
                Bn.dlm_attn_masked(q, k, v, n, p, mode, 64, out)
        finally:
            Bn.dlm_set_attn_tiles_per_unit(0)
        torch.cuda.synchronize()
        assert Bn.device_error(clear=True) == 0
        outs.append(out)
    assert torch.equal(outs[0], outs[1])


def test_workload_tiles_bit_identical():
    """The whole 32 x 512 launch with one and with two query tiles per unit:
    every (sequence, head) pair bit-identical whichever slot ran it."""
    from paper_2608_02625_gb300 import binding as Bn, synth_gpu
    w = workloads.get("c3_batch32_512")
    q, k, v = synth_gpu.qkv(w, 0, dev())
    n = w.seq_lens()
    outs = []
    for tiles in (1, 2):
        Bn.dlm_set_attn_tiles_per_unit(tiles)
        try:
            outs.append(gpu_attn(q, k, v, n))
        finally:
            Bn.dlm_set_attn_tiles_per_unit(0)
    assert torch.equal(outs[0], outs[1])

