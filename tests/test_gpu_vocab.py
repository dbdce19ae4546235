"""Step A2 (vocabulary reduction) on the GPU against the oracle.

argmax is bit-exact (exact compare, lowest index wins); conf and lse are within
the relative tolerances of gpu_util."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import check_vocab, dev, host_logit_rows
from paper_2608_02625_gb300 import synth, workloads

pytestmark = pytest.mark.gpu


def gpu_vocab(x: torch.Tensor):
    from paper_2608_02625_gb300 import binding as Bn
    N = x.shape[0] if x.dim() == 2 else x.shape[0] * x.shape[1]
    am = torch.full((N,), -1, dtype=torch.int32, device=x.device)
    cf = torch.full((N,), -1.0, dtype=torch.float32, device=x.device)
    ls = torch.full((N,), -1.0, dtype=torch.float32, device=x.device)
    Bn.dlm_vocab_confidence(x, am, cf, ls)
    torch.cuda.synchronize()
    return am.cpu().numpy(), cf.cpu().numpy(), ls.cpu().numpy()


def to_dev(x_f32: np.ndarray, dtype: str) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(x_f32, dtype=np.float32))
    return (t.to(torch.bfloat16) if dtype == "bf16" else t).to(dev())


@pytest.mark.parametrize("name", ["c1_tiny_f32", "c2_single_512"])
def test_workload_all_rows(name):
    w = workloads.get(name)
    from paper_2608_02625_gb300 import synth_gpu
    x = synth_gpu.logits(w, 0, dev())
    am, cf, ls = gpu_vocab(x)
    rows = np.arange(w.N)
    ref = oracle.vocab_confidence(host_logit_rows(w, 0, rows))
    check_vocab(am, cf, ls, *ref, where=name)


@pytest.mark.parametrize("name", ["c3_batch32_512", "c4_long_2048", "c5_heavy_4step"])
def test_workload_sampled_rows(name):
    """Full-size launch; the oracle recomputes ~180 rows one by one (random,
    and at the edges of waves of CTAs and of sequences)."""
    w = workloads.get(name)
    from paper_2608_02625_gb300 import synth_gpu
    tok, msk = w.initial_state()
    t_tok = torch.from_numpy(tok.reshape(-1)).to(dev())
    t_msk = torch.from_numpy(msk.reshape(-1)).to(dev())
    x = synth_gpu.logits(w, 0, dev(), t_tok, t_msk)
    am, cf, ls = gpu_vocab(x)
    rng = np.random.default_rng(5)
    # 160 random rows, plus rows at the edges of waves of resident CTAs (4 per
    # SM on 152 SMs) and of sequences.
    wave = 4 * 152
    edges = [r for k in range(1, 4) for r in (k * wave - 1, k * wave) if r < w.N]
    seq_edges = [r for b in (0, 1, w.B // 2, w.B - 1) for r in (b * w.L, b * w.L + w.L - 1)]
    rows = np.unique(np.concatenate([[0, w.N - 1], edges, seq_edges, rng.integers(0, w.N, 160)]))
    ref = oracle.vocab_confidence(host_logit_rows(w, 0, rows, tok.reshape(-1)[rows], msk.reshape(-1)[rows]))
    check_vocab(am[rows], cf[rows], ls[rows], *ref, where=name)
    del x
    torch.cuda.empty_cache()


def planted(N, V, seed, sigma=3.0):
    rng = np.random.default_rng(seed)
    return (rng.standard_normal((N, V)) * sigma).astype(np.float32)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("N,V", [(1, 1), (3, 7), (2, 8), (5, 1001), (64, 4096), (1, 151552), (7, 151553),
                                 (300, 32000)])
def test_shapes(dtype, N, V):
    x = planted(N, V, N * 7 + V)
    t = to_dev(x, dtype)
    ref = oracle.vocab_confidence(t.float().cpu().numpy())
    check_vocab(*gpu_vocab(t), *ref, where=f"{dtype} {N}x{V}")


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_ties_and_neg_inf(dtype):
    N, V = 6, 151552
    x = planted(N, V, 3)
    x[0, [5, 77777, 150000]] = 40.0          # ties in different threads / cluster chunks
    x[1, :] = -np.inf
    x[1, [123456, 99]] = [2.0, 2.0]          # only two finite entries, tied
    x[2, ::3] = -np.inf
    x[3, :] = 1.5                            # all equal
    x[4, V - 1] = 50.0                       # maximum at the last index
    x[5, 0] = 50.0
    t = to_dev(x, dtype)
    am, cf, ls = gpu_vocab(t)
    ref = oracle.vocab_confidence(t.float().cpu().numpy())
    check_vocab(am, cf, ls, *ref, where="ties")
    assert am[0] == 5 and am[1] == 99 and am[3] == 0 and am[4] == V - 1 and am[5] == 0


def test_strided_rows_and_3d():
    N, V = 40, 5000
    wide = to_dev(planted(N, V + 24, 11), "bf16")
    x = wide[:, 8:8 + V]                     # rows 16-byte aligned, row stride V + 24
    ref = oracle.vocab_confidence(x.float().cpu().numpy())
    check_vocab(*gpu_vocab(x), *ref, where="strided")
    x3 = to_dev(planted(4 * 10, V, 12), "bf16").reshape(4, 10, V)
    ref3 = oracle.vocab_confidence(x3.reshape(40, V).float().cpu().numpy())
    check_vocab(*gpu_vocab(x3), *ref3, where="3d")
    odd = wide[:, 3:3 + V]                   # rows not 16-byte aligned: scalar path
    ref_odd = oracle.vocab_confidence(odd.float().cpu().numpy())
    check_vocab(*gpu_vocab(odd), *ref_odd, where="unaligned")


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("N,V,pad", [(1000, 1003, 5), (2000, 64, 0), (700, 40000, 8), (900, 12, 4)])
def test_many_rows_ragged(dtype, N, V, pad):
    """More rows than one wave of resident CTAs (the staged scan), with row
    lengths that leave a scalar tail, tiny rows (most threads idle) and padded
    row strides."""
    x = planted(N, V + pad, N + V)
    t = to_dev(x, dtype)[:, :V]
    ref = oracle.vocab_confidence(t.float().cpu().numpy())
    check_vocab(*gpu_vocab(t), *ref, where=f"{dtype} {N}x{V}+{pad}")


@pytest.mark.parametrize("dtype,N,V", [("bf16", 200, 151552), ("f32", 160, 65536), ("bf16", 100, 151552)])
def test_split_rows_several_per_cluster(dtype, N, V):
    """Few long rows (at most two per SM): each row is split over a cluster, and
    with these counts a cluster takes several rows in turn (alternating partial
    slots); ties planted across the chunk boundaries of a cluster."""
    x = planted(N, V, N + V + 1)
    chunk = V // 8
    for r in range(0, N, 7):
        x[r, [chunk - 1, 3 * chunk + 5, V - 1]] = 30.0   # equal maxima in different CTAs' chunks
    t = to_dev(x, dtype)
    am, cf, ls = gpu_vocab(t)
    ref = oracle.vocab_confidence(t.float().cpu().numpy())
    check_vocab(am, cf, ls, *ref, where=f"{dtype} {N}x{V}")
    assert all(am[r] == chunk - 1 for r in range(0, N, 7))


def test_c4_zipf_full_size_planted_ties():
    """The long-draft workload at full size (16384 rows of the Zipf(1.1) prior
    plus N(0, 1)), with equal maxima planted in sampled rows at positions that
    fall to different threads, warps and staging slots of the row kernel, and
    to different CTAs' chunks of the split-row clusters (a 256-row slice); the
    lowest index must win everywhere."""
    from paper_2608_02625_gb300 import synth_gpu
    w = workloads.get("c4_long_2048")
    x = synth_gpu.logits(w, 0, dev())
    V = w.V
    rng = np.random.default_rng(44)
    rows = np.unique(np.concatenate([[0, 1, 255, w.N - 1], rng.integers(0, w.N, 24)]))
    pos = np.array([V // 8 - 1, 3 * (V // 8) + 5, V // 2 + 2048 * 8 + 3, V - 1])   # first planted index wins
    peak = float(x[torch.from_numpy(rows).to(dev())].float().max().item()) + 16.0   # exact in bf16 (an integer)
    peak = float(torch.tensor(peak).to(torch.bfloat16).float())
    for r in rows:
        x[int(r), torch.from_numpy(pos).to(dev())] = peak
    am, cf, ls = gpu_vocab(x)
    ref = oracle.vocab_confidence(host_rows_planted(w, rows, pos, peak))
    check_vocab(am[rows], cf[rows], ls[rows], *ref, where="c4 planted ties")
    assert np.all(am[rows] == pos[0])
    sl = rows[rows < 256]
    sub = x[:256]
    ref_s = oracle.vocab_confidence(host_rows_planted(w, sl, pos, peak))
    outs = gpu_vocab(sub)
    check_vocab(outs[0][sl], outs[1][sl], outs[2][sl], *ref_s, where="c4 planted ties, 256 rows, clusters")
    assert np.all(outs[0][sl] == pos[0])
    del x
    torch.cuda.empty_cache()


def host_rows_planted(w, rows, pos, peak):
    x = host_logit_rows(w, 0, rows)
    x[:, pos] = np.float32(peak)
    return x
