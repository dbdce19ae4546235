"""The vocabulary projection fused with the per-position reduction
(dlm_lmhead_confidence) on the GPU against the oracle's lm_head_confidence.

Inputs are host-generated (seeded numpy), rounded to bf16 on the host, and the
oracle evaluates the projection of those exact values in fp64. The GPU
accumulates the logits in fp32, so:
* argmax: identical wherever the oracle's two largest logits of the row are
  more than LOGIT_MARGIN apart; elsewhere the GPU's choice must be within
  LOGIT_MARGIN of the maximum (both are correct answers to within rounding);
* lse within LSE_ATOL + 2e-5 |lse|, conf within CONF_RTOL_LMH relative:
  fp32 accumulation over d = 2048 products of magnitude ~1/sqrt(d) leaves
  absolute logit errors of order 1e-5, and conf = exp(m - lse) inherits the
  error of m - lse."""
import math

import numpy as np
import pytest
import torch

import oracle
from gpu_util import dev

pytestmark = pytest.mark.gpu

LOGIT_MARGIN = 1e-3
LSE_ATOL = 1e-4
LSE_RTOL = 2e-5
CONF_RTOL_LMH = 2e-4


def make_inputs(N, V, d, seed, peak_frac=0.1, peak=8.0):
    """hidden ~ N(0, 1), weight ~ N(0, 1/d), with a planted logit bump of
    `peak` on a random token for a fraction of the rows; bf16-rounded."""
    rng = np.random.default_rng(seed)
    h = rng.standard_normal((N, d), dtype=np.float32)
    w = (rng.standard_normal((V, d), dtype=np.float32) / np.float32(math.sqrt(d)))
    rows = np.nonzero(rng.random(N) < peak_frac)[0]
    toks = rng.integers(0, V, rows.size)
    for r, t in zip(rows, toks):
        h[r] += peak * w[t] / np.float32(np.dot(w[t], w[t]))
    hb = torch.from_numpy(h).to(torch.bfloat16)
    wb = torch.from_numpy(w).to(torch.bfloat16)
    return hb, wb


def gpu_lmhead(hb, wb):
    from paper_2608_02625_gb300 import binding as Bn
    d = dev()
    N = hb.shape[0] if hb.dim() == 2 else hb.shape[0] * hb.shape[1]
    am = torch.full((N,), -1, dtype=torch.int32, device=d)
    cf = torch.full((N,), -1.0, dtype=torch.float32, device=d)
    ls = torch.full((N,), -1.0, dtype=torch.float32, device=d)
    ws = torch.empty(Bn.dlm_lmhead_workspace_bytes(N), dtype=torch.uint8, device=d)
    Bn.dlm_lmhead_confidence(hb, wb, am, cf, ls, ws)
    torch.cuda.synchronize()
    assert Bn.device_error(clear=True) == 0
    return am.cpu().numpy(), cf.cpu().numpy(), ls.cpu().numpy()


def check(gpu, h_rows, w, where):
    """gpu: (argmax, conf, lse) of the given rows; h_rows, w: the bf16 values as float."""
    am, cf, ls = (np.asarray(a) for a in gpu)
    logits = oracle.lm_head_logits(h_rows, w)
    am_ref, cf_ref, ls_ref = oracle.vocab_confidence(logits)
    top2 = np.sort(logits, axis=1)[:, -2:] if logits.shape[1] > 1 else np.concatenate([logits, logits - 1e9], 1)
    gap = top2[:, 1] - top2[:, 0]
    clear = gap > LOGIT_MARGIN
    bad = clear & (am != am_ref)
    assert not bad.any(), f"{where}: argmax differs at clear rows {np.nonzero(bad)[0][:8]}"
    mx = logits.max(axis=1)
    chosen = logits[np.arange(len(am)), np.clip(am, 0, logits.shape[1] - 1)]
    assert np.all((am >= 0) & (am < logits.shape[1]) & (chosen >= mx - LOGIT_MARGIN)), f"{where}: argmax not a max"
    el = np.abs(ls.astype(np.float64) - ls_ref)
    assert np.all(el <= LSE_ATOL + LSE_RTOL * np.abs(ls_ref)), f"{where}: lse err {el.max():.3g}"
    ec = np.abs(cf.astype(np.float64) - cf_ref) / cf_ref
    assert np.all(ec <= CONF_RTOL_LMH), f"{where}: conf rel err {ec.max():.3g}"
    return int((~clear).sum())


@pytest.mark.parametrize("N,V,d", [(300, 1000, 64), (128, 256, 128), (300, 1000, 512), (1, 7, 64), (129, 257, 192),
                                   (1000, 20000, 2048)])
def test_vs_oracle_all_rows(N, V, d):
    """Ragged row blocks and vocabulary tiles, several widths, a single row,
    a vocabulary smaller than one tile."""
    hb, wb = make_inputs(N, V, d, seed=N + V + d)
    gpu = gpu_lmhead(hb.to(dev()), wb.to(dev()))
    check(gpu, hb.float().numpy(), wb.float().numpy(), f"N={N} V={V} d={d}")


def test_strided_and_3d_hidden():
    hb, wb = make_inputs(2 * 150, 3000, 256, seed=4)
    full = torch.zeros(300, 256 + 64, dtype=torch.bfloat16)
    full[:, :256] = hb
    hv = full.to(dev())[:, :256]                   # row stride 320 elements
    assert hv.stride(0) == 320
    gpu = gpu_lmhead(hv, wb.to(dev()))
    check(gpu, hb.float().numpy(), wb.float().numpy(), "strided hidden")
    gpu3 = gpu_lmhead(hb.to(dev()).reshape(2, 150, 256), wb.to(dev()))
    check(gpu3, hb.float().numpy(), wb.float().numpy(), "3-D hidden")


def test_ties_take_the_lowest_index():
    """Duplicate weight rows give exactly equal logits: the lowest vocabulary
    index must win, within a tile, across tiles and across splits."""
    N, V, d = 256, 4096, 128
    hb, wb = make_inputs(N, V, d, seed=8, peak_frac=0.5, peak=10.0)
    w = wb.clone()
    am0 = oracle.lm_head_confidence(hb.float().numpy(), w.float().numpy())[0]
    dup = (am0.astype(np.int64) * 7 + 1111) % V          # a copy of each row's argmax weight elsewhere
    w[torch.from_numpy(dup)] = w[torch.from_numpy(am0.astype(np.int64))]
    gpu = gpu_lmhead(hb.to(dev()), w.to(dev()))
    ref_am = oracle.lm_head_confidence(hb.float().numpy(), w.float().numpy())[0]
    np.testing.assert_array_equal(gpu[0], ref_am)


def test_full_size_sampled_rows():
    """The 32 x 512 batch's 16384 rows against a 151552-token vocabulary at
    d = 2048 in one launch; the oracle recomputes 24 sampled rows."""
    N, V, d = 16384, 151552, 2048
    hb, wb = make_inputs(N, V, d, seed=99)
    gpu = gpu_lmhead(hb.to(dev()), wb.to(dev()))
    rng = np.random.default_rng(3)
    rows = np.unique(np.concatenate([[0, 127, 128, N - 1], rng.integers(0, N, 20)]))
    check(tuple(a[rows] for a in gpu), hb[rows].float().numpy(), wb.float().numpy(), "full size")
