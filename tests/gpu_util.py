"""Helpers of the GPU parity tests.

Oracle inputs are always regenerated on the host from the seeded generator
(paper_2608_02625_gb300.synth), never read back from the CUDA path; the device
generator is checked bit-for-bit against the host one in test_gpu_synth.py.
"""
from __future__ import annotations

import numpy as np
import torch

from paper_2608_02625_gb300 import synth
from paper_2608_02625_gb300.workloads import Workload
from oracle import remask_count

# Tolerances (problem statement: attention max abs error 2e-2 in bf16, 1e-5 in
# fp32; conf / lse: relative 2e-5, derived from fp32 accumulation of <= V
# terms each with an exp2 of relative error ~2^-22).
ATTN_TOL_BF16 = 2e-2
ATTN_TOL_F32 = 1e-5
# Bounds scaled to the output, which a small systematic error would break
# even where 2e-2 absolute is loose (outputs of order 0.05 on paper-shaped
# inputs). The kernel's bf16 roundings: each softmax numerator is rounded to
# bf16 (round to nearest even, relative error <= 2^-8) before the PV product
# and the row sum adds the same rounded values, so the output is an exactly
# normalised average of v with perturbed weights; the output is then rounded
# to bf16 (<= 2^-8 |out|). The worst case is about 2 * 2^-8 |out|, and the
# round-to-nearest errors average out. Hence, against the fp64 oracle:
#   max |err|                  <= 2^-7  max|ref|   (measured <= 5.6e-3)
#   mean |err|                 <= 2^-8  mean|ref|  (measured <= 2.3e-3)
#   |mean (err * sign(ref))|   <= 2^-10 mean|ref|  (measured <= 5e-4; rounding
#                                                   towards zero would give ~2^-9)
ATTN_MAX_REL_BF16 = 2.0 ** -7
ATTN_MEAN_REL_BF16 = 2.0 ** -8
ATTN_BIAS_REL_BF16 = 2.0 ** -10
LSE_RTOL = 2e-5
CONF_RTOL = 2e-5

# Figures the parity tests report besides asserting them: attention error
# statistics per case and the number of update positions left out of the
# exact comparison by the decision-margin protocol. conftest prints them in
# pytest's terminal summary and writes them as JSON to $DLM_TEST_REPORT if set.
REPORT = {"attention_errors": [], "margin_limited": [], "notes": []}


def report(kind: str, **fields):
    REPORT[kind].append(fields)


def dev():
    return torch.device("cuda", 0)


def bf16_f32(bits: np.ndarray) -> np.ndarray:
    return synth.bf16_bits_to_f32(bits)


def host_qkv_seq(w: Workload, step: int, which: int, b: int, H: int) -> np.ndarray:
    """Host copy of q (which=S_Q), k or v for sequence b: fp32 [L, H, D]."""
    seed = w.step_seed(step)
    per = w.L * H * w.D
    sigma = w.qkv_sigma
    x = synth.qkv_host(seed, which, (w.B, w.L, H, w.D), sigma, w.dtype, flat_offset=b * per, count=per)
    x = bf16_f32(x) if w.dtype == "bf16" else x
    return x.reshape(w.L, H, w.D)


def host_logit_rows(w: Workload, step: int, rows, tokens=None, mask=None) -> np.ndarray:
    """Host copy of logits rows (fp32 values of the stored dtype)."""
    x = w.logit_spec(step).rows_f32(rows, tokens, mask)
    if w.dtype == "bf16":
        x = bf16_f32(synth.f32_to_bf16_bits(x))
    return x


def check_update_margin(gpu, ref, amb, where=""):
    """Decision-margin parity of the update: GPU (tokens, mask, n_edits) against
    the oracle's, computed from the oracle's own vocabulary outputs. They must be
    identical at every position outside `amb`, and n_edits identical for every
    sequence without an ambiguous position."""
    g_tok, g_msk, g_ne = gpu
    diff = (g_tok != ref[0]) | (g_msk != ref[1])
    assert not np.any(diff & ~amb), f"{where}: update differs at unambiguous positions {np.argwhere(diff & ~amb)[:8]}"
    for b in range(g_tok.shape[0]):
        if not amb[b].any():
            assert g_ne[b] == ref[2][b], f"{where}: n_edits of sequence {b}"
    report("margin_limited", where=where, positions=int(amb.sum()), checked=int(amb.size),
           differing=int(diff.sum()))
    return int(amb.sum())


def check_vocab(am_gpu, conf_gpu, lse_gpu, am_ref, conf_ref, lse_ref, where=""):
    am_gpu, conf_gpu, lse_gpu = (np.asarray(a) for a in (am_gpu, conf_gpu, lse_gpu))
    bad = np.nonzero(am_gpu != am_ref)[0]
    assert bad.size == 0, f"{where} argmax differs at rows {bad[:8]}: gpu {am_gpu[bad[:8]]} ref {am_ref[bad[:8]]}"
    rl = np.abs(lse_gpu.astype(np.float64) - lse_ref) / np.maximum(1.0, np.abs(lse_ref))
    rc = np.abs(conf_gpu.astype(np.float64) - conf_ref) / np.maximum(conf_ref, 1e-30)
    assert rl.max() <= LSE_RTOL, f"{where} lse rel err {rl.max():.3g}"
    assert rc.max() <= CONF_RTOL, f"{where} conf rel err {rc.max():.3g}"
    return float(rl.max()), float(rc.max())


def ambiguous_positions(w: Workload, step: int, conf_ref: np.ndarray, state, argmax_ref, prompt, seqlen):
    """Positions where a decision of the update could flip within the conf
    tolerance: an edit candidate with |conf - tau| within 2 CONF_RTOL conf, or,
    when the k-th and (k+1)-th smallest response confs are that close, every
    position whose conf lies between them (widened by the tolerance), since
    the remask set could then differ. Returns a bool [B, L] array."""
    return ambiguous_for(w.edit_threshold[step], w.remask_k, w.remask_frac, conf_ref, state, argmax_ref, prompt,
                         seqlen)


def ambiguous_for(edit_threshold, remask_k, remask_frac, conf_ref, state, argmax_ref, prompt, seqlen):
    """ambiguous_positions for explicit update parameters."""
    tok, msk = state
    tau = np.float32(edit_threshold)
    B, L = tok.shape
    amb = np.zeros((B, L), dtype=bool)
    for b in range(B):
        p, n = int(prompt[b]), int(seqlen[b])
        c = conf_ref[b, p:n].astype(np.float64)
        tol = CONF_RTOL * np.maximum(c, 1e-30) * 2
        edit_cand = (msk[b, p:n] == 0) & (argmax_ref[b, p:n] != tok[b, p:n])
        amb[b, p:n] |= edit_cand & (np.abs(c - float(tau)) <= tol)
        k = remask_count(remask_k, remask_frac, n - p)
        if 0 < k < n - p:
            srt = np.sort(c)
            lo, hi = srt[k - 1], srt[k]          # the last remasked and the first kept conf
            t_lo, t_hi = 2 * CONF_RTOL * max(lo, 1e-30), 2 * CONF_RTOL * max(hi, 1e-30)
            if hi - lo <= t_lo + t_hi:
                amb[b, p:n] |= (c >= lo - t_lo) & (c <= hi + t_hi)
    return amb
