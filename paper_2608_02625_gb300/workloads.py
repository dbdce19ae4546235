"""Synthetic workloads of the refine step, shaped like the paper's 384/512-token
generation runs (Sec. 5.2: responses of up to 384 or 512 tokens; Table 10:
a 384x4 refine schedule).

Each workload fixes shapes, value distributions and update parameters. The
numbers come from the problem statement of this library; where it leaves a
value open the reading used here is stated beside the field.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

from . import synth


def attended_pairs(n: int, p: int, mask_mode: int, block: int) -> int:
    """(query, key) pairs a sequence of n positions (prompt p) attends to under
    an attention mask: 0 full, 1 block-causal, 2 block-local (dlmrefine.h)."""
    if mask_mode == 0:
        return n * n
    p = min(max(p, 0), n)
    i = np.arange(p, n)
    start = p + ((i - p) // block) * block
    end = np.minimum(n, start + block)
    own = end if mask_mode == 1 else p + (end - start)
    return int(p * p + own.sum())


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int
    L: int
    Hq: int
    Hkv: int
    D: int
    V: int
    dtype: str                 # "f32" or "bf16": q/k/v/out and logits
    qkv_sigma: float
    logit_sigma: float
    prompt_lo: int             # prompt length range (inclusive)
    prompt_hi: int
    resp_len: int              # n_b = min(L, p_b + resp_len)
    mask_frac: float           # fraction of response positions masked at step 0
    peak_frac: tuple           # per step: fraction of rows with a planted peak
    peak_base: float
    peak_width: float
    peak_current: float        # P(peak token = current token) at filled positions
    zipf_s: float | None
    edit_threshold: tuple      # per step
    remask_k: int              # >= 0 fixed k; < 0 -> floor(remask_frac * r_b)
    remask_frac: float
    steps: int = 1
    seed: int = 0

    @property
    def mask_id(self) -> int:
        # Outside [0, V): a prediction can never equal the mask token.
        return self.V

    @property
    def N(self) -> int:
        return self.B * self.L

    def prompt_lens(self) -> np.ndarray:
        return synth.prompt_lengths(self.seed, self.B, self.prompt_lo, self.prompt_hi)

    def seq_lens(self) -> np.ndarray:
        p = self.prompt_lens().astype(np.int64)
        return np.minimum(self.L, p + self.resp_len).astype(np.int32)

    def step_seed(self, s: int) -> int:
        return self.seed if s == 0 else synth.step_seed(self.seed, s)

    def logit_spec(self, s: int = 0) -> synth.LogitSpec:
        return synth.LogitSpec(self.V, self.logit_sigma, self.step_seed(s),
                               peak_frac=self.peak_frac[s], peak_base=self.peak_base,
                               peak_width=self.peak_width, peak_current=self.peak_current,
                               zipf_s=self.zipf_s)

    def initial_state(self):
        """(tokens int32[B,L], mask uint8[B,L]) before the first refine step:
        prompt and draft tokens uniform in V, a seeded set of exactly
        floor(mask_frac * r_b) response positions masked (token = mask_id)."""
        tok = synth.drafts(self.seed, self.B, self.L, self.V)
        m = synth.response_masks(self.seed, self.B, self.L, self.prompt_lens(), self.seq_lens(),
                                 self.mask_frac)
        tok = np.where(m == 1, self.mask_id, tok).astype(np.int32)
        return tok, m

    def attn_flops(self, mask_mode: int = 0, block: int = 64) -> float:
        """Algorithmic FLOPs of one attention call: 4 * Hq * D per attended
        (query, key) pair; sum_b 4 * Hq * n_b^2 * D without a mask."""
        pairs = sum(attended_pairs(int(n), int(p), mask_mode, block)
                    for n, p in zip(self.seq_lens(), self.prompt_lens()))
        return float(4.0 * self.Hq * self.D * pairs)

    def logit_bytes(self) -> int:
        esz = 2 if self.dtype == "bf16" else 4
        return self.N * self.V * esz

    def vocab_bytes(self) -> int:
        """Algorithmic bytes of one vocabulary reduction: logits read once plus
        argmax, conf and lse written (4 B each) per row."""
        return self.logit_bytes() + 12 * self.N

    def refined_tokens(self) -> int:
        return int(np.sum(self.seq_lens().astype(np.int64) - self.prompt_lens()))


def _peak(sigma: float, V: int):
    # "+8" peak: 8 above the typical row maximum of V draws of N(0, sigma)
    # (about 4.25 sigma at V = 151552), jittered by U[-4, 4) so that the
    # confidences of peaked rows straddle the edit thresholds.
    typical_max = 4.25 * sigma
    return typical_max + 8.0 - 4.0, 8.0


_C2_BASE, _C2_WIDTH = _peak(3.0, 151552)

WORKLOADS = {
    # Tiny CPU-checkable step (fp32). Every row gets a planted argmax whose
    # logit exceeds the bound 6*sigma of all other entries by 0.5 + U[0, 0.5).
    "c1_tiny_f32": Workload(
        "c1_tiny_f32", B=1, L=128, Hq=4, Hkv=2, D=64, V=1024, dtype="f32",
        qkv_sigma=1.0, logit_sigma=2.0, prompt_lo=64, prompt_hi=64, resp_len=64,
        mask_frac=0.5, peak_frac=(1.0,), peak_base=6 * 2.0 + 0.5, peak_width=0.5,
        peak_current=0.0, zipf_s=None, edit_threshold=(0.9,), remask_k=8, remask_frac=0.0),
    # One paper-shaped sequence: 128 prompt + 384 response, fully drafted.
    "c2_single_512": Workload(
        "c2_single_512", B=1, L=512, Hq=32, Hkv=4, D=128, V=151552, dtype="bf16",
        qkv_sigma=1 / math.sqrt(128), logit_sigma=3.0, prompt_lo=128, prompt_hi=128,
        resp_len=384, mask_frac=0.0, peak_frac=(0.1,), peak_base=_C2_BASE,
        peak_width=_C2_WIDTH, peak_current=0.0, zipf_s=None, edit_threshold=(0.8,),
        remask_k=38, remask_frac=0.0),
    # Batched refine: 32 sequences, prompts U{64..256}, n_b = min(512, p_b + 384),
    # 25% of the response masked. Threshold and k not stated: 0.8 and
    # floor(0.1 * r_b), as in the single-sequence and long-draft workloads.
    "c3_batch32_512": Workload(
        "c3_batch32_512", B=32, L=512, Hq=32, Hkv=4, D=128, V=151552, dtype="bf16",
        qkv_sigma=1 / math.sqrt(128), logit_sigma=3.0, prompt_lo=64, prompt_hi=256,
        resp_len=384, mask_frac=0.25, peak_frac=(0.1,), peak_base=_C2_BASE,
        peak_width=_C2_WIDTH, peak_current=0.0, zipf_s=None, edit_threshold=(0.8,),
        remask_k=-1, remask_frac=0.1),
    # Long draft: 512 prompt + 1536 response; logits from a Zipf(1.1) prior
    # (shifted per position) plus N(0, 1). Threshold not stated: 0.8.
    "c4_long_2048": Workload(
        "c4_long_2048", B=8, L=2048, Hq=32, Hkv=4, D=128, V=151552, dtype="bf16",
        qkv_sigma=1 / math.sqrt(128), logit_sigma=1.0, prompt_lo=512, prompt_hi=512,
        resp_len=1536, mask_frac=0.0, peak_frac=(0.0,), peak_base=0.0, peak_width=0.0,
        peak_current=0.0, zipf_s=1.1, edit_threshold=(0.8,), remask_k=-1, remask_frac=0.1),
    # Heavy batch, four consecutive steps; step s plants peaks on a fraction
    # (0.1, 0.3, 0.5, 0.7) of positions, on the current token with prob. 0.5.
    "c5_heavy_4step": Workload(
        "c5_heavy_4step", B=128, L=640, Hq=16, Hkv=2, D=128, V=151552, dtype="bf16",
        qkv_sigma=1 / math.sqrt(128), logit_sigma=3.0, prompt_lo=256, prompt_hi=256,
        resp_len=384, mask_frac=0.0, peak_frac=(0.1, 0.3, 0.5, 0.7), peak_base=_C2_BASE,
        peak_width=_C2_WIDTH, peak_current=0.5, zipf_s=None,
        edit_threshold=(0.9, 0.7, 0.5, 0.5), remask_k=16, remask_frac=0.0, steps=4),
}

ORDER = ["c1_tiny_f32", "c2_single_512", "c3_batch32_512", "c4_long_2048", "c5_heavy_4step"]


def get(name: str) -> Workload:
    if name in WORKLOADS:
        return WORKLOADS[name]
    for k in WORKLOADS:
        if k.startswith(name):
            return WORKLOADS[k]
    raise KeyError(name)


def scaled(w: Workload, **kw) -> Workload:
    """A copy of ``w`` with some fields replaced (smaller parity cases)."""
    return dataclasses.replace(w, **kw)
