"""Seeded synthetic inputs for the refine step (host side, numpy).

This module generates inputs only. It computes nothing the refine step
computes (no softmax, no maximum, no selection): it turns a seed and an
element index into a number, the same way on the host (here) and on the
device (``csrc/synth.cu``, library ``libdlmsynth.so``), bit for bit, so that
tensors of tens of GB can be generated in HBM at full speed while any slice of
them can be regenerated on the host for the CPU oracle.

Generator definition
--------------------
* ``mix64`` is the output function of SplitMix64 (Steele, Lea & Flood,
  "Fast splittable pseudorandom number generators", OOPSLA 2014), with the
  multipliers of the published reference implementation.
* A *stream key* is ``mix64(mix64(seed) ^ (stream * 0xD1B54A32D192ED03))``.
* Draw ``i`` of a stream is ``mix64(key + i * 0x9E3779B97F4A7C15)`` (mod 2^64):
  the counter-based form of SplitMix64, so every draw is addressable.
* A *normal* for element ``e`` sums the twelve 16-bit lanes of draws
  ``3e, 3e+1, 3e+2`` (an Irwin-Hall sum of 12 uniforms), subtracts the mean
  393210, converts the integer to fp32 (exact: |z| < 2^24) and multiplies once,
  rounding to nearest, by ``c = fp32(sigma) * 2^-16``. The result is bounded:
  ``|x| < 6 * sigma``.
* A *uniform integer* in ``[0, n)`` is ``(hi32(draw) * n) >> 32``.
* A *unit float* in ``[0, 1)`` is ``(draw >> 40) * 2^-24`` (exact in fp32).
* bf16 values are the fp32 values rounded to nearest-even on the bit pattern.

Every fp32 operation here is a single IEEE operation rounded to nearest
(numpy does not contract ``a * b + c``); the device twin uses ``__fmul_rn`` and
``__fadd_rn`` so that neither side fuses a multiply-add.
"""
from __future__ import annotations

import numpy as np

MASK64 = (1 << 64) - 1
GOLDEN = 0x9E3779B97F4A7C15
STREAM_MUL = 0xD1B54A32D192ED03
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB
IH_MEAN = 393210  # 12 * (2^16 - 1) / 2

# Stream ids: one per kind of input, so that inputs never share draws.
S_Q, S_K, S_V = 1, 2, 3
S_LOGIT = 4
S_PEAK = 5
S_DRAFT = 6
S_MASK = 7
S_PROMPT = 8
S_SHIFT = 9
S_STEP = 10


def mix64_int(z: int) -> int:
    """SplitMix64 output function on a Python int (mod 2^64)."""
    z &= MASK64
    z = ((z ^ (z >> 30)) * _M1) & MASK64
    z = ((z ^ (z >> 27)) * _M2) & MASK64
    return z ^ (z >> 31)


def stream_key(seed: int, stream: int) -> int:
    return mix64_int(mix64_int(seed) ^ ((stream * STREAM_MUL) & MASK64))


def step_seed(seed: int, step: int) -> int:
    """Seed of refine step ``step`` of a multi-step workload."""
    return stream_key(seed, S_STEP + (step << 8))


def _mix64(z: np.ndarray) -> np.ndarray:
    z = z ^ (z >> np.uint64(30))
    z = z * np.uint64(_M1)
    z = z ^ (z >> np.uint64(27))
    z = z * np.uint64(_M2)
    return z ^ (z >> np.uint64(31))


def draws(key: int, idx) -> np.ndarray:
    """Draws ``idx`` (uint64 array) of the stream with key ``key``."""
    idx = np.asarray(idx, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix64(np.uint64(key) + idx * np.uint64(GOLDEN))


def _lane_sum(d: np.ndarray) -> np.ndarray:
    m = np.uint64(0xFFFF)
    return ((d & m) + ((d >> np.uint64(16)) & m) + ((d >> np.uint64(32)) & m)
            + (d >> np.uint64(48))).astype(np.int64)


def normal_scale(sigma: float) -> np.float32:
    """The fp32 multiplier ``fp32(sigma) * 2^-16`` (exact power-of-two scaling)."""
    return np.float32(np.float32(sigma) * np.float32(2.0 ** -16))


def normals(key: int, idx, sigma: float) -> np.ndarray:
    """fp32 Irwin-Hall(12) normals for element indices ``idx``."""
    idx = np.asarray(idx, dtype=np.uint64)
    three = np.uint64(3)
    s = (_lane_sum(draws(key, idx * three)) + _lane_sum(draws(key, idx * three + np.uint64(1)))
         + _lane_sum(draws(key, idx * three + np.uint64(2))))
    z = (s - IH_MEAN).astype(np.float32)
    return (z * normal_scale(sigma)).astype(np.float32)


def uniform_int(key: int, idx, n: int) -> np.ndarray:
    hi = draws(key, idx) >> np.uint64(32)
    return ((hi * np.uint64(n)) >> np.uint64(32)).astype(np.int64)


def unit_float(key: int, idx) -> np.ndarray:
    d = draws(key, idx) >> np.uint64(40)
    return (d.astype(np.float32) * np.float32(2.0 ** -24)).astype(np.float32)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (nearest-even); returns the uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# ---------------------------------------------------------------------------
# Tensors of a workload (host twins of the device generator)
# ---------------------------------------------------------------------------

def qkv_host(seed: int, which: int, shape, sigma: float, dtype: str, flat_offset: int = 0,
             count: int | None = None) -> np.ndarray:
    """Elements ``[flat_offset, flat_offset + count)`` of q (which=S_Q), k or v.

    The tensor is indexed in row-major order of ``shape`` = (B, L, H, D).
    Returns fp32 values (dtype "f32") or bf16 bit patterns (dtype "bf16").
    """
    total = int(np.prod(shape))
    if count is None:
        count = total - flat_offset
    idx = np.arange(flat_offset, flat_offset + count, dtype=np.uint64)
    x = normals(stream_key(seed, which), idx, sigma)
    return f32_to_bf16_bits(x) if dtype == "bf16" else x


def peak_threshold(frac: float) -> int:
    """Integer threshold on hi32(draw) that selects a fraction ``frac`` of rows."""
    return min(int(round(frac * 4294967296.0)), 4294967296)


class LogitSpec:
    """Parameters of the synthetic logits of one refine step.

    Row ``r`` (position ``r % L`` of sequence ``r // L``) holds
    ``base[v] + sigma * N_rv`` where ``base`` is zero or a table (the Zipf
    prior, indexed at ``(v + shift_r) % V``); a *peaked* row then has one token
    ``t_r`` set to ``peak_base + peak_width * u_r``.

    * ``peak_frac``: fraction of rows that are peaked (1.0 = every row).
    * ``peak_current``: probability that the peak token is the row's current
      token (0 = always uniform); masked positions always get a uniform token.
    """

    def __init__(self, V, sigma, seed, peak_frac=0.0, peak_base=0.0, peak_width=0.0,
                 peak_current=0.0, zipf_s=None):
        self.V = int(V)
        self.sigma = float(sigma)
        self.seed = int(seed)
        self.peak_frac = float(peak_frac)
        self.peak_base = float(peak_base)
        self.peak_width = float(peak_width)
        self.peak_current = float(peak_current)
        self.zipf_s = zipf_s

    def zipf_table(self) -> np.ndarray | None:
        """fp32 table ``-s * ln(1 + j)``, computed on the host once and copied to
        the device, so both sides add the same fp32 values."""
        if self.zipf_s is None:
            return None
        j = np.arange(self.V, dtype=np.float64)
        return (-self.zipf_s * np.log1p(j)).astype(np.float32)

    def peak_plan(self, rows: np.ndarray, tokens: np.ndarray | None = None,
                  mask: np.ndarray | None = None):
        """(is_peaked bool[n], token int64[n], value fp32[n]) for the given rows.

        ``tokens``/``mask`` are the current token and mask at those rows (only
        read when ``peak_current > 0``)."""
        rows = np.asarray(rows, dtype=np.uint64)
        key = stream_key(self.seed, S_PEAK)
        four = np.uint64(4)
        d0 = draws(key, rows * four) >> np.uint64(32)
        d1 = draws(key, rows * four + np.uint64(1)) >> np.uint64(32)
        is_peak = d0 < np.uint64(peak_threshold(self.peak_frac))
        tok = uniform_int(key, rows * four + np.uint64(2), self.V)
        if self.peak_current > 0.0 and tokens is not None:
            use_cur = d1 < np.uint64(peak_threshold(self.peak_current))
            filled = np.asarray(mask) == 0
            tok = np.where(use_cur & filled, np.asarray(tokens, dtype=np.int64), tok)
        u = unit_float(key, rows * four + np.uint64(3))
        val = (u * np.float32(self.peak_width)).astype(np.float32) + np.float32(self.peak_base)
        return is_peak, tok, val.astype(np.float32)

    def rows_f32(self, rows, tokens=None, mask=None) -> np.ndarray:
        """fp32 logits of the given rows, shape [len(rows), V]."""
        rows = np.asarray(rows, dtype=np.int64)
        V = self.V
        key = stream_key(self.seed, S_LOGIT)
        out = np.empty((len(rows), V), dtype=np.float32)
        table = self.zipf_table()
        shift_key = stream_key(self.seed, S_SHIFT)
        is_peak, tok, val = self.peak_plan(rows, tokens, mask)
        v = np.arange(V, dtype=np.uint64)
        for n, r in enumerate(rows):
            x = normals(key, np.uint64(r) * np.uint64(V) + v, self.sigma)
            if table is not None:
                sh = int(uniform_int(shift_key, np.array([r], dtype=np.uint64), V)[0])
                x = (table[(np.arange(V) + sh) % V] + x).astype(np.float32)
            if is_peak[n]:
                x[tok[n]] = val[n]
            out[n] = x
        return out


def prompt_lengths(seed: int, B: int, lo: int, hi: int) -> np.ndarray:
    """Per-sequence prompt lengths uniform in ``lo..hi`` (inclusive)."""
    if lo == hi:
        return np.full(B, lo, dtype=np.int32)
    key = stream_key(seed, S_PROMPT)
    return (lo + uniform_int(key, np.arange(B, dtype=np.uint64), hi - lo + 1)).astype(np.int32)


def drafts(seed: int, B: int, L: int, V: int) -> np.ndarray:
    """Draft tokens uniform in [0, V), shape [B, L] (prompt positions included)."""
    key = stream_key(seed, S_DRAFT)
    return uniform_int(key, np.arange(B * L, dtype=np.uint64), V).reshape(B, L).astype(np.int32)


def response_masks(seed: int, B: int, L: int, prompt_lens, seq_lens, frac: float) -> np.ndarray:
    """Mask exactly floor(frac * r_b) response positions of each sequence: those
    whose draw is smallest (index breaks ties). uint8 [B, L]."""
    key = stream_key(seed, S_MASK)
    m = np.zeros((B, L), dtype=np.uint8)
    for b in range(B):
        p, n = int(prompt_lens[b]), int(seq_lens[b])
        r = n - p
        cnt = int(np.floor(np.float64(np.float32(frac)) * r))
        if cnt <= 0:
            continue
        d = draws(key, np.arange(b * L + p, b * L + n, dtype=np.uint64))
        order = np.lexsort((np.arange(r), d))
        m[b, p + order[:cnt]] = 1
    return m
