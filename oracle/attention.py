"""Oracle step A1: non-causal (bidirectional) GQA attention -- test infrastructure.

Sec. 4.2: the refiner applies bidirectional correction over the entire
sequence, so every valid position attends to every valid position (no causal
or block mask; Sec. 3.3 describes the block-causal pattern this replaces).
The paper does not give the architecture; the readings used here are

* softmax scale 1/sqrt(D) (standard scaled dot-product attention);
* grouped-query attention with contiguous groups: query head h reads key/value
  head floor(h * Hkv / Hq);
* keys j >= n_b (padding) are excluded; query rows i >= n_b output 0.

Definition, for each b, h and i < n_b:
    s_j   = (q_i . k_j) / sqrt(D)            for j < n_b
    w_j   = exp(s_j - max_j s_j)
    out_i = sum_j w_j v_j / sum_j w_j

Mask variants (the same attention over a subset of keys per query):

* block-causal -- the attention of block-autoregressive diffusion (Sec. 3.3):
  the response [p_b, n_b) is cut into blocks of `block` positions starting at
  p_b; a query attends to the prompt and to its own and earlier blocks, never
  to later ones; prompt queries attend to the prompt only;
* block-local -- the "local 64-token refinement" of the causal ablation
  (Sec. 5.3, Sec. 6.3, Appendix C.4): a response query attends to the prompt
  and to its own block only; prompt queries attend to the prompt only.

The readings (blocks start at the prompt length; the prompt is context for
every query and attends only to itself under both variants) are this
oracle's; the paper describes the patterns in words.
"""
from __future__ import annotations

import math

import numpy as np


def kv_head(h: int, Hq: int, Hkv: int) -> int:
    """Key/value head read by query head h (contiguous grouping)."""
    return (h * Hkv) // Hq


def score_scale(D: int) -> float:
    return 1.0 / math.sqrt(D)


MASK_FULL = 0
MASK_BLOCK_CAUSAL = 1
MASK_BLOCK_LOCAL = 2


def block_index(i: int, p: int, block: int) -> int:
    """Block of position i: response blocks 0, 1, ... of `block` positions
    starting at the prompt length p; prompt positions are block -1."""
    return -1 if i < p else (i - p) // block


def key_allowed(i: int, j: int, p: int, block: int, mode: int) -> bool:
    """May query i attend to key j (both < n)?"""
    if mode == MASK_FULL:
        return True
    if j < p:
        return True                      # the prompt is context for every query
    bi, bj = block_index(i, p, block), block_index(j, p, block)
    if mode == MASK_BLOCK_CAUSAL:
        return bj <= bi
    if mode == MASK_BLOCK_LOCAL:
        return bj == bi
    raise ValueError(f"unknown mask mode {mode}")


def key_mask(n: int, p: int = 0, block: int = 1, mode: int = MASK_FULL) -> np.ndarray:
    """Which keys each query of a length-n sequence may attend to (n x n bool):
    all of them for the refiner's bidirectional pass."""
    return np.array([[key_allowed(i, j, p, block, mode) for j in range(n)] for i in range(n)], dtype=bool)


def bidir_attn(q, k, v, seq_lens, mask_mode: int = MASK_FULL, block: int = 1, prompt_lens=None) -> np.ndarray:
    """q [B,L,Hq,D], k/v [B,L,Hkv,D] (any real dtype), seq_lens int [B];
    mask_mode / block / prompt_lens (int [B], clamped to [0, n_b]) select a
    mask variant.

    Returns fp64 [B,L,Hq,D]."""
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    B, L, Hq, D = q.shape
    Hkv = k.shape[2]
    out = np.zeros((B, L, Hq, D), dtype=np.float64)
    for b in range(B):
        n = min(max(int(seq_lens[b]), 0), L)
        if n == 0:
            continue
        p = 0 if prompt_lens is None else min(max(int(prompt_lens[b]), 0), n)
        allowed = key_mask(n, p, block, mask_mode)
        for h in range(Hq):
            g = kv_head(h, Hq, Hkv)
            Q = q[b, :n, h, :]
            K = k[b, :n, g, :]
            Vv = v[b, :n, g, :]
            s = np.where(allowed, (Q @ K.T) * score_scale(D), -np.inf)
            w = np.exp(s - s.max(axis=1, keepdims=True))
            out[b, :n, h, :] = (w @ Vv) / w.sum(axis=1, keepdims=True)
    return out
