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
"""
from __future__ import annotations

import math

import numpy as np


def kv_head(h: int, Hq: int, Hkv: int) -> int:
    """Key/value head read by query head h (contiguous grouping)."""
    return (h * Hkv) // Hq


def score_scale(D: int) -> float:
    return 1.0 / math.sqrt(D)


def key_mask(n: int) -> np.ndarray:
    """Which keys each query of a length-n sequence may attend to: all of them
    (an n x n matrix of True; a causal decoder would use the lower triangle)."""
    return np.ones((n, n), dtype=bool)


def bidir_attn(q, k, v, seq_lens) -> np.ndarray:
    """q [B,L,Hq,D], k/v [B,L,Hkv,D] (any real dtype), seq_lens int [B].

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
        for h in range(Hq):
            g = kv_head(h, Hq, Hkv)
            Q = q[b, :n, h, :]
            K = k[b, :n, g, :]
            Vv = v[b, :n, g, :]
            s = np.where(key_mask(n), (Q @ K.T) * score_scale(D), -np.inf)
            w = np.exp(s - s.max(axis=1, keepdims=True))
            out[b, :n, h, :] = (w @ Vv) / w.sum(axis=1, keepdims=True)
    return out
