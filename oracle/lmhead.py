"""Oracle of the vocabulary projection fused with step A2 -- test infrastructure.

The refiner predicts every position's token from its final hidden state
(Sec. 4.2: each revisable position gets a distribution over the vocabulary);
the logits a pass reduces are the output projection of those states,
    logits[r, v] = sum_k hidden[r, k] * weight[v, k]      (hidden [N, d], weight [V, d]),
and the fused operation returns, for each row r, exactly what
vocab.vocab_confidence returns for that row of logits (argmax with ties to the
lowest index, maximum softmax probability, log-sum-exp), without storing the
N x V logits. The width d is not given by the paper; it is a parameter.

The projection is evaluated in fp64 (inputs converted exactly), block by block
over the vocabulary so that memory stays bounded.
"""
from __future__ import annotations

import numpy as np

from .vocab import vocab_confidence


def lm_head_logits(hidden, weight, block: int = 8192) -> np.ndarray:
    """fp64 logits [N, V] = hidden @ weight^T."""
    h = np.asarray(hidden, dtype=np.float64)
    w = np.asarray(weight)
    N, V = h.shape[0], w.shape[0]
    out = np.empty((N, V), dtype=np.float64)
    for v0 in range(0, V, block):
        out[:, v0:v0 + block] = project(h, np.asarray(w[v0:v0 + block], dtype=np.float64))
    return out


def project(h: np.ndarray, w_block: np.ndarray) -> np.ndarray:
    """One vocabulary block of logits: h [N, d] times w_block [v, d]^T."""
    return h @ w_block.T


def lm_head_confidence(hidden, weight):
    """(argmax int32[N], conf f32[N], lse f32[N]) of hidden @ weight^T."""
    return vocab_confidence(lm_head_logits(hidden, weight))
