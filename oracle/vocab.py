"""Oracle step A2: per-position reduction over the vocabulary -- test infrastructure.

The refiner's confidence of a position is the largest softmax probability of
its logits, and its prediction is the token that attains it (the confidences
that Table 10's refine threshold and Appendix C.4's "confident edits", Table 11 refer
to). For a row x of V logits:

    m      = max_v x_v
    argmax = the lowest v with x_v == m        (ties break to the lowest index)
    S      = sum_v exp(x_v - m)
    lse    = m + ln S                          (log-sum-exp)
    conf   = exp(m - lse) = 1 / S              (maximum softmax probability)

Inputs are converted exactly to fp64; S, lse and conf are evaluated in fp64 and
rounded once to fp32. Entries may be -inf; NaN is outside the contract.
"""
from __future__ import annotations

import numpy as np


def first_argmax(x: np.ndarray) -> np.ndarray:
    """Lowest index attaining the row maximum (np.argmax returns the first)."""
    return np.argmax(x, axis=1)


def vocab_confidence(logits, chunk_rows: int = 256):
    """logits [N, V] (any real dtype). Returns (argmax int32[N], conf f32[N], lse f32[N])."""
    logits = np.asarray(logits)
    N = logits.shape[0]
    am = np.empty(N, dtype=np.int32)
    conf = np.empty(N, dtype=np.float32)
    lse = np.empty(N, dtype=np.float32)
    for r0 in range(0, N, chunk_rows):
        x = logits[r0:r0 + chunk_rows].astype(np.float64)
        m = x.max(axis=1)
        S = np.exp(x - m[:, None]).sum(axis=1)
        am[r0:r0 + chunk_rows] = first_argmax(x)
        lse[r0:r0 + chunk_rows] = (m + np.log(S)).astype(np.float32)
        conf[r0:r0 + chunk_rows] = (1.0 / S).astype(np.float32)
    return am, conf, lse


def token_prob(logits, tokens, lse):
    """Softmax probability of a given token of each row: p_r = exp(x_{r,t_r} - lse_r).

    logits [N, V], tokens int [N], lse [N] (the row's log-sum-exp, as given).
    Evaluated in fp64 and rounded once to fp32; a token outside [0, V) gives 0.
    With t_r the row's argmax this is conf_r (exp(m - lse) = 1 / S)."""
    logits = np.asarray(logits)
    tokens = np.asarray(tokens).reshape(-1)
    lse = np.asarray(lse, dtype=np.float64).reshape(-1)
    N, V = logits.shape
    out = np.zeros(N, dtype=np.float32)
    for r in range(N):
        t = int(tokens[r])
        if 0 <= t < V:
            out[r] = np.float32(softmax_prob(np.float64(logits[r, t]), lse[r]))
    return out


def softmax_prob(x_t: float, lse: float) -> float:
    """exp(x_t - lse): one entry of softmax(x) given the row's log-sum-exp."""
    return float(np.exp(x_t - lse))
