"""Oracle step A3: the refine update (commit / edit / remask) -- test infrastructure.

Sec. 4.2 fixes the frame: prompt tokens never change, draft tokens may be
revised at any response position. The per-pass rule is LLaDA2.1 token editing
(Sec. 5.1, Appendix C.4 with Table 11: editing stops when no confident edits remain), which
the paper does not spell out; the reading implemented here is, for each
sequence b with prompt length p_b and valid length n_b (response [p_b, n_b),
r_b = n_b - p_b):

1. prompt [0, p_b) and padding [n_b, L) are copied unchanged;
2. each response position i becomes unmasked and takes
     argmax_i  if it was masked                               (commit),
     argmax_i  if argmax_i != token_i and conf_i >= tau       (edit; counted),
     token_i   otherwise;
3. k_b = remask_k if remask_k >= 0 else floor(remask_frac * r_b), capped at r_b;
4. the k_b response positions that come first in the order
   (conf ascending, index ascending) are remasked: mask 1, token mask_id;
5. n_edits_b = number of edits in step 2 (commits are not edits; an edit that
   is remasked in step 4 still counts).

The threshold compare and the remask order use the fp32 values as given
(-0.0 and +0.0 compare equal). seq_lens is clamped to [0, L] and prompt_lens
to [0, n_b].

Variant (a second reading of step 4, when ``tok_prob`` is given): the remask
order ranks each response position by the probability of the token it holds
after step 2 -- conf_i when that token is the argmax (commit, edit, or a kept
token equal to the argmax), else tok_prob_i, the softmax probability of the
kept token (``vocab.token_prob``) -- so the least likely resulting tokens are
remasked. The paper does not fix which of the two rankings its editing rule
uses; the default is the first.
"""
from __future__ import annotations

import math

import numpy as np


def clamp_lengths(p: int, n: int, L: int):
    n = min(max(int(n), 0), L)
    p = min(max(int(p), 0), n)
    return p, n


def remask_count(remask_k: int, remask_frac: float, r: int) -> int:
    """k_b: fixed count, or floor(remask_frac * r_b) with remask_frac taken as the
    fp32 value given (the fp64 product of a 24-bit mantissa and r_b < 2^29 is
    exact), capped at r_b."""
    if remask_k >= 0:
        k = int(remask_k)
    else:
        k = int(math.floor(float(np.float32(remask_frac)) * r))
    return max(0, min(k, r))


def is_edit(pred: int, tok: int, c: float, tau: float) -> bool:
    return pred != tok and c >= tau


def remask_order(conf_vals, positions):
    """Positions sorted by (conf ascending, index ascending)."""
    return sorted(positions, key=lambda i: (conf_vals[i], i))


def resulting_token_prob(new_tok: int, pred: int, c: float, tp: float) -> float:
    """Probability of the token a position holds after step 2 (variant ranking)."""
    return c if new_tok == pred else tp


def refine_update(tokens, mask, argmax, conf, *, edit_threshold, remask_k, remask_frac,
                  mask_id, prompt_lens, seq_lens, tok_prob=None):
    """tokens int [B,L], mask uint8 [B,L], argmax int [B,L], conf f32 [B,L];
    tok_prob f32 [B,L] or None (variant ranking, see the module docstring).

    Returns (new_tokens int32[B,L], new_mask uint8[B,L], n_edits int32[B])."""
    tokens = np.asarray(tokens)
    mask = np.asarray(mask)
    argmax = np.asarray(argmax)
    conf32 = np.asarray(conf, dtype=np.float32)
    tp32 = None if tok_prob is None else np.asarray(tok_prob, dtype=np.float32)
    B, L = tokens.shape
    tau = float(np.float32(edit_threshold))
    new_tok = np.array(tokens, dtype=np.int32, copy=True)
    new_mask = np.array(mask, dtype=np.uint8, copy=True)
    n_edits = np.zeros(B, dtype=np.int32)
    for b in range(B):
        p, n = clamp_lengths(prompt_lens[b], seq_lens[b], L)
        tok = [int(t) for t in tokens[b]]
        msk = [int(x) for x in mask[b]]
        pred = [int(x) for x in argmax[b]]
        c = [float(x) for x in conf32[b]]
        edits = 0
        for i in range(p, n):
            if msk[i]:
                new_tok[b, i] = pred[i]
            elif is_edit(pred[i], tok[i], c[i], tau):
                new_tok[b, i] = pred[i]
                edits += 1
            else:
                new_tok[b, i] = tok[i]
            new_mask[b, i] = 0
        k = remask_count(remask_k, remask_frac, n - p)
        rank = c
        if tp32 is not None:
            rank = list(c)
            for i in range(p, n):
                rank[i] = resulting_token_prob(int(new_tok[b, i]), pred[i], c[i], float(tp32[b, i]))
        for i in remask_order(rank, range(p, n))[:k]:
            new_mask[b, i] = 1
            new_tok[b, i] = mask_id
        n_edits[b] = edits
    return new_tok, new_mask, n_edits
