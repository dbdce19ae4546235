"""Planted mistakes in the oracle (on the CPU only) must each fail some pin.

Every mutation below is a plausible slip in writing the method down: a causal
mask, a wrong softmax scale, interleaved instead of contiguous GQA groups, the
last instead of the first maximum, a strict threshold, ties broken towards the
higher index, a rounded-up remask count, a block-causal mask that drops the
query's own block, a block-local mask without the prompt, a resulting-token ranking that
ignores which positions end with their argmax, a sign slip in a token's
probability, a projection that pairs the wrong feature indices, and in the
multi-pass loop: a budget off by one, a stop as soon as one sequence makes no
edit, commits counted as edits, a stop rule that ignores the edits. If a pin
suite let one through, the oracle could carry that slip undetected."""
import math

import numpy as np
import pytest

import oracle_pins as P
from oracle import attention as oatt
from oracle import update as oupd
from oracle import lmhead as olmh
from oracle import vocab as ovoc
from oracle import loop as oloop

MUTATIONS = {
    "causal_mask": (oatt, "key_mask", lambda n, p=0, block=1, mode=0: np.tril(np.ones((n, n), dtype=bool)),
                    P.ATTN_PINS),
    "block_causal_strict": (oatt, "key_allowed",
                            lambda i, j, p, b, mode: True if mode == 0 else (
                                j < p or (oatt.block_index(j, p, b) < oatt.block_index(i, p, b) if mode == 1
                                          else oatt.block_index(j, p, b) == oatt.block_index(i, p, b))),
                            P.ATTN_PINS),
    "local_without_prompt": (oatt, "key_allowed",
                             lambda i, j, p, b, mode: True if mode == 0 else (
                                 (j < p or oatt.block_index(j, p, b) <= oatt.block_index(i, p, b)) if mode == 1
                                 else oatt.block_index(j, p, b) == oatt.block_index(i, p, b)),
                             P.ATTN_PINS),
    "scale_1_over_D": (oatt, "score_scale", lambda D: 1.0 / D, P.ATTN_PINS),
    "interleaved_gqa": (oatt, "kv_head", lambda h, Hq, Hkv: h % Hkv, P.ATTN_PINS),
    "last_argmax": (ovoc, "first_argmax",
                    lambda x: x.shape[1] - 1 - np.argmax(x[:, ::-1], axis=1), P.VOCAB_PINS),
    "strict_threshold": (oupd, "is_edit", lambda p, t, c, tau: p != t and c > tau, P.UPDATE_PINS),
    "ties_high_index": (oupd, "remask_order",
                        lambda cv, pos: sorted(pos, key=lambda i: (cv[i], -i)), P.UPDATE_PINS),
    "result_rank_ignores_argmax": (oupd, "resulting_token_prob", lambda nt, pred, c, tp: tp, P.UPDATE_PINS),
    "token_prob_sign": (ovoc, "softmax_prob", lambda x, lse: float(np.exp(lse - x)), P.VOCAB_PINS),
    "projection_reversed_features": (olmh, "project", lambda h, w: h @ w[:, ::-1].T, P.VOCAB_PINS),
    "loop_budget_plus_one": (oloop, "more_passes", lambda ne, passes, mx: passes <= mx and bool(np.any(ne > 0)),
                             P.LOOP_PINS),
    "loop_stops_per_sequence": (oloop, "more_passes", lambda ne, passes, mx: passes < mx and bool(np.all(ne > 0)),
                                P.LOOP_PINS),
    "loop_ignores_edits": (oloop, "more_passes", lambda ne, passes, mx: passes < mx, P.LOOP_PINS),
    "loop_counts_commits": (oloop, "refine_update",
                            lambda tok, msk, am, cf, **kw: (lambda r: (r[0], r[1], r[2] + np.asarray(msk).sum(
                                axis=1).astype(np.int32)))(oupd.refine_update(tok, msk, am, cf, **kw)),
                            P.LOOP_PINS),
    "ceil_remask_count": (oupd, "remask_count",
                          lambda k, f, r: max(0, min(k if k >= 0 else
                                                     math.ceil(float(np.float32(f)) * r), r)),
                          P.UPDATE_PINS),
}


# A planted mask slip can leave a query row with no keys (a NaN row): expected.
@pytest.mark.filterwarnings("ignore:invalid value encountered:RuntimeWarning")
@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_mutation_is_caught(name, monkeypatch):
    mod, attr, fn, pins = MUTATIONS[name]
    monkeypatch.setattr(mod, attr, fn)
    failed = []
    for pin in pins:
        try:
            pin()
        except AssertionError:
            failed.append(pin.__name__)
    assert failed, f"mutation {name} passed every pin"
