"""Pins of the CPU oracle: checks against things other than the oracle itself.

Each ``pin_*`` function raises AssertionError when the oracle disagrees with
a brute-force loop, a torch fp64 library routine, a closed form, an invariant
or a hand-worked example. ``test_oracle_*.py`` runs them as tests;
``test_oracle_mutations.py`` plants plausible mistakes in the oracle and checks
that some pin fails for each.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np
import torch

import oracle
from oracle import attention as oatt
from oracle import update as oupd
from oracle import vocab as ovoc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- attention

def brute_attention(q, k, v, seq_lens):
    """Pure-Python loops: per query, per key, per dim (tiny inputs only).

    Uses the log-sum-exp form (stable) rather than max subtraction, with the
    kv head taken as h // (Hq // Hkv)."""
    B, L, Hq, D = q.shape
    Hkv = k.shape[2]
    grp = Hq // Hkv
    out = np.zeros((B, L, Hq, D))
    for b in range(B):
        n = int(seq_lens[b])
        for h in range(Hq):
            g = h // grp
            for i in range(n):
                s = [sum(float(q[b, i, h, d]) * float(k[b, j, g, d]) for d in range(D)) / math.sqrt(D)
                     for j in range(n)]
                mx = max(s)
                lse = mx + math.log(sum(math.exp(x - mx) for x in s))
                for d in range(D):
                    out[b, i, h, d] = sum(math.exp(s[j] - lse) * float(v[b, j, g, d]) for j in range(n))
    return out


def _rand_qkv(rng, B, L, Hq, Hkv, D, scale=1.0):
    return (rng.standard_normal((B, L, Hq, D)) * scale, rng.standard_normal((B, L, Hkv, D)) * scale,
            rng.standard_normal((B, L, Hkv, D)))


def pin_attn_brute_force():
    rng = np.random.default_rng(11)
    q, k, v = _rand_qkv(rng, 2, 5, 4, 2, 3)
    sl = np.array([5, 3])
    got = oracle.bidir_attn(q, k, v, sl)
    ref = brute_attention(q, k, v, sl)
    assert np.abs(got - ref).max() < 1e-12


def pin_attn_torch_sdpa():
    """torch CPU fp64 scaled_dot_product_attention (no mask = non-causal)."""
    rng = np.random.default_rng(12)
    B, L, Hq, Hkv, D = 2, 48, 8, 2, 16
    q, k, v = _rand_qkv(rng, B, L, Hq, Hkv, D)
    sl = np.array([48, 29])
    got = oracle.bidir_attn(q, k, v, sl)
    for b in range(B):
        n = int(sl[b])
        tq = torch.from_numpy(q[b, :n]).permute(1, 0, 2)               # [Hq, n, D]
        tk = torch.from_numpy(k[b, :n]).permute(1, 0, 2).repeat_interleave(Hq // Hkv, 0)
        tv = torch.from_numpy(v[b, :n]).permute(1, 0, 2).repeat_interleave(Hq // Hkv, 0)
        ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, is_causal=False)
        assert np.abs(got[b, :n] - ref.permute(1, 0, 2).numpy()).max() < 1e-12
        assert np.all(got[b, n:] == 0.0)


def pin_attn_identical_keys_mean():
    """All keys equal: softmax is uniform, out = mean of v over j < n."""
    rng = np.random.default_rng(13)
    B, L, Hq, Hkv, D = 1, 9, 2, 1, 4
    q = rng.standard_normal((B, L, Hq, D))
    k = np.broadcast_to(rng.standard_normal(D), (B, L, Hkv, D)).copy()
    v = rng.standard_normal((B, L, Hkv, D))
    n = 7
    got = oracle.bidir_attn(q, k, v, [n])
    assert np.abs(got[0, :n] - v[0, :n, 0].mean(axis=0)).max() < 1e-12


def pin_attn_dominant_key():
    """One key whose score exceeds all others by >= 50: out = its value."""
    B, L, Hq, Hkv, D = 1, 6, 1, 1, 4
    q = np.zeros((B, L, Hq, D)); q[..., 0] = 1.0
    k = np.zeros((B, L, Hkv, D)); k[0, 4, 0, 0] = 100.0 * math.sqrt(D)   # score 100 vs 0
    v = np.arange(L * D, dtype=np.float64).reshape(B, L, Hkv, D)
    got = oracle.bidir_attn(q, k, v, [L])
    assert np.abs(got[0, :, 0] - v[0, 4, 0]).max() < 1e-12


def pin_attn_single_position():
    rng = np.random.default_rng(14)
    q, k, v = _rand_qkv(rng, 1, 4, 2, 2, 8)
    got = oracle.bidir_attn(q, k, v, [1])
    assert np.abs(got[0, 0] - v[0, 0]).max() < 1e-12
    assert np.all(got[0, 1:] == 0.0)


def pin_attn_two_key_closed_form():
    """Two keys with scores a, b (before scaling): out = sigma(a-b) v0 + sigma(b-a) v1
    with the 1/sqrt(D) scale applied: weights e^{a/sD} / (e^{a/sD} + e^{b/sD})."""
    D = 16
    q = np.zeros((1, 2, 1, D)); q[0, :, 0, 0] = 1.0
    k = np.zeros((1, 2, 1, D)); k[0, 0, 0, 0] = 3.0; k[0, 1, 0, 0] = -1.0
    v = np.zeros((1, 2, 1, D)); v[0, 0, 0, 1] = 1.0; v[0, 1, 0, 2] = 1.0
    got = oracle.bidir_attn(q, k, v, [2])
    w0 = 1.0 / (1.0 + math.exp((-1.0 - 3.0) / 4.0))
    assert abs(got[0, 0, 0, 1] - w0) < 1e-14 and abs(got[0, 0, 0, 2] - (1 - w0)) < 1e-14


def pin_attn_permutation_invariance():
    """Non-causal: jointly permuting (k_j, v_j) over j < n changes nothing."""
    rng = np.random.default_rng(15)
    q, k, v = _rand_qkv(rng, 1, 12, 4, 2, 8)
    n = 10
    perm = np.concatenate([rng.permutation(n), np.arange(n, 12)])
    a = oracle.bidir_attn(q, k, v, [n])
    b = oracle.bidir_attn(q, k[:, perm], v[:, perm], [n])
    assert np.abs(a - b).max() < 1e-12


def pin_attn_gqa_grouping():
    """Hq = 4, Hkv = 2: heads 0,1 read kv head 0 and heads 2,3 read kv head 1,
    i.e. equal to MHA on kv heads repeated in contiguous groups."""
    rng = np.random.default_rng(16)
    q, k, v = _rand_qkv(rng, 1, 7, 4, 2, 5)
    got = oracle.bidir_attn(q, k, v, [7])
    k_rep = np.repeat(k, 2, axis=2)
    v_rep = np.repeat(v, 2, axis=2)
    ref = brute_attention(q, k_rep, v_rep, [7])
    assert np.abs(got - ref).max() < 1e-12


def pin_attn_padding_and_empty():
    rng = np.random.default_rng(17)
    q, k, v = _rand_qkv(rng, 3, 6, 2, 1, 4)
    v[1, 4:] = np.nan       # padding keys must not be read
    k[1, 4:] = np.inf
    got = oracle.bidir_attn(q, k, v, [6, 4, 0])
    assert np.all(got[2] == 0.0)
    assert np.all(got[1, 4:] == 0.0)
    assert np.all(np.isfinite(got))


def key_ranges(i, n, p, block, mode):
    """The keys query i may use, written as index ranges (an independent
    statement of the block variants): block-causal [0, end_i), block-local
    [0, p) + [start_i, end_i), with start_i / end_i the bounds of i's block;
    prompt queries [0, p)."""
    if mode == 0:
        return [(0, n)]
    if i < p:
        return [(0, p)]
    start = p + ((i - p) // block) * block
    end = min(n, start + block)
    return [(0, end)] if mode == 1 else [(0, p), (start, end)]


def brute_masked(q, k, v, seq_lens, prompt_lens, block, mode):
    B, L, Hq, D = q.shape
    grp = Hq // k.shape[2]
    out = np.zeros((B, L, Hq, D))
    for b in range(B):
        n, p = int(seq_lens[b]), int(prompt_lens[b])
        for h in range(Hq):
            g = h // grp
            for i in range(n):
                js = [j for lo, hi in key_ranges(i, n, p, block, mode) for j in range(lo, hi)]
                s = [float(np.dot(q[b, i, h], k[b, j, g])) / math.sqrt(D) for j in js]
                mx = max(s)
                w = [math.exp(x - mx) for x in s]
                out[b, i, h] = sum(wj * v[b, j, g] for wj, j in zip(w, js)) / sum(w)
    return out


def pin_attn_masks_brute_force():
    """Both block variants against loops over the key ranges, several block
    sizes, prompts and lengths (including blocks cut by n)."""
    rng = np.random.default_rng(18)
    q, k, v = _rand_qkv(rng, 3, 13, 2, 1, 4)
    sl, pl = np.array([13, 11, 5]), np.array([3, 0, 5])
    for mode in (1, 2):
        for block in (1, 2, 4, 20):
            got = oracle.bidir_attn(q, k, v, sl, mask_mode=mode, block=block, prompt_lens=pl)
            ref = brute_masked(q, k, v, sl, pl, block, mode)
            assert np.abs(got - ref).max() < 1e-12, (mode, block)


def pin_attn_masks_torch_sdpa():
    """torch fp64 scaled_dot_product_attention with a boolean mask built from
    the key ranges."""
    rng = np.random.default_rng(19)
    B, L, Hq, Hkv, D = 1, 40, 4, 2, 8
    q, k, v = _rand_qkv(rng, B, L, Hq, Hkv, D)
    n, p = 37, 6
    for mode, block in ((1, 8), (2, 8), (1, 5)):
        got = oracle.bidir_attn(q, k, v, [n], mask_mode=mode, block=block, prompt_lens=[p])
        m = torch.zeros(n, n, dtype=torch.bool)
        for i in range(n):
            for lo, hi in key_ranges(i, n, p, block, mode):
                m[i, lo:hi] = True
        tq = torch.from_numpy(q[0, :n]).permute(1, 0, 2)
        tk = torch.from_numpy(k[0, :n]).permute(1, 0, 2).repeat_interleave(Hq // Hkv, 0)
        tv = torch.from_numpy(v[0, :n]).permute(1, 0, 2).repeat_interleave(Hq // Hkv, 0)
        ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, attn_mask=m)
        assert np.abs(got[0, :n] - ref.permute(1, 0, 2).numpy()).max() < 1e-12


def pin_attn_masks_properties():
    """Block-causal with one block covering the response is the full attention
    for response queries; block-local with the response as one block is the
    same; changing keys/values of a later block leaves block-causal outputs of
    earlier blocks unchanged; prompt queries see only the prompt."""
    rng = np.random.default_rng(20)
    q, k, v = _rand_qkv(rng, 1, 16, 2, 2, 4)
    n, p = 16, 4
    full = oracle.bidir_attn(q, k, v, [n])
    for mode in (1, 2):
        one = oracle.bidir_attn(q, k, v, [n], mask_mode=mode, block=n - p, prompt_lens=[p])
        assert np.abs(one[0, p:] - full[0, p:]).max() < 1e-12
        prompt_only = oracle.bidir_attn(q, k, v, [p])
        assert np.abs(one[0, :p] - prompt_only[0, :p]).max() < 1e-12
    a = oracle.bidir_attn(q, k, v, [n], mask_mode=1, block=4, prompt_lens=[p])
    k2, v2 = k.copy(), v.copy()
    k2[0, 12:] += 3.0
    v2[0, 12:] -= 2.0
    b = oracle.bidir_attn(q, k2, v2, [n], mask_mode=1, block=4, prompt_lens=[p])
    assert np.abs(a[0, :12] - b[0, :12]).max() < 1e-12 and np.abs(a[0, 12:] - b[0, 12:]).max() > 1e-3


ATTN_PINS = [pin_attn_brute_force, pin_attn_torch_sdpa, pin_attn_identical_keys_mean,
             pin_attn_dominant_key, pin_attn_single_position, pin_attn_two_key_closed_form,
             pin_attn_permutation_invariance, pin_attn_gqa_grouping, pin_attn_padding_and_empty,
             pin_attn_masks_brute_force, pin_attn_masks_torch_sdpa, pin_attn_masks_properties]


# ---------------------------------------------------------------- vocab

def pin_vocab_uniform_row():
    V = 1000
    x = np.full((1, V), 2.5)
    am, conf, lse = oracle.vocab_confidence(x)
    assert am[0] == 0
    assert conf[0] == np.float32(1.0 / V)
    assert lse[0] == np.float32(2.5 + math.log(V))


def pin_vocab_single_finite():
    V = 64
    x = np.full((1, V), -np.inf); x[0, 17] = -3.25
    am, conf, lse = oracle.vocab_confidence(x)
    assert am[0] == 17 and conf[0] == 1.0 and lse[0] == np.float32(-3.25)


def pin_vocab_two_valued_closed_form():
    V, a, b, t = 500, 4.0, 1.5, 123
    x = np.full((1, V), b); x[0, t] = a
    am, conf, lse = oracle.vocab_confidence(x)
    c = math.exp(a) / (math.exp(a) + (V - 1) * math.exp(b))
    assert am[0] == t
    assert abs(float(conf[0]) - c) <= 1e-7 * c
    ref_lse = math.log(math.exp(a) + (V - 1) * math.exp(b))
    assert abs(float(lse[0]) - ref_lse) <= 1e-7 * ref_lse


def pin_vocab_ties_lowest_index():
    x = np.zeros((2, 16)); x[0, 7] = 5.0; x[0, 3] = 5.0
    x[1, 15] = -1.0; x[1, :15] = -2.0; x[1, 9] = -1.0
    am, _, _ = oracle.vocab_confidence(x)
    assert am[0] == 3 and am[1] == 9


def pin_vocab_torch():
    rng = np.random.default_rng(21)
    x = rng.standard_normal((33, 4096)) * 3.0
    x[5, 100] = 40.0
    am, conf, lse = oracle.vocab_confidence(x)
    t = torch.from_numpy(x)
    ref_lse = torch.logsumexp(t, dim=1).numpy()
    ref_conf = torch.softmax(t, dim=1).max(dim=1).values.numpy()
    ref_am = torch.argmax(t, dim=1).numpy()
    assert np.array_equal(am, ref_am)
    assert np.all(np.abs(lse.astype(np.float64) - ref_lse) <= 1e-7 * np.abs(ref_lse))
    assert np.all(np.abs(conf.astype(np.float64) - ref_conf) <= 1e-7 * ref_conf)


def pin_token_prob_closed_forms():
    """Uniform row: 1/V for every token; two-valued row in closed form; a token
    outside [0, V) gives 0; the argmax's probability is the confidence."""
    V = 300
    x = np.full((3, V), 1.25)
    x[1, 40] = 3.0
    lse = np.array([1.25 + math.log(V), math.log(math.exp(3.0) + (V - 1) * math.exp(1.25)), 0.0])
    p = oracle.token_prob(x, np.array([7, 40, V]), lse)
    assert abs(float(p[0]) - 1.0 / V) <= 1e-7 / V
    c = math.exp(3.0) / (math.exp(3.0) + (V - 1) * math.exp(1.25))
    assert abs(float(p[1]) - c) <= 1e-7 * c
    assert p[2] == 0.0
    rng = np.random.default_rng(23)
    y = rng.standard_normal((9, 2000)) * 3.0
    am, conf, lse32 = oracle.vocab_confidence(y)
    pa = oracle.token_prob(y, am, lse32)
    assert np.all(np.abs(pa.astype(np.float64) - conf) <= 1e-5 * conf)


def pin_token_prob_torch():
    """Against torch fp64 log_softmax + gather, and the probabilities of all
    tokens of a row summing to 1."""
    rng = np.random.default_rng(24)
    x = rng.standard_normal((17, 3000)) * 2.5
    tok = rng.integers(0, 3000, 17)
    t = torch.from_numpy(x)
    lse = torch.logsumexp(t, dim=1).numpy()
    p = oracle.token_prob(x, tok, lse)
    ref = torch.exp(torch.log_softmax(t, dim=1).gather(1, torch.from_numpy(tok)[:, None])[:, 0]).numpy()
    assert np.all(np.abs(p.astype(np.float64) - ref) <= 1e-6 * ref + 1e-30)
    row = np.repeat(x[:1], 3000, axis=0)
    tot = oracle.token_prob(row, np.arange(3000), np.full(3000, lse[0])).astype(np.float64).sum()
    assert abs(tot - 1.0) <= 1e-5


def pin_lmhead_brute_force():
    """Tiny case with explicit dot products and a max / sum written out."""
    rng = np.random.default_rng(25)
    h = rng.standard_normal((3, 5))
    w = rng.standard_normal((7, 5))
    am, conf, lse = oracle.lm_head_confidence(h, w)
    for r in range(3):
        x = [sum(h[r, k] * w[v, k] for k in range(5)) for v in range(7)]
        mx = max(x)
        S = sum(math.exp(t - mx) for t in x)
        assert am[r] == x.index(mx)
        assert abs(float(lse[r]) - (mx + math.log(S))) <= 1e-6 * max(1.0, abs(mx))
        assert abs(float(conf[r]) - 1.0 / S) <= 1e-6 / S


def pin_lmhead_torch():
    """torch fp64 matmul + logsumexp / softmax / argmax, with the vocabulary
    spread over several projection blocks."""
    rng = np.random.default_rng(26)
    h = rng.standard_normal((9, 64))
    w = rng.standard_normal((3000, 64)) / 8.0
    logits = oracle.lm_head_logits(h, w, block=1000)
    t = torch.from_numpy(h) @ torch.from_numpy(w).T
    assert np.abs(logits - t.numpy()).max() <= 1e-12
    am, conf, lse = oracle.lm_head_confidence(h, w)
    assert np.array_equal(am, torch.argmax(t, dim=1).numpy())
    assert np.all(np.abs(lse - torch.logsumexp(t, 1).numpy()) <= 1e-6 * np.abs(lse))
    c = torch.softmax(t, 1).max(1).values.numpy()
    assert np.all(np.abs(conf - c) <= 1e-6 * c)


def pin_lmhead_one_hot_weights():
    """Weight rows that pick single hidden coordinates: the logits are those
    coordinates, so the reduction of the projection is the reduction of the
    selected columns."""
    rng = np.random.default_rng(27)
    h = rng.standard_normal((4, 6))
    sel = np.array([5, 0, 3, 3, 1])
    w = np.eye(6)[sel]
    got = oracle.lm_head_confidence(h, w)
    ref = oracle.vocab_confidence(h[:, sel])
    for a, b in zip(got, ref):
        assert np.array_equal(a, b)


VOCAB_PINS = [pin_vocab_uniform_row, pin_vocab_single_finite, pin_vocab_two_valued_closed_form,
              pin_vocab_ties_lowest_index, pin_vocab_torch, pin_token_prob_closed_forms, pin_token_prob_torch,
              pin_lmhead_brute_force, pin_lmhead_torch, pin_lmhead_one_hot_weights]


# ---------------------------------------------------------------- update

def golden_cases():
    with open(os.path.join(GOLDEN, "update_hand_examples.json")) as f:
        return json.load(f)["cases"]


def run_case(c):
    tok = np.array([c["tokens"]], dtype=np.int32)
    m = np.array([c["mask"]], dtype=np.uint8)
    am = np.array([c["argmax"]], dtype=np.int32)
    cf = np.array([c["conf"]], dtype=np.float32)
    tp = np.array([c["tok_prob"]], dtype=np.float32) if "tok_prob" in c else None
    return oracle.refine_update(tok, m, am, cf, edit_threshold=c["edit_threshold"],
                                remask_k=c["remask_k"], remask_frac=c["remask_frac"],
                                mask_id=c["mask_id"], prompt_lens=[c["prompt_len"]],
                                seq_lens=[c["seq_len"]], tok_prob=tp)


def pin_update_golden():
    for c in golden_cases():
        nt, nm, ne = run_case(c)
        assert nt[0].tolist() == c["expect_tokens"], c["name"]
        assert nm[0].tolist() == c["expect_mask"], c["name"]
        assert int(ne[0]) == c["expect_n_edits"], c["name"]


def random_update_case(rng, B=6, L=40, V=50, ties=False):
    p = rng.integers(0, L // 2 + 1, B)
    n = np.minimum(L, p + rng.integers(0, L + 1, B))
    tok = rng.integers(0, V, (B, L)).astype(np.int32)
    m = (rng.random((B, L)) < 0.3).astype(np.uint8)
    tok[m == 1] = V
    am = np.where(rng.random((B, L)) < 0.5, tok, rng.integers(0, V, (B, L))).astype(np.int32)
    am[m == 1] = rng.integers(0, V, int(m.sum()))
    if ties:
        cf = rng.choice(np.array([0.0, 0.25, 0.5], dtype=np.float32), (B, L))
    else:
        cf = rng.random((B, L)).astype(np.float32)
    return dict(tokens=tok, mask=m, argmax=am, conf=cf, prompt_lens=p, seq_lens=n, V=V)


def check_update_invariants(case, out, tau, k_fn, mask_id):
    tok, m, am, cf = case["tokens"], case["mask"], case["argmax"], case["conf"]
    nt, nm, ne = out
    B, L = tok.shape
    for b in range(B):
        p, n = int(case["prompt_lens"][b]), int(case["seq_lens"][b])
        r = n - p
        outside = np.r_[0:p, n:L]
        assert np.array_equal(nt[b, outside], tok[b, outside])
        assert np.array_equal(nm[b, outside], m[b, outside])
        resp = np.arange(p, n)
        k = k_fn(r)
        assert int(nm[b, resp].sum()) == min(k, r)
        sel = resp[nm[b, resp] == 1]
        keep = resp[nm[b, resp] == 0]
        assert np.all(nt[b, sel] == mask_id)
        for i in keep:
            assert nt[b, i] in (am[b, i], tok[b, i])
            if m[b, i] == 1:
                assert nt[b, i] == am[b, i]
            elif am[b, i] != nt[b, i]:
                assert cf[b, i] < np.float32(tau)
        if len(sel) and len(keep):
            worst_sel = max((float(cf[b, i]), i) for i in sel)
            best_keep = min((float(cf[b, i]), i) for i in keep)
            assert worst_sel < best_keep
        filled = resp[m[b, resp] == 0]
        edits = sum(1 for i in filled if am[b, i] != tok[b, i] and cf[b, i] >= np.float32(tau))
        assert int(ne[b]) == edits <= r


def pin_update_invariants():
    rng = np.random.default_rng(31)
    for trial in range(30):
        case = random_update_case(rng, ties=trial % 2 == 1)
        tau = float(rng.choice([0.0, 0.25, 0.5, 0.9]))
        k = int(rng.integers(-1, 12))
        frac = 0.3
        out = oracle.refine_update(case["tokens"], case["mask"], case["argmax"], case["conf"],
                                   edit_threshold=tau, remask_k=k, remask_frac=frac,
                                   mask_id=case["V"], prompt_lens=case["prompt_lens"],
                                   seq_lens=case["seq_lens"])
        kf = (lambda r: k) if k >= 0 else (lambda r: int(math.floor(float(np.float32(frac)) * r)))
        check_update_invariants(case, out, tau, kf, case["V"])


def pin_update_rank_count():
    """Selection by an O(r^2) rank count: position i is remasked iff fewer than
    k response positions j have (conf_j, j) < (conf_i, i)."""
    rng = np.random.default_rng(32)
    for trial in range(20):
        case = random_update_case(rng, B=3, L=30, ties=True)
        k = int(rng.integers(0, 20))
        _, nm, _ = oracle.refine_update(case["tokens"], case["mask"], case["argmax"], case["conf"],
                                        edit_threshold=0.5, remask_k=k, remask_frac=0.0,
                                        mask_id=case["V"], prompt_lens=case["prompt_lens"],
                                        seq_lens=case["seq_lens"])
        for b in range(3):
            p, n = int(case["prompt_lens"][b]), int(case["seq_lens"][b])
            c = case["conf"][b]
            for i in range(p, n):
                rank = sum(1 for j in range(p, n) if (c[j] < c[i]) or (c[j] == c[i] and j < i))
                assert (nm[b, i] == 1) == (rank < k)


def pin_update_remask_fraction():
    """k_b = floor(fp32(frac) * r_b): 38 of 384 and 153 of 1536 at frac 0.1."""
    assert oupd.remask_count(-1, 0.1, 384) == 38
    assert oupd.remask_count(-1, 0.1, 1536) == 153
    assert oupd.remask_count(-1, 0.25, 3) == 0
    assert oupd.remask_count(-1, 1.0, 7) == 7
    assert oupd.remask_count(5, 0.9, 3) == 3


def pin_update_result_ranking():
    """Ranking by the resulting token's probability: with tok_prob = conf it is
    the default ranking; otherwise position i is remasked iff fewer than k
    response positions j have (key_j, j) < (key_i, i), key = conf where the
    position ends with its argmax and tok_prob elsewhere (O(r^2) rank count);
    steps 1-2 and the edit count do not depend on the ranking."""
    rng = np.random.default_rng(33)
    for trial in range(20):
        case = random_update_case(rng, B=3, L=30, ties=trial % 2 == 0)
        k = int(rng.integers(0, 20))
        args = dict(edit_threshold=0.5, remask_k=k, remask_frac=0.0, mask_id=case["V"],
                    prompt_lens=case["prompt_lens"], seq_lens=case["seq_lens"])
        base = oracle.refine_update(case["tokens"], case["mask"], case["argmax"], case["conf"], **args)
        same = oracle.refine_update(case["tokens"], case["mask"], case["argmax"], case["conf"],
                                    tok_prob=case["conf"], **args)
        for x, y in zip(base, same):
            assert np.array_equal(x, y)
        tp = rng.choice(np.array([0.0, 0.1, 0.5], dtype=np.float32), (3, 30)) if trial % 2 == 0 else \
            rng.random((3, 30)).astype(np.float32)
        nt, nm, ne = oracle.refine_update(case["tokens"], case["mask"], case["argmax"], case["conf"],
                                          tok_prob=tp, **args)
        assert np.array_equal(ne, base[2])
        unmasked = (nm == 0) & (base[1] == 0)
        assert np.array_equal(nt[unmasked], base[0][unmasked])
        am, cf = case["argmax"], case["conf"]
        for b in range(3):
            p, n = int(case["prompt_lens"][b]), int(case["seq_lens"][b])
            after = [int(am[b, i]) if case["mask"][b, i] or (am[b, i] != case["tokens"][b, i] and
                                                              cf[b, i] >= np.float32(0.5))
                     else int(case["tokens"][b, i]) for i in range(30)]
            key = [float(cf[b, i]) if after[i] == int(am[b, i]) else float(tp[b, i]) for i in range(30)]
            for i in range(p, n):
                rank = sum(1 for j in range(p, n) if (key[j] < key[i]) or (key[j] == key[i] and j < i))
                assert (nm[b, i] == 1) == (rank < k)


UPDATE_PINS = [pin_update_golden, pin_update_invariants, pin_update_rank_count,
               pin_update_remask_fraction, pin_update_result_ranking]


# ---------------------------------------------------------------- multi-pass loop

def loop_golden_cases():
    with open(os.path.join(GOLDEN, "loop_hand_examples.json")) as f:
        return json.load(f)["cases"]


def run_loop_case(c, max_passes=None):
    logits = np.log(np.array(c["probs"], dtype=np.float64))   # [pass, B, L, V]

    def logits_for(tok, msk, t):
        return logits[min(t, len(logits) - 1)].reshape(-1, c["V"])

    return oracle.refine_passes(np.array(c["tokens"]), np.array(c["mask"]), logits_for,
                                max_passes=c["max_passes"] if max_passes is None else max_passes,
                                edit_threshold=c["edit_threshold"], remask_k=c["remask_k"],
                                remask_frac=c["remask_frac"], mask_id=c["mask_id"],
                                prompt_lens=c["prompt_lens"], seq_lens=c["seq_lens"])


def pin_loop_golden():
    """Hand-worked passes (tests/golden/loop_hand_examples.json): a batch-level
    stop after the first pass without a confident edit, and pass budgets."""
    for c in loop_golden_cases():
        r = run_loop_case(c)
        assert r["passes"] == c["expect_passes"], c["name"]
        assert r["tokens"].tolist() == c["expect_tokens"], c["name"]
        assert r["mask"].tolist() == c["expect_mask"], c["name"]
        assert r["n_edits"].tolist() == c["expect_n_edits"], c["name"]


def _loop_state(rng, B=3, L=24, V=16):
    p = rng.integers(0, L // 3, B)
    n = np.minimum(L, p + rng.integers(1, L, B))
    tok = rng.integers(0, V, (B, L)).astype(np.int32)
    msk = (rng.random((B, L)) < 0.3).astype(np.uint8)
    tok[msk == 1] = V
    return tok, msk, p, n


def pin_loop_unreachable_threshold():
    """A threshold above 1 admits no edit (a confidence is at most 1): one
    pass, whatever the budget, equal to one refine_update."""
    rng = np.random.default_rng(41)
    for trial in range(10):
        tok, msk, p, n = _loop_state(rng)
        x = rng.standard_normal((tok.size, 16)) * 3
        for budget in (1, 2, 7):
            r = oracle.refine_passes(tok, msk, lambda t, m, i: x, max_passes=budget, edit_threshold=1.5,
                                     remask_k=2, remask_frac=0.0, mask_id=16, prompt_lens=p, seq_lens=n)
            assert r["passes"] == 1 and not r["n_edits"].any()


def pin_loop_commits_only_stop():
    """Masked positions committed but every filled prediction equal to its
    token: commits are not edits, so the first pass is the last."""
    rng = np.random.default_rng(42)
    tok, msk, p, n = _loop_state(rng)
    V = 16
    pred = np.where(msk == 1, rng.integers(0, V, tok.shape), tok)
    x = np.full((tok.size, V), -5.0)
    x[np.arange(tok.size), pred.reshape(-1)] = 5.0
    r = oracle.refine_passes(tok, msk, lambda t, m, i: x, max_passes=9, edit_threshold=0.5, remask_k=0,
                             remask_frac=0.0, mask_id=V, prompt_lens=p, seq_lens=n)
    assert r["passes"] == 1
    for b in range(tok.shape[0]):
        resp = np.arange(p[b], n[b])
        assert np.array_equal(r["tokens"][b, resp], pred[b, resp])     # every masked position committed
        assert not r["mask"][b, resp].any()


def pin_loop_budget():
    """Predictions that flip every pass between two tokens with probability
    ~0.9 edit every filled response position every pass: the loop runs exactly
    max_passes passes, and the final tokens follow the parity of the count."""
    B, L, V = 2, 10, 8
    p, n = np.array([3, 0]), np.array([10, 7])
    tok = np.zeros((B, L), dtype=np.int32)
    msk = np.zeros((B, L), dtype=np.uint8)

    def logits_for(t, m, i):
        x = np.full((B * L, V), -3.0)
        x[:, 1 if i % 2 == 0 else 0] = 3.0   # pass 0 predicts 1, pass 1 predicts 0, ...
        return x

    for budget in range(1, 6):
        r = oracle.refine_passes(tok, msk, logits_for, max_passes=budget, edit_threshold=0.8, remask_k=0,
                                 remask_frac=0.0, mask_id=V, prompt_lens=p, seq_lens=n)
        assert r["passes"] == budget
        want = 1 if budget % 2 == 1 else 0
        for b in range(B):
            assert np.all(r["tokens"][b, p[b]:n[b]] == want)
            assert np.all(r["tokens"][b, :p[b]] == 0) and np.all(r["tokens"][b, n[b]:] == 0)
        assert np.all(r["n_edits"] == n - p)


LOOP_PINS = [pin_loop_golden, pin_loop_unreachable_threshold, pin_loop_commits_only_stop, pin_loop_budget]

ALL_PINS = ATTN_PINS + VOCAB_PINS + UPDATE_PINS + LOOP_PINS
