"""Steps A2 + A3 fused in one launch (dlm_refine_step) on the GPU.

Vocabulary outputs: against the oracle on host-regenerated logits (argmax
exact, conf / lse within the tolerances of the separate call) and against the
separate dlm_vocab_confidence call. Update outputs: against the oracle's update
computed from the oracle's own argmax / conf under the decision-margin protocol
(identical wherever no conf lies within tolerance of a decision boundary), and
bit for bit against dlm_refine_update run on the fused call's argmax / conf
(the update is integer work and exact fp32 comparisons, so equal inputs give
equal outputs). Each case runs twice on one workspace, which must be zero again
after every call."""
import numpy as np
import pytest
import torch

import oracle
import oracle_pins as P
from gpu_util import CONF_RTOL, LSE_RTOL, ambiguous_for, check_update_margin, check_vocab, dev, host_logit_rows
from paper_2608_02625_gb300 import workloads

pytestmark = pytest.mark.gpu


def new_outputs(B, L, tok, msk, inplace):
    d = dev()
    am = torch.full((B, L), -5, dtype=torch.int32, device=d)
    cf = torch.full((B, L), -1.0, dtype=torch.float32, device=d)
    ls = torch.full((B, L), -1.0, dtype=torch.float32, device=d)
    ne = torch.full((B,), -1, dtype=torch.int32, device=d)
    if inplace:
        nt, nm = tok.clone(), msk.clone()
    else:
        nt, nm = torch.full_like(tok, -7), torch.full_like(msk, 7)
    return am, cf, ls, nt, nm, ne


def run_fused(logits, tok, msk, params, ws, inplace=False):
    from paper_2608_02625_gb300 import binding as Bn
    B, L = tok.shape
    am, cf, ls, nt, nm, ne = new_outputs(B, L, tok, msk, inplace)
    src_tok, src_msk = (nt, nm) if inplace else (tok, msk)
    Bn.dlm_refine_step(logits, src_tok, src_msk, params, am, cf, ls, nt, nm, ne, ws)
    torch.cuda.synchronize()
    assert Bn.device_error(clear=True) == 0
    assert int(ws.abs().sum()) == 0, "workspace not left zero"
    return [t.cpu().numpy() for t in (am, cf, ls, nt, nm, ne)]


def run_separate(logits, tok, msk, params):
    from paper_2608_02625_gb300 import binding as Bn
    B, L = tok.shape
    am, cf, ls, nt, nm, ne = new_outputs(B, L, tok, msk, False)
    Bn.dlm_vocab_confidence(logits, am.view(-1), cf.view(-1), ls.view(-1))
    Bn.dlm_refine_update(tok, msk, am, cf, params, nt, nm, ne)
    torch.cuda.synchronize()
    assert Bn.device_error(clear=True) == 0
    return [t.cpu().numpy() for t in (am, cf, ls, nt, nm, ne)]


def oracle_update_parity(fz, tok, msk, pn, ref_vocab, where):
    """Oracle vocabulary outputs -> oracle update; compare with the fused call's."""
    shp = tok.shape
    am_ref, cf_ref = ref_vocab[0].reshape(shp), ref_vocab[1].reshape(shp)
    ref = oracle.refine_update(tok, msk, am_ref, cf_ref, **pn)
    amb = ambiguous_for(pn["edit_threshold"], pn["remask_k"], pn["remask_frac"], cf_ref, (tok, msk), am_ref,
                        pn["prompt_lens"], pn["seq_lens"])
    check_update_margin((fz[3], fz[4], fz[5]), ref, amb, where)


def gpu_update_from(fz, tok, msk, params):
    """dlm_refine_update on the fused call's own argmax / conf."""
    from paper_2608_02625_gb300 import binding as Bn
    d = dev()
    B = tok.shape[0]
    out = Bn.dlm_refine_update(tok, msk, torch.from_numpy(fz[0]).to(d), torch.from_numpy(fz[1]).to(d), params,
                               torch.empty_like(tok), torch.empty_like(msk),
                               torch.empty(B, dtype=torch.int32, device=d))
    torch.cuda.synchronize()
    return [t.cpu().numpy() for t in out]


def assert_equal_outputs(a, b, names, where):
    for n, x, y in zip(names, a, b):
        assert np.array_equal(x, y), f"{where}: {n} differs at {np.argwhere(x != y)[:8].tolist()}"


def check_vs_separate(fz, sep, where):
    assert np.array_equal(fz[0], sep[0]), f"{where}: argmax differs from the separate call"
    rc = np.abs(fz[1].astype(np.float64) - sep[1]) / np.maximum(sep[1], 1e-30)
    rl = np.abs(fz[2].astype(np.float64) - sep[2]) / np.maximum(1.0, np.abs(sep[2]))
    assert rc.max() <= 2 * CONF_RTOL and rl.max() <= 2 * LSE_RTOL, f"{where}: conf/lse vs separate call"


@pytest.mark.parametrize("name", workloads.ORDER)
def test_workload_full_size(name):
    """Every workload at full size (step 0), in the launch configuration a
    fused step uses; the oracle checks one sampled sequence."""
    from paper_2608_02625_gb300 import binding as Bn
    from paper_2608_02625_gb300 import synth_gpu
    w = workloads.get(name)
    d = dev()
    tok_np, msk_np = w.initial_state()
    tok, msk = torch.from_numpy(tok_np).to(d), torch.from_numpy(msk_np).to(d)
    logits = synth_gpu.logits(w, 0, d, tok, msk)
    prompt = torch.from_numpy(w.prompt_lens()).to(d)
    seqlen = torch.from_numpy(w.seq_lens()).to(d)
    params = Bn.RefineParams(w.edit_threshold[0], w.remask_k, w.remask_frac, w.mask_id, prompt, seqlen)
    ws = torch.zeros(Bn.dlm_refine_step_workspace_bytes(w.B) // 4, dtype=torch.int32, device=d)
    fz = run_fused(logits, tok, msk, params, ws)
    again = run_fused(logits, tok, msk, params, ws)
    names = ("argmax", "conf", "lse", "tokens", "mask", "n_edits")
    assert_equal_outputs(again, fz, names, f"{name} second call")
    sep = run_separate(logits, tok, msk, params)
    check_vs_separate(fz, sep, name)
    # the update of the fused call equals dlm_refine_update on the fused call's argmax / conf
    assert_equal_outputs(fz[3:], gpu_update_from(fz, tok, msk, params), names[3:], f"{name} vs dlm_refine_update")
    # oracle on one sampled sequence: vocabulary, then the update from the oracle's own outputs
    b = w.B // 2
    rows = np.arange(b * w.L, (b + 1) * w.L)
    x = host_logit_rows(w, 0, rows, tok_np[b], msk_np[b])   # the state of the sampled rows
    ref_v = oracle.vocab_confidence(x)
    check_vocab(fz[0][b], fz[1][b], fz[2][b], *ref_v, where=name)
    pn = dict(edit_threshold=w.edit_threshold[0], remask_k=w.remask_k, remask_frac=w.remask_frac,
              mask_id=w.mask_id, prompt_lens=w.prompt_lens()[b:b + 1], seq_lens=w.seq_lens()[b:b + 1])
    sub = [a[b:b + 1] for a in fz]
    oracle_update_parity(sub, tok_np[b:b + 1], msk_np[b:b + 1], pn, ref_v, f"{name} oracle update")


def random_logits(rng, N, V, dtype, ties):
    x = rng.standard_normal((N, V)).astype(np.float32) * 2.0
    if ties:   # repeat each row's maximum at a later index
        j = np.argmax(x, axis=1)
        later = np.minimum(V - 1, j + 1 + rng.integers(0, max(1, V // 2), N))
        x[np.arange(N), later] = x[np.arange(N), j]
    if V > 3:
        x[rng.random((N, V)) < 0.01] = -np.inf
    if dtype == "bf16":
        x = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    return x


@pytest.mark.parametrize("seed", range(8))
@pytest.mark.parametrize("L,V,dtype", [(1, 7, "f32"), (37, 1000, "bf16"), (37, 4099, "f32"), (300, 2049, "bf16"),
                                       (129, 1, "bf16")])
def test_random_ragged(seed, L, V, dtype):
    """Ragged lengths (empty sequences and full ones), odd V (scalar loads), ties,
    -inf entries, both remask modes, in-place update, 3-D and row-strided logits."""
    from paper_2608_02625_gb300 import binding as Bn
    rng = np.random.default_rng(97 * seed + L + V)
    d = dev()
    B = int(rng.integers(1, 10))
    case = P.random_update_case(rng, B=B, L=L, V=max(V, 2), ties=seed % 2 == 0)
    case["seq_lens"][0] = 0 if seed % 4 == 1 else case["seq_lens"][0]
    case["seq_lens"][-1] = L if seed % 4 == 2 else case["seq_lens"][-1]
    case["prompt_lens"] = np.minimum(case["prompt_lens"], case["seq_lens"])
    x = random_logits(rng, B * L, V, dtype, ties=seed % 2 == 1)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    pad = 8 if seed % 3 == 0 else 0
    full = torch.from_numpy(np.pad(x, ((0, 0), (0, pad)))).to(tdt).to(d)
    logits = full[:, :V]
    if seed % 3 == 1:
        logits = logits.reshape(B, L, V)
    tau = float(rng.choice([0.0, 0.3, 0.9, 1.0]))
    k = int(rng.integers(-1, L + 2)) if seed % 2 else -1
    frac = float(rng.random())
    tok = torch.from_numpy(case["tokens"]).to(d)
    msk = torch.from_numpy(case["mask"]).to(d)
    prompt = torch.from_numpy(case["prompt_lens"].astype(np.int32)).to(d)
    seqlen = torch.from_numpy(case["seq_lens"].astype(np.int32)).to(d)
    params = Bn.RefineParams(tau, k, frac, case["V"], prompt, seqlen)
    ws = torch.zeros(B, dtype=torch.int32, device=d)
    inplace = seed % 4 == 3
    fz = run_fused(logits, tok, msk, params, ws, inplace=inplace)
    again = run_fused(logits, tok, msk, params, ws, inplace=inplace)
    names = ("argmax", "conf", "lse", "tokens", "mask", "n_edits")
    assert_equal_outputs(again, fz, names, "second call")
    ref_v = oracle.vocab_confidence(x)
    check_vocab(fz[0].reshape(-1), fz[1].reshape(-1), fz[2].reshape(-1), *ref_v, where=f"L={L} V={V}")
    pn = dict(edit_threshold=tau, remask_k=k, remask_frac=frac, mask_id=case["V"],
              prompt_lens=case["prompt_lens"], seq_lens=case["seq_lens"])
    oracle_update_parity(fz, case["tokens"], case["mask"], pn, ref_v, f"L={L} V={V} oracle update")
    assert_equal_outputs(fz[3:], gpu_update_from(fz, tok, msk, params), names[3:], f"L={L} V={V} vs update call")
    check_vs_separate(fz, run_separate(logits, tok, msk, params), f"L={L} V={V}")


def test_empty_batch_needs_no_workspace():
    from paper_2608_02625_gb300 import binding as Bn
    d = dev()
    z = lambda *s, dt=torch.int32: torch.empty(s, dtype=dt, device=d)
    params = Bn.RefineParams(0.5, 1, 0.0, 9, z(0), z(0))
    Bn.dlm_refine_step(z(0, 16, dt=torch.bfloat16), z(0, 4), z(0, 4, dt=torch.uint8), params,
                       z(0, 4), z(0, 4, dt=torch.float32), z(0, 4, dt=torch.float32), z(0, 4),
                       z(0, 4, dt=torch.uint8), z(0), z(0))
    torch.cuda.synchronize()


@pytest.mark.parametrize("r", [1023, 1024, 1025])
def test_key_cache_boundary(r):
    """The fused step's update at the capacity of its shared-memory key cache
    (four keys per thread of the 256-thread vocabulary block: 1024 response
    positions) and one past it: equal to the separate update on the same
    predictions, and to the oracle under the decision-margin protocol."""
    from paper_2608_02625_gb300 import binding as Bn
    rng = np.random.default_rng(9000 + r)
    d = dev()
    B, L, V = 2, r + 30, 64
    case = P.random_update_case(rng, B=B, L=L, V=V, ties=False)
    case["prompt_lens"] = np.array([0, 30])
    case["seq_lens"] = case["prompt_lens"] + r
    x = random_logits(rng, B * L, V, "bf16", ties=True)
    logits = torch.from_numpy(x).to(torch.bfloat16).to(d)
    tok = torch.from_numpy(case["tokens"]).to(d)
    msk = torch.from_numpy(case["mask"]).to(d)
    prompt = torch.from_numpy(case["prompt_lens"].astype(np.int32)).to(d)
    seqlen = torch.from_numpy(case["seq_lens"].astype(np.int32)).to(d)
    params = Bn.RefineParams(0.5, -1, 0.1, case["V"], prompt, seqlen)
    ws = torch.zeros(B, dtype=torch.int32, device=d)
    fz = run_fused(logits, tok, msk, params, ws)
    names = ("tokens", "mask", "n_edits")
    assert_equal_outputs(fz[3:], gpu_update_from(fz, tok, msk, params), names, f"r={r} vs update call")
    ref_v = oracle.vocab_confidence(x)
    pn = dict(edit_threshold=0.5, remask_k=-1, remask_frac=0.1, mask_id=case["V"],
              prompt_lens=case["prompt_lens"], seq_lens=case["seq_lens"])
    oracle_update_parity(fz, case["tokens"], case["mask"], pn, ref_v, f"r={r} oracle update")

