"""Remask ranking by the probability of each position's resulting token on the
GPU: dlm_token_prob against the oracle's token_prob (relative tolerance of the
other vocabulary outputs), and dlm_refine_update_ranked against the oracle's
refine_update(tok_prob=...) bit for bit, on the same host-generated inputs."""
import numpy as np
import pytest
import torch

import oracle
import oracle_pins as P
from gpu_util import CONF_RTOL, dev, host_logit_rows
from paper_2608_02625_gb300 import workloads

pytestmark = pytest.mark.gpu


def gpu_token_prob(x: torch.Tensor, tokens: np.ndarray, lse: np.ndarray):
    from paper_2608_02625_gb300 import binding as Bn
    d = x.device
    t = torch.from_numpy(np.ascontiguousarray(tokens, dtype=np.int32)).to(d)
    ls = torch.from_numpy(np.ascontiguousarray(lse, dtype=np.float32)).to(d)
    pr = torch.full(t.shape, -1.0, dtype=torch.float32, device=d)
    Bn.dlm_token_prob(x, t, ls, pr)
    torch.cuda.synchronize()
    return pr.cpu().numpy()


def check_prob(gpu, ref, where):
    gpu = gpu.astype(np.float64).reshape(-1)
    ref = ref.astype(np.float64).reshape(-1)
    bad = np.abs(gpu - ref) > CONF_RTOL * ref + 1e-37
    assert not bad.any(), f"{where}: token_prob differs at {np.argwhere(bad)[:8].ravel()} gpu {gpu[bad][:4]} ref {ref[bad][:4]}"


@pytest.mark.parametrize("dtype,N,V,layout", [("f32", 37, 1000, "2d"), ("bf16", 64, 4099, "2d"),
                                              ("bf16", 40, 2048, "strided"), ("f32", 30, 7, "3d"),
                                              ("bf16", 16, 151552, "2d")])
def test_token_prob_vs_oracle(dtype, N, V, layout):
    rng = np.random.default_rng(N + V)
    x = (rng.standard_normal((N, V)) * 3.0).astype(np.float32)
    x[rng.random((N, V)) < 0.01] = -np.inf
    if dtype == "bf16":
        x = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    tok = rng.integers(0, V, N).astype(np.int32)
    tok[0] = V          # outside [0, V): probability 0
    tok[1] = -1
    am, _, lse = oracle.vocab_confidence(x)
    tok[2] = am[2]      # the argmax: the confidence
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    if layout == "strided":
        full = torch.from_numpy(np.pad(x, ((0, 0), (0, 8)))).to(tdt).to(dev())
        xt = full[:, :V]
    else:
        xt = torch.from_numpy(x).to(tdt).to(dev())
        if layout == "3d":
            xt = xt.reshape(2, N // 2, V)
    gpu = gpu_token_prob(xt, tok, lse)
    ref = oracle.token_prob(x, tok, lse)
    assert gpu[0] == 0.0 and gpu[1] == 0.0
    check_prob(gpu, ref, f"{dtype} N={N} V={V} {layout}")


def run_ranked(tok, msk, am, cf, tp, *, tau, k, frac, mask_id, prompt, seqlen, inplace=False):
    from paper_2608_02625_gb300 import binding as Bn
    d = dev()
    g = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a, dtype=dt)).to(d)
    t_tok, t_msk = g(tok, np.int32), g(msk, np.uint8)
    B = tok.shape[0]
    ne = torch.full((B,), -1, dtype=torch.int32, device=d)
    nt, nm = (t_tok, t_msk) if inplace else (torch.full_like(t_tok, -7), torch.full_like(t_msk, 7))
    params = Bn.RefineParams(tau, k, frac, mask_id, g(prompt, np.int32), g(seqlen, np.int32))
    Bn.dlm_refine_update_ranked(t_tok, t_msk, g(am, np.int32), g(cf, np.float32), g(tp, np.float32), params,
                                nt, nm, ne)
    torch.cuda.synchronize()
    assert Bn.device_error(clear=True) == 0
    return nt.cpu().numpy(), nm.cpu().numpy(), ne.cpu().numpy()


def same(gpu, ref, where):
    for name, g, r in zip(("tokens", "mask", "n_edits"), gpu, ref):
        assert np.array_equal(g, r), f"{where}: {name} differs at {np.argwhere(g != r)[:8].tolist()}"


@pytest.mark.parametrize("case", P.golden_cases(), ids=lambda c: c["name"])
def test_golden_cases(case):
    """Every hand-worked case; without a tok_prob of its own a case ranks by
    tok_prob = conf, which must reproduce its default-ranking result."""
    tok = np.array([case["tokens"]]); msk = np.array([case["mask"]])
    am = np.array([case["argmax"]]); cf = np.array([case["conf"]], dtype=np.float32)
    tp = np.array([case.get("tok_prob", case["conf"])], dtype=np.float32)
    gpu = run_ranked(tok, msk, am, cf, tp, tau=case["edit_threshold"], k=case["remask_k"],
                     frac=case["remask_frac"], mask_id=case["mask_id"], prompt=[case["prompt_len"]],
                     seqlen=[case["seq_len"]])
    assert gpu[0][0].tolist() == case["expect_tokens"]
    assert gpu[1][0].tolist() == case["expect_mask"]
    assert int(gpu[2][0]) == case["expect_n_edits"]


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("L", [1, 37, 512, 3000])
def test_random_vs_oracle(seed, L):
    rng = np.random.default_rng(7000 + 1000 * L + seed)
    B = 5
    case = P.random_update_case(rng, B=B, L=L, V=40, ties=seed % 2 == 0)
    if seed % 3 == 0:
        tp = rng.choice(np.array([0.0, 0.3, 0.5], dtype=np.float32), (B, L))   # ties across both key kinds
        case["conf"] = rng.choice(np.array([0.3, 0.5, 0.9], dtype=np.float32), (B, L))
    else:
        tp = (rng.random((B, L)) * case["conf"]).astype(np.float32)
    tau = float(rng.choice([0.0, 0.3, 0.5, 1.0]))
    k = int(rng.integers(-1, L + 2))
    frac = float(rng.random())
    ref = oracle.refine_update(case["tokens"], case["mask"], case["argmax"], case["conf"], edit_threshold=tau,
                               remask_k=k, remask_frac=frac, mask_id=case["V"], prompt_lens=case["prompt_lens"],
                               seq_lens=case["seq_lens"], tok_prob=tp)
    for inplace in (False, True):
        gpu = run_ranked(case["tokens"], case["mask"], case["argmax"], case["conf"], tp, tau=tau, k=k, frac=frac,
                         mask_id=case["V"], prompt=case["prompt_lens"], seqlen=case["seq_lens"], inplace=inplace)
        same(gpu, ref, f"L={L} seed={seed} inplace={inplace}")


@pytest.mark.parametrize("name", ["c3_batch32_512", "c4_long_2048", "c5_heavy_4step"])
def test_full_size_state(name):
    """The workload's batch and lengths in the bench's launch configuration,
    with host-generated predictions, confidences and kept-token probabilities."""
    w = workloads.get(name)
    tok, msk = w.initial_state()
    rng = np.random.default_rng(11)
    am = rng.integers(0, w.V, (w.B, w.L)).astype(np.int32)
    am = np.where(rng.random((w.B, w.L)) < 0.4, np.where(msk == 1, am, tok), am).astype(np.int32)
    cf = rng.random((w.B, w.L)).astype(np.float32)
    tp = (rng.random((w.B, w.L)) * cf).astype(np.float32)
    p, n = w.prompt_lens(), w.seq_lens()
    tau = w.edit_threshold[0]
    ref = oracle.refine_update(tok, msk, am, cf, edit_threshold=tau, remask_k=w.remask_k, remask_frac=w.remask_frac,
                               mask_id=w.mask_id, prompt_lens=p, seq_lens=n, tok_prob=tp)
    gpu = run_ranked(tok, msk, am, cf, tp, tau=tau, k=w.remask_k, frac=w.remask_frac, mask_id=w.mask_id,
                     prompt=p, seqlen=n)
    same(gpu, ref, name)


def test_workload_rows_chain():
    """c3 rows at full size: GPU vocabulary reduction, then dlm_token_prob of the
    current tokens from the GPU's lse, against the oracle's token_prob from the
    oracle's own lse on the host-regenerated rows."""
    from paper_2608_02625_gb300 import binding as Bn
    from paper_2608_02625_gb300 import synth_gpu
    w = workloads.get("c3_batch32_512")
    d = dev()
    tok, msk = w.initial_state()
    x = synth_gpu.logits(w, 0, d, torch.from_numpy(tok.reshape(-1)).to(d), torch.from_numpy(msk.reshape(-1)).to(d))
    am = torch.empty(w.N, dtype=torch.int32, device=d)
    cf = torch.empty(w.N, dtype=torch.float32, device=d)
    ls = torch.empty(w.N, dtype=torch.float32, device=d)
    pr = torch.empty(w.N, dtype=torch.float32, device=d)
    Bn.dlm_vocab_confidence(x, am, cf, ls)
    Bn.dlm_token_prob(x, torch.from_numpy(tok.reshape(-1)).to(d), ls, pr)
    torch.cuda.synchronize()
    rng = np.random.default_rng(12)
    rows = np.unique(np.concatenate([[0, w.N - 1], rng.integers(0, w.N, 40)]))
    xr = host_logit_rows(w, 0, rows, tok.reshape(-1)[rows], msk.reshape(-1)[rows])
    _, _, lse_ref = oracle.vocab_confidence(xr)
    ref = oracle.token_prob(xr, tok.reshape(-1)[rows], lse_ref)
    # the GPU used its own lse (within 2e-5 relative of the oracle's): allow for it
    gpu = pr.cpu().numpy()[rows].astype(np.float64)
    lse_err = np.abs(ls.cpu().numpy()[rows].astype(np.float64) - lse_ref) + 1e-7
    assert np.all(np.abs(gpu - ref) <= (CONF_RTOL + 2 * lse_err) * ref + 1e-37)


@pytest.mark.parametrize("r", [2047, 2048, 2049])
def test_key_cache_boundary(r):
    """The ranked update at the capacity of the shared-memory key cache (2048
    response positions) and one past it: keys of both kinds, with ties."""
    rng = np.random.default_rng(5000 + r)
    L = r + 40
    case = P.random_update_case(rng, B=3, L=L, V=40, ties=True)
    case["prompt_lens"] = np.array([0, 17, 40])
    case["seq_lens"] = case["prompt_lens"] + r
    tp = rng.choice(np.array([0.0, 0.25, 0.5], dtype=np.float32), (3, L))
    ref = oracle.refine_update(case["tokens"], case["mask"], case["argmax"], case["conf"], edit_threshold=0.25,
                               remask_k=-1, remask_frac=0.1, mask_id=case["V"], prompt_lens=case["prompt_lens"],
                               seq_lens=case["seq_lens"], tok_prob=tp)
    gpu = run_ranked(case["tokens"], case["mask"], case["argmax"], case["conf"], tp, tau=0.25, k=-1, frac=0.1,
                     mask_id=case["V"], prompt=case["prompt_lens"], seqlen=case["seq_lens"])
    same(gpu, ref, f"r={r}")

