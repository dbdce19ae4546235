"""Step A3 (refine update) on the GPU against the oracle: bit-exact."""
import numpy as np
import pytest
import torch

import oracle
import oracle_pins as P
from gpu_util import dev
from paper_2608_02625_gb300 import workloads

pytestmark = pytest.mark.gpu


def run_gpu(tok, msk, am, cf, *, tau, k, frac, mask_id, prompt, seqlen, inplace=False):
    from paper_2608_02625_gb300 import binding as Bn
    d = dev()
    t_tok = torch.from_numpy(np.ascontiguousarray(tok, dtype=np.int32)).to(d)
    t_msk = torch.from_numpy(np.ascontiguousarray(msk, dtype=np.uint8)).to(d)
    t_am = torch.from_numpy(np.ascontiguousarray(am, dtype=np.int32)).to(d)
    t_cf = torch.from_numpy(np.ascontiguousarray(cf, dtype=np.float32)).to(d)
    B = tok.shape[0]
    ne = torch.full((B,), -1, dtype=torch.int32, device=d)
    if inplace:
        nt, nm = t_tok, t_msk
    else:
        nt = torch.full_like(t_tok, -7)
        nm = torch.full_like(t_msk, 7)
    params = Bn.RefineParams(tau, k, frac, mask_id, torch.tensor(np.asarray(prompt, dtype=np.int32), device=d),
                             torch.tensor(np.asarray(seqlen, dtype=np.int32), device=d))
    Bn.dlm_refine_update(t_tok, t_msk, t_am, t_cf, params, nt, nm, ne)
    torch.cuda.synchronize()
    return nt.cpu().numpy(), nm.cpu().numpy(), ne.cpu().numpy()


def assert_same(gpu, ref, where=""):
    for name, g, r in zip(("tokens", "mask", "n_edits"), gpu, ref):
        assert np.array_equal(g, r), f"{where}: {name} differs at {np.argwhere(g != r)[:8].tolist()}"


@pytest.mark.parametrize("case", [c for c in P.golden_cases() if "tok_prob" not in c], ids=lambda c: c["name"])
def test_golden_cases(case):
    """The default-ranking cases (cases with a tok_prob are for dlm_refine_update_ranked)."""
    tok = np.array([case["tokens"]]); msk = np.array([case["mask"]])
    am = np.array([case["argmax"]]); cf = np.array([case["conf"]], dtype=np.float32)
    gpu = run_gpu(tok, msk, am, cf, tau=case["edit_threshold"], k=case["remask_k"], frac=case["remask_frac"],
                  mask_id=case["mask_id"], prompt=[case["prompt_len"]], seqlen=[case["seq_len"]])
    assert gpu[0][0].tolist() == case["expect_tokens"]
    assert gpu[1][0].tolist() == case["expect_mask"]
    assert int(gpu[2][0]) == case["expect_n_edits"]


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("L", [1, 37, 512, 3000])
def test_random_vs_oracle(seed, L):
    rng = np.random.default_rng(1000 * L + seed)
    B = 5
    case = P.random_update_case(rng, B=B, L=L, V=40, ties=seed % 2 == 0)
    if seed % 3 == 0:   # near-ties: neighbouring fp32 values
        base = np.float32(0.3)
        case["conf"] = (base + rng.integers(0, 4, (B, L)) * np.finfo(np.float32).eps * base).astype(np.float32)
    tau = float(rng.choice([0.0, 0.3, 0.5, 1.0]))
    k = int(rng.integers(-1, L + 2))
    frac = float(rng.random())
    ref = oracle.refine_update(case["tokens"], case["mask"], case["argmax"], case["conf"], edit_threshold=tau,
                               remask_k=k, remask_frac=frac, mask_id=case["V"], prompt_lens=case["prompt_lens"],
                               seq_lens=case["seq_lens"])
    for inplace in (False, True):
        gpu = run_gpu(case["tokens"], case["mask"], case["argmax"], case["conf"], tau=tau, k=k, frac=frac,
                      mask_id=case["V"], prompt=case["prompt_lens"], seqlen=case["seq_lens"], inplace=inplace)
        assert_same(gpu, ref, f"L={L} seed={seed} inplace={inplace}")


@pytest.mark.parametrize("name", workloads.ORDER)
def test_full_size_workload_state(name):
    """Every workload's batch and lengths, in the launch configuration of the bench,
    with host-generated predictions and confidences (ties and near-ties included)."""
    w = workloads.get(name)
    tok, msk = w.initial_state()
    rng = np.random.default_rng(7)
    am = rng.integers(0, w.V, (w.B, w.L)).astype(np.int32)
    am = np.where(rng.random((w.B, w.L)) < 0.3, np.where(msk == 1, am, tok), am).astype(np.int32)
    cf = rng.choice(np.array([0.1, 0.5, 0.8, 0.95], dtype=np.float32), (w.B, w.L))
    cf = np.where(rng.random((w.B, w.L)) < 0.5, rng.random((w.B, w.L)).astype(np.float32), cf).astype(np.float32)
    p, n = w.prompt_lens(), w.seq_lens()
    for s in range(w.steps):
        tau = w.edit_threshold[s]
        ref = oracle.refine_update(tok, msk, am, cf, edit_threshold=tau, remask_k=w.remask_k,
                                   remask_frac=w.remask_frac, mask_id=w.mask_id, prompt_lens=p, seq_lens=n)
        gpu = run_gpu(tok, msk, am, cf, tau=tau, k=w.remask_k, frac=w.remask_frac, mask_id=w.mask_id,
                      prompt=p, seqlen=n)
        assert_same(gpu, ref, f"{name} step {s}")
        tok, msk = ref[0], ref[1]


def test_length_clamp_sets_error_word():
    from paper_2608_02625_gb300 import binding as Bn
    Bn.device_error(clear=True)
    tok = np.arange(8, dtype=np.int32)[None]
    msk = np.zeros((1, 8), np.uint8)
    cf = np.linspace(0, 1, 8, dtype=np.float32)[None]
    gpu = run_gpu(tok, msk, tok, cf, tau=0.5, k=2, frac=0.0, mask_id=99, prompt=[3], seqlen=[50])
    ref = oracle.refine_update(tok, msk, tok, cf, edit_threshold=0.5, remask_k=2, remask_frac=0.0, mask_id=99,
                               prompt_lens=[3], seq_lens=[50])
    assert_same(gpu, ref, "clamped")
    assert Bn.device_error(clear=True) & 0x1
    assert Bn.device_error(clear=True) == 0


@pytest.mark.parametrize("lo,hi", [(0, 64), (64, 128), (300, 512), (100, 101)])
def test_editable_window(lo, hi):
    """Refining one window [p_b + lo, p_b + hi) of each response: the window's
    bounds go in prompt_lens / seq_lens. Inside it the rules apply as to a
    response (against the oracle with the same bounds); everything outside,
    masked positions included, is unchanged."""
    rng = np.random.default_rng(lo * 7 + hi)
    B, L, V = 4, 640, 1000
    case = P.random_update_case(rng, B=B, L=L, V=V)
    p = np.array([256, 128, 0, 600]); n = np.array([640, 500, 640, 640])
    wlo = np.minimum(n, p + lo); whi = np.minimum(n, p + hi)
    ref = oracle.refine_update(case["tokens"], case["mask"], case["argmax"], case["conf"], edit_threshold=0.5,
                               remask_k=3, remask_frac=0.0, mask_id=V, prompt_lens=wlo, seq_lens=whi)
    gpu = run_gpu(case["tokens"], case["mask"], case["argmax"], case["conf"], tau=0.5, k=3, frac=0.0, mask_id=V,
                  prompt=wlo, seqlen=whi)
    assert_same(gpu, ref, f"window [{lo}, {hi})")
    for b in range(B):
        out = np.r_[0:wlo[b], whi[b]:L]
        assert np.array_equal(gpu[0][b, out], case["tokens"][b, out])
        assert np.array_equal(gpu[1][b, out], case["mask"][b, out])


@pytest.mark.parametrize("r", [2047, 2048, 2049])
def test_key_cache_boundary(r):
    """Responses at the capacity of the shared-memory key cache (four keys per
    thread of the 512-thread update: 2048 positions) and one past it, heavy
    ties included, against the oracle."""
    rng = np.random.default_rng(r)
    L = r + 40
    case = P.random_update_case(rng, B=3, L=L, V=40, ties=True)
    case["prompt_lens"] = np.array([0, 17, 40])
    case["seq_lens"] = case["prompt_lens"] + r
    for k, frac in ((-1, 0.1), (r // 3, 0.0), (1, 0.0)):
        ref = oracle.refine_update(case["tokens"], case["mask"], case["argmax"], case["conf"], edit_threshold=0.25,
                                   remask_k=k, remask_frac=frac, mask_id=case["V"], prompt_lens=case["prompt_lens"],
                                   seq_lens=case["seq_lens"])
        gpu = run_gpu(case["tokens"], case["mask"], case["argmax"], case["conf"], tau=0.25, k=k, frac=frac,
                      mask_id=case["V"], prompt=case["prompt_lens"], seqlen=case["seq_lens"])
        assert_same(gpu, ref, f"r={r} k={k}")

