"""Block-causal and block-local attention (dlm_attn_masked) on the GPU against
the oracle's mask variants, with the tolerances of the unmasked attention
tests: bf16 max abs error 2e-2 and the output-scaled bounds, fp32 1e-5;
rows i >= n_b exactly zero. The full mode through the same entry point must
equal dlm_bidir_attn bit for bit."""
import math

import numpy as np
import pytest
import torch

import oracle
from gpu_util import ATTN_TOL_BF16, ATTN_TOL_F32, dev, host_qkv_seq
from paper_2608_02625_gb300 import workloads
from test_gpu_attn import compare, rand_qkv

pytestmark = pytest.mark.gpu

CAUSAL, LOCAL = 1, 2


def gpu_masked(q, k, v, seq_lens, prompt_lens, mode, block):
    from paper_2608_02625_gb300 import binding as Bn
    d = q.device
    out = torch.full(q.shape, float("nan"), dtype=q.dtype, device=d)
    sl = torch.tensor(np.asarray(seq_lens, dtype=np.int32), device=d)
    pl = torch.tensor(np.asarray(prompt_lens, dtype=np.int32), device=d) if prompt_lens is not None else None
    Bn.dlm_attn_masked(q, k, v, sl, pl, mode, block, out)
    torch.cuda.synchronize()
    assert Bn.device_error(clear=True) == 0
    return out


def run(B, L, Hq, Hkv, D, sl, pl, mode, block, sigma, dtype, seed):
    q, k, v = rand_qkv(B, L, Hq, Hkv, D, sigma, dtype, seed)
    ref = oracle.bidir_attn(q.float().numpy(), k.float().numpy(), v.float().numpy(), sl, mask_mode=mode,
                            block=block, prompt_lens=pl if pl is not None else [0] * B)
    out = gpu_masked(q.to(dev()), k.to(dev()), v.to(dev()), sl, pl, mode, block)
    where = f"mode {mode} block {block} B{B} L{L} {Hq}/{Hkv} D{D} sl {sl} pl {pl}"
    if dtype == "f32":
        return compare(out, ref, sl, ATTN_TOL_F32, where=where)
    return compare(out, ref, sl, ATTN_TOL_BF16, where=where + f" sigma {sigma:.3g}")


@pytest.mark.parametrize("mode", [CAUSAL, LOCAL])
@pytest.mark.parametrize("block", [64, 32, 100, 128, 1000])
@pytest.mark.parametrize("B,L,Hq,Hkv,D,sl,pl", [
    (2, 512, 8, 2, 128, [512, 300], [128, 37]),       # GQA pairs share rows; prompt cut mid sub-tile
    (2, 300, 2, 2, 128, [300, 129], [0, 64]),         # MHA: a unit's two tiles are different row blocks
    (3, 256, 4, 2, 64, [256, 1, 200], [256, 0, 200]),  # all-prompt sequences, n = 1, D = 64
    (1, 640, 4, 1, 128, [640], [256]),                 # c5-shaped lengths
])
def test_bf16_vs_oracle(B, L, Hq, Hkv, D, sl, pl, mode, block):
    run(B, L, Hq, Hkv, D, sl, pl, mode, block, 1 / math.sqrt(D), "bf16", seed=B * L + block + mode)


@pytest.mark.parametrize("mode,block", [(CAUSAL, 64), (LOCAL, 64), (CAUSAL, 7), (LOCAL, 33)])
def test_bf16_peaked(mode, block):
    run(2, 384, 4, 2, 128, [384, 250], [64, 100], mode, block, 1.0, "bf16", seed=block)


@pytest.mark.parametrize("mode,block", [(CAUSAL, 64), (LOCAL, 64), (CAUSAL, 5), (LOCAL, 48)])
def test_f32_vs_oracle(mode, block):
    run(2, 200, 4, 2, 64, [200, 77], [40, 0], mode, block, 1.0, "f32", seed=7 + block)


def test_no_prompt_lens_means_zero():
    run(1, 256, 2, 1, 128, [256], None, LOCAL, 64, 1 / math.sqrt(128), "bf16", seed=5)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_full_mode_equals_bidir(dtype):
    from paper_2608_02625_gb300 import binding as Bn
    q, k, v = (t.to(dev()) for t in rand_qkv(2, 300, 4, 2, 128, 1.0, dtype, 9))
    sl = [300, 170]
    a = gpu_masked(q, k, v, sl, [50, 20], 0, 64)
    b = torch.empty_like(a)
    Bn.dlm_bidir_attn(q, k, v, torch.tensor(sl, dtype=torch.int32, device=dev()), b)
    torch.cuda.synchronize()
    assert torch.equal(a, b)


def test_prompt_clamp_sets_error_word():
    from paper_2608_02625_gb300 import binding as Bn
    q, k, v = (t.to(dev()) for t in rand_qkv(1, 128, 2, 1, 128, 0.1, "bf16", 2))
    out = torch.empty_like(q)
    Bn.dlm_attn_masked(q, k, v, torch.tensor([100], dtype=torch.int32, device=dev()),
                       torch.tensor([500], dtype=torch.int32, device=dev()), CAUSAL, 64, out)
    torch.cuda.synchronize()
    assert Bn.device_error(clear=True) & 0x1
    ref = oracle.bidir_attn(q.float().cpu().numpy(), k.float().cpu().numpy(), v.float().cpu().numpy(), [100],
                            mask_mode=CAUSAL, block=64, prompt_lens=[500])
    compare(out, ref, [100], ATTN_TOL_BF16, where="clamped prompt")


@pytest.mark.parametrize("mode", [CAUSAL, LOCAL])
def test_full_size_sampled(mode):
    """c3 at full size with 64-token blocks (the drafting block size); the
    oracle recomputes sampled (sequence, head) pairs from host-regenerated q, k, v."""
    from paper_2608_02625_gb300 import synth, synth_gpu
    w = workloads.get("c3_batch32_512")
    d = dev()
    q, k, v = synth_gpu.qkv(w, 0, d)
    sl, pl = w.seq_lens(), w.prompt_lens()
    out = gpu_masked(q, k, v, sl, pl, mode, 64).float().cpu().numpy()
    for b, h in ((0, 0), (7, 13), (31, 31)):
        qs = host_qkv_seq(w, 0, synth.S_Q, b, w.Hq)[:, h:h + 1]
        g = (h * w.Hkv) // w.Hq
        ks = host_qkv_seq(w, 0, synth.S_K, b, w.Hkv)[:, g:g + 1]
        vs = host_qkv_seq(w, 0, synth.S_V, b, w.Hkv)[:, g:g + 1]
        ref = oracle.bidir_attn(qs[None], ks[None], vs[None], [sl[b]], mask_mode=mode, block=64, prompt_lens=[pl[b]])
        err = np.abs(out[b, :, h] - ref[0, :, 0])
        assert err.max() <= ATTN_TOL_BF16, f"mode {mode} b {b} h {h}: {err.max()}"


@pytest.mark.parametrize("mode", [CAUSAL, LOCAL])
def test_workload_full_size(mode):
    """The 32 x 512 workload with its prompt lengths under both block masks (64-token
    blocks, the bench's setting): the whole batch in one launch, the oracle on
    sampled (sequence, query head) pairs from host-generated inputs."""
    from paper_2608_02625_gb300 import synth, synth_gpu
    w = workloads.get("c3_batch32_512")
    q, k, v = synth_gpu.qkv(w, 0, dev())
    n, pl = w.seq_lens(), w.prompt_lens()
    out = gpu_masked(q, k, v, n, pl, mode, 64)
    g_out = out.float()
    for b, heads in ((0, (0, 31)), (9, (5,)), (22, (13, 26)), (31, (7,))):
        hq = host_qkv_seq(w, 0, synth.S_Q, b, w.Hq)
        hk = host_qkv_seq(w, 0, synth.S_K, b, w.Hkv)
        hv = host_qkv_seq(w, 0, synth.S_V, b, w.Hkv)
        for h in heads:
            g = (h * w.Hkv) // w.Hq
            ref = oracle.bidir_attn(hq[None, :, h:h + 1], hk[None, :, g:g + 1], hv[None, :, g:g + 1], [n[b]],
                                    mask_mode=mode, block=64, prompt_lens=[pl[b]])
            compare(g_out[b:b + 1, :, h:h + 1], ref, [n[b]], ATTN_TOL_BF16, where=f"c3 mode {mode} b={b} h={h}")

