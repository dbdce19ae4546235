"""Memory safety of every entry point: outputs are views inside larger buffers
filled with a canary byte, with gaps between rows where the layout allows;
after each call the bytes outside the views must still hold the canary, and
the results must equal those of the same call on plain contiguous outputs."""
import numpy as np
import pytest
import torch

from gpu_util import dev

pytestmark = pytest.mark.gpu

CANARY = 0xA5
PAD = 256  # elements before and after every view (16-byte aligned for every dtype here)


class Guarded:
    """A view of `shape` inside a canary-filled buffer; `gap` extra elements
    after each innermost row (0 keeps the view contiguous)."""

    def __init__(self, shape, dtype, gap=0):
        shape = tuple(shape)
        inner = shape[-1] + gap
        outer = int(np.prod(shape[:-1])) if len(shape) > 1 else 1
        self.buf = torch.empty(2 * PAD + outer * inner, dtype=dtype, device=dev())
        self.buf.view(torch.uint8).fill_(CANARY)
        body = self.buf[PAD:PAD + outer * inner].view(*shape[:-1], inner) if len(shape) > 1 else \
            self.buf[PAD:PAD + inner]
        self.view = body[..., :shape[-1]]
        self.mask = torch.ones(self.buf.numel(), dtype=torch.bool, device=dev())
        idx = torch.arange(self.buf.numel(), device=dev()).as_strided(self.view.shape, self.view.stride(),
                                                                     self.view.storage_offset())
        self.mask[idx.reshape(-1)] = False  # positions inside the view

    def untouched(self) -> bool:
        outside = self.buf.view(torch.uint8).view(-1, self.buf.element_size())[self.mask]
        return bool((outside == CANARY).all())


def _sync():
    torch.cuda.synchronize()
    from paper_2608_02625_gb300 import binding as Bn
    assert Bn.device_error(clear=True) == 0


@pytest.mark.parametrize("dtype,D", [(torch.bfloat16, 128), (torch.bfloat16, 64), (torch.float32, 64)])
@pytest.mark.parametrize("mode", [0, 1, 2])
def test_attention_writes_only_its_output(dtype, D, mode):
    from paper_2608_02625_gb300 import binding as Bn
    g = torch.Generator().manual_seed(D + mode)
    B, L, Hq, Hkv = 2, 200, 4, 2
    q, k, v = [torch.randn(B, L, H, D, generator=g).to(dtype).to(dev()) for H in (Hq, Hkv, Hkv)]
    n = torch.tensor([200, 77], dtype=torch.int32, device=dev())
    p = torch.tensor([64, 13], dtype=torch.int32, device=dev())
    ref = torch.empty_like(q)
    out = Guarded((B, L, Hq, D), dtype, gap=64)
    for o in (ref, out.view):
        if mode == 0:
            Bn.dlm_bidir_attn(q, k, v, n, o)
        else:
            Bn.dlm_attn_masked(q, k, v, n, p, mode, 32, o)
    _sync()
    assert out.untouched()
    assert torch.equal(out.view, ref)


@pytest.mark.parametrize("N,V", [(5, 151552), (700, 4096), (40, 1003)])
def test_vocab_writes_only_its_outputs(N, V):
    from paper_2608_02625_gb300 import binding as Bn
    g = torch.Generator().manual_seed(N + V)
    logits = (torch.randn(N, V, generator=g) * 3).to(torch.bfloat16).to(dev())
    outs = [Guarded((N,), t) for t in (torch.int32, torch.float32, torch.float32)]
    ref = [torch.empty(N, dtype=t, device=dev()) for t in (torch.int32, torch.float32, torch.float32)]
    Bn.dlm_vocab_confidence(logits, *[o.view for o in outs])
    Bn.dlm_vocab_confidence(logits, *ref)
    _sync()
    assert all(o.untouched() for o in outs)
    assert all(torch.equal(o.view, r) for o, r in zip(outs, ref))
    prob = Guarded((N,), torch.float32)
    tokens = torch.randint(0, V, (N,), generator=g, dtype=torch.int32).to(dev())
    Bn.dlm_token_prob(logits, tokens, ref[2], prob.view)
    _sync()
    assert prob.untouched()


def _update_inputs(B, L, V, seed):
    g = torch.Generator().manual_seed(seed)
    tok = torch.randint(0, V, (B, L), generator=g, dtype=torch.int32)
    msk = (torch.rand(B, L, generator=g) < 0.25).to(torch.uint8)
    am = torch.randint(0, V, (B, L), generator=g, dtype=torch.int32)
    cf = torch.rand(B, L, generator=g, dtype=torch.float32)
    return [t.to(dev()) for t in (tok, msk, am, cf)]


@pytest.mark.parametrize("ranked", [False, True])
def test_update_writes_only_its_outputs(ranked):
    from paper_2608_02625_gb300 import binding as Bn
    B, L, V = 3, 300, 1000
    tok, msk, am, cf = _update_inputs(B, L, V, 7)
    prm = Bn.RefineParams(0.5, -1, 0.2, V, torch.tensor([10, 50, 0], dtype=torch.int32, device=dev()),
                          torch.tensor([300, 200, 1], dtype=torch.int32, device=dev()))
    outs = [Guarded((B, L), torch.int32, gap=4), Guarded((B, L), torch.uint8, gap=16), Guarded((B,), torch.int32)]
    ref = [torch.empty_like(tok), torch.empty_like(msk), torch.empty(B, dtype=torch.int32, device=dev())]
    tp = torch.rand(B, L, generator=torch.Generator().manual_seed(3)).to(dev())
    for o in ([x.view for x in outs], ref):
        if ranked:
            Bn.dlm_refine_update_ranked(tok, msk, am, cf, tp, prm, *o)
        else:
            Bn.dlm_refine_update(tok, msk, am, cf, prm, *o)
    _sync()
    assert all(o.untouched() for o in outs)
    assert all(torch.equal(o.view, r) for o, r in zip(outs, ref))


@pytest.mark.parametrize("static", [False, True])
def test_fused_step_writes_only_its_outputs(static):
    from paper_2608_02625_gb300 import binding as Bn
    B, L, V = 2, 96, 40000
    g = torch.Generator().manual_seed(11)
    logits = (torch.randn(B * L, V, generator=g) * 3).to(torch.bfloat16).to(dev())
    tok, msk, _, _ = _update_inputs(B, L, V, 12)
    prm = Bn.RefineParams(0.3, 5, 0.0, V, torch.tensor([16, 40], dtype=torch.int32, device=dev()),
                          torch.tensor([96, 90], dtype=torch.int32, device=dev()))
    outs = [Guarded((B, L), t) for t in (torch.int32, torch.float32, torch.float32)] + \
        [Guarded((B, L), torch.int32, gap=4), Guarded((B, L), torch.uint8, gap=16), Guarded((B,), torch.int32)]
    ref = [torch.empty(B, L, dtype=t, device=dev()) for t in (torch.int32, torch.float32, torch.float32)] + \
        [torch.empty_like(tok), torch.empty_like(msk), torch.empty(B, dtype=torch.int32, device=dev())]
    ws = Guarded((Bn.dlm_refine_step_workspace_bytes(B) // 4,), torch.int32)
    ws.view.zero_()
    if static:
        Bn.dlm_refine_step_static(logits, tok, msk, prm, *[o.view for o in outs])
    else:
        Bn.dlm_refine_step(logits, tok, msk, prm, *[o.view for o in outs], ws.view)
    wr = torch.zeros(Bn.dlm_refine_step_workspace_bytes(B) // 4, dtype=torch.int32, device=dev())
    Bn.dlm_refine_step(logits, tok, msk, prm, *ref, wr)
    _sync()
    assert all(o.untouched() for o in outs) and ws.untouched()
    assert all(torch.equal(o.view, r) for o, r in zip(outs, ref))
    assert int(ws.view.abs().sum()) == 0  # the counters are left zero


def test_lmhead_writes_only_its_outputs():
    from paper_2608_02625_gb300 import binding as Bn
    N, V, d = 300, 5000, 128
    g = torch.Generator().manual_seed(21)
    hid = torch.randn(N, d, generator=g).to(torch.bfloat16).to(dev())
    wt = (torch.randn(V, d, generator=g) / d ** 0.5).to(torch.bfloat16).to(dev())
    outs = [Guarded((N,), t) for t in (torch.int32, torch.float32, torch.float32)]
    ref = [torch.empty(N, dtype=t, device=dev()) for t in (torch.int32, torch.float32, torch.float32)]
    nbytes = Bn.dlm_lmhead_workspace_bytes(N)
    ws = Guarded((nbytes,), torch.uint8)
    Bn.dlm_lmhead_confidence(hid, wt, *[o.view for o in outs], ws.view)
    Bn.dlm_lmhead_confidence(hid, wt, *ref, torch.empty(nbytes, dtype=torch.uint8, device=dev()))
    _sync()
    assert all(o.untouched() for o in outs) and ws.untouched()
    assert all(torch.equal(o.view, r) for o, r in zip(outs, ref))
