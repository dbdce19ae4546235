"""dlm_refine_step_static: the fused step on the library's static scratch,
for callers that cannot allocate device memory.

Collected last (conftest orders test_zz_* files after the others) and written
to pass both alone in a fresh process, where its first call sets the device
up, and after every other test. Each case makes two static calls in a row and
checks both against dlm_refine_step with a caller-provided workspace, within
the tolerances of the other vocabulary tests (the two run the same kernel, so
the results are in fact identical)."""
import numpy as np
import pytest
import torch

from gpu_util import CONF_RTOL, LSE_RTOL, dev

pytestmark = pytest.mark.gpu


def outputs(B, L):
    d = dev()
    return [torch.full((B, L), -5, dtype=torch.int32, device=d),
            torch.full((B, L), -1.0, dtype=torch.float32, device=d),
            torch.full((B, L), -1.0, dtype=torch.float32, device=d),
            torch.full((B, L), -7, dtype=torch.int32, device=d),
            torch.full((B, L), 7, dtype=torch.uint8, device=d),
            torch.full((B,), -1, dtype=torch.int32, device=d)]


def close(a, b, where):
    am, cf, ls, nt, nm, ne = (t.cpu().numpy() for t in a)
    am2, cf2, ls2, nt2, nm2, ne2 = (t.cpu().numpy() for t in b)
    assert np.array_equal(am, am2), f"{where}: argmax"
    assert np.all(np.abs(cf.astype(np.float64) - cf2) <= CONF_RTOL * np.maximum(cf2, 1e-30)), f"{where}: conf"
    assert np.all(np.abs(ls.astype(np.float64) - ls2) <= LSE_RTOL * np.maximum(1.0, np.abs(ls2))), f"{where}: lse"
    for n, x, y in (("tokens", nt, nt2), ("mask", nm, nm2), ("n_edits", ne, ne2)):
        assert np.array_equal(x, y), f"{where}: {n} differs at {np.argwhere(x != y)[:8].tolist()}"


def case(B, L, V, seed):
    from paper_2608_02625_gb300 import binding as Bn
    d = dev()
    g = torch.Generator(device="cpu").manual_seed(seed)
    logits = (torch.randn((B * L, V), generator=g) * 3.0).to(torch.bfloat16).to(d)
    tok = torch.randint(0, V, (B, L), generator=g, dtype=torch.int32).to(d)
    msk = (torch.rand((B, L), generator=g) < 0.25).to(torch.uint8).to(d)
    prompt = torch.randint(0, L // 2 + 1, (B,), generator=g, dtype=torch.int32)
    seqlen = torch.minimum(prompt + torch.randint(0, L + 1, (B,), generator=g, dtype=torch.int32),
                           torch.tensor(L, dtype=torch.int32))
    params = Bn.RefineParams(0.8, -1, 0.1, V, prompt.to(d), seqlen.to(d))
    return logits, tok, msk, params


@pytest.mark.parametrize("B,L,V", [(32, 512, 151552), (5, 37, 4099), (1, 1, 8)])
def test_static_matches_workspace_call_twice(B, L, V):
    from paper_2608_02625_gb300 import binding as Bn
    logits, tok, msk, params = case(B, L, V, seed=B * 1000 + L)
    ws = torch.zeros(Bn.dlm_refine_step_workspace_bytes(B) // 4, dtype=torch.int32, device=dev())
    ref = outputs(B, L)
    Bn.dlm_refine_step(logits, tok, msk, params, *ref, ws)
    for call in range(2):
        got = outputs(B, L)
        Bn.dlm_refine_step_static(logits, tok, msk, params, *got)
        torch.cuda.synchronize()
        assert Bn.device_error(clear=True) == 0
        close(got, ref, f"B={B} L={L} V={V} static call {call + 1}")


def test_larger_then_smaller_batch():
    """The scratch keeps the last call's contents; a call with a smaller batch
    after a larger one still starts from cleared counters."""
    from paper_2608_02625_gb300 import binding as Bn
    for B, L, V in ((40, 64, 1000), (3, 64, 1000)):
        logits, tok, msk, params = case(B, L, V, seed=7 + B)
        ws = torch.zeros(B, dtype=torch.int32, device=dev())
        ref = outputs(B, L)
        Bn.dlm_refine_step(logits, tok, msk, params, *ref, ws)
        got = outputs(B, L)
        Bn.dlm_refine_step_static(logits, tok, msk, params, *got)
        torch.cuda.synchronize()
        close(got, ref, f"B={B}")


def test_no_device_memory_taken():
    """After the first call (device set-up, kernel loaded), further calls leave
    the device's free memory unchanged."""
    from paper_2608_02625_gb300 import binding as Bn
    B, L, V = 8, 128, 2048
    logits, tok, msk, params = case(B, L, V, seed=3)
    got = outputs(B, L)
    Bn.dlm_refine_step_static(logits, tok, msk, params, *got)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(2):
        Bn.dlm_refine_step_static(logits, tok, msk, params, *got)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0


def test_batch_above_maximum_rejected():
    from paper_2608_02625_gb300 import binding as Bn
    d = dev()
    B, L, V = 4097, 1, 16
    z = lambda *s, dt=torch.int32: torch.zeros(s, dtype=dt, device=d)
    params = Bn.RefineParams(0.5, 1, 0.0, V, z(B), z(B))
    with pytest.raises(Bn.DlmError) as e:
        Bn.dlm_refine_step_static(z(B * L, V, dt=torch.bfloat16), z(B, L), z(B, L, dt=torch.uint8), params,
                                  z(B, L), z(B, L, dt=torch.float32), z(B, L, dt=torch.float32), z(B, L),
                                  z(B, L, dt=torch.uint8), z(B))
    assert e.value.status == -3 and "4096" in str(e.value)
