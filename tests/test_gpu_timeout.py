"""The bounded waits give up instead of hanging: a kernel waiting, through the
wait routine every pipelined kernel uses, on a barrier nothing arrives on
returns after its budget with DLM_DEVERR_TIMEOUT in the device error word,
and the context stays usable (a following attention call is correct)."""
import time

import numpy as np
import pytest
import torch

import oracle
from gpu_util import ATTN_TOL_BF16, dev

pytestmark = pytest.mark.gpu

DLM_DEVERR_TIMEOUT = 0x2


@pytest.mark.parametrize("budget_ns", [1000, 1000000, 50000000])
def test_wait_gives_up_after_its_budget(budget_ns):
    from paper_2608_02625_gb300 import binding as Bn
    torch.cuda.set_device(dev())
    assert Bn.device_error(clear=True) == 0
    t0 = time.perf_counter()
    Bn.dlm_selftest_wait_timeout(budget_ns)
    torch.cuda.synchronize()
    elapsed = time.perf_counter() - t0
    assert Bn.device_error(clear=True) == DLM_DEVERR_TIMEOUT
    assert elapsed >= budget_ns * 1e-9 and elapsed < budget_ns * 1e-9 + 1.0
    # The context is still usable: a small attention call is correct and clean.
    g = torch.Generator().manual_seed(2)
    q = torch.randn(1, 160, 4, 128, generator=g).to(torch.bfloat16)
    k = torch.randn(1, 160, 2, 128, generator=g).to(torch.bfloat16)
    v = torch.randn(1, 160, 2, 128, generator=g).to(torch.bfloat16)
    out = torch.empty(q.shape, dtype=torch.bfloat16, device=dev())
    Bn.dlm_bidir_attn(q.to(dev()), k.to(dev()), v.to(dev()), torch.tensor([150], dtype=torch.int32, device=dev()),
                      out)
    torch.cuda.synchronize()
    assert Bn.device_error(clear=True) == 0
    ref = oracle.bidir_attn(q.float().numpy(), k.float().numpy(), v.float().numpy(), [150])
    assert np.abs(out.float().cpu().numpy() - ref).max() <= ATTN_TOL_BF16
