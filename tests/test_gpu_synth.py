"""The device generator reproduces the host generator bit for bit."""
import numpy as np
import pytest
import torch

from gpu_util import dev
from paper_2608_02625_gb300 import synth, workloads

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_normals_bitwise(dtype):
    from paper_2608_02625_gb300 import synth_gpu
    n, e0 = 100003, 12345
    t = torch.empty(n, dtype=torch.bfloat16 if dtype == "bf16" else torch.float32, device=dev())
    key = synth.stream_key(9, synth.S_K)
    synth_gpu.fill_normal_(t, key, 0.7, e0)
    host = synth.normals(key, np.arange(e0, e0 + n, dtype=np.uint64), 0.7)
    if dtype == "bf16":
        got = t.view(torch.int16).cpu().numpy().view(np.uint16)
        assert np.array_equal(got, synth.f32_to_bf16_bits(host))
    else:
        assert np.array_equal(t.cpu().numpy().view(np.uint32), host.view(np.uint32))


@pytest.mark.parametrize("name", ["c1_tiny_f32", "c4_long_2048", "c5_heavy_4step"])
def test_logit_rows_bitwise(name):
    from paper_2608_02625_gb300 import synth_gpu
    w = workloads.get(name)
    rows = np.array([0, 1, 17, 300, 1023]) % w.N
    tok, msk = w.initial_state()
    tok, msk = tok.reshape(-1), msk.reshape(-1)
    rng = np.random.default_rng(0)
    tok = np.where(rng.random(tok.size) < 0.5, tok, w.mask_id).astype(np.int32)   # some current tokens
    msk = (tok == w.mask_id).astype(np.uint8)
    for step in range(w.steps):
        spec = w.logit_spec(step)
        dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
        out = torch.empty((len(rows), w.V), dtype=dt, device=dev())
        for i, r in enumerate(rows):
            synth_gpu.fill_logits_(out[i:i + 1], spec, int(r), torch.from_numpy(tok[r:r + 1]).to(dev()),
                                   torch.from_numpy(msk[r:r + 1]).to(dev()))
        host = spec.rows_f32(rows, tok[rows], msk[rows])
        if w.dtype == "bf16":
            assert np.array_equal(out.view(torch.int16).cpu().numpy().view(np.uint16), synth.f32_to_bf16_bits(host))
        else:
            assert np.array_equal(out.cpu().numpy().view(np.uint32), host.view(np.uint32))
