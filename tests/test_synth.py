"""Host side of the seeded input generator (no GPU)."""
import numpy as np
import torch

from paper_2608_02625_gb300 import synth, workloads


def test_mix64_known_values():
    # SplitMix64 with state 0: the first outputs of the published generator
    # (state advances by the golden gamma before mixing).
    z = 0
    outs = []
    for _ in range(3):
        z = (z + synth.GOLDEN) & synth.MASK64
        outs.append(synth.mix64_int(z))
    assert outs == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]
    # The counter form draws(key, i) = mix64(key + i * gamma) is the same sequence.
    d = synth.draws(0, np.arange(1, 4, dtype=np.uint64))
    assert [int(x) for x in d] == outs


def test_normals_bounded_and_moments():
    x = synth.normals(synth.stream_key(3, synth.S_Q), np.arange(200000, dtype=np.uint64), 2.0)
    assert x.dtype == np.float32
    assert np.all(np.abs(x) < 12.0)
    assert abs(float(x.mean())) < 0.02
    assert abs(float(x.std()) - 2.0) < 0.02


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(100000) * 10.0 ** rng.integers(-6, 6, 100000)).astype(np.float32)
    ours = synth.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


def test_uniform_int_range_and_slices():
    key = synth.stream_key(1, synth.S_DRAFT)
    u = synth.uniform_int(key, np.arange(50000, dtype=np.uint64), 151552)
    assert u.min() >= 0 and u.max() < 151552
    # Any slice regenerates identically (counter-based).
    u2 = synth.uniform_int(key, np.arange(1000, 2000, dtype=np.uint64), 151552)
    assert np.array_equal(u[1000:2000], u2)


def test_workload_structure():
    w = workloads.get("c3")
    p, n = w.prompt_lens(), w.seq_lens()
    assert p.min() >= 64 and p.max() <= 256
    assert np.array_equal(n, np.minimum(512, p + 384))
    tok, m = w.initial_state()
    for b in range(w.B):
        r = int(n[b] - p[b])
        assert int(m[b].sum()) == r // 4
        assert m[b, :p[b]].sum() == 0 and m[b, n[b]:].sum() == 0
    assert np.all(tok[m == 1] == w.mask_id)
    assert np.all(tok[m == 0] < w.V)


def test_planted_peaks_c1():
    w = workloads.get("c1")
    spec = w.logit_spec(0)
    x = spec.rows_f32(np.arange(8))
    is_peak, tok, val = spec.peak_plan(np.arange(8))
    assert is_peak.all()
    for r in range(8):
        others = np.delete(x[r], tok[r])
        assert x[r, tok[r]] == val[r]
        assert x[r, tok[r]] - others.max() >= 0.5
