"""Host logic of the bench's FLOP accounting for masked attention."""
import itertools

from oracle import attention as oatt
from paper_2608_02625_gb300 import workloads


def test_attended_pairs_match_the_oracle_masks():
    for n, p, mode, block in itertools.product((1, 7, 13, 64), (0, 3, 64), (0, 1, 2), (1, 4, 64)):
        if p > n:
            continue
        assert workloads.attended_pairs(n, p, mode, block) == int(oatt.key_mask(n, p, block, mode).sum())


def test_full_attention_flops():
    w = workloads.get("c3_batch32_512")
    n = w.seq_lens().astype(float)
    assert w.attn_flops() == float((4.0 * w.Hq * w.D * n * n).sum())
    assert w.attn_flops(1, 64) < w.attn_flops() and w.attn_flops(2, 64) < w.attn_flops(1, 64)
