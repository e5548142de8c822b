"""Host-side arithmetic of the benchmark, checked on CPU against brute force.

The benchmark reports effective TFLOP/s as 4 * head_dim FLOPs (Q K^T and P V)
per computed (query, key) pair: B^2 pairs for an off-diagonal block of the
support and B(B+1)/2 for the diagonal one (causal mask, Eq. 2; support
restriction, Eqs. 7-8).  Here that count is compared with an explicit
element-wise mask on small random supports, and the all-blocks support with
the dense count.
"""
import numpy as np
import pytest

import bench
from paper_2609_27373_gb300 import synth


def _brute_pairs(idx, counts, seqlen, block):
    """Computed (query, key) pairs per kv-head row, from an explicit mask."""
    B, Hkv, nb, _ = idx.shape
    total = 0
    q = np.arange(seqlen)[:, None]
    k = np.arange(seqlen)[None, :]
    causal = k <= q
    for b in range(B):
        for g in range(Hkv):
            allowed = np.zeros((seqlen, seqlen), dtype=bool)
            for qb in range(nb):
                for kb in idx[b, g, qb, : counts[b, g, qb]]:
                    allowed[qb * block:(qb + 1) * block, kb * block:(kb + 1) * block] = True
            total += int(np.count_nonzero(allowed & causal))
    return total


@pytest.mark.parametrize("block,seqlen,n_heads,n_kv_heads", [(32, 256, 2, 2), (64, 512, 4, 2), (128, 640, 2, 1)])
def test_sparse_flops_count_the_computed_pairs(block, seqlen, n_heads, n_kv_heads):
    head_dim = 64
    nb = seqlen // block
    idx, counts = synth.random_support(1, n_kv_heads, nb, cap=5, seed=block + seqlen, density=0.4)
    pairs = _brute_pairs(idx, counts, seqlen, block)
    group = n_heads // n_kv_heads
    assert bench.sparse_flops(idx, counts, n_heads, head_dim, block) == 4.0 * head_dim * pairs * group


def test_all_blocks_support_counts_the_dense_flops():
    batch, n_heads, n_kv_heads, seqlen, head_dim, block = 2, 4, 2, 512, 96, 64
    idx, counts = synth.all_blocks_support(batch, n_kv_heads, seqlen // block)
    assert bench.sparse_flops(idx, counts, n_heads, head_dim, block) == bench.dense_flops(batch, n_heads, seqlen,
                                                                                          head_dim)


def test_pair_count_of_a_block():
    for block in (32, 64, 128):
        mask = np.tril(np.ones((block, block), dtype=bool))
        assert bench.pair_count(block, True) == int(mask.sum())
        assert bench.pair_count(block, False) == block * block
