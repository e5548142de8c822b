"""wise_support_mass (routing diagnostic) through the C ABI against the oracle.

The retained mass of a support is the share of one step's unrestricted
attention (its block mass, Eq. 5) that falls inside the support.  The GPU
sums the fp32 masses it is given; the oracle sums the same fp32 values in
fp64, so the two agree to fp32 rounding of a short sum.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_27373_gb300 import synth, wise
from gpu_helpers import to_dev

pytestmark = pytest.mark.gpu


def _mass(shape, Q, K, V):
    nb = shape.n_blocks
    mass = torch.empty((shape.batch, shape.n_heads, nb, nb), dtype=torch.float32, device="cuda")
    O = torch.empty((shape.batch, shape.n_heads, shape.seqlen, shape.head_dim), dtype=torch.bfloat16, device="cuda")
    wise.wise_full_attn_accumulate(shape, Q, K, V, O, mass, 0)
    return mass


@pytest.mark.parametrize("B,H,Hkv,L,D,blk,cap", [(1, 8, 8, 2048, 128, 128, 6), (2, 8, 2, 1536, 64, 64, 9)])
def test_retained_mass_matches_oracle(B, H, Hkv, L, D, blk, cap):
    shape = wise.Shape(B, L, H, Hkv, D, blk)
    nb = shape.n_blocks
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=40, std=1.5, v_std=1.0)
    mass = _mass(shape, to_dev(Q), to_dev(K), to_dev(V))
    idx, counts = synth.random_support(B, Hkv, nb, cap, seed=41, density=0.4)
    out = torch.full((B, H, nb), -7.0, dtype=torch.float32, device="cuda")
    wise.wise_support_mass(shape, mass, torch.from_numpy(idx).cuda(), torch.from_numpy(counts).cuda(), out)
    assert wise.wise_get_status() == wise.WISE_OK
    want = orc.support_mass(mass.cpu().numpy(), idx, counts, H)
    got = out.cpu().numpy().astype(np.float64)
    assert np.abs(got - want).max() <= 1e-5
    assert 0.0 < got.min() and got.max() <= 1.0 + 1e-5


def test_retained_mass_of_every_block_is_one():
    B, H, Hkv, L, D, blk = 1, 4, 4, 1024, 128, 128
    shape = wise.Shape(B, L, H, Hkv, D, blk)
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=42)
    mass = _mass(shape, to_dev(Q), to_dev(K), to_dev(V))
    idx, counts = synth.all_blocks_support(B, Hkv, shape.n_blocks)
    out = torch.empty((B, H, shape.n_blocks), dtype=torch.float32, device="cuda")
    wise.wise_support_mass(shape, mass, torch.from_numpy(idx).cuda(), torch.from_numpy(counts).cuda(), out)
    assert wise.wise_get_status() == wise.WISE_OK
    assert np.abs(out.cpu().numpy() - 1.0).max() <= 1e-5


def test_retained_mass_skips_and_reports_invalid_entries():
    B, H, Hkv, L, D, blk = 1, 2, 1, 512, 64, 128
    shape = wise.Shape(B, L, H, Hkv, D, blk)
    nb = shape.n_blocks
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=43)
    mass = _mass(shape, to_dev(Q), to_dev(K), to_dev(V))
    idx = np.full((B, Hkv, nb, 3), -1, dtype=np.int32)
    counts = np.zeros((B, Hkv, nb), dtype=np.int32)
    idx[0, 0, 2] = [2, 1, 3]  # only 2 is valid (1 is not ascending, 3 is beyond the query block)
    counts[0, 0, 2] = 3
    idx[0, 0, 3] = [0, 3, -1]
    counts[0, 0, 3] = 2
    out = torch.empty((B, H, nb), dtype=torch.float32, device="cuda")
    wise.wise_support_mass(shape, mass, torch.from_numpy(idx).cuda(), torch.from_numpy(counts).cuda(), out)
    assert wise.wise_get_status() == wise.WISE_ERR_BAD_SUPPORT
    want = orc.support_mass(mass.cpu().numpy(), idx, counts, H)
    assert np.abs(out.cpu().numpy() - want).max() <= 1e-6
    assert np.all(out.cpu().numpy()[:, :, :2] == 0.0)
