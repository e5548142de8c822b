"""Run-to-run determinism of the kernels: repeated launches on the same
inputs give bit-identical outputs, block masses and supports.  The attention
kernel keeps several tensor-core operations in flight that reuse tensor
memory in issue order; a reuse hazard would show up here as differences
between runs or between the sparse (all blocks) and dense kernels."""
import numpy as np
import pytest
import torch

from paper_2609_27373_gb300 import synth, wise
from gpu_helpers import to_dev

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("B,H,Hkv,L,D,blk", [(1, 32, 32, 4096, 128, 128), (2, 6, 3, 2048, 96, 128),
                                             (1, 8, 8, 1536, 64, 64)])
def test_repeated_launches_are_bit_identical(B, H, Hkv, L, D, blk):
    shape = wise.Shape(B, L, H, Hkv, D, blk)
    nb = shape.n_blocks
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=91, std=1.3, v_std=1.0)
    dq, dk, dv = to_dev(Q), to_dev(K), to_dev(V)
    idx, counts = synth.random_support(B, Hkv, nb, 8, seed=5, density=0.6)
    di, dc = torch.from_numpy(idx).cuda(), torch.from_numpy(counts).cuda()
    all_idx, all_counts = synth.all_blocks_support(B, Hkv, nb)
    dai, dac = torch.from_numpy(all_idx).cuda(), torch.from_numpy(all_counts).cuda()
    ref_o = ref_m = ref_s = ref_d = None
    for rep in range(6):
        O = torch.empty_like(dq)
        mass = torch.empty((B, H, nb, nb), dtype=torch.float32, device="cuda")
        wise.wise_full_attn_accumulate(shape, dq, dk, dv, O, mass, 0)
        Os = torch.empty_like(dq)
        wise.wise_sparse_attn(shape, dq, dk, dv, di, dc, Os)
        Od = torch.empty_like(dq)
        wise.wise_sparse_attn(shape, dq, dk, dv, dai, dac, Od)
        torch.cuda.synchronize()
        if rep == 0:
            ref_o, ref_m, ref_s, ref_d = O.clone(), mass.clone(), Os.clone(), Od.clone()
            assert torch.equal(Od.view(torch.int16), O.view(torch.int16))
        else:
            assert torch.equal(O.view(torch.int16), ref_o.view(torch.int16))
            assert torch.equal(mass, ref_m)
            assert torch.equal(Os.view(torch.int16), ref_s.view(torch.int16))
            assert torch.equal(Od.view(torch.int16), ref_d.view(torch.int16))
    assert wise.wise_get_status() == wise.WISE_OK
