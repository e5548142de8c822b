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
                                             (1, 8, 8, 1536, 64, 64), (1, 8, 4, 2048, 128, 32)])
def test_repeated_launches_are_bit_identical(B, H, Hkv, L, D, blk):
    shape = wise.Shape(B, L, H, Hkv, D, blk)
    nb = shape.n_blocks
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=91, std=1.3, v_std=1.0)
    dq, dk, dv = to_dev(Q), to_dev(K), to_dev(V)
    idx, counts = synth.random_support(B, Hkv, nb, 8, seed=5, density=0.6)
    di, dc = torch.from_numpy(idx).cuda(), torch.from_numpy(counts).cuda()
    all_idx, all_counts = synth.all_blocks_support(B, Hkv, nb)
    dai, dac = torch.from_numpy(all_idx).cuda(), torch.from_numpy(all_counts).cuda()
    ref = None
    for rep in range(6):
        O = torch.empty_like(dq)
        mass = torch.empty((B, H, nb, nb), dtype=torch.float32, device="cuda")
        wise.wise_full_attn_accumulate(shape, dq, dk, dv, O, mass, 0)
        Op = torch.empty_like(dq)
        wise.wise_full_attn_accumulate(shape, dq, dk, dv, Op)
        Os = torch.empty_like(dq)
        wise.wise_sparse_attn(shape, dq, dk, dv, di, dc, Os)
        Od = torch.empty_like(dq)
        wise.wise_sparse_attn(shape, dq, dk, dv, dai, dac, Od)
        torch.cuda.synchronize()
        assert wise.wise_get_status() == wise.WISE_OK
        outs = [O, mass, Op, Os, Od]
        if rep == 0:
            ref = [x.clone() for x in outs]
            # the sparse kernel with every block equals the dense kernel
            assert torch.equal(Od.view(torch.int16), Op.view(torch.int16))
        else:
            names = ["dense+mass O", "block mass", "dense O", "sparse O", "all-blocks sparse O"]
            for name, x, y in zip(names, outs, ref):
                iv = torch.int32 if x.dtype == torch.float32 else torch.int16
                assert torch.equal(x.view(iv), y.view(iv)), f"rep {rep}: {name} differs from rep 0"
    assert wise.wise_get_status() == wise.WISE_OK
