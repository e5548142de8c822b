"""wise_full_attn_accumulate_noalloc: block-mass attention without any device
allocation by the library.

Some callers cannot let a library call cudaMalloc: their device memory is
handed out by another allocator that has reserved the pool, or they run a
serving loop that cannot take the device-wide synchronisation cudaMalloc and
cudaFree may cause.  This entry point keeps its scratch in a fixed array
compiled into libwise.so.  Through the C ABI, it must give the same output
and block mass as wise_full_attn_accumulate on two calls in a row (a first
step that overwrites the mass and a second that accumulates), and refuse a
problem whose scratch would not fit.  This file is collected last so that a
run stopping at its first failure has already run every other test.
"""
import os
import subprocess
import sys
import textwrap

import numpy as np
import pytest
import torch

from paper_2609_27373_gb300 import synth, wise
from gpu_helpers import MASS_MAX_ABS, assert_close_o, bf16_dev_to_f64, to_dev

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("B,H,Hkv,L,D,blk", [(1, 8, 8, 2048, 128, 128), (2, 4, 2, 1024, 64, 64),
                                             (1, 6, 6, 768, 96, 128), (1, 4, 4, 1024, 128, 32)])
def test_noalloc_matches_the_allocating_entry_point_on_two_calls(B, H, Hkv, L, D, blk):
    assert torch.cuda.is_available()
    shape = wise.Shape(B, L, H, Hkv, D, blk)
    nb = shape.n_blocks
    steps = [synth.random_qkv(B, H, Hkv, L, D, seed=s, std=1.5, v_std=1.0) for s in (31, 32)]
    mass_ref = torch.zeros((B, H, nb, nb), dtype=torch.float32, device="cuda")
    mass_new = torch.full((B, H, nb, nb), 7.0, dtype=torch.float32, device="cuda")
    for step, (Q, K, V) in enumerate(steps):
        dQ, dK, dV = to_dev(Q), to_dev(K), to_dev(V)
        O_ref = torch.empty_like(dQ)
        O_new = torch.empty_like(dQ)
        wise.wise_full_attn_accumulate(shape, dQ, dK, dV, O_ref, mass_ref, step)
        wise.wise_full_attn_accumulate_noalloc(shape, dQ, dK, dV, O_new, mass_new, step)
        torch.cuda.synchronize()
        assert_close_o(bf16_dev_to_f64(O_new), bf16_dev_to_f64(O_ref), what=f"call {step + 1}")
        diff = np.abs(mass_new.cpu().numpy().astype(np.float64) - mass_ref.cpu().numpy())
        assert diff.max() <= MASS_MAX_ABS, f"call {step + 1}: block mass differs by {diff.max():.3e}"
    assert wise.wise_get_status() == wise.WISE_OK


def test_noalloc_rejects_a_problem_beyond_its_scratch():
    # 32 heads x 256 query tiles >= one CTA per SM, each needing about 256 blocks * 1 KB:
    # far more than the 8 MiB array.
    shape = wise.Shape(1, 32768, 32, 8, 128, 128)
    Q = torch.zeros((1, 32, 32768, 128), dtype=torch.bfloat16, device="cuda")
    K = torch.zeros((1, 8, 32768, 128), dtype=torch.bfloat16, device="cuda")
    O = torch.empty_like(Q)
    mass = torch.zeros((1, 32, 256, 256), dtype=torch.float32, device="cuda")
    with pytest.raises(wise.WiseError) as e:
        wise.wise_full_attn_accumulate_noalloc(shape, Q, K, K, O, mass, 0)
    assert e.value.code == wise.WISE_ERR_UNSUPPORTED
    assert wise.wise_get_status() == wise.WISE_OK


_FRESH_PROCESS = textwrap.dedent("""
    import sys, torch
    sys.path.insert(0, sys.argv[1])
    from paper_2609_27373_gb300 import synth, wise
    wise.load()
    B, H, L, D, blk = 1, 8, 2048, 128, 128
    shape = wise.Shape(B, L, H, H, D, blk)
    nb = shape.n_blocks
    to = lambda x: torch.from_numpy(x.view("int16")).view(torch.bfloat16).cuda()
    Q, K, V = (to(x) for x in synth.random_qkv(B, H, H, L, D, seed=3))
    O = torch.empty_like(Q)
    mass = torch.zeros((B, H, nb, nb), dtype=torch.float32, device="cuda")
    torch.cuda.synchronize()
    # Plain dense attention (no scratch) loads the library's module first.
    wise.wise_full_attn_accumulate(shape, Q, K, V, O)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for step in range(3):
        wise.wise_full_attn_accumulate_noalloc(shape, Q, K, V, O, mass, step)
    torch.cuda.synchronize()
    free1 = torch.cuda.mem_get_info()[0]
    print(free0, free1, wise.wise_get_status())
""")


def test_noalloc_allocates_nothing_in_a_fresh_process():
    # A fresh process whose first block-mass calls are the no-allocation
    # ones: free device memory must not change across them.  (The allocating
    # entry point would take its scratch, several MiB, with cudaMalloc on its
    # first call; modules are loaded eagerly so that loading a kernel is not
    # mistaken for an allocation.)
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, CUDA_MODULE_LOADING="EAGER")
    r = subprocess.run([sys.executable, "-c", _FRESH_PROCESS, root], capture_output=True, text=True, env=env,
                       timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    free0, free1, status = (int(x) for x in r.stdout.split()[-3:])
    assert status == wise.WISE_OK
    assert free1 == free0, f"device memory changed by {free0 - free1} bytes across the no-allocation calls"
