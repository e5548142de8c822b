"""Failure detection on the GPU: a kernel wait that runs out is reported, and
the device stays usable.

Every wait inside the attention kernels is bounded by the launch's limit
(wise_set_wait_limit_ns, 2 s by default).  Here the limit is set to 1 ns for
one call on a 4K problem, so that the first wait that does not succeed at
once gives up: the kernel sets its abort flag and the status word, lets the
copies and products already in flight finish (those waits keep the 2 s
limit), frees its tensor memory and returns.  The host then reads
WISE_ERR_TIMEOUT from wise_get_status(), and a normal call on the same
device still matches the oracle.  No GPU fault, trap or endless wait is
involved: the wait that runs out is an ordinary bounded wait given a short
limit.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_27373_gb300 import synth, wise
from gpu_helpers import assert_close_o, bf16_dev_to_f64, empty_like_q, to_dev

pytestmark = pytest.mark.gpu


def _short_limit_call(fn, tries=3):
    # A wait whose phase completes while the waiting thread is suspended in
    # its first probe never consults the clock, so one launch is not certain
    # to run out; a few launches make it so.
    status = wise.WISE_OK
    wise.wise_set_wait_limit_ns(1)
    try:
        for _ in range(tries):
            fn()
            status = wise.wise_get_status()
            if status != wise.WISE_OK:
                break
    finally:
        wise.wise_set_wait_limit_ns(0)
    return status


@pytest.mark.parametrize("mode", ["dense", "dense_mass", "sparse"])
def test_a_wait_that_runs_out_is_reported_and_the_device_stays_usable(mode):
    assert torch.cuda.is_available()
    wise.load()
    assert wise.wise_get_status() == wise.WISE_OK
    B, H, L, D, blk = 1, 32, 4096, 128, 128
    shape = wise.Shape(B, L, H, H, D, blk)
    nb = shape.n_blocks
    Q, K, V = (to_dev(x) for x in synth.random_qkv(B, H, H, L, D, seed=5))
    O = torch.empty_like(Q)
    mass = torch.zeros((B, H, nb, nb), dtype=torch.float32, device="cuda")
    idx, counts = synth.random_support(B, H, nb, 8, seed=6, density=0.5)
    di, dc = torch.from_numpy(idx).cuda(), torch.from_numpy(counts).cuda()

    def call():
        if mode == "dense":
            wise.wise_full_attn_accumulate(shape, Q, K, V, O)
        elif mode == "dense_mass":
            wise.wise_full_attn_accumulate(shape, Q, K, V, O, mass, 0)
        else:
            wise.wise_sparse_attn(shape, Q, K, V, di, dc, O)

    call()  # warm-up with the default limit (loads the kernel, allocates the mass scratch)
    assert wise.wise_get_status() == wise.WISE_OK
    assert _short_limit_call(call) == wise.WISE_ERR_TIMEOUT
    # The status word was cleared by the read; the device and the library
    # work normally again, with the default limit.
    assert wise.wise_get_status() == wise.WISE_OK
    b2 = (1, 2, 2, 640, 128, 128)
    Bs, Hs, Hkv, Ls, Ds, blks = b2
    Qs, Ks, Vs = synth.random_qkv(Bs, Hs, Hkv, Ls, Ds, seed=9)
    small = wise.Shape(Bs, Ls, Hs, Hkv, Ds, blks)
    Os = empty_like_q(Qs)
    wise.wise_full_attn_accumulate(small, to_dev(Qs), to_dev(Ks), to_dev(Vs), Os)
    torch.cuda.synchronize()
    want, _ = orc.full_attention(Qs, Ks, Vs, blks, with_mass=False)
    assert_close_o(bf16_dev_to_f64(Os), want)
    assert wise.wise_get_status() == wise.WISE_OK
    # And the large call itself completes with the default limit.
    call()
    assert wise.wise_get_status() == wise.WISE_OK


def test_wait_limit_setter_restores_the_default():
    wise.load()
    wise.wise_set_wait_limit_ns(5_000_000)
    wise.wise_set_wait_limit_ns(0)
    with pytest.raises(ValueError):
        wise.wise_set_wait_limit_ns(-1)
