"""Freeze-A control and the support overlap through the C ABI, against the
oracle.

wise_freeze_a_attn: O = Abar V, Abar the frozen step's attention restricted
to the support and renormalised (the oracle forms A, restricts and
renormalises it, in fp64); tolerance of the attention outputs.
wise_support_overlap: exact integer counts, compared bit for bit.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_27373_gb300 import synth, wise
from gpu_helpers import assert_close_o, bf16_dev_to_f64, to_dev

pytestmark = pytest.mark.gpu


def _f64(bits):
    return synth.bf16_bits_to_f32(bits).astype(np.float64)


@pytest.mark.parametrize("B,H,Hkv,L,D,blk,cap", [(1, 4, 4, 1152, 128, 128, 5), (2, 4, 2, 704, 64, 64, 6),
                                                 (1, 3, 1, 640, 96, 128, 3)])
def test_freeze_a_matches_the_definition(B, H, Hkv, L, D, blk, cap):
    """Frozen Q, K of one step, V of another step, a random support spanning
    several tiles and a ragged last query tile; N(0, 1) logits as in the
    workloads (sharper rows make the bf16 roundings of P and O alone approach
    the max-abs bound)."""
    shape = wise.Shape(B, L, H, Hkv, D, blk)
    Q0, K0, _ = synth.random_qkv(B, H, Hkv, L, D, seed=60)
    _, _, V1 = synth.random_qkv(B, H, Hkv, L, D, seed=61)
    idx, counts = synth.random_support(B, Hkv, shape.n_blocks, cap, seed=62, density=0.5)
    O = torch.empty((B, H, L, D), dtype=torch.bfloat16, device="cuda")
    wise.wise_freeze_a_attn(shape, to_dev(Q0), to_dev(K0), to_dev(V1), torch.from_numpy(idx).cuda(),
                            torch.from_numpy(counts).cuda(), O)
    assert wise.wise_get_status() == wise.WISE_OK
    want = orc.freeze_a(_f64(Q0), _f64(K0), _f64(V1), idx, counts, blk)
    assert_close_o(bf16_dev_to_f64(O), want, "Freeze-A O")


def test_freeze_a_with_current_q_k_is_the_sparse_step():
    """Freezing at the current step is the sparse step itself, bit for bit."""
    B, H, Hkv, L, D, blk = 1, 4, 2, 1024, 128, 128
    shape = wise.Shape(B, L, H, Hkv, D, blk)
    Q, K, V = (to_dev(x) for x in synth.random_qkv(B, H, Hkv, L, D, seed=63))
    idx, counts = synth.random_support(B, Hkv, shape.n_blocks, 4, seed=64)
    di, dc = torch.from_numpy(idx).cuda(), torch.from_numpy(counts).cuda()
    O1 = torch.empty_like(Q)
    O2 = torch.empty_like(Q)
    wise.wise_freeze_a_attn(shape, Q, K, V, di, dc, O1)
    wise.wise_sparse_attn(shape, Q, K, V, di, dc, O2)
    assert wise.wise_get_status() == wise.WISE_OK
    assert torch.equal(O1.view(torch.int16), O2.view(torch.int16))


def _overlap(shape, ia, ca, ib, cb):
    out = torch.full((shape.batch, 2), -1, dtype=torch.int64, device="cuda")
    wise.wise_support_overlap(shape, torch.from_numpy(ia).cuda(), torch.from_numpy(ca).cuda(),
                              torch.from_numpy(ib).cuda(), torch.from_numpy(cb).cuda(), out)
    return out.cpu().numpy()


@pytest.mark.parametrize("B,Hkv,L,blk,cap_a,cap_b", [(2, 3, 4096, 128, 8, 5), (3, 2, 2048, 64, 11, 11),
                                                     (1, 8, 32768, 128, 15, 32)])
def test_overlap_matches_oracle(B, Hkv, L, blk, cap_a, cap_b):
    shape = wise.Shape(B, L, Hkv, Hkv, 128, blk)
    nb = shape.n_blocks
    ia, ca = synth.random_support(B, Hkv, nb, cap_a, seed=65, density=0.4)
    ib, cb = synth.random_support(B, Hkv, nb, cap_b, seed=66, density=0.6)
    got = _overlap(shape, ia, ca, ib, cb)
    assert wise.wise_get_status() == wise.WISE_OK
    np.testing.assert_array_equal(got, orc.support_overlap(ia, ca, ib, cb))
    same = _overlap(shape, ia, ca, ia, ca)
    np.testing.assert_array_equal(same[:, 0], ca.sum(axis=(1, 2)))
    np.testing.assert_array_equal(same[:, 1], ca.sum(axis=(1, 2)))


def test_overlap_skips_and_reports_malformed_entries():
    B, Hkv, L, blk, cap = 1, 2, 1024, 128, 4
    shape = wise.Shape(B, L, Hkv, Hkv, 128, blk)
    nb = shape.n_blocks
    ia, ca = synth.random_support(B, Hkv, nb, cap, seed=67, density=0.5)
    ib, cb = synth.random_support(B, Hkv, nb, cap, seed=68, density=0.5)
    ia[0, 0, 5, 0] = 7          # beyond query block 5
    ib[0, 1, 3, 1] = ib[0, 1, 3, 0]  # repeated entry
    cb[0, 1, 6] = cap + 3       # count over the row width
    got = _overlap(shape, ia, ca, ib, cb)
    assert wise.wise_get_status() == wise.WISE_ERR_BAD_SUPPORT
    np.testing.assert_array_equal(got, orc.support_overlap(ia, ca, ib, cb))


def test_overlap_of_empty_supports_is_zero():
    B, Hkv, L, blk = 2, 2, 512, 128
    shape = wise.Shape(B, L, Hkv, Hkv, 128, blk)
    nb = shape.n_blocks
    idx = np.full((B, Hkv, nb, 3), -1, dtype=np.int32)
    counts = np.zeros((B, Hkv, nb), dtype=np.int32)
    got = _overlap(shape, idx, counts, idx, counts)
    assert wise.wise_get_status() == wise.WISE_OK
    np.testing.assert_array_equal(got, np.zeros((B, 2), dtype=np.int64))


def test_rolling_working_sets_of_consecutive_steps():
    """The appendix statistic on a synthetic trajectory: W(t) = union of the
    eta sets of steps t-3..t (WS_UNION), overlap of W(t-1) and W(t) on the
    GPU equals the oracle's sets built from the same GPU masses."""
    B, H, Hkv, L, D, blk = 1, 4, 2, 1024, 64, 64
    shape = wise.Shape(B, L, H, Hkv, D, blk)
    nb = shape.n_blocks
    steps = 6
    wl = synth.WORKLOADS["4k"].scaled(batch=B, seqlen=L, n_heads=H, n_kv_heads=Hkv, head_dim=D, block=blk,
                                      steps=steps, seed=9)
    traj = synth.Trajectory(wl)
    masses = torch.empty((steps, B, H, nb, nb), dtype=torch.float32, device="cuda")
    O = torch.empty((B, H, L, D), dtype=torch.bfloat16, device="cuda")
    for t in range(steps):
        Q, K, V = (to_dev(x) for x in traj.step(t))
        wise.wise_full_attn_accumulate(shape, Q, K, V, O, masses[t], 0)
    sets = []
    for t in (steps - 2, steps - 1):
        lo = max(0, t - 3)
        idx = torch.empty((B, Hkv, nb, nb), dtype=torch.int32, device="cuda")
        cnt = torch.empty((B, Hkv, nb), dtype=torch.int32, device="cuda")
        wise.wise_select_working_set(shape, wise.WS_UNION, masses[lo:t + 1].contiguous(), idx, cnt, eta=0.95,
                                     n_sink=1, n_local=1)
        sets.append((idx.cpu().numpy(), cnt.cpu().numpy()))
    got = _overlap(shape, sets[0][0], sets[0][1], sets[1][0], sets[1][1])
    assert wise.wise_get_status() == wise.WISE_OK
    np.testing.assert_array_equal(got, orc.support_overlap(sets[0][0], sets[0][1], sets[1][0], sets[1][1]))
    j = got[0, 0] / got[0, 1]
    assert 0.5 < j <= 1.0
