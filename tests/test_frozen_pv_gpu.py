"""Freeze-A with a stored distribution through the C ABI, against the oracle.

wise_freeze_a_probs stores Abar (the frozen step's attention restricted to the
support and renormalised) as row-max-relative bf16 128 x 128 tiles in the
order of each query tile's support walk and a per-row 1 / sum; the test
gathers the tiles back into a dense [L, L] matrix, scales the rows and
compares with the oracle's Abar (bf16 rounding of values <= 1: max-abs 4e-3;
masked entries exactly 0).  wise_frozen_pv (O = Abar V) is compared
with the oracle's Freeze-A output at the attention tolerance, and with the
recomputing entry point wise_freeze_a_attn.
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


def _walk(idx, counts, b, g, qt, S, n_blocks):
    """Key tiles of query tile qt: those holding a used entry of one of its S
    query blocks' lists, ascending."""
    tiles = set()
    for q in range(qt * S, min(qt * S + S, n_blocks)):
        n = min(max(int(counts[b, g, q]), 0), idx.shape[3])
        prev = -1
        for v in idx[b, g, q, :n]:
            v = int(v)
            if 0 <= v <= q and v > prev:
                tiles.add(v // S)
                prev = v
    return sorted(tiles)


def _gather(P, inv_l, shape, idx, counts):
    B, H, Hkv, L = shape.batch, shape.n_heads, shape.n_kv_heads, shape.seqlen
    S = 128 // shape.block
    nqt = (L + 127) // 128
    Pd = bf16_dev_to_f64(P) * inv_l.cpu().numpy().astype(np.float64)[:, None, :, None]
    dense = np.zeros((B, H, L, L))
    for b in range(B):
        for h in range(H):
            for qt in range(nqt):
                u = (b * H + h) * nqt + qt
                rows = slice(qt * 128, min(qt * 128 + 128, L))
                nr = rows.stop - rows.start
                for t, kt in enumerate(_walk(idx, counts, b, h // (H // Hkv), qt, S, shape.n_blocks)):
                    cols = slice(kt * 128, min(kt * 128 + 128, L))
                    dense[b, h, rows, cols] = Pd[u, t, :nr, :cols.stop - cols.start]
    return dense


CASES = [(1, 4, 4, 1152, 128, 128, 5), (2, 4, 2, 704, 64, 64, 6), (1, 2, 1, 640, 96, 32, 12),
         (1, 3, 3, 512, 128, 32, 9)]


@pytest.mark.parametrize("B,H,Hkv,L,D,blk,cap", CASES)
def test_stored_distribution_and_frozen_pv_match_the_definition(B, H, Hkv, L, D, blk, cap):
    shape = wise.Shape(B, L, H, Hkv, D, blk)
    nb = shape.n_blocks
    Q0, K0, _ = synth.random_qkv(B, H, Hkv, L, D, seed=70)
    _, _, V1 = synth.random_qkv(B, H, Hkv, L, D, seed=71)
    idx, counts = synth.random_support(B, Hkv, nb, cap, seed=72, density=0.5)
    di, dc = torch.from_numpy(idx).cuda(), torch.from_numpy(counts).cuda()
    n_units = B * H * ((L + 127) // 128)
    tile_cap = wise.freeze_tile_cap(shape, cap)
    P = torch.zeros((n_units, tile_cap, 128, 128), dtype=torch.bfloat16, device="cuda")
    inv_l = torch.empty((n_units, 128), dtype=torch.float32, device="cuda")
    wise.wise_freeze_a_probs(shape, to_dev(Q0), to_dev(K0), di, dc, P, inv_l)
    O = torch.empty((B, H, L, D), dtype=torch.bfloat16, device="cuda")
    wise.wise_frozen_pv(shape, P, inv_l, to_dev(V1), di, dc, O)
    assert wise.wise_get_status() == wise.WISE_OK
    abar = orc.freeze_a_distribution(_f64(Q0), _f64(K0), idx, counts, blk)
    got = _gather(P, inv_l, shape, idx, counts)
    assert np.abs(got - abar).max() <= 4e-3
    assert np.all(got[abar == 0.0] == 0.0)
    want = orc.freeze_a(_f64(Q0), _f64(K0), _f64(V1), idx, counts, blk)
    assert_close_o(bf16_dev_to_f64(O), want, "frozen P V")
    O2 = torch.empty_like(O)
    wise.wise_freeze_a_attn(shape, to_dev(Q0), to_dev(K0), to_dev(V1), di, dc, O2)
    assert_close_o(bf16_dev_to_f64(O), bf16_dev_to_f64(O2).astype(np.float64), "frozen P V vs recomputed")


def test_frozen_pv_at_the_4k_workload_size():
    """The 4K workload's shape and selected support; two sampled heads of the
    output checked against the oracle's Freeze-A (fp64)."""
    wl = synth.WORKLOADS["4k"]
    shape, sel = wise.shape_of(wl), wise.select_of(wl)
    layer = wise.WiseAttention(shape, sel, wl.n_discovery)
    traj = synth.Trajectory(wl)
    for t in range(wl.n_discovery + 1):
        Q, K, V = traj.step(t)
        O = torch.empty(Q.shape, dtype=torch.bfloat16, device="cuda")
        layer.step(t, to_dev(Q), to_dev(K), to_dev(V), O)
    _, _, V1 = traj.step(wl.n_discovery + 1)
    n_units = wl.batch * wl.n_heads * (wl.seqlen // 128)
    tile_cap = wise.freeze_tile_cap(shape, wl.cap)
    P = torch.empty((n_units, tile_cap, 128, 128), dtype=torch.bfloat16, device="cuda")
    inv_l = torch.empty((n_units, 128), dtype=torch.float32, device="cuda")
    wise.wise_freeze_a_probs(shape, to_dev(Q), to_dev(K), layer.idx, layer.counts, P, inv_l)
    Of = torch.empty_like(O)
    wise.wise_frozen_pv(shape, P, inv_l, to_dev(V1), layer.idx, layer.counts, Of)
    assert wise.wise_get_status() == wise.WISE_OK
    heads = [3, 20]  # no GQA in this workload: kv head = query head
    idx, counts = layer.idx.cpu().numpy()[:, heads], layer.counts.cpu().numpy()[:, heads]
    want = orc.freeze_a(_f64(Q)[:, heads], _f64(K)[:, heads], _f64(V1)[:, heads], idx, counts, wl.block)
    assert_close_o(bf16_dev_to_f64(Of)[:, heads], want, "frozen P V, 4K")


def test_tile_cap_below_the_walk_bound_is_rejected():
    shape = wise.Shape(1, 512, 2, 2, 64, 64)
    idx, counts = synth.random_support(1, 2, shape.n_blocks, 4, seed=1)
    P = torch.empty((8, 3, 128, 128), dtype=torch.bfloat16, device="cuda")
    inv_l = torch.empty((8, 128), dtype=torch.float32, device="cuda")
    Q = torch.zeros((1, 2, 512, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(wise.WiseError):
        wise.wise_freeze_a_probs(shape, Q, Q, torch.from_numpy(idx).cuda(), torch.from_numpy(counts).cuda(), P,
                                 inv_l)
