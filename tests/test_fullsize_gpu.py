"""Parity at the full sizes of the five benchmark workloads, through the same
C-ABI calls and launch configuration the benchmark times.

Each workload runs its discovery steps (dense attention + block mass), one
selection and its first late step on the GPU.  The oracle checks sampled
(batch, head, query block) units of the first discovery step's output, of the
accumulated block mass and of the late step's output, and the whole support
(idx/counts) bit for bit from the GPU's fp32 block mass.  The 4K workload is
also checked on every unit (test_4k_every_unit), for its first and last late
steps.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_27373_gb300 import synth, wise
from gpu_helpers import MASS_MAX_ABS, MASS_ROWSUM, assert_close_o, bf16_dev_to_f64, empty_like_q, sample_units, to_dev, units_of

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["4k", "4k_b4_d96", "16k", "32k_gqa", "4k_b32"])
def test_workload_at_full_size(name):
    wl = synth.WORKLOADS[name]
    shape, sel = wise.shape_of(wl), wise.select_of(wl)
    layer = wise.WiseAttention(shape, sel, wl.n_discovery)
    traj = synth.Trajectory(wl)
    units = sample_units(wl.batch, wl.n_heads, wl.n_blocks, 10, seed=wl.seed)
    ref_mass = None
    for t in range(wl.n_discovery + 1):
        Q, K, V = traj.step(t)
        O = empty_like_q(Q)
        layer.step(t, to_dev(Q), to_dev(K), to_dev(V), O)
        torch.cuda.synchronize()
        if t < wl.n_discovery:
            want, r = orc.full_attention(Q, K, V, wl.block, units=units, with_mass=True)
            ref_mass = r if ref_mass is None else ref_mass + r
            if t == 0:
                assert_close_o(units_of(bf16_dev_to_f64(O), units, wl.block), want, what=f"{name} dense")
        else:
            got_mass = layer.blockmass.cpu().numpy().astype(np.float64)
            got_rows = np.stack([got_mass[b, h, q] for b, h, q in units])
            assert np.abs(got_rows - ref_mass).max() <= wl.n_discovery * MASS_MAX_ABS
            idx, counts = layer.idx.cpu().numpy(), layer.counts.cpu().numpy()
            wi, wc = orc.select_support(layer.blockmass.cpu().numpy(), wl.n_kv_heads, wl.block, wl.sel_mode,
                                        wl.n_sink, wl.n_local, wl.topk, wl.eta, wl.cap)
            np.testing.assert_array_equal(counts, wc)
            np.testing.assert_array_equal(idx, wi)
            assert counts.max() <= wl.cap and counts.min() >= 1
            want = orc.sparse_attention(Q, K, V, idx, counts, wl.block, units=units)
            assert_close_o(units_of(bf16_dev_to_f64(O), units, wl.block), want, what=f"{name} sparse")
    assert wise.wise_get_status() == wise.WISE_OK


def test_4k_every_unit():
    """The 4K workload with every (head, query block) unit checked: the first
    discovery step's output and block mass, the block mass accumulated over
    the four discovery steps, the selected support (bit-exact from the GPU's
    own mass) and two late steps (the first, t = 4, and the last, t = 31)."""
    wl = synth.WORKLOADS["4k"]
    shape, sel = wise.shape_of(wl), wise.select_of(wl)
    layer = wise.WiseAttention(shape, sel, wl.n_discovery)
    traj = synth.Trajectory(wl)
    ref_mass = None
    late_t = (wl.n_discovery, wl.steps - 1)
    for t in range(wl.steps):
        Q, K, V = traj.step(t)
        if t >= wl.n_discovery and t not in late_t:
            continue  # the support is fixed: skipped late steps change no state
        O = empty_like_q(Q)
        layer.step(t, to_dev(Q), to_dev(K), to_dev(V), O)
        torch.cuda.synchronize()
        if t < wl.n_discovery:
            want, r = orc.full_attention(Q, K, V, wl.block, with_mass=True)
            ref_mass = r if ref_mass is None else ref_mass + r
            if t == 0:
                assert_close_o(bf16_dev_to_f64(O), want, what="4k discovery step 0, every unit")
                got0 = layer.blockmass.cpu().numpy().astype(np.float64)
                assert np.abs(got0 - r).max() <= MASS_MAX_ABS
                assert np.abs(got0.sum(-1) - 1.0).max() <= MASS_ROWSUM
        else:
            if t == wl.n_discovery:
                got_mass = layer.blockmass.cpu().numpy()
                assert np.abs(got_mass.astype(np.float64) - ref_mass).max() <= wl.n_discovery * MASS_MAX_ABS
                wi, wc = orc.select_support(got_mass, wl.n_kv_heads, wl.block, wl.sel_mode, wl.n_sink, wl.n_local,
                                            wl.topk, wl.eta, wl.cap)
                np.testing.assert_array_equal(layer.counts.cpu().numpy(), wc)
                np.testing.assert_array_equal(layer.idx.cpu().numpy(), wi)
            want = orc.sparse_attention(Q, K, V, layer.idx.cpu().numpy(), layer.counts.cpu().numpy(), wl.block)
            assert_close_o(bf16_dev_to_f64(O), want, what=f"4k late step {t}, every unit")
    assert wise.wise_get_status() == wise.WISE_OK
