"""A whole recurrent trajectory captured as one CUDA graph and replayed.

The trajectory is the path of Table 2's "full trajectory" row: the discovery
steps (dense attention + block mass, Eqs. 2 and 5), one support selection
(Eq. 6) and the late steps (Eqs. 7-8), all through the C ABI.  Captured once
and replayed, it must give (i) a support that is bit-exact against the
oracle's selection run on the replay's own fp32 block mass, (ii) late-step
outputs within the O tolerance of the fp64 oracle, and (iii) every output,
block mass and support bit-identical to the same trajectory run eagerly.  A
second replay must reproduce the first bit for bit.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_27373_gb300 import synth, wise
from gpu_helpers import assert_close_o, bf16_dev_to_f64, sample_units, to_dev, units_of

pytestmark = pytest.mark.gpu


def _run(layer, steps, outs):
    for t, (Q, K, V) in enumerate(steps):
        layer.step(t, Q, K, V, outs[t])


@pytest.mark.parametrize("name", ["tiny", "4k"])
def test_trajectory_graph_replay_matches_oracle_and_eager(name):
    assert torch.cuda.is_available()
    wl = synth.WORKLOADS[name]
    shape, sel = wise.shape_of(wl), wise.select_of(wl)
    traj = synth.Trajectory(wl)
    checked = {wl.n_discovery, wl.steps - 1}  # first and last late steps
    host, steps = {}, []
    for t in range(wl.steps):
        bits = traj.step(t)
        if t in checked:
            host[t] = bits
        steps.append(tuple(to_dev(x) for x in bits))
    outs_e = [torch.empty_like(s[0]) for s in steps]
    outs_g = [torch.empty_like(s[0]) for s in steps]
    # Eager run first (its first block-mass call sets up the library's
    # scratch, which must happen outside a capture).
    eager = wise.WiseAttention(shape, sel, wl.n_discovery)
    _run(eager, steps, outs_e)
    torch.cuda.synchronize()
    assert wise.wise_get_status() == wise.WISE_OK

    layer = wise.WiseAttention(shape, sel, wl.n_discovery)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        _run(layer, steps, outs_g)
    g.replay()
    torch.cuda.synchronize()
    assert wise.wise_get_status() == wise.WISE_OK

    # (i) the support, bit-exact from the replay's own mass
    mass = layer.blockmass.cpu().numpy()
    wi, wc = orc.select_support(mass, wl.n_kv_heads, wl.block, wl.sel_mode, wl.n_sink, wl.n_local, wl.topk, wl.eta,
                                wl.cap)
    np.testing.assert_array_equal(layer.counts.cpu().numpy(), wc)
    np.testing.assert_array_equal(layer.idx.cpu().numpy(), wi)
    # (iii) bit-identical to the eager trajectory
    assert torch.equal(layer.blockmass, eager.blockmass)
    assert torch.equal(layer.idx, eager.idx) and torch.equal(layer.counts, eager.counts)
    for t in range(wl.steps):
        assert torch.equal(outs_g[t].view(torch.int16), outs_e[t].view(torch.int16)), f"step {t}"
    # (ii) late steps against the oracle on the replay's support
    units = None if name == "tiny" else sample_units(wl.batch, wl.n_heads, wl.n_blocks, 12, seed=wl.seed + 7)
    for t in sorted(checked):
        Q, K, V = host[t]
        want = orc.sparse_attention(Q, K, V, wi, wc, wl.block, units=units)
        got = bf16_dev_to_f64(outs_g[t])
        if units is not None:
            got = units_of(got, units, wl.block)
        assert_close_o(got, want, what=f"{name} late step {t}")
    # A second replay reproduces the first.
    first = [o.clone() for o in outs_g]
    g.replay()
    torch.cuda.synchronize()
    for t in range(wl.steps):
        assert torch.equal(outs_g[t].view(torch.int16), first[t].view(torch.int16)), f"replay 2, step {t}"
    assert wise.wise_get_status() == wise.WISE_OK
