"""wise_select_working_set (Eq. 6 union and the intervention controls)
through the C ABI: bit-exact against the oracle run on the GPU's fp32
per-step masses (both use the same exact fixed-point rule)."""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_27373_gb300 import synth, wise
from gpu_helpers import to_dev

pytestmark = pytest.mark.gpu


def _step_masses(shape, n_steps, seed):
    nb = shape.n_blocks
    out = torch.empty((n_steps, shape.batch, shape.n_heads, nb, nb), dtype=torch.float32, device="cuda")
    O = torch.empty((shape.batch, shape.n_heads, shape.seqlen, shape.head_dim), dtype=torch.bfloat16, device="cuda")
    for s in range(n_steps):
        Q, K, V = synth.random_qkv(shape.batch, shape.n_heads, shape.n_kv_heads, shape.seqlen, shape.head_dim,
                                   seed=seed + s, std=1.6, v_std=1.0)
        wise.wise_full_attn_accumulate(shape, to_dev(Q), to_dev(K), to_dev(V), O, out[s], 0)
    return out


@pytest.mark.parametrize("B,H,Hkv,L,D,blk", [(1, 4, 4, 2048, 64, 128), (2, 4, 2, 1024, 64, 64)])
def test_working_sets_match_oracle(B, H, Hkv, L, D, blk):
    shape = wise.Shape(B, L, H, Hkv, D, blk)
    nb = shape.n_blocks
    masses = _step_masses(shape, 4, seed=60)
    m_host = masses.cpu().numpy()

    def run(mode, m, **kw):
        idx = torch.full((B, Hkv, nb, nb), -9, dtype=torch.int32, device="cuda")
        cnt = torch.full((B, Hkv, nb), -9, dtype=torch.int32, device="cuda")
        wise.wise_select_working_set(shape, mode, m, idx, cnt, **kw)
        return idx.cpu().numpy(), cnt.cpu().numpy()

    union = run(wise.WS_UNION, masses, eta=0.95)
    want = orc.working_set(0, m_host, Hkv, eta=0.95)
    assert np.array_equal(union[0], want[0]) and np.array_equal(union[1], want[1])
    static = run(wise.WS_STATIC, masses[:1], eta=0.95, n_sink=1, n_local=1)
    want = orc.working_set(1, m_host[:1], Hkv, eta=0.95, n_sink=1, n_local=1)
    assert np.array_equal(static[0], want[0]) and np.array_equal(static[1], want[1])
    ref_i, ref_c = (torch.from_numpy(x).cuda() for x in union)
    for mode, omode in ((wise.WS_MASS_MATCHED, 2), (wise.WS_SIZE_MATCHED, 3)):
        got = run(mode, masses[:1], ref_idx=ref_i, ref_counts=ref_c)
        want = orc.working_set(omode, m_host[:1], Hkv, ref_idx=union[0], ref_counts=union[1])
        assert np.array_equal(got[0], want[0]) and np.array_equal(got[1], want[1])
    assert wise.wise_get_status() == wise.WISE_OK
    # the union holds every step's own coverage set, so it is at least as large
    assert np.all(union[1] >= static[1] - 2)


def test_working_set_feeds_the_sparse_kernel():
    # The paper's working set of 4 steps, then attention restricted to it,
    # against the oracle's support-restricted attention on that support.
    B, H, Hkv, L, D, blk = 1, 2, 2, 1024, 64, 128
    shape = wise.Shape(B, L, H, Hkv, D, blk)
    nb = shape.n_blocks
    masses = _step_masses(shape, 4, seed=70)
    idx = torch.empty((B, Hkv, nb, nb), dtype=torch.int32, device="cuda")
    cnt = torch.empty((B, Hkv, nb), dtype=torch.int32, device="cuda")
    wise.wise_select_working_set(shape, wise.WS_UNION, masses, idx, cnt, eta=0.95)
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=74)
    O = torch.empty((B, H, L, D), dtype=torch.bfloat16, device="cuda")
    wise.wise_sparse_attn(shape, to_dev(Q), to_dev(K), to_dev(V), idx, cnt, O)
    assert wise.wise_get_status() == wise.WISE_OK
    from gpu_helpers import assert_close_o, bf16_dev_to_f64
    want = orc.sparse_attention(Q, K, V, idx.cpu().numpy(), cnt.cpu().numpy(), blk)
    assert_close_o(bf16_dev_to_f64(O), want, what="sparse on the Eq. 6 working set")


def test_working_set_rejects_a_short_row_width():
    shape = wise.Shape(1, 1024, 2, 2, 64, 128)
    masses = torch.zeros((1, 1, 2, 8, 8), dtype=torch.float32, device="cuda")
    idx = torch.empty((1, 2, 8, 7), dtype=torch.int32, device="cuda")
    cnt = torch.empty((1, 2, 8), dtype=torch.int32, device="cuda")
    with pytest.raises(wise.WiseError) as e:
        wise.wise_select_working_set(shape, wise.WS_STATIC, masses, idx, cnt)
    assert e.value.code == wise.WISE_ERR_INVALID_ARG
