"""GPU parity of the three kernels against the fp64 oracle, through the C ABI.

Sizes are small enough for the oracle to finish in seconds yet span several
128-row query tiles, ragged tails (a half query tile with block 64, a quarter
or three quarters of one with block 32), head dims 64/96/128, blocks
32/64/128, grouped-query attention and batch > 1.
Tolerances: O within max-abs 1e-2 and rel-L2 5e-3 of fp64; per-step block
mass within 1e-4; supports bit-exact against the oracle's selection run on
the GPU's own fp32 masses.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_27373_gb300 import synth, wise
from gpu_helpers import (MASS_MAX_ABS, MASS_ROWSUM, assert_close_o, bf16_dev_to_f64, empty_like_q, to_dev)

pytestmark = pytest.mark.gpu

CASES = {
    "d128_b128": (1, 2, 2, 640, 128, 128),
    "d64_b64_ragged": (1, 3, 3, 576, 64, 64),
    "d96_b128_batch2": (2, 3, 3, 512, 96, 128),
    "d128_gqa": (1, 4, 2, 512, 128, 128),
    "d128_b64_gqa": (1, 2, 1, 384, 128, 64),
    "d96_b64": (1, 2, 2, 320, 96, 64),
    "d64_single_block": (1, 1, 1, 128, 64, 128),
    # Block 32 (the paper's default): four query and four key blocks per tile.
    "d128_b32": (1, 2, 2, 640, 128, 32),
    "d64_b32_gqa_ragged": (1, 4, 2, 480, 64, 32),
    "d96_b32_batch2": (2, 2, 1, 352, 96, 32),
}


def _inputs(name, seed=0, std=1.0):
    B, H, Hkv, L, D, blk = CASES[name]
    # V stays N(0, 1) (as in the workloads) so |O| stays where a bf16 output
    # rounding is below the max-abs bound; std sharpens the attention only.
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=seed + sum(name.encode()) % 1000, std=std, v_std=1.0)
    return wise.Shape(B, L, H, Hkv, D, blk), Q, K, V


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    wise.load()
    assert wise.wise_get_status() == wise.WISE_OK


def _dense(shape, Q, K, V, mass=None, step=0):
    dQ, dK, dV = to_dev(Q), to_dev(K), to_dev(V)
    O = empty_like_q(Q)
    wise.wise_full_attn_accumulate(shape, dQ, dK, dV, O, mass, step)
    torch.cuda.synchronize()
    return O


@pytest.mark.parametrize("name", list(CASES))
def test_dense_attention_matches_oracle(name):
    shape, Q, K, V = _inputs(name)
    O = _dense(shape, Q, K, V)
    want, _ = orc.full_attention(Q, K, V, shape.block, with_mass=False)
    assert_close_o(bf16_dev_to_f64(O), want)
    assert wise.wise_get_status() == wise.WISE_OK


@pytest.mark.parametrize("name", list(CASES))
def test_block_mass_matches_oracle_and_accumulates(name):
    shape, Q, K, V = _inputs(name, std=2.0)
    nb = shape.n_blocks
    mass = torch.full((shape.batch, shape.n_heads, nb, nb), 7.0, dtype=torch.float32, device="cuda")
    O0 = _dense(shape, Q, K, V, mass, step=0)
    m0 = mass.cpu().numpy().astype(np.float64)
    _, r_ref = orc.full_attention(Q, K, V, shape.block)
    # Q/K at std 2 give logits of std 4: sharp rows whose bf16 P and O
    # roundings alone approach 1e-2, so O is checked bit for bit against the
    # plain dense kernel (whose parity is tested at workload scale) instead.
    assert np.abs(m0 - r_ref).max() <= MASS_MAX_ABS
    assert np.abs(m0.sum(-1) - 1.0).max() <= MASS_ROWSUM
    assert np.all(np.triu(m0, k=1) == 0.0), "step 0 must overwrite the whole row"
    # the plain dense variant gives the same O up to bf16 rounding of the last bit
    O_plain = _dense(shape, Q, K, V)
    a, b = bf16_dev_to_f64(O_plain), bf16_dev_to_f64(O0)
    ulp = np.exp2(np.floor(np.log2(np.maximum(np.maximum(np.abs(a), np.abs(b)), 1e-30))) - 7)
    assert np.all(np.abs(a - b) <= ulp)
    # a second step accumulates
    Q2, K2, V2 = synth.random_qkv(shape.batch, shape.n_heads, shape.n_kv_heads, shape.seqlen, shape.head_dim,
                                  seed=77, std=2.0, v_std=1.0)
    _dense(shape, Q2, K2, V2, mass, step=1)
    m01 = mass.cpu().numpy().astype(np.float64)
    _, r2 = orc.full_attention(Q2, K2, V2, shape.block)
    assert np.abs(m01 - (r_ref + r2)).max() <= 2 * MASS_MAX_ABS
    assert np.abs(m01.sum(-1) - 2.0).max() <= 2 * MASS_ROWSUM


SELECTIONS = [
    wise.Select(1, 1, wise.WISE_SEL_TOPK, 2, 0.0, 4),
    wise.Select(1, 2, wise.WISE_SEL_TOPK, 3, 0.0, 6),
    wise.Select(1, 1, wise.WISE_SEL_COVERAGE, 0, 0.95, 8),
    wise.Select(2, 1, wise.WISE_SEL_COVERAGE, 0, 0.5, 5),
    wise.Select(0, 1, wise.WISE_SEL_COVERAGE, 0, 1.0, 64),
]


@pytest.mark.parametrize("sel", SELECTIONS, ids=lambda s: f"m{s.mode}k{s.topk}e{s.eta}c{s.cap}s{s.n_sink}l{s.n_local}")
@pytest.mark.parametrize("name", ["d128_b128", "d64_b64_ragged", "d128_gqa", "d96_b128_batch2", "d64_b32_gqa_ragged"])
def test_selection_is_bit_exact(name, sel):
    shape, Q, K, V = _inputs(name, std=2.0)
    nb = shape.n_blocks
    mass = torch.empty((shape.batch, shape.n_heads, nb, nb), dtype=torch.float32, device="cuda")
    _dense(shape, Q, K, V, mass, step=0)
    idx = torch.empty((shape.batch, shape.n_kv_heads, nb, sel.cap), dtype=torch.int32, device="cuda")
    counts = torch.empty((shape.batch, shape.n_kv_heads, nb), dtype=torch.int32, device="cuda")
    wise.wise_select_support(shape, sel, mass, idx, counts)
    want_idx, want_counts = orc.select_support(mass.cpu().numpy(), shape.n_kv_heads, shape.block, sel.mode,
                                               sel.n_sink, sel.n_local, sel.topk, sel.eta, sel.cap)
    np.testing.assert_array_equal(counts.cpu().numpy(), want_counts)
    np.testing.assert_array_equal(idx.cpu().numpy(), want_idx)


def test_selection_on_adversarial_masses_is_bit_exact():
    """Ties, zeros, negatives, NaN, huge values and values a few ulps apart."""
    rng = np.random.default_rng(3)
    B, H, Hkv, nb = 2, 8, 2, 40
    m = rng.choice(np.array([0.0, 0.25, 0.25, 0.5, 1e-8, -1.0, np.nan, 5000.0], np.float32), size=(B, H, nb, nb))
    m += np.float32(1e-7) * rng.integers(0, 3, size=m.shape).astype(np.float32)
    shape = wise.Shape(B, nb * 64, H, Hkv, 64, 64)
    dm = torch.from_numpy(m).cuda()
    for sel in SELECTIONS + [wise.Select(3, 3, wise.WISE_SEL_TOPK, 40, 0.0, 40)]:
        idx = torch.empty((B, Hkv, nb, sel.cap), dtype=torch.int32, device="cuda")
        counts = torch.empty((B, Hkv, nb), dtype=torch.int32, device="cuda")
        wise.wise_select_support(shape, sel, dm, idx, counts)
        wi, wc = orc.select_support(m, Hkv, 64, sel.mode, sel.n_sink, sel.n_local, sel.topk, sel.eta, sel.cap)
        np.testing.assert_array_equal(counts.cpu().numpy(), wc)
        np.testing.assert_array_equal(idx.cpu().numpy(), wi)


def _sparse(shape, Q, K, V, idx, counts):
    O = empty_like_q(Q)
    wise.wise_sparse_attn(shape, to_dev(Q), to_dev(K), to_dev(V), torch.from_numpy(idx).cuda(),
                          torch.from_numpy(counts).cuda(), O)
    torch.cuda.synchronize()
    return O


@pytest.mark.parametrize("name", list(CASES))
def test_sparse_attention_matches_oracle(name):
    shape, Q, K, V = _inputs(name)
    idx, counts = synth.random_support(shape.batch, shape.n_kv_heads, shape.n_blocks, 5, seed=4)
    O = _sparse(shape, Q, K, V, idx, counts)
    want = orc.sparse_attention(Q, K, V, idx, counts, shape.block)
    assert_close_o(bf16_dev_to_f64(O), want)
    assert wise.wise_get_status() == wise.WISE_OK


@pytest.mark.parametrize("name", list(CASES))
def test_sparse_with_all_blocks_equals_dense(name):
    """Eq. 8 with R == 0 is Eq. 2: same output bits as the dense kernel."""
    shape, Q, K, V = _inputs(name)
    idx, counts = synth.all_blocks_support(shape.batch, shape.n_kv_heads, shape.n_blocks)
    O_sp = _sparse(shape, Q, K, V, idx, counts)
    O_dn = _dense(shape, Q, K, V)
    assert torch.equal(O_sp.view(torch.int16), O_dn.view(torch.int16))


def test_sparse_rows_without_support_are_zero():
    shape, Q, K, V = _inputs("d64_b64_ragged")
    idx, counts = synth.random_support(shape.batch, shape.n_kv_heads, shape.n_blocks, 4, seed=5)
    counts[0, 1, :] = 0          # a whole head without support
    counts[0, 0, 3] = 0          # one query block without support
    O = _sparse(shape, Q, K, V, idx, counts)
    want = orc.sparse_attention(Q, K, V, idx, counts, shape.block)
    got = bf16_dev_to_f64(O)
    assert np.all(got[0, 1] == 0.0)
    assert np.all(got[0, 0, 3 * 64:4 * 64] == 0.0)
    assert_close_o(got, want)


@pytest.mark.parametrize("name", ["d128_b128", "d64_b64_ragged", "d128_b32", "d64_b32_gqa_ragged"])
def test_inconsistent_support_is_skipped_and_flagged(name):
    """Blocks 32 and 64 take their tile schedules from the staging warp, block
    128 from the producer's own merge: both keep the same entries."""
    shape, Q, K, V = _inputs(name)
    nb = shape.n_blocks
    idx, counts = synth.random_support(shape.batch, shape.n_kv_heads, nb, 4, seed=6)
    bad_idx, bad_counts = idx.copy(), counts.copy()
    if counts[0, 0, 2] < 4:
        bad_idx[0, 0, 2, counts[0, 0, 2]] = nb + 5  # beyond the row's count: ignored, no flag
    bad_idx[0, 1, 3, :] = [3, 1, 1, -1]             # unordered, duplicate
    bad_counts[0, 1, 3] = 3
    bad_counts[0, 1, 4] = 99                        # over cap: clamped
    O = _sparse(shape, Q, K, V, bad_idx, bad_counts)
    assert wise.wise_get_status() == wise.WISE_ERR_BAD_SUPPORT
    assert wise.wise_get_status() == wise.WISE_OK, "the status word is cleared by reading it"
    # the kernel keeps each row's valid ascending prefix entries
    fixed_idx, fixed_counts = bad_idx.copy(), bad_counts.copy()
    fixed_idx[0, 1, 3, :] = [3, -1, -1, -1]
    fixed_counts[0, 1, 3] = 1
    fixed_counts[0, 1, 4] = counts[0, 1, 4]
    want = orc.sparse_attention(Q, K, V, fixed_idx, fixed_counts, shape.block)
    assert_close_o(bf16_dev_to_f64(O), want)


@pytest.mark.parametrize("name", ["d128_b32", "d64_b32_gqa_ragged", "d64_b64_ragged", "d128_b64_gqa"])
def test_staged_and_merged_schedules_agree(name):
    """Blocks 32 and 64 take their tile schedules from the staging warp while
    cap * (128 / B) <= 128, else from the producer's own merge of the lists.
    The same support, stored once at the largest staged cap and once with one
    more (empty) column, must give the same output bits, valid or not."""
    shape, Q, K, V = _inputs(name)
    nb, S = shape.n_blocks, 128 // shape.block
    cap = 128 // S
    idx, counts = synth.random_support(shape.batch, shape.n_kv_heads, nb, cap, seed=7, density=0.6)
    # one malformed row (unordered, duplicate, out of range) in both layouts
    q = min(5, nb - 1)
    idx[0, 0, q, :4] = [q, 0, 0, nb + 3]
    counts[0, 0, q] = 4
    wide = np.full(idx.shape[:-1] + (cap + 1,), -1, dtype=np.int32)
    wide[..., :cap] = idx
    O_staged = _sparse(shape, Q, K, V, idx, counts)
    st_staged = wise.wise_get_status()
    O_merged = _sparse(shape, Q, K, V, wide, counts)
    st_merged = wise.wise_get_status()
    assert st_staged == st_merged == wise.WISE_ERR_BAD_SUPPORT
    assert torch.equal(O_staged.view(torch.int16), O_merged.view(torch.int16))
    fixed_idx, fixed_counts = idx.copy(), counts.copy()
    fixed_idx[0, 0, q, :4] = [q, -1, -1, -1]
    fixed_counts[0, 0, q] = 1
    want = orc.sparse_attention(Q, K, V, fixed_idx, fixed_counts, shape.block)
    assert_close_o(bf16_dev_to_f64(O_staged), want)


def test_tiny_workload_trajectory_end_to_end():
    """The tiny workload (L=512, 4 heads, d=64, block 64): 3 discovery steps,
    one selection, 5 late steps, through the WiseAttention driver."""
    wl = synth.WORKLOADS["tiny"]
    shape, sel = wise.shape_of(wl), wise.select_of(wl)
    layer = wise.WiseAttention(shape, sel, wl.n_discovery)
    traj = synth.Trajectory(wl)
    acc = None
    for t in range(wl.steps):
        Q, K, V = traj.step(t)
        O = empty_like_q(Q)
        layer.step(t, to_dev(Q), to_dev(K), to_dev(V), O)
        torch.cuda.synchronize()
        if t < wl.n_discovery:
            want, r = orc.full_attention(Q, K, V, wl.block)
            acc = r if acc is None else acc + r
            assert np.abs(layer.blockmass.cpu().numpy() - acc).max() <= (t + 1) * MASS_MAX_ABS
        else:
            if t == wl.n_discovery:
                gi, gc = layer.idx.cpu().numpy(), layer.counts.cpu().numpy()
                wi, wc = orc.select_support(layer.blockmass.cpu().numpy(), wl.n_kv_heads, wl.block, wl.sel_mode,
                                            wl.n_sink, wl.n_local, wl.topk, wl.eta, wl.cap)
                np.testing.assert_array_equal(gc, wc)
                np.testing.assert_array_equal(gi, wi)
            want = orc.sparse_attention(Q, K, V, gi, gc, wl.block)
        assert_close_o(bf16_dev_to_f64(O), want, what=f"step {t}")
    assert wise.wise_get_status() == wise.WISE_OK
