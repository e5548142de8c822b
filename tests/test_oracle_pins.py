"""Pins of the fp64 oracle to facts fixed by the paper and by mathematics.

None of these tests compares the oracle with itself.  Each one checks it
against a library routine (torch's fp64 scaled-dot-product attention and
softmax), a closed form, an invariant the equations imply, a hand-derived
case, or an exhaustive search over the definition, chosen so that a dropped
term, a wrong sign, a swapped index or a transposed operand fails at least
one of them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2609_27373_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bf16_vals(bits):
    return synth.bf16_bits_to_f32(bits).astype(np.float64)


def expand_kv(x, group):
    return np.repeat(x, group, axis=1)


def sdpa_reference(Q, K, V, group, attn_mask=None, is_causal=False, scale=None):
    """torch fp64 scaled_dot_product_attention on the widened bf16 values."""
    q = torch.from_numpy(bf16_vals(Q))
    k = torch.from_numpy(expand_kv(bf16_vals(K), group))
    v = torch.from_numpy(expand_kv(bf16_vals(V), group))
    m = None if attn_mask is None else torch.from_numpy(attn_mask)
    return torch.nn.functional.scaled_dot_product_attention(q, k, v, attn_mask=m, is_causal=is_causal,
                                                            scale=scale).numpy()


# --------------------------------------------------------------------------- Eq. 2

@pytest.mark.parametrize("B,H,Hkv,L,D,blk", [(2, 4, 2, 48, 8, 16), (1, 3, 3, 40, 5, 8), (1, 2, 1, 12, 3, 4)])
def test_full_attention_equals_library_causal_sdpa(B, H, Hkv, L, D, blk):
    """Eq. 2 with a causal M is torch's causal scaled-dot-product attention
    (scale 1/sqrt(d_h)); GQA heads share their group's K/V."""
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=11 + L)
    O, _ = orc.full_attention(Q, K, V, blk)
    ref = sdpa_reference(Q, K, V, H // Hkv, is_causal=True)
    np.testing.assert_allclose(O, ref, rtol=0, atol=1e-12)


def test_full_attention_custom_scale():
    Q, K, V = synth.random_qkv(1, 2, 2, 16, 4, seed=3)
    O, _ = orc.full_attention(Q, K, V, 4, scale=0.37)
    ref = sdpa_reference(Q, K, V, 1, is_causal=True, scale=0.37)
    np.testing.assert_allclose(O, ref, rtol=0, atol=1e-12)


def test_one_hot_routing_closed_form():
    """Query i aims at key j*(i) <= i with logit 16, every other admissible
    logit is 0: O_i = (e^16 V_j* + sum_{j<=i, j!=j*} V_j) / (e^16 + i)."""
    L = D = 16
    rng = np.random.default_rng(5)
    target = np.array([rng.integers(0, i + 1) for i in range(L)])
    K = np.zeros((1, 1, L, D), np.float32)
    Q = np.zeros((1, 1, L, D), np.float32)
    for j in range(L):
        K[0, 0, j, j] = 8.0
    for i in range(L):
        Q[0, 0, i, target[i]] = 8.0          # logit = (8*8) / sqrt(16) = 16
    V = rng.standard_normal((1, 1, L, D)).astype(np.float32)
    Qb, Kb, Vb = (synth.f32_to_bf16_bits(x) for x in (Q, K, V))
    O, _ = orc.full_attention(Qb, Kb, Vb, 4)
    v = bf16_vals(Vb)[0, 0]
    for i in range(L):
        others = [j for j in range(i + 1) if j != target[i]]
        want = (math.exp(16.0) * v[target[i]] + v[others].sum(axis=0)) / (math.exp(16.0) + i)
        np.testing.assert_allclose(O[0, 0, i], want, rtol=0, atol=1e-12)


def test_zero_queries_closed_form():
    """Q = 0 makes every admissible logit equal: A_ij = 1/(i+1) for j <= i, so
    O_i = mean_{j<=i} V_j and r_qb = (1/B) sum_{i in I_q} |{j in I_b: j<=i}|/(i+1)."""
    L, D, blk = 24, 6, 4
    _, K, V = synth.random_qkv(1, 1, 1, L, D, seed=9)
    Q = np.zeros((1, 1, L, D), np.uint16)
    O, M = orc.full_attention(Q, K, V, blk)
    v = bf16_vals(V)[0, 0]
    want_o = np.cumsum(v, axis=0) / np.arange(1, L + 1)[:, None]
    np.testing.assert_allclose(O[0, 0], want_o, rtol=0, atol=1e-13)
    nb = L // blk
    want_m = np.zeros((nb, nb))
    for q in range(nb):
        for b in range(nb):
            for i in range(q * blk, (q + 1) * blk):
                n_keys = sum(1 for j in range(b * blk, (b + 1) * blk) if j <= i)
                want_m[q, b] += n_keys / (i + 1) / blk
    np.testing.assert_allclose(M[0, 0], want_m, rtol=0, atol=1e-14)


# --------------------------------------------------------------------------- Eq. 5

def test_block_mass_equals_library_softmax_block_sums():
    """Eq. 5 from torch's fp64 softmax of the causally masked logits, summed
    over key blocks and averaged over the |I_q| = B query rows."""
    B, H, Hkv, L, D, blk = 1, 4, 2, 32, 8, 8
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=21)
    _, M = orc.full_attention(Q, K, V, blk)
    q = torch.from_numpy(bf16_vals(Q))
    k = torch.from_numpy(expand_kv(bf16_vals(K), H // Hkv))
    logits = q @ k.transpose(-1, -2) / math.sqrt(D)
    causal = torch.ones(L, L, dtype=torch.bool).tril()
    A = torch.softmax(logits.masked_fill(~causal, float("-inf")), dim=-1)
    nb = L // blk
    want = A.reshape(B, H, nb, blk, nb, blk).sum(dim=(3, 5)) / blk
    np.testing.assert_allclose(M, want.numpy(), rtol=0, atol=1e-14)


def test_block_mass_rows_sum_to_one_and_are_causal():
    """Rows of A sum to 1 (Eq. 2), hence sum_b r_qb = 1 (Eq. 5); r_qb = 0 for b > q."""
    Q, K, V = synth.random_qkv(2, 3, 3, 64, 16, seed=4, std=2.0)
    _, M = orc.full_attention(Q, K, V, 16)
    np.testing.assert_allclose(M.sum(-1), 1.0, rtol=0, atol=1e-13)
    assert np.all(np.triu(M, k=1) == 0.0)
    assert np.all(M >= 0.0)


def test_units_pack_the_same_rows():
    Q, K, V = synth.random_qkv(2, 4, 2, 32, 8, seed=8)
    O, M = orc.full_attention(Q, K, V, 8)
    units = [(1, 3, 2), (0, 0, 0), (1, 1, 3)]
    Ou, Mu = orc.full_attention(Q, K, V, 8, units=units)
    for n, (b, h, q) in enumerate(units):
        np.testing.assert_array_equal(Ou[n], O[b, h, q * 8:(q + 1) * 8])
        np.testing.assert_array_equal(Mu[n], M[b, h, q])
    idx, counts = synth.random_support(2, 2, 4, 3, seed=1)
    Os = orc.sparse_attention(Q, K, V, idx, counts, 8)
    Osu = orc.sparse_attention(Q, K, V, idx, counts, 8, units=units)
    for n, (b, h, q) in enumerate(units):
        np.testing.assert_array_equal(Osu[n], Os[b, h, q * 8:(q + 1) * 8])


def test_bad_arguments_are_rejected():
    Q, K, V = synth.random_qkv(1, 2, 2, 16, 4, seed=0)
    with pytest.raises(ValueError):
        orc.full_attention(Q, K, V, 5)                     # L % B != 0
    with pytest.raises(ValueError):
        orc.full_attention(Q, K, V, 4, units=[(0, 2, 0)])  # head out of range
    idx = np.full((1, 2, 4, 2), 7, np.int32)
    with pytest.raises(ValueError):
        orc.sparse_attention(Q, K, V, idx, np.ones((1, 2, 4), np.int32), 4)  # block 7 >= nKB


# --------------------------------------------------------------------------- Eqs. 7-8

def test_sparse_with_all_blocks_equals_full():
    """R == 0 when every admissible block is in the support (Eq. 8 -> Eq. 2)."""
    B, H, Hkv, L, D, blk = 2, 4, 2, 64, 8, 16
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=12)
    idx, counts = synth.all_blocks_support(B, Hkv, L // blk)
    O_full, _ = orc.full_attention(Q, K, V, blk)
    O_sp = orc.sparse_attention(Q, K, V, idx, counts, blk)
    np.testing.assert_allclose(O_sp, O_full, rtol=0, atol=1e-14)


def test_sparse_equals_library_masked_sdpa():
    """Eq. 8 is softmax(QK^T/sqrt(d) + M + R)V: torch SDPA with the boolean
    mask (j <= i) and (b(j) in B_q(i))."""
    B, H, Hkv, L, D, blk = 2, 4, 2, 64, 8, 8
    nb = L // blk
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=13)
    idx, counts = synth.random_support(B, Hkv, nb, 4, seed=2)
    O = orc.sparse_attention(Q, K, V, idx, counts, blk)
    grp = H // Hkv
    mask = np.zeros((B, H, L, L), dtype=bool)
    for b in range(B):
        for h in range(H):
            for q in range(nb):
                for kb in idx[b, h // grp, q, : counts[b, h // grp, q]]:
                    mask[b, h, q * blk:(q + 1) * blk, kb * blk:(kb + 1) * blk] = True
    mask &= np.tril(np.ones((L, L), dtype=bool))
    ref = sdpa_reference(Q, K, V, grp, attn_mask=mask)
    np.testing.assert_allclose(O, ref, rtol=0, atol=1e-12)


def test_sparse_diagonal_only_is_blockwise_causal_attention():
    """With B_q = {q} every query block attends causally inside itself only."""
    L, D, blk = 32, 8, 8
    nb = L // blk
    Q, K, V = synth.random_qkv(1, 2, 2, L, D, seed=14)
    idx = np.arange(nb, dtype=np.int32).reshape(1, 1, nb, 1).repeat(2, axis=1)
    counts = np.ones((1, 2, nb), np.int32)
    O = orc.sparse_attention(Q, K, V, idx, counts, blk)
    q = bf16_vals(Q).reshape(1, 2, nb, blk, D)
    k = bf16_vals(K).reshape(1, 2, nb, blk, D)
    v = bf16_vals(V).reshape(1, 2, nb, blk, D)
    ref = torch.nn.functional.scaled_dot_product_attention(torch.from_numpy(q), torch.from_numpy(k),
                                                           torch.from_numpy(v), is_causal=True).numpy()
    np.testing.assert_allclose(O, ref.reshape(1, 2, L, D), rtol=0, atol=1e-12)


def test_sparse_empty_support_rows_are_zero():
    L, D, blk = 32, 4, 8
    Q, K, V = synth.random_qkv(1, 1, 1, L, D, seed=15)
    idx = np.full((1, 1, 4, 2), -1, np.int32)
    counts = np.zeros((1, 1, 4), np.int32)
    O = orc.sparse_attention(Q, K, V, idx, counts, blk)
    assert np.all(O == 0.0)


# --------------------------------------------------------------------------- Eq. 6

def _run_case(case):
    nb, q, group = case["nb"], case["q"], case["group"]
    m = np.zeros((1, group, nb, nb), np.float32)
    for h, row in enumerate(case["masses"]):
        m[0, h, q] = [float("nan") if x == "nan" else x for x in row]
    mode = synth.SEL_TOPK if case["mode"] == "topk" else synth.SEL_COVERAGE
    idx, counts = orc.select_support(m, 1, 1, mode, case["n_sink"], case["n_local"], case["topk"],
                                     case["eta"], case["cap"])
    return idx[0, 0, q], counts[0, 0, q]


with open(os.path.join(GOLDEN, "selection_cases.json")) as _f:
    _CASES = json.load(_f)["cases"]


@pytest.mark.parametrize("case", _CASES, ids=[c["name"] for c in _CASES])
def test_selection_golden_cases(case):
    row, n = _run_case(case)
    assert n == len(case["expect"]), case["why"]
    assert row[:n].tolist() == case["expect"], case["why"]
    assert np.all(row[n:] == -1)


def _u(x):
    x = np.float32(x)
    if not (x > 0):
        return 0
    return int(math.floor(float(min(x, np.float32(4096.0))) * 2.0 ** 32))


@pytest.mark.parametrize("seed", range(12))
def test_coverage_is_minimum_cardinality_by_exhaustive_search(seed):
    """Eq. 6 defines B_q as argmin |B| s.t. sum_{b in B} r_qb >= eta.  Search
    every superset of the forced blocks: the selected set must reach the
    threshold, have the minimum size, and carry the maximum mass among sets
    of that size."""
    rng = np.random.default_rng(seed)
    nb = 9
    q = nb - 1
    group = 1 + seed % 2
    m = np.zeros((1, group, nb, nb), np.float32)
    m[0, :, q] = rng.dirichlet(np.full(nb, 0.4), size=group).astype(np.float32)
    eta = float(rng.choice([0.5, 0.8, 0.9, 0.95]))
    n_sink, n_local = 1, 1 + seed % 2
    idx, counts = orc.select_support(m, 1, 1, synth.SEL_COVERAGE, n_sink, n_local, 0, eta, nb)
    got = set(idx[0, 0, q, : counts[0, 0, q]].tolist())
    U = [sum(_u(m[0, h, q, kb]) for h in range(group)) for kb in range(nb)]
    T = sum(U)
    e16 = int(math.floor(eta * 65536 + 0.5))
    forced = set(range(n_sink)) | set(range(q - n_local + 1, q + 1))
    cands = [kb for kb in range(nb) if kb not in forced]

    def ok(S):
        return sum(U[kb] for kb in S) * 65536 >= e16 * T

    best = None
    for r in range(len(cands) + 1):
        sets = [forced | set(c) for c in itertools.combinations(cands, r)]
        good = [S for S in sets if ok(S)]
        if good:
            best = (r, max(sum(U[kb] for kb in S) for S in good))
            break
    assert ok(got)
    assert len(got) == len(forced) + best[0]
    assert sum(U[kb] for kb in got) == best[1]


@pytest.mark.parametrize("seed", range(6))
def test_topk_matches_library_stable_ranking(seed):
    """Top-k keeps the k best candidates under (pooled mass desc, index asc):
    numpy's lexsort of the pooled fixed-point masses gives the same set."""
    rng = np.random.default_rng(100 + seed)
    B, H, Hkv, nb = 2, 4, 2, 12
    m = rng.random((B, H, nb, nb)).astype(np.float32)
    m[..., :, 3] = m[..., :, 4]           # planted exact ties between blocks 3 and 4
    k, cap, n_sink, n_local = 3, 6, 1, 2
    idx, counts = orc.select_support(m, Hkv, 1, synth.SEL_TOPK, n_sink, n_local, k, 0.0, cap)
    grp = H // Hkv
    for b in range(B):
        for g in range(Hkv):
            for q in range(nb):
                U = np.array([sum(_u(m[b, h, q, kb]) for h in range(g * grp, (g + 1) * grp))
                              for kb in range(q + 1)], dtype=object)
                forced = set(range(min(n_sink, q + 1))) | set(range(max(0, q - n_local + 1), q + 1))
                cands = np.array([kb for kb in range(q + 1) if kb not in forced], dtype=np.int64)
                if len(cands):
                    keys = np.array([U[kb] for kb in cands], dtype=np.float64)
                    order = np.lexsort((cands, -keys))
                    pick = set(cands[order[: min(k, cap - len(forced))]].tolist())
                else:
                    pick = set()
                want = sorted(forced | pick)
                assert counts[b, g, q] == len(want)
                assert idx[b, g, q, : len(want)].tolist() == want


def test_selection_rejects_bad_parameters():
    m = np.zeros((1, 1, 4, 4), np.float32)
    with pytest.raises(ValueError):
        orc.select_support(m, 1, 1, synth.SEL_TOPK, 1, 1, 2, 0.0, 1)      # cap < forced
    with pytest.raises(ValueError):
        orc.select_support(m, 1, 1, synth.SEL_COVERAGE, 1, 1, 0, 1.5, 4)  # eta > 1
    with pytest.raises(ValueError):
        orc.select_support(m, 1, 1, synth.SEL_TOPK, 1, 0, 2, 0.0, 4)      # no diagonal


# --------------------------------------------------------------------------- end to end (sanity)

def test_planted_blocks_are_recovered_on_the_tiny_workload():
    """Statistical sanity of generator + oracle (not a parity check): after
    the discovery steps, top-k selection recovers the planted key blocks."""
    wl = synth.WORKLOADS["tiny"]
    traj = synth.Trajectory(wl)
    acc = None
    for t in range(wl.n_discovery):
        Q, K, V = traj.step(t)
        _, M = orc.full_attention(Q, K, V, wl.block)
        acc = M if acc is None else acc + M
    idx, counts = orc.select_support(acc.astype(np.float32), wl.n_kv_heads, wl.block, wl.sel_mode, wl.n_sink,
                                     wl.n_local, wl.topk, wl.eta, wl.cap)
    hit = tot = 0
    for g in range(wl.n_kv_heads):
        for q in range(wl.n_blocks):
            chosen = set(idx[0, g, q, : counts[0, g, q]].tolist())
            for p in traj.planted[0][g][q]:
                tot += 1
                hit += p in chosen
    assert tot > 0 and hit / tot >= 0.9
    np.testing.assert_allclose(acc.sum(-1), wl.n_discovery, atol=1e-12)


# ---------------------------------------------------------------- retained mass (routing diagnostic)

def test_retained_mass_of_the_full_support_is_one():
    # Every admissible block kept: the retained fraction is the whole row of
    # Eq. 5, which sums to 1 (rows of A sum to 1).
    B, H, Hkv, L, D, blk = 1, 4, 2, 64, 16, 8
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=21)
    _, mass = orc.full_attention(Q, K, V, blk, with_mass=True)
    idx, counts = synth.all_blocks_support(B, Hkv, L // blk)
    r = orc.support_mass(mass, idx, counts, H)
    assert np.allclose(r, 1.0, atol=1e-12)


def test_retained_mass_of_complementary_supports_adds_to_one():
    # Split the admissible blocks of every row into two disjoint supports: the
    # two retained fractions add to the whole row (pins that no term is lost
    # or counted twice, and that each query head reads its own row).
    B, H, Hkv, L, D, blk = 2, 6, 3, 96, 16, 16
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=22)
    _, mass = orc.full_attention(Q, K, V, blk, with_mass=True)
    nb = L // blk
    rng = np.random.default_rng(5)
    a = np.full((B, Hkv, nb, nb), -1, dtype=np.int32)
    c = np.full_like(a, -1)
    na = np.zeros((B, Hkv, nb), dtype=np.int32)
    nc = np.zeros_like(na)
    for b, g, q in itertools.product(range(B), range(Hkv), range(nb)):
        pick = rng.random(q + 1) < 0.5
        sa, sc = np.flatnonzero(pick), np.flatnonzero(~pick)
        a[b, g, q, : len(sa)], na[b, g, q] = sa, len(sa)
        c[b, g, q, : len(sc)], nc[b, g, q] = sc, len(sc)
    ra = orc.support_mass(mass, a, na, H)
    rc = orc.support_mass(mass, c, nc, H)
    assert np.allclose(ra + rc, 1.0, atol=1e-12)
    assert ra.min() >= 0.0 and rc.min() >= 0.0


def test_retained_mass_hand_case_with_group_lists_and_invalid_entries():
    # 2 query heads sharing one kv-group list; 3 query blocks.  Masses are
    # chosen by hand; invalid entries (negative, beyond the query block, not
    # ascending) are skipped, as the attention kernels skip them.
    mass = np.zeros((1, 2, 3, 3))
    mass[0, 0] = [[1.0, 0, 0], [0.25, 0.75, 0], [0.5, 0.125, 0.375]]
    mass[0, 1] = [[1.0, 0, 0], [0.5, 0.5, 0], [0.0625, 0.4375, 0.5]]
    idx = np.array([[[[0, -1, -1], [1, 0, 1], [-3, 2, 0]]]], dtype=np.int32)
    counts = np.array([[[1, 3, 3]]], dtype=np.int32)
    r = orc.support_mass(mass, idx, counts, 2)
    # q=0: {0}; q=1: {1} (0 and the repeated 1 are not ascending); q=2: {2} (-3 and 0 after 2 skipped)
    want = np.array([[[1.0, 0.75, 0.375], [1.0, 0.5, 0.5]]])
    assert np.array_equal(r, want)


# ---------------------------------------------------------------- working sets of Eq. 6 and the controls

def _ws_units(x):
    x = float(np.float32(x))
    return 0 if not x > 0 else int(math.floor(min(x, 4096.0) * 2.0 ** 32))


def _rows(masses, group):
    """Pooled fixed-point masses per (step, b, g, q) row, for brute force."""
    S, B, H, nq, _ = masses.shape
    for st, b, g, q in itertools.product(range(S), range(B), range(H // group), range(nq)):
        yield st, b, g, q, [sum(_ws_units(masses[st, b, h, q, kb]) for h in range(g * group, (g + 1) * group))
                            for kb in range(q + 1)]


def _min_cover(U, forced, need):
    """Exhaustive search: the smallest size of a set holding `forced` whose
    mass satisfies need(mass)."""
    rest = [kb for kb in range(len(U)) if kb not in forced]
    for k in range(len(rest) + 1):
        for extra in itertools.combinations(rest, k):
            if need(sum(U[kb] for kb in forced) + sum(U[kb] for kb in extra)):
                return len(forced) + k
    return None


@pytest.mark.parametrize("n_sink,n_local", [(0, 0), (1, 1)])
def test_static_set_is_a_minimum_eta_cover_by_exhaustive_search(n_sink, n_local):
    rng = np.random.default_rng(31)
    masses = rng.dirichlet(np.ones(7), size=(1, 1, 2, 7)).astype(np.float32)  # rows of 7 blocks
    masses = np.tril(masses.reshape(1, 1, 2, 7, 7))  # only admissible blocks kb <= q carry mass
    eta = 0.8
    eta16 = int(math.floor(float(np.float32(eta)) * 65536 + 0.5))
    idx, counts = orc.working_set(1, masses, 2, eta=eta, n_sink=n_sink, n_local=n_local)
    for _, b, g, q, U in _rows(masses, 1):
        forced = {kb for kb in range(q + 1) if kb < n_sink or kb > q - n_local}
        total = sum(U)
        sel = idx[b, g, q, : counts[b, g, q]]
        assert set(forced) <= set(sel.tolist())
        assert sum(U[kb] for kb in sel) * 65536 >= eta16 * total
        assert counts[b, g, q] == _min_cover(U, forced, lambda s: s * 65536 >= eta16 * total)


def test_union_is_the_union_of_the_per_step_sets():
    rng = np.random.default_rng(32)
    masses = np.tril(rng.random((3, 1, 2, 6, 6))).astype(np.float32)
    masses /= masses.sum(-1, keepdims=True)
    u_idx, u_cnt = orc.working_set(0, masses, 1, eta=0.9, n_sink=1, n_local=1)
    per = [orc.working_set(1, masses[s:s + 1], 1, eta=0.9, n_sink=1, n_local=1) for s in range(3)]
    for b, g, q in itertools.product(range(1), range(1), range(6)):
        want = set()
        for idx, cnt in per:
            want |= set(idx[b, g, q, : cnt[b, g, q]].tolist())
        assert sorted(want) == u_idx[b, g, q, : u_cnt[b, g, q]].tolist()
    # the same step twice adds nothing
    twice = np.concatenate([masses[:1], masses[:1]])
    a = orc.working_set(0, twice, 1, eta=0.9)
    b1 = orc.working_set(1, masses[:1], 1, eta=0.9)
    assert np.array_equal(a[0], b1[0]) and np.array_equal(a[1], b1[1])


def test_mass_and_size_matched_controls_by_exhaustive_search():
    rng = np.random.default_rng(33)
    nq = 7
    masses = np.tril(rng.random((1, 1, 3, nq, nq))).astype(np.float32)
    masses /= masses.sum(-1, keepdims=True)
    # reference working set: a random admissible subset of each row
    ref_idx = np.full((1, 3, nq, nq), -1, dtype=np.int32)
    ref_cnt = np.zeros((1, 3, nq), dtype=np.int32)
    for g, q in itertools.product(range(3), range(nq)):
        s = sorted(rng.choice(q + 1, size=rng.integers(1, q + 2), replace=False).tolist())
        ref_idx[0, g, q, : len(s)], ref_cnt[0, g, q] = s, len(s)
    mm = orc.working_set(2, masses, 3, ref_idx=ref_idx, ref_counts=ref_cnt)
    sm = orc.working_set(3, masses, 3, ref_idx=ref_idx, ref_counts=ref_cnt)
    for _, b, g, q, U in _rows(masses, 1):
        ref = ref_idx[b, g, q, : ref_cnt[b, g, q]].tolist()
        target = sum(U[kb] for kb in ref)
        m_sel = mm[0][b, g, q, : mm[1][b, g, q]].tolist()
        assert sum(U[kb] for kb in m_sel) >= target
        assert len(m_sel) == _min_cover(U, set(), lambda s: s >= target) <= len(ref)
        s_sel = sm[0][b, g, q, : sm[1][b, g, q]].tolist()
        assert len(s_sel) == len(ref)
        best = max(sum(U[kb] for kb in c) for c in itertools.combinations(range(q + 1), len(ref)))
        assert sum(U[kb] for kb in s_sel) == best
    # against its own coverage set, the mass-matched control is that set
    st = orc.working_set(1, masses, 3, eta=0.9)
    same = orc.working_set(2, masses, 3, ref_idx=st[0], ref_counts=st[1])
    assert np.array_equal(same[0], st[0]) and np.array_equal(same[1], st[1])


def test_working_set_hand_case_with_gqa_pooling():
    # 2 query heads pooled into one kv group, one step, q = 3 (4 admissible
    # blocks).  Pooled masses (halves): head 0 [0.5, 0.25, 0.125, 0.125],
    # head 1 [0.125, 0.5, 0.25, 0.125] -> pooled [0.625, 0.75, 0.375, 0.25] of
    # total 2.  eta = 0.6 needs 1.2: ranked 1 (0.75), 0 (0.625) -> {0, 1}.
    m = np.zeros((1, 1, 2, 4, 4), dtype=np.float32)
    m[0, 0, 0, 3] = [0.5, 0.25, 0.125, 0.125]
    m[0, 0, 1, 3] = [0.125, 0.5, 0.25, 0.125]
    idx, counts = orc.working_set(1, m, 1, eta=0.6)
    assert idx[0, 0, 3, : counts[0, 0, 3]].tolist() == [0, 1]
    # with the diagonal forced: {3} holds 0.25, then 1 (1.0), then 0 (1.625 >= 1.2)
    idx, counts = orc.working_set(1, m, 1, eta=0.6, n_local=1)
    assert idx[0, 0, 3, : counts[0, 0, 3]].tolist() == [0, 1, 3]
    # size matched against a 2-block reference with the diagonal forced: {3} + top 1 -> {1, 3}
    ref = np.array([[[[0, 2, -1, -1]] * 4]], dtype=np.int32)
    rc = np.full((1, 1, 4), 2, dtype=np.int32)
    idx, counts = orc.working_set(3, m, 1, n_local=1, ref_idx=ref, ref_counts=rc)
    assert idx[0, 0, 3, : counts[0, 0, 3]].tolist() == [1, 3]


# ---------------------------------------------- rolling-set overlap (appendix)

def _lists(rows, cap):
    """rows: {(g, q): [entries]} for B = 1 -> idx [1,Hkv,nQB,cap], counts."""
    Hkv = 1 + max(g for g, _ in rows)
    nq = 1 + max(q for _, q in rows)
    idx = np.full((1, Hkv, nq, cap), -1, dtype=np.int32)
    counts = np.zeros((1, Hkv, nq), dtype=np.int32)
    for (g, q), ent in rows.items():
        idx[0, g, q, :len(ent)] = ent
        counts[0, g, q] = len(ent)
    return idx, counts


def test_overlap_hand_case_with_invalid_entries():
    """Two supports over 2 kv heads x 3 query blocks, counted by hand: each
    row shares exactly one block, and the rows hold 1, 2, 3 distinct blocks in
    the union, so |A & B| = 6 and |A | B| = 12 (Jaccard 1/2).  A repeated
    entry and an entry beyond its query block are skipped."""
    a = {(0, 0): [0], (0, 1): [0, 1, 1], (0, 2): [0, 2], (1, 0): [0], (1, 1): [1], (1, 2): [0, 1, 2]}
    b = {(0, 0): [0], (0, 1): [1], (0, 2): [1, 2], (1, 0): [0], (1, 1): [0, 1], (1, 2): [2, 5]}
    ia, ca = _lists(a, 4)
    ib, cb = _lists(b, 4)
    np.testing.assert_array_equal(orc.support_overlap(ia, ca, ib, cb), [[6, 12]])
    np.testing.assert_array_equal(orc.support_overlap(ib, cb, ia, ca), [[6, 12]])


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_overlap_identities_on_random_supports(seed):
    """|A & A| = |A | A| = |A| = sum of counts for well-formed lists;
    inclusion-exclusion |A & B| + |A | B| = |A| + |B|; supports without a
    common block have an empty intersection."""
    B, Hkv, nb = 2, 3, 9
    ia, ca = synth.random_support(B, Hkv, nb, 5, seed=seed)
    ib, cb = synth.random_support(B, Hkv, nb, 7, seed=seed + 10)
    self_ov = orc.support_overlap(ia, ca, ia, ca)
    np.testing.assert_array_equal(self_ov[:, 0], ca.sum(axis=(1, 2)))
    np.testing.assert_array_equal(self_ov[:, 1], ca.sum(axis=(1, 2)))
    ov = orc.support_overlap(ia, ca, ib, cb)
    np.testing.assert_array_equal(ov[:, 0] + ov[:, 1], ca.sum(axis=(1, 2)) + cb.sum(axis=(1, 2)))
    # Even blocks only against odd blocks only.
    ev, cev = ia.copy(), ca.copy()
    od, cod = ia.copy(), ca.copy()
    for arr, cnt, parity in ((ev, cev, 0), (od, cod, 1)):
        for bb in range(B):
            for g in range(Hkv):
                for q in range(nb):
                    keep = [v for v in range(q + 1) if v % 2 == parity]
                    arr[bb, g, q, :] = -1
                    arr[bb, g, q, :len(keep[:5])] = keep[:5]
                    cnt[bb, g, q] = len(keep[:5])
    ov = orc.support_overlap(ev, cev, od, cod)
    assert (ov[:, 0] == 0).all() and (ov[:, 1] == cev.sum(axis=(1, 2)) + cod.sum(axis=(1, 2))).all()


# ------------------------------------------------------------ Freeze-A (appendix)

def test_freeze_a_with_the_frozen_values_is_the_sparse_attention_of_that_step():
    """With V = the frozen step's V, Abar V is that step's support-restricted
    attention: softmax-then-restrict-and-renormalise (the control's definition)
    equals restrict-then-softmax (Eqs. 7-8, the C oracle)."""
    B, H, Hkv, L, D, blk = 2, 4, 2, 64, 8, 8
    Q, K, V = synth.random_qkv(B, H, Hkv, L, D, seed=21)
    idx, counts = synth.random_support(B, Hkv, L // blk, 4, seed=22)
    got = orc.freeze_a(bf16_vals(Q), bf16_vals(K), bf16_vals(V), idx, counts, blk)
    want = orc.sparse_attention(Q, K, V, idx, counts, blk)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)


def test_freeze_a_with_every_block_is_full_attention_on_the_new_values():
    """With the all-blocks support Abar = A: O = A(Q0, K0) V, i.e. torch's
    causal SDPA with the frozen Q and K and the new V."""
    B, H, Hkv, L, D, blk = 1, 3, 3, 40, 5, 8
    Q, K, V0 = synth.random_qkv(B, H, Hkv, L, D, seed=23)
    _, _, V1 = synth.random_qkv(B, H, Hkv, L, D, seed=24)
    idx, counts = synth.all_blocks_support(B, Hkv, L // blk)
    got = orc.freeze_a(bf16_vals(Q), bf16_vals(K), bf16_vals(V1), idx, counts, blk)
    ref = sdpa_reference(Q, K, V1, 1, is_causal=True)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)


def test_freeze_a_rows_are_convex_combinations_of_supported_values():
    """Abar rows are distributions over the supported admissible keys: with V
    = one-hot columns marking whether a key is supported, O sums to 1 on the
    supported column and 0 elsewhere."""
    B, H, Hkv, L, D, blk = 1, 2, 1, 32, 4, 8
    Q, K, _ = synth.random_qkv(B, H, Hkv, L, D, seed=25)
    idx, counts = synth.random_support(B, Hkv, L // blk, 2, seed=26)
    # For the rows of query block q: V column 0 marks the keys whose block is
    # in q's support, column 1 the others.
    got_rows = []
    for q in range(L // blk):
        inside = np.zeros((B, Hkv, L, 2))
        sup = set(int(v) for v in idx[0, 0, q, :counts[0, 0, q]])
        for j in range(L):
            inside[0, 0, j, 0 if j // blk in sup else 1] = 1.0
        O = orc.freeze_a(bf16_vals(Q), bf16_vals(K), inside, idx, counts, blk)
        got_rows.append(O[0, :, q * blk:(q + 1) * blk, :])
    got = np.stack(got_rows)
    np.testing.assert_allclose(got[..., 0], 1.0, rtol=0, atol=1e-12)
    np.testing.assert_allclose(got[..., 1], 0.0, rtol=0, atol=1e-12)


def test_freeze_a_distribution_rows_are_normalised_on_the_support():
    """Abar is a distribution over the admissible supported keys of each row
    (rows of a query block with an empty list are 0), zero elsewhere."""
    B, H, Hkv, L, D, blk = 1, 2, 1, 48, 4, 8
    Q, K, _ = synth.random_qkv(B, H, Hkv, L, D, seed=27)
    idx, counts = synth.random_support(B, Hkv, L // blk, 3, seed=28)
    counts[0, 0, 2] = 0
    abar = orc.freeze_a_distribution(bf16_vals(Q), bf16_vals(K), idx, counts, blk)
    for h in range(H):
        for i in range(L):
            q = i // blk
            sup = set(int(v) for v in idx[0, 0, q, :counts[0, 0, q]])
            allowed = np.array([(j // blk in sup) and j <= i for j in range(L)])
            assert np.all(abar[0, h, i, ~allowed] == 0.0)
            want = 1.0 if allowed.any() else 0.0
            assert abs(abar[0, h, i].sum() - want) < 1e-12
