"""Python front end of the fp64 CPU oracle (wise_oracle.c).

TEST INFRASTRUCTURE ONLY: the tests, the smoke check and the benchmark's CPU
baseline may use this module; the library never imports it.  It compiles the
C oracle with the host gcc (OpenMP) into oracle/_build/ and calls it through
ctypes.  Each function states the equation of the paper it evaluates.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "wise_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libwise_oracle.so")
_lock = threading.Lock()
_lib = None


class _Shape(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int), ("seqlen", ctypes.c_int), ("n_heads", ctypes.c_int),
                ("n_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int), ("block", ctypes.c_int),
                ("scale", ctypes.c_double)]


class _Select(ctypes.Structure):
    _fields_ = [("n_sink", ctypes.c_int), ("n_local", ctypes.c_int), ("mode", ctypes.c_int),
                ("topk", ctypes.c_int), ("eta", ctypes.c_float), ("cap", ctypes.c_int)]


def build(force: bool = False) -> str:
    """Compile the C oracle (gcc -O2 -fopenmp) if it is missing or stale."""
    with _lock:
        if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
            os.makedirs(_BUILD, exist_ok=True)
            tmp = _LIB_PATH + f".{os.getpid()}.tmp"
            subprocess.check_call(["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"])
            os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        lib.wo_full_attention.argtypes = [ctypes.POINTER(_Shape), P, P, P, ctypes.c_long, P, P, P]
        lib.wo_sparse_attention.argtypes = [ctypes.POINTER(_Shape), P, P, P, P, P, ctypes.c_int,
                                            ctypes.c_long, P, P]
        lib.wo_select_support.argtypes = [ctypes.POINTER(_Shape), ctypes.POINTER(_Select), P, P, P]
        lib.wo_max_threads.restype = ctypes.c_int
        lib.wo_set_threads.argtypes = [ctypes.c_int]
        _lib = lib
    return _lib


def set_threads(n: int) -> None:
    _load().wo_set_threads(int(n))


def max_threads() -> int:
    return int(_load().wo_max_threads())


def _shape(batch, seqlen, n_heads, n_kv_heads, head_dim, block, scale=0.0):
    return _Shape(batch, seqlen, n_heads, n_kv_heads, head_dim, block, float(scale or 0.0))


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p) if a is not None else None


def _bits(a):
    a = np.ascontiguousarray(a)
    if a.dtype != np.uint16:
        raise TypeError("bf16 inputs are passed as uint16 bit patterns")
    return a


def _units(units):
    if units is None:
        return None, 0
    u = np.ascontiguousarray(np.asarray(units, dtype=np.int32).reshape(-1, 3))
    return u, len(u)


def full_attention(Q, K, V, block, units=None, scale=None, with_mass=True):
    """Eq. 2 (causal mask) and Eq. 5.

    Q [B,H,L,D], K/V [B,Hkv,L,D] as bf16 bits.  Returns (O, mass) in float64:
    O [B,H,L,D] and mass [B,H,nQB,nKB] for all query blocks, or packed per
    listed (b, h, q) unit: O [n,block,D], mass [n,nKB].
    """
    Q, K, V = _bits(Q), _bits(K), _bits(V)
    B, H, L, D = Q.shape
    Hkv = K.shape[1]
    nb = L // block
    u, n = _units(units)
    if u is None:
        O = np.zeros((B, H, L, D), dtype=np.float64)
        M = np.zeros((B, H, nb, nb), dtype=np.float64) if with_mass else None
    else:
        O = np.zeros((n, block, D), dtype=np.float64)
        M = np.zeros((n, nb), dtype=np.float64) if with_mass else None
    sh = _shape(B, L, H, Hkv, D, block, scale)
    rc = _load().wo_full_attention(ctypes.byref(sh), _ptr(Q), _ptr(K), _ptr(V), n, _ptr(u), _ptr(O), _ptr(M))
    if rc != 0:
        raise ValueError("oracle full_attention rejected its arguments")
    return O, M


def sparse_attention(Q, K, V, idx, counts, block, units=None, scale=None):
    """Eqs. 7-8: attention restricted to the block support (idx, counts)."""
    Q, K, V = _bits(Q), _bits(K), _bits(V)
    B, H, L, D = Q.shape
    Hkv = K.shape[1]
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    counts = np.ascontiguousarray(counts, dtype=np.int32)
    cap = idx.shape[-1]
    u, n = _units(units)
    O = np.zeros((B, H, L, D) if u is None else (n, block, D), dtype=np.float64)
    sh = _shape(B, L, H, Hkv, D, block, scale)
    rc = _load().wo_sparse_attention(ctypes.byref(sh), _ptr(Q), _ptr(K), _ptr(V), _ptr(idx), _ptr(counts),
                                     cap, n, _ptr(u), _ptr(O))
    if rc != 0:
        raise ValueError("oracle sparse_attention rejected its arguments")
    return O


def select_support(blockmass, n_kv_heads, block, mode, n_sink, n_local, topk, eta, cap):
    """Eq. 6 in single-pass form: forced sink/local blocks, then top-k or
    cumulative-mass coverage over the pooled fixed-point masses.

    blockmass [B,H,nQB,nKB] float32.  Returns idx [B,Hkv,nQB,cap] int32
    (ascending, -1 padded) and counts [B,Hkv,nQB] int32.
    """
    m = np.ascontiguousarray(blockmass, dtype=np.float32)
    B, H, nq, nk = m.shape
    if nq != nk:
        raise ValueError("blockmass must be square in its last two dims")
    idx = np.empty((B, n_kv_heads, nq, cap), dtype=np.int32)
    counts = np.empty((B, n_kv_heads, nq), dtype=np.int32)
    sh = _shape(B, nq * block, H, n_kv_heads, 1, block)
    sel = _Select(int(n_sink), int(n_local), int(mode), int(topk), float(eta), int(cap))
    rc = _load().wo_select_support(ctypes.byref(sh), ctypes.byref(sel), _ptr(m), _ptr(idx), _ptr(counts))
    if rc != 0:
        raise ValueError("oracle select_support rejected its arguments")
    return idx, counts


def support_mass(blockmass, idx, counts, n_heads):
    """Retained mass of a support (appendix "Experimental details",
    evaluation metrics: the fraction of the unrestricted attention mass that
    falls inside the frozen support), per query-head row: the row's block
    masses r_qb (Eq. 5) summed over the key blocks of its kv-group's support
    list, in fp64.  List entries that are negative, beyond the query block or
    not strictly above the last accepted entry are skipped, as the attention
    kernels skip them.

    blockmass [B,H,nQB,nKB]; idx [B,Hkv,nQB,cap]; counts [B,Hkv,nQB].
    Returns retained [B,H,nQB] float64.
    """
    m = np.asarray(blockmass, dtype=np.float64)
    B, H, nq, _ = m.shape
    Hkv = idx.shape[1]
    if H != n_heads or H % Hkv:
        raise ValueError("head counts do not match")
    group = H // Hkv
    out = np.zeros((B, H, nq), dtype=np.float64)
    for b in range(B):
        for h in range(H):
            for q in range(nq):
                n = int(counts[b, h // group, q])
                n = min(max(n, 0), idx.shape[3])
                prev = -1
                total = 0.0
                for v in idx[b, h // group, q, :n]:
                    v = int(v)
                    if 0 <= v <= q and v > prev:
                        total += m[b, h, q, v]
                        prev = v
                out[b, h, q] = total
    return out


def _mass_units(x):
    """Fixed-point mass of the selection rule: floor(min(x, 4096) * 2^32) for
    x > 0, else 0 (exact for fp32 inputs)."""
    x = float(np.float32(x))
    if not x > 0.0:
        return 0
    return int(np.floor(min(x, 4096.0) * 4294967296.0))


def working_set(mode, step_masses, n_kv_heads, eta=0.95, n_sink=0, n_local=0, ref_idx=None, ref_counts=None):
    """Working sets of Eq. 6 (the union over the discovery window of each
    step's smallest block set reaching eta of the mass) and the intervention
    controls of the appendix ("Experimental details"): Static (the first
    step's eta set), MassMatched (the first step's smallest top set whose mass
    reaches the first-step mass of a reference working set) and SizeMatched
    (the first step's top blocks, as many as the reference set holds).

    Same arithmetic as the selection rule of select_support: masses pooled
    over the kv-group's query heads in exact fixed point, ranking by pooled
    mass (descending) then block (ascending), forced blocks
    {0..n_sink-1} U {q-n_local+1..q} in every set, coverage reached when
    cum * 65536 >= floor(eta * 65536 + 0.5) * admissible total.

    step_masses [n_steps,B,H,nQB,nKB] fp32 (mode 0 may use several steps,
    the others exactly one).  Returns idx [B,Hkv,nQB,nQB] int32 (ascending,
    -1 padded) and counts [B,Hkv,nQB].
    """
    m = np.asarray(step_masses, dtype=np.float32)
    S, B, H, nq, nk = m.shape
    if nq != nk or H % n_kv_heads:
        raise ValueError("bad shapes")
    if mode != 0 and S != 1:
        raise ValueError("one step for the controls")
    group = H // n_kv_heads
    eta16 = int(np.floor(float(np.float32(eta)) * 65536.0 + 0.5))
    idx = np.full((B, n_kv_heads, nq, nq), -1, dtype=np.int32)
    counts = np.zeros((B, n_kv_heads, nq), dtype=np.int32)
    for b in range(B):
        for g in range(n_kv_heads):
            for q in range(nq):
                adm = list(range(q + 1))
                forced = {kb for kb in adm if kb < n_sink or kb > q - n_local}

                def pooled(st):
                    return {kb: sum(_mass_units(m[st, b, h, q, kb]) for h in range(g * group, (g + 1) * group))
                            for kb in adm}

                def ranked(U):
                    return sorted((kb for kb in adm if kb not in forced), key=lambda kb: (-U[kb], kb))

                if mode in (0, 1):
                    chosen = set(forced)
                    for st in range(S):
                        U = pooled(st)
                        total = sum(U.values())
                        cum = sum(U[kb] for kb in forced)
                        sel = set(forced)
                        for kb in ranked(U):
                            if cum * 65536 >= eta16 * total:
                                break
                            sel.add(kb)
                            cum += U[kb]
                        chosen |= sel
                else:
                    U = pooled(0)
                    n = min(max(int(ref_counts[b, g, q]), 0), ref_idx.shape[3])
                    ref, prev = [], -1
                    for v in ref_idx[b, g, q, :n]:
                        v = int(v)
                        if 0 <= v <= q and v > prev:
                            ref.append(v)
                            prev = v
                    chosen = set(forced)
                    cum = sum(U[kb] for kb in forced)
                    if mode == 2:
                        target = sum(U[kb] for kb in ref)
                        for kb in ranked(U):
                            if cum >= target:
                                break
                            chosen.add(kb)
                            cum += U[kb]
                    else:
                        for kb in ranked(U)[: max(0, len(ref) - len(forced))]:
                            chosen.add(kb)
                s = sorted(chosen)
                idx[b, g, q, : len(s)] = s
                counts[b, g, q] = len(s)
    return idx, counts


def _used_blocks(idx_row, n, q):
    """Entries of a support list that the attention kernels use: the first n
    (clamped to the row width), skipping entries that are negative, beyond
    query block q or not strictly above the last accepted entry."""
    n = min(max(int(n), 0), len(idx_row))
    out, prev = [], -1
    for v in idx_row[:n]:
        v = int(v)
        if 0 <= v <= q and v > prev:
            out.append(v)
            prev = v
    return out


def support_overlap(idx_a, counts_a, idx_b, counts_b):
    """Overlap of two block supports (appendix "Stability of the Deployed
    Working Set"): the working set of an example is the collection of active
    (head, query block, key block) triples, and the rolling-set Jaccard of two
    consecutive steps is |W(t-1) & W(t)| / |W(t-1) | W(t)|.  Returns int64
    [B, 2]: per batch element the sizes of the intersection and of the union,
    from Python sets.  idx [B,Hkv,nQB,cap], counts [B,Hkv,nQB]."""
    B, Hkv, nq = np.asarray(counts_a).shape
    out = np.zeros((B, 2), dtype=np.int64)
    for b in range(B):
        wa, wb = set(), set()
        for g in range(Hkv):
            for q in range(nq):
                wa.update((g, q, v) for v in _used_blocks(idx_a[b, g, q], counts_a[b, g, q], q))
                wb.update((g, q, v) for v in _used_blocks(idx_b[b, g, q], counts_b[b, g, q], q))
        out[b, 0] = len(wa & wb)
        out[b, 1] = len(wa | wb)
    return out


def freeze_a_distribution(Q0, K0, idx, counts, block, scale=None):
    """Abar of the Freeze-A control (appendix "Experimental details",
    intervention controls), in the order the paper defines it: A = the
    unrestricted causal attention of the frozen step (softmax of
    scale * Q0 K0^T + M, Eq. 2), then A restricted to the key blocks of the
    support and renormalised over the admissible keys.  fp64 numpy, [B,H,L,L];
    rows whose restricted mass is zero are 0.  Q0 [B,H,L,d], K0 [B,Hkv,L,d],
    idx [B,Hkv,nQB,cap], counts [B,Hkv,nQB]."""
    Q0 = np.asarray(Q0, dtype=np.float64)
    K0 = np.asarray(K0, dtype=np.float64)
    B, H, L, d = Q0.shape
    Hkv = K0.shape[1]
    group = H // Hkv
    sc = 1.0 / np.sqrt(d) if scale is None else float(scale)
    nq = L // block
    causal = np.tril(np.ones((L, L), dtype=bool))
    out = np.zeros((B, H, L, L), dtype=np.float64)
    for b in range(B):
        for h in range(H):
            g = h // group
            s = sc * (Q0[b, h] @ K0[b, g].T)
            s = np.where(causal, s, -np.inf)
            a = np.exp(s - s.max(axis=1, keepdims=True))
            a /= a.sum(axis=1, keepdims=True)
            keep = np.zeros((L, L), dtype=bool)
            for q in range(nq):
                for v in _used_blocks(idx[b, g, q], counts[b, g, q], q):
                    keep[q * block:(q + 1) * block, v * block:(v + 1) * block] = True
            abar = np.where(keep & causal, a, 0.0)
            tot = abar.sum(axis=1, keepdims=True)
            out[b, h] = np.divide(abar, tot, out=np.zeros_like(abar), where=tot > 0)
    return out


def freeze_a(Q0, K0, V, idx, counts, block, scale=None):
    """Freeze-A output O = Abar V with the current step's V [B,Hkv,L,dv]
    (Abar from freeze_a_distribution).  fp64, [B,H,L,dv]."""
    abar = freeze_a_distribution(Q0, K0, idx, counts, block, scale)
    V = np.asarray(V, dtype=np.float64)
    B, H = abar.shape[:2]
    group = H // V.shape[1]
    out = np.zeros((B, H, abar.shape[2], V.shape[3]), dtype=np.float64)
    for b in range(B):
        for h in range(H):
            out[b, h] = abar[b, h] @ V[b, h // group]
    return out
