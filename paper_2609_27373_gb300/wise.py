"""ctypes binding of libwise.so with the same names as its C entry points.

Only argument marshalling happens here: every step of the path runs in the
library's CUDA kernels.  Tensors are torch CUDA tensors (PyTorch supplies the
device memory and the stream); shapes and dtypes are checked before the call
so that a wrong tensor fails here rather than inside a kernel.  There is no
fallback: if the library is missing the import fails loudly.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os

import torch

from . import build as _build

WISE_OK = 0
WISE_ERR_INVALID_ARG = -1
WISE_ERR_UNSUPPORTED = -2
WISE_ERR_SHAPE = -3
WISE_ERR_CUDA = -4
WISE_ERR_TIMEOUT = -5
WISE_ERR_BAD_SUPPORT = -6
WISE_SEL_TOPK = 0
WISE_SEL_COVERAGE = 1

EXPORTS = ("wise_full_attn_accumulate", "wise_full_attn_accumulate_noalloc", "wise_select_support",
           "wise_sparse_attn", "wise_freeze_a_attn", "wise_freeze_a_probs", "wise_frozen_pv", "wise_support_mass",
           "wise_support_overlap",
           "wise_select_working_set", "wise_get_status", "wise_set_wait_limit_ns", "wise_status_string",
           "wise_version")
NOALLOC_SCRATCH_BYTES = 8 << 20


class WiseError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: {status_string(code)} ({code})")
        self.code = code


class wise_shape_t(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int), ("seqlen", ctypes.c_int), ("n_heads", ctypes.c_int),
                ("n_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int), ("block", ctypes.c_int),
                ("scale", ctypes.c_float)]


class wise_select_t(ctypes.Structure):
    _fields_ = [("n_sink", ctypes.c_int), ("n_local", ctypes.c_int), ("mode", ctypes.c_int),
                ("topk", ctypes.c_int), ("eta", ctypes.c_float), ("cap", ctypes.c_int)]


@dataclasses.dataclass(frozen=True)
class Shape:
    batch: int
    seqlen: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    block: int
    scale: float = 0.0

    @property
    def n_blocks(self) -> int:
        return self.seqlen // self.block

    def c(self) -> wise_shape_t:
        return wise_shape_t(self.batch, self.seqlen, self.n_heads, self.n_kv_heads, self.head_dim, self.block,
                            float(self.scale))


@dataclasses.dataclass(frozen=True)
class Select:
    n_sink: int
    n_local: int
    mode: int
    topk: int
    eta: float
    cap: int

    def c(self) -> wise_select_t:
        return wise_select_t(self.n_sink, self.n_local, self.mode, self.topk, float(self.eta), self.cap)


_lib = None


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """Loads libwise.so (building it first if it is missing or stale)."""
    global _lib
    if _lib is None:
        path = _build.build() if build_if_missing else _build.LIB
        if not os.path.exists(path):
            raise ImportError(f"libwise.so not built at {path}")
        lib = ctypes.CDLL(path)
        P = ctypes.c_void_p
        lib.wise_full_attn_accumulate.argtypes = [ctypes.POINTER(wise_shape_t), P, P, P, P, P, ctypes.c_int, P]
        lib.wise_full_attn_accumulate_noalloc.argtypes = [ctypes.POINTER(wise_shape_t), P, P, P, P, P, ctypes.c_int,
                                                          P]
        lib.wise_select_support.argtypes = [ctypes.POINTER(wise_shape_t), ctypes.POINTER(wise_select_t), P, P, P, P]
        lib.wise_sparse_attn.argtypes = [ctypes.POINTER(wise_shape_t), P, P, P, P, P, ctypes.c_int, P, P]
        lib.wise_freeze_a_attn.argtypes = [ctypes.POINTER(wise_shape_t), P, P, P, P, P, ctypes.c_int, P, P]
        lib.wise_freeze_a_probs.argtypes = [ctypes.POINTER(wise_shape_t), P, P, P, P, ctypes.c_int, P, P,
                                            ctypes.c_int, P]
        lib.wise_frozen_pv.argtypes = [ctypes.POINTER(wise_shape_t), P, P, ctypes.c_int, P, P, P, ctypes.c_int, P, P]
        lib.wise_support_mass.argtypes = [ctypes.POINTER(wise_shape_t), P, P, P, ctypes.c_int, P, P]
        I = ctypes.c_int
        lib.wise_support_overlap.argtypes = [ctypes.POINTER(wise_shape_t), P, P, I, P, P, I, P, P]
        lib.wise_select_working_set.argtypes = [ctypes.POINTER(wise_shape_t), I, ctypes.c_float, I, I, P, I, P, P,
                                                I, P, P, I, P]
        lib.wise_get_status.argtypes = [P]
        lib.wise_set_wait_limit_ns.argtypes = [ctypes.c_ulonglong]
        lib.wise_status_string.argtypes = [ctypes.c_int]
        lib.wise_status_string.restype = ctypes.c_char_p
        lib.wise_version.restype = ctypes.c_int
        _lib = lib
    return _lib


def status_string(code: int) -> str:
    return load().wise_status_string(int(code)).decode()


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _ptr(t) -> ctypes.c_void_p:
    return ctypes.c_void_p(0 if t is None else t.data_ptr())


def _check(t, name, shape, dtype):
    if t is None:
        raise ValueError(f"{name} is required")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def _qkvo(shape: Shape, Q, K, V, O):
    qs = (shape.batch, shape.n_heads, shape.seqlen, shape.head_dim)
    ks = (shape.batch, shape.n_kv_heads, shape.seqlen, shape.head_dim)
    _check(Q, "Q", qs, torch.bfloat16)
    _check(K, "K", ks, torch.bfloat16)
    _check(V, "V", ks, torch.bfloat16)
    _check(O, "O", qs, torch.bfloat16)


def wise_full_attn_accumulate(shape: Shape, Q, K, V, O, blockmass=None, step: int = 0, stream=None) -> None:
    """Dense causal attention (Eq. 2) of one step; with `blockmass` the step's
    block attention mass (Eq. 5) is written (step 0) or accumulated (step > 0)
    into it, fp32 [batch, n_heads, nQB, nKB]."""
    _qkvo(shape, Q, K, V, O)
    if blockmass is not None:
        nb = shape.n_blocks
        _check(blockmass, "blockmass", (shape.batch, shape.n_heads, nb, nb), torch.float32)
    sh = shape.c()
    rc = load().wise_full_attn_accumulate(ctypes.byref(sh), _ptr(Q), _ptr(K), _ptr(V), _ptr(O), _ptr(blockmass),
                                          int(step), _stream(stream))
    if rc != WISE_OK:
        raise WiseError(rc, "wise_full_attn_accumulate")


def wise_full_attn_accumulate_noalloc(shape: Shape, Q, K, V, O, blockmass, step: int = 0, stream=None) -> None:
    """wise_full_attn_accumulate with block mass, without any device
    allocation by the library: its scratch is a fixed 8 MiB array compiled
    into libwise.so.  For callers whose device memory is managed elsewhere or
    who cannot afford cudaMalloc's synchronisation; problems whose scratch
    would exceed the array are rejected (WiseError, WISE_ERR_UNSUPPORTED)."""
    _qkvo(shape, Q, K, V, O)
    nb = shape.n_blocks
    _check(blockmass, "blockmass", (shape.batch, shape.n_heads, nb, nb), torch.float32)
    sh = shape.c()
    rc = load().wise_full_attn_accumulate_noalloc(ctypes.byref(sh), _ptr(Q), _ptr(K), _ptr(V), _ptr(O),
                                                  _ptr(blockmass), int(step), _stream(stream))
    if rc != WISE_OK:
        raise WiseError(rc, "wise_full_attn_accumulate_noalloc")


def wise_select_support(shape: Shape, sel: Select, blockmass, idx, counts, stream=None) -> None:
    """Support selection (Eq. 6) into idx int32 [batch, n_kv_heads, nQB, cap]
    and counts int32 [batch, n_kv_heads, nQB]."""
    nb = shape.n_blocks
    _check(blockmass, "blockmass", (shape.batch, shape.n_heads, nb, nb), torch.float32)
    _check(idx, "idx", (shape.batch, shape.n_kv_heads, nb, sel.cap), torch.int32)
    _check(counts, "counts", (shape.batch, shape.n_kv_heads, nb), torch.int32)
    sh, se = shape.c(), sel.c()
    rc = load().wise_select_support(ctypes.byref(sh), ctypes.byref(se), _ptr(blockmass), _ptr(idx), _ptr(counts),
                                    _stream(stream))
    if rc != WISE_OK:
        raise WiseError(rc, "wise_select_support")


def wise_sparse_attn(shape: Shape, Q, K, V, idx, counts, O, stream=None) -> None:
    """Support-restricted attention (Eqs. 7-8) of one late step."""
    _qkvo(shape, Q, K, V, O)
    nb = shape.n_blocks
    if idx is None or idx.dim() != 4:
        raise ValueError("idx must be int32 [batch, n_kv_heads, nQB, cap]")
    cap = idx.shape[-1]
    _check(idx, "idx", (shape.batch, shape.n_kv_heads, nb, cap), torch.int32)
    _check(counts, "counts", (shape.batch, shape.n_kv_heads, nb), torch.int32)
    sh = shape.c()
    rc = load().wise_sparse_attn(ctypes.byref(sh), _ptr(Q), _ptr(K), _ptr(V), _ptr(idx), _ptr(counts), int(cap),
                                 _ptr(O), _stream(stream))
    if rc != WISE_OK:
        raise WiseError(rc, "wise_sparse_attn")


def wise_freeze_a_attn(shape: Shape, Q_frozen, K_frozen, V, idx, counts, O, stream=None) -> None:
    """Freeze-A control: the within-support attention distribution of a past
    step (its Q and K) applied to the current V, O = Abar V."""
    _qkvo(shape, Q_frozen, K_frozen, V, O)
    nb = shape.n_blocks
    if idx is None or idx.dim() != 4:
        raise ValueError("idx must be int32 [batch, n_kv_heads, nQB, cap]")
    cap = idx.shape[-1]
    _check(idx, "idx", (shape.batch, shape.n_kv_heads, nb, cap), torch.int32)
    _check(counts, "counts", (shape.batch, shape.n_kv_heads, nb), torch.int32)
    sh = shape.c()
    rc = load().wise_freeze_a_attn(ctypes.byref(sh), _ptr(Q_frozen), _ptr(K_frozen), _ptr(V), _ptr(idx),
                                   _ptr(counts), int(cap), _ptr(O), _stream(stream))
    if rc != WISE_OK:
        raise WiseError(rc, "wise_freeze_a_attn")


def freeze_tile_cap(shape: Shape, cap: int) -> int:
    """Smallest tile_cap the stored-distribution calls accept for support
    lists of row width `cap`."""
    return min((shape.seqlen + 127) // 128, (128 // shape.block) * cap)


def wise_freeze_a_probs(shape: Shape, Q_frozen, K_frozen, idx, counts, P, inv_l, stream=None) -> None:
    """Stores Abar of the frozen step as P bf16 [n_units, tile_cap, 128, 128]
    (row-max-relative exponentials) and inv_l fp32 [n_units, 128]."""
    _check(Q_frozen, "Q_frozen", (shape.batch, shape.n_heads, shape.seqlen, shape.head_dim), torch.bfloat16)
    _check(K_frozen, "K_frozen", (shape.batch, shape.n_kv_heads, shape.seqlen, shape.head_dim), torch.bfloat16)
    cap = _support(shape, idx, counts)
    tile_cap = _p_tiles(shape, P, inv_l)
    sh = shape.c()
    rc = load().wise_freeze_a_probs(ctypes.byref(sh), _ptr(Q_frozen), _ptr(K_frozen), _ptr(idx), _ptr(counts), cap,
                                    _ptr(P), _ptr(inv_l), tile_cap, _stream(stream))
    if rc != WISE_OK:
        raise WiseError(rc, "wise_freeze_a_probs")


def wise_frozen_pv(shape: Shape, P, inv_l, V, idx, counts, O, stream=None) -> None:
    """O = Abar V from the P and inv_l that wise_freeze_a_probs stored."""
    _check(V, "V", (shape.batch, shape.n_kv_heads, shape.seqlen, shape.head_dim), torch.bfloat16)
    _check(O, "O", (shape.batch, shape.n_heads, shape.seqlen, shape.head_dim), torch.bfloat16)
    cap = _support(shape, idx, counts)
    tile_cap = _p_tiles(shape, P, inv_l)
    sh = shape.c()
    rc = load().wise_frozen_pv(ctypes.byref(sh), _ptr(P), _ptr(inv_l), tile_cap, _ptr(V), _ptr(idx), _ptr(counts),
                               cap, _ptr(O), _stream(stream))
    if rc != WISE_OK:
        raise WiseError(rc, "wise_frozen_pv")


def _support(shape: Shape, idx, counts) -> int:
    if idx is None or idx.dim() != 4:
        raise ValueError("idx must be int32 [batch, n_kv_heads, nQB, cap]")
    cap = int(idx.shape[3])
    _check(idx, "idx", (shape.batch, shape.n_kv_heads, shape.n_blocks, cap), torch.int32)
    _check(counts, "counts", (shape.batch, shape.n_kv_heads, shape.n_blocks), torch.int32)
    return cap


def _p_tiles(shape: Shape, P, inv_l) -> int:
    n_units = shape.batch * shape.n_heads * ((shape.seqlen + 127) // 128)
    if P is None or P.dim() != 4:
        raise ValueError("P must be bf16 [n_units, tile_cap, 128, 128]")
    _check(P, "P", (n_units, int(P.shape[1]), 128, 128), torch.bfloat16)
    _check(inv_l, "inv_l", (n_units, 128), torch.float32)
    return int(P.shape[1])


def wise_support_overlap(shape: Shape, idx_a, counts_a, idx_b, counts_b, inter_union, stream=None) -> None:
    """inter_union int64 [batch, 2] (device; bit pattern of the C API's
    unsigned counts) = per batch element the number of (kv head, query block,
    key block) triples in both supports and in either."""
    nb = shape.n_blocks
    caps = []
    for name, idx, counts in (("idx_a", idx_a, counts_a), ("idx_b", idx_b, counts_b)):
        if idx is None or idx.dim() != 4:
            raise ValueError(f"{name} must be int32 [batch, n_kv_heads, nQB, cap]")
        caps.append(int(idx.shape[3]))
        _check(idx, name, (shape.batch, shape.n_kv_heads, nb, caps[-1]), torch.int32)
        _check(counts, "counts" + name[3:], (shape.batch, shape.n_kv_heads, nb), torch.int32)
    _check(inter_union, "inter_union", (shape.batch, 2), torch.int64)
    sh = shape.c()
    rc = load().wise_support_overlap(ctypes.byref(sh), _ptr(idx_a), _ptr(counts_a), caps[0], _ptr(idx_b),
                                     _ptr(counts_b), caps[1], _ptr(inter_union), _stream(stream))
    if rc != WISE_OK:
        raise WiseError(rc, "wise_support_overlap")


def wise_support_mass(shape: Shape, blockmass, idx, counts, retained, stream=None) -> None:
    """Routing diagnostic: retained[b, h, q] = sum of blockmass[b, h, q, kb]
    over the support list of the kv-group of h (fp32 [batch, n_heads, nQB]).
    With one step's mass this is the fraction of that step's full attention
    kept by the support."""
    nb = shape.n_blocks
    _check(blockmass, "blockmass", (shape.batch, shape.n_heads, nb, nb), torch.float32)
    if idx is None or idx.dim() != 4:
        raise ValueError("idx must be int32 [batch, n_kv_heads, nQB, cap]")
    cap = int(idx.shape[3])
    _check(idx, "idx", (shape.batch, shape.n_kv_heads, nb, cap), torch.int32)
    _check(counts, "counts", (shape.batch, shape.n_kv_heads, nb), torch.int32)
    _check(retained, "retained", (shape.batch, shape.n_heads, nb), torch.float32)
    sh = shape.c()
    rc = load().wise_support_mass(ctypes.byref(sh), _ptr(blockmass), _ptr(idx), _ptr(counts), cap, _ptr(retained),
                                  _stream(stream))
    if rc != WISE_OK:
        raise WiseError(rc, "wise_support_mass")


WS_UNION, WS_STATIC, WS_MASS_MATCHED, WS_SIZE_MATCHED = 0, 1, 2, 3


def wise_select_working_set(shape: Shape, mode: int, step_masses, idx, counts, eta: float = 0.95, n_sink: int = 0,
                            n_local: int = 0, ref_idx=None, ref_counts=None, stream=None) -> None:
    """The paper's working set (WS_UNION: union of the per-step eta coverage
    sets of the given steps, Eq. 6) or one of its controls (WS_STATIC,
    WS_MASS_MATCHED, WS_SIZE_MATCHED against ref_idx / ref_counts).
    step_masses fp32 [n_steps, batch, n_heads, nQB, nKB]; idx int32
    [batch, n_kv_heads, nQB, cap >= nQB], counts int32 [batch, n_kv_heads, nQB]."""
    nb = shape.n_blocks
    if step_masses is None or step_masses.dim() != 5:
        raise ValueError("step_masses must be fp32 [n_steps, batch, n_heads, nQB, nKB]")
    n_steps = int(step_masses.shape[0])
    _check(step_masses, "step_masses", (n_steps, shape.batch, shape.n_heads, nb, nb), torch.float32)
    if idx is None or idx.dim() != 4:
        raise ValueError("idx must be int32 [batch, n_kv_heads, nQB, cap]")
    cap = int(idx.shape[3])
    _check(idx, "idx", (shape.batch, shape.n_kv_heads, nb, cap), torch.int32)
    _check(counts, "counts", (shape.batch, shape.n_kv_heads, nb), torch.int32)
    ref_cap = 0
    if ref_idx is not None:
        ref_cap = int(ref_idx.shape[3])
        _check(ref_idx, "ref_idx", (shape.batch, shape.n_kv_heads, nb, ref_cap), torch.int32)
        _check(ref_counts, "ref_counts", (shape.batch, shape.n_kv_heads, nb), torch.int32)
    sh = shape.c()
    rc = load().wise_select_working_set(ctypes.byref(sh), int(mode), float(eta), int(n_sink), int(n_local),
                                        _ptr(step_masses), n_steps, _ptr(ref_idx), _ptr(ref_counts), ref_cap,
                                        _ptr(idx), _ptr(counts), cap, _stream(stream))
    if rc != WISE_OK:
        raise WiseError(rc, "wise_select_working_set")


def wise_get_status(stream=None) -> int:
    """Synchronizes the stream and returns (and clears) the device status word."""
    return int(load().wise_get_status(_stream(stream)))


def wise_set_wait_limit_ns(ns: int) -> None:
    """Limit of each internal wait of the attention kernels for later launches (0 = the 2 s default)."""
    if ns < 0:
        raise ValueError("ns must be >= 0")
    rc = load().wise_set_wait_limit_ns(int(ns))
    if rc != WISE_OK:
        raise WiseError(rc, "wise_set_wait_limit_ns")


def wise_version() -> int:
    return int(load().wise_version())


def shape_of(wl) -> Shape:
    """Shape of a synth.Workload."""
    return Shape(wl.batch, wl.seqlen, wl.n_heads, wl.n_kv_heads, wl.head_dim, wl.block)


def select_of(wl) -> Select:
    """Selection rule of a synth.Workload."""
    return Select(wl.n_sink, wl.n_local, wl.sel_mode, wl.topk, wl.eta, wl.cap)


class WiseAttention:
    """One attention layer's WISE state across a recurrent trajectory (Sec. 5).

    Steps 0 .. n_discovery-1 run dense attention and accumulate block mass;
    the first later step selects the support once; every later step runs
    support-restricted attention on that fixed support.  Q/K/V are supplied
    fresh at every step (they are recomputed by the model, Sec. 5.2).
    """

    def __init__(self, shape: Shape, sel: Select, n_discovery: int, device=None):
        if n_discovery < 1:
            raise ValueError("at least one discovery step is needed")
        self.shape, self.sel, self.n_discovery = shape, sel, n_discovery
        dev = torch.device("cuda") if device is None else torch.device(device)
        nb = shape.n_blocks
        self.blockmass = torch.zeros((shape.batch, shape.n_heads, nb, nb), dtype=torch.float32, device=dev)
        self.idx = torch.full((shape.batch, shape.n_kv_heads, nb, sel.cap), -1, dtype=torch.int32, device=dev)
        self.counts = torch.zeros((shape.batch, shape.n_kv_heads, nb), dtype=torch.int32, device=dev)
        self.selected = False

    def step(self, t: int, Q, K, V, O, stream=None) -> None:
        if t < self.n_discovery:
            wise_full_attn_accumulate(self.shape, Q, K, V, O, self.blockmass, t, stream)
            return
        if not self.selected:
            wise_select_support(self.shape, self.sel, self.blockmass, self.idx, self.counts, stream)
            self.selected = True
        wise_sparse_attn(self.shape, Q, K, V, self.idx, self.counts, O, stream)
