"""Host-side checks of the C-ABI library: it builds for sm_103a, loads, exports
every entry point declared in include/wise.h, and rejects bad arguments
before touching a device.  No kernel is launched here."""
import ctypes
import os
import re

import pytest

from paper_2609_27373_gb300 import wise

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_entry_points():
    text = open(os.path.join(ROOT, "include", "wise.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(wise_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_entry_points()
    for n in ("wise_full_attn_accumulate", "wise_select_support", "wise_sparse_attn"):
        assert n in names
    assert set(names) == set(wise.EXPORTS)


def test_library_exports_every_declared_symbol():
    lib = wise.load()
    for name in declared_entry_points():
        assert hasattr(lib, name), name


def test_status_strings_and_version():
    assert wise.status_string(wise.WISE_OK) == "ok"
    for code in range(-6, 0):
        assert wise.status_string(code) != "unknown status"
    assert wise.status_string(-99) == "unknown status"
    assert wise.wise_version() >= 100


def _shape(**kw):
    d = dict(batch=1, seqlen=256, n_heads=2, n_kv_heads=2, head_dim=128, block=128, scale=0.0)
    d.update(kw)
    return wise.wise_shape_t(*d.values())


NULL = ctypes.c_void_p(0)


@pytest.mark.parametrize("kw,code", [
    (dict(block=16), wise.WISE_ERR_UNSUPPORTED),
    (dict(head_dim=80), wise.WISE_ERR_UNSUPPORTED),
    (dict(n_heads=3, n_kv_heads=2), wise.WISE_ERR_UNSUPPORTED),
    (dict(seqlen=200), wise.WISE_ERR_SHAPE),
    (dict(batch=-1), wise.WISE_ERR_INVALID_ARG),
    (dict(scale=-1.0), wise.WISE_ERR_INVALID_ARG),
    (dict(), wise.WISE_ERR_INVALID_ARG),          # NULL tensors
])
def test_attention_argument_checks(kw, code):
    lib = wise.load()
    sh = _shape(**kw)
    assert lib.wise_full_attn_accumulate(ctypes.byref(sh), NULL, NULL, NULL, NULL, NULL, 0, NULL) == code
    assert lib.wise_sparse_attn(ctypes.byref(sh), NULL, NULL, NULL, NULL, NULL, 4, NULL, NULL) == code


def test_empty_problems_are_a_no_op():
    lib = wise.load()
    for sh in (_shape(batch=0), _shape(seqlen=0)):
        assert lib.wise_full_attn_accumulate(ctypes.byref(sh), NULL, NULL, NULL, NULL, NULL, 0, NULL) == 0
        assert lib.wise_sparse_attn(ctypes.byref(sh), NULL, NULL, NULL, NULL, NULL, 4, NULL, NULL) == 0


@pytest.mark.parametrize("kw,code", [
    (dict(block=16), wise.WISE_ERR_UNSUPPORTED),
    (dict(head_dim=80), wise.WISE_ERR_UNSUPPORTED),
    (dict(seqlen=200), wise.WISE_ERR_SHAPE),
    (dict(batch=0, block=16), wise.WISE_ERR_UNSUPPORTED),   # empty, but still an invalid shape
    (dict(seqlen=0, head_dim=80), wise.WISE_ERR_UNSUPPORTED),
    (dict(batch=0), wise.WISE_OK),                           # empty and valid: a no-op
])
def test_noalloc_entry_point_checks_like_the_allocating_one(kw, code):
    # The same checks, in the same order, as wise_full_attn_accumulate with a
    # block-mass buffer (all of them run before any device is touched).
    lib = wise.load()
    sh = _shape(**kw)
    mass = ctypes.c_void_p(0x1000)
    assert lib.wise_full_attn_accumulate(ctypes.byref(sh), NULL, NULL, NULL, NULL, mass, 0, NULL) == code
    assert lib.wise_full_attn_accumulate_noalloc(ctypes.byref(sh), NULL, NULL, NULL, NULL, mass, 0, NULL) == code
    assert lib.wise_full_attn_accumulate_noalloc(ctypes.byref(sh), NULL, NULL, NULL, NULL, NULL, 0, NULL) == \
        wise.WISE_ERR_INVALID_ARG


def test_misaligned_pointer_is_rejected():
    lib = wise.load()
    sh = _shape()
    p = ctypes.c_void_p(0x1000 + 8)
    assert lib.wise_full_attn_accumulate(ctypes.byref(sh), p, p, p, p, NULL, 0, NULL) == wise.WISE_ERR_INVALID_ARG


@pytest.mark.parametrize("sel,code", [
    (wise.wise_select_t(1, 1, 0, 2, 0.0, 1), wise.WISE_ERR_INVALID_ARG),     # cap < forced blocks
    (wise.wise_select_t(1, 0, 0, 2, 0.0, 4), wise.WISE_ERR_INVALID_ARG),     # no diagonal
    (wise.wise_select_t(1, 1, 1, 0, 1.5, 4), wise.WISE_ERR_INVALID_ARG),     # eta > 1
    (wise.wise_select_t(1, 1, 7, 0, 0.5, 4), wise.WISE_ERR_INVALID_ARG),     # unknown mode
    (wise.wise_select_t(-1, 1, 0, 2, 0.0, 4), wise.WISE_ERR_INVALID_ARG),    # negative sink
    (wise.wise_select_t(1, 1, 0, 2, 0.0, 4), wise.WISE_ERR_INVALID_ARG),     # NULL buffers
])
def test_selection_argument_checks(sel, code):
    lib = wise.load()
    sh = _shape()
    assert lib.wise_select_support(ctypes.byref(sh), ctypes.byref(sel), NULL, NULL, NULL, NULL) == code
