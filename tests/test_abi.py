"""The C ABI library: it builds, loads and exports every declared entry point;
host-side argument checks reject bad requests before touching the device."""

import ctypes
import os
import re

import pytest

from paper_2608_02703_gb300 import archead
from paper_2608_02703_gb300.build import INCLUDE, build


@pytest.fixture(scope="module")
def lib():
    build()
    return archead.load()


def declared_functions():
    with open(os.path.join(INCLUDE, "archead.h")) as f:
        text = f.read()
    return sorted(set(re.findall(r"ARCHEAD_API\s+[\w\s\*]*?\b(archead_\w+)\s*\(", text)))


def test_header_declares_the_abi():
    names = declared_functions()
    for must in ("archead_pack_create", "archead_forward", "archead_forward_ce", "archead_destroy"):
        assert must in names
    assert set(names) == set(archead.EXPORTED)


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert ctypes.cast(getattr(lib, name), ctypes.c_void_p).value


def test_status_strings(lib):
    for code, name in [(0, "ARCHEAD_OK"), (1, "ARCHEAD_ERR_INVALID_ARG"), (2, "ARCHEAD_ERR_UNSUPPORTED"),
                       (3, "ARCHEAD_ERR_OOM"), (4, "ARCHEAD_ERR_CUDA"), (5, "ARCHEAD_ERR_DEVICE_TIMEOUT"),
                       (6, "ARCHEAD_ERR_TARGET_RANGE")]:
        assert archead.archead_status_string(code) == name
    assert archead.archead_status_string(99) == "ARCHEAD_ERR_UNKNOWN"


def _desc(**kw):
    d = archead.archead_desc(vocab=100, hidden=256, core_rank=8, corr_rank=4, group_size=64, format=0)
    dummy = ctypes.c_void_p(16)  # never dereferenced: the checks below fail first
    for name, _ in archead.archead_desc._fields_[6:]:
        setattr(d, name, dummy)
    for k, v in kw.items():
        setattr(d, k, v)
    return d


@pytest.mark.parametrize("bad", [
    dict(vocab=0), dict(hidden=100), dict(hidden=32), dict(group_size=48), dict(group_size=16),
    dict(hidden=192, group_size=128), dict(core_rank=-1), dict(core_rank=257), dict(corr_rank=300),
    dict(format=2), dict(format=-1), dict(format=1, res_row_scale=None), dict(res_codes=None), dict(res_scales=None), dict(core_u=None), dict(corr_b_scale=None),
])
def test_pack_create_rejects_bad_desc(lib, bad):
    out = ctypes.c_void_p(1234)
    st = lib.archead_pack_create(ctypes.byref(_desc(**bad)), None, ctypes.byref(out))
    assert st == archead.ERR_INVALID_ARG
    assert out.value is None


def test_pack_create_null_args(lib):
    out = ctypes.c_void_p()
    assert lib.archead_pack_create(None, None, ctypes.byref(out)) == archead.ERR_INVALID_ARG
    assert lib.archead_pack_create(ctypes.byref(_desc()), None, None) == archead.ERR_INVALID_ARG


def test_null_pack_calls(lib):
    assert lib.archead_forward(None, None, 1, None, 0, None) == archead.ERR_INVALID_ARG
    assert lib.archead_forward_ce(None, None, 1, None, None, None) == archead.ERR_INVALID_ARG
    assert lib.archead_forward_host(None, None, 1, None, 0, None) == archead.ERR_INVALID_ARG
    assert lib.archead_debug_dequant(None, 0, 0, 1, None, None) == archead.ERR_INVALID_ARG
    assert lib.archead_sync_status(None, None) == archead.ERR_INVALID_ARG
    assert lib.archead_set_wait_budget(None, 10) == archead.ERR_INVALID_ARG
    assert lib.archead_debug_wait_timeout(None, None) == archead.ERR_INVALID_ARG
    assert lib.archead_profile_enable(None, 1) == archead.ERR_INVALID_ARG
    assert lib.archead_pack_bytes(None) == -1
    assert lib.archead_device_bytes(None) == -1
    lib.archead_destroy(None)
