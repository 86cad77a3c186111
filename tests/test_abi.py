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


def test_abi_version(lib):
    with open(os.path.join(INCLUDE, "archead.h")) as f:
        declared = int(re.search(r"#define ARCHEAD_ABI_VERSION (\d+)", f.read()).group(1))
    assert lib.archead_abi_version() == declared == archead.archead_abi_version() == 2


def test_pack_create_ex_reads_only_the_callers_struct(lib):
    """A struct of version 1 (up to corr_b_scale) is accepted for the INT8
    format; fields past desc_size read as absent even if the memory behind
    them is set, so the paper's format (which needs res_row_scale) is
    refused; a struct shorter than version 1 is refused."""
    v1 = archead.archead_desc.res_row_scale.offset
    out = ctypes.c_void_p(1234)
    assert lib.archead_pack_create_ex(ctypes.byref(_desc()), v1 - 8, None, ctypes.byref(out)) == archead.ERR_INVALID_ARG
    assert out.value is None
    assert lib.archead_pack_create_ex(None, v1, None, ctypes.byref(out)) == archead.ERR_INVALID_ARG
    sc4 = _desc(format=1)  # res_row_scale set, but past the size given
    assert lib.archead_pack_create_ex(ctypes.byref(sc4), v1, None, ctypes.byref(out)) == archead.ERR_INVALID_ARG
    # A version-1 INT8 struct reaches the shape checks (an invalid shape is reported as such).
    assert lib.archead_pack_create_ex(ctypes.byref(_desc(hidden=100)), v1, None,
                                      ctypes.byref(out)) == archead.ERR_INVALID_ARG


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


C_CLIENT = r"""
#include <stdio.h>
#include <string.h>
#include "archead.h"

/* A plain C client: the header must compile as C11 and the library must be
   callable without C++ (argument checks only; no device is needed). */
int main(void) {
  archead_desc d;
  archead_pack *pack = (archead_pack *)1;
  memset(&d, 0, sizeof d);
  d.vocab = 100; d.hidden = 256; d.core_rank = 8; d.corr_rank = 4; d.group_size = 64;
  d.format = ARCHEAD_FORMAT_SC4;  /* res_row_scale left NULL: rejected */
  if (archead_pack_create(&d, NULL, &pack) != ARCHEAD_ERR_INVALID_ARG || pack != NULL) return 1;
  if (archead_forward(NULL, NULL, 1, NULL, ARCHEAD_OUT_BF16, NULL) != ARCHEAD_ERR_INVALID_ARG) return 2;
  if (strcmp(archead_status_string(ARCHEAD_ERR_UNSUPPORTED), "ARCHEAD_ERR_UNSUPPORTED") != 0) return 3;
  if (archead_pack_bytes(NULL) != -1) return 4;
  archead_destroy(NULL);
  printf("c client ok\n");
  return 0;
}
"""


def test_plain_c_client_compiles_links_and_runs(lib, tmp_path):
    import subprocess

    src = tmp_path / "client.c"
    src.write_text(C_CLIENT)
    exe = tmp_path / "client"
    libdir = os.path.dirname(archead.library_path())
    subprocess.run(["gcc", "-std=c11", "-Wall", "-Werror", "-pedantic", f"-I{INCLUDE}", str(src), "-o", str(exe),
                    f"-L{libdir}", "-larchead", f"-Wl,-rpath,{libdir}"], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True)
    assert out.returncode == 0, out.stdout + out.stderr
    assert "c client ok" in out.stdout
