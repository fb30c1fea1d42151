"""The C-ABI library loads and exports every symbol include/dms.h declares (no GPU calls)."""
import os
import re
import subprocess

import pytest

import paper_2506_05345_gb300 as dms
from paper_2506_05345_gb300 import _native

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "dms.h")


def _declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(dms_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(_native.LIB_PATH):
        from paper_2506_05345_gb300 import build
        build.build()
    return dms.library()


def test_header_declares_the_boundary():
    names = _declared_functions()
    for required in ("dms_cache_create", "dms_append_and_evict", "dms_decode_attention",
                     "dms_cache_stats"):
        assert required in names
    assert set(names) == set(_native.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in _declared_functions():
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", _native.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (dms_[a-z_]+)\b", out))
    assert set(_declared_functions()) <= exported


def test_status_strings(lib):
    assert _native.status_string(0) == "ok"
    assert "capacity" in _native.status_string(3)
    assert _native.status_string(99) == "unknown status"


def test_struct_layouts_match_header():
    import ctypes
    assert ctypes.sizeof(_native.dms_options) == 4 + 4 + 8 + 4 + 4 + 4 + 20
    assert ctypes.sizeof(_native.dms_stats) == 6 * 8 + 4 * 4


def test_invalid_arguments_rejected_on_host(lib):
    """Host-side checks run before any device call (no GPU needed)."""
    opt = _native.dms_options()
    opt.batch = 1
    code, h = dms.dms_cache_create(1, 8, 64, 16, 100, opt)  # head_dim must be 128
    assert code == _native.DMS_ERR_INVALID_ARGUMENT and h is None
    code, h = dms.dms_cache_create(0, 8, 128, 16, 100, opt)
    assert code == _native.DMS_ERR_INVALID_ARGUMENT
    code, h = dms.dms_cache_create(1, 8, 128, -1, 100, opt)
    assert code == _native.DMS_ERR_INVALID_ARGUMENT
    opt.batch = 0
    code, h = dms.dms_cache_create(1, 8, 128, 16, 100, opt)
    assert code == _native.DMS_ERR_INVALID_ARGUMENT
    opt.batch = 1024
    code, h = dms.dms_cache_create(1, 8, 128, 16, 100, opt)  # 8192 heads > 4096
    assert code == _native.DMS_ERR_INVALID_ARGUMENT
    assert lib.dms_append_and_evict(None, 0, None, None, None, 1, None) == 1
    assert lib.dms_decode_attention(None, 0, None, None, 4, 0.0, None) == 1
    assert lib.dms_decode_plan(None, 0, 4, None, None, None) == 1
    assert lib.dms_selftest_stale_flag(None, 0, 2000000) == 1


def test_kv_format_options_checked_on_host(lib):
    """The fp8 page format is taken only by the tiled decode kernel; unknown formats and
    nonzero reserved fields are rejected before any device call."""
    opt = _native.dms_options()
    opt.batch = 1
    opt.kv_format = _native.DMS_KV_FP8_E4M3
    opt.decode_kernel = _native.DMS_DECODE_SIMPLE
    code, h = dms.dms_cache_create(1, 2, 128, 16, 100, opt)
    assert code == _native.DMS_ERR_INVALID_ARGUMENT and h is None
    opt.decode_kernel = 4  # no such decode kernel
    opt.kv_format = 0
    code, h = dms.dms_cache_create(1, 2, 128, 16, 100, opt)
    assert code == _native.DMS_ERR_INVALID_ARGUMENT and h is None
    opt.decode_kernel = _native.DMS_DECODE_TILED
    opt.kv_format = 2
    code, h = dms.dms_cache_create(1, 2, 128, 16, 100, opt)
    assert code == _native.DMS_ERR_INVALID_ARGUMENT and h is None
    opt.kv_format = 0
    opt.reserved[2] = 1
    code, h = dms.dms_cache_create(1, 2, 128, 16, 100, opt)
    assert code == _native.DMS_ERR_INVALID_ARGUMENT and h is None
    assert lib.dms_cache_export_kv(None, 0, None, None, None, None) == 1
