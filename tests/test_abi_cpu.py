"""CPU checks of the C ABI: the library loads, exports exactly what
include/kvr.h declares, and its host-only arithmetic and argument checks
behave (no compute call needs a GPU here)."""
import ctypes
import os
import re

import pytest

from conftest import ROOT


def _declared():
    src = open(os.path.join(ROOT, "include", "kvr.h")).read()
    return sorted(set(re.findall(r"^KVR_API\s+[\w\s\*]+?\b(kvr_\w+)\s*\(", src, flags=re.M)))


@pytest.fixture(scope="module")
def kvr():
    from paper_2606_13361_gb300 import build
    build.build_library()
    from paper_2606_13361_gb300 import kvr as k
    return k


def test_library_exports_every_declared_symbol(kvr):
    decl = _declared()
    assert len(decl) >= 20
    lib = ctypes.CDLL(kvr.LIB_PATH)
    for name in decl:
        assert hasattr(lib, name), name
    assert sorted(kvr.EXPORTED) == decl


def test_sizes_match_the_paper_shapes(kvr):
    qwen = kvr.make_desc(36, 32, 8, 128, max_positions=40960)
    assert kvr.kvr_artifact_bytes(qwen, 1) == 147456
    assert kvr.kvr_artifact_bytes(qwen, 3774) == 3774 * 147456
    assert kvr.kvr_page_bytes(qwen) == 128 * 147456
    pool = kvr.kvr_pool_bytes(qwen, 64, 10)
    assert pool >= 10 * 128 * 147456
    bad = kvr.make_desc(36, 30, 8, 128, max_positions=1024)  # 30 % 8 != 0
    assert kvr.kvr_artifact_bytes(bad, 10) == 0
    assert kvr.kvr_pool_bytes(kvr.make_desc(1, 4, 1, 96, 1024), 1, 1) == 0  # head_dim 96


def test_status_strings_and_version(kvr):
    for s in range(9):
        assert kvr.kvr_status_string(s)
    assert kvr.kvr_status_string(99) == "unknown status"
    assert kvr.kvr_version() >= 100


def test_create_rejects_bad_arguments_before_any_cuda_call(kvr):
    d = kvr.make_desc(1, 4, 1, 64, max_positions=1024)
    out = ctypes.c_void_p()
    st = kvr.lib.kvr_create(ctypes.byref(d), None, 1 << 20, 4, 0, None, ctypes.byref(out))
    assert st == kvr.KVR_ERR_INVALID_ARG and "pool" in kvr.kvr_last_error()
    bad = kvr.make_desc(1, 4, 1, 64, max_positions=1024, dtype=7)
    st = kvr.lib.kvr_create(ctypes.byref(bad), ctypes.c_void_p(1 << 20), 1 << 20, 4, 0, None,
                            ctypes.byref(out))
    assert st == kvr.KVR_ERR_INVALID_ARG and "BF16" in kvr.kvr_last_error()
    assert kvr.lib.kvr_destroy(None) == kvr.KVR_ERR_INVALID_ARG
    assert kvr.lib.kvr_sync_status(None, None) == kvr.KVR_ERR_INVALID_ARG
    n = ctypes.c_int32()
    assert kvr.lib.kvr_seq_open(None, ctypes.byref(n)) == kvr.KVR_ERR_INVALID_ARG
