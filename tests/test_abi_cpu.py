"""CPU checks of the C ABI: the library loads, exports exactly what
include/kvr.h declares, and its host-only arithmetic and argument checks
behave (no compute call needs a GPU here)."""
import ctypes
import os
import re

import numpy as np
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
    assert kvr.lib.kvr_selftest_wait_timeout(None, None) == kvr.KVR_ERR_INVALID_ARG
    m8 = kvr.kvr_artifact_meta(0, kvr.KVR_DTYPE_Q8, 10)
    s8 = ctypes.c_int32()
    assert kvr.lib.kvr_load_kv_q8_resident(None, ctypes.byref(m8), None, 1, None, ctypes.byref(s8)) == \
        kvr.KVR_ERR_INVALID_ARG
    n = ctypes.c_int32()
    assert kvr.lib.kvr_seq_open(None, ctypes.byref(n)) == kvr.KVR_ERR_INVALID_ARG


def test_artifact_header_round_trip_and_layout(kvr, tmp_path):
    """Algorithm 1 stores m = (model, dtype, L) with (K, V); the container's
    header carries it in a fixed little-endian layout."""
    import struct
    import numpy as np
    d = kvr.make_desc(2, 4, 1, 64, max_positions=4096, model_id=0x1122334455667788)
    meta = kvr.kvr_artifact_meta(d.model_id, kvr.KVR_DTYPE_BF16, 300)
    h = kvr.kvr_artifact_write_header(d, meta)
    assert len(h) == kvr.KVR_ARTIFACT_HEADER_BYTES == 64
    fields = struct.unpack("<4sIQIIIIIIQ16s", h)
    assert fields == (b"KVRA", 1, 0x1122334455667788, kvr.KVR_DTYPE_BF16, 300, 2, 1, 64, 0,
                      2 * 2 * 1 * 300 * 64 * 2, bytes(16))
    m, n = kvr.kvr_artifact_read_header(d, h)
    assert (m.model_id, m.dtype, m.L, n) == (d.model_id, 1, 300, kvr.kvr_artifact_bytes(d, 300))
    payload = np.random.default_rng(5).integers(0, 256, n, dtype=np.uint8)
    path = tmp_path / "a.kvra"
    kvr.save_artifact(path, d, meta, payload)
    assert os.path.getsize(path) == 64 + n
    m2, back = kvr.read_artifact(path, d)
    assert m2.L == 300 and np.array_equal(back, payload)
    # the int8 encoding of the same model (Sec. 5): its own payload size
    q8 = kvr.kvr_artifact_meta(d.model_id, kvr.KVR_DTYPE_Q8, 300)
    hq = kvr.kvr_artifact_write_header(d, q8)
    assert struct.unpack_from("<I", hq, 16)[0] == kvr.KVR_DTYPE_Q8
    mq, nq = kvr.kvr_artifact_read_header(d, hq)
    assert mq.dtype == kvr.KVR_DTYPE_Q8 and nq == kvr.kvr_artifact_bytes_q8(d, 300) == 16 + 2 * 2 * 300 * 64


def test_artifact_header_rejects_foreign_and_malformed(kvr):
    """Algorithm 2 loads only an artifact whose metadata matches the model:
    another model id, dtype or shape is META_MISMATCH; a header that is not a
    container (magic, version, payload size) is INVALID_ARG."""
    d = kvr.make_desc(2, 4, 1, 64, max_positions=4096, model_id=7)
    h = bytearray(kvr.kvr_artifact_write_header(d, kvr.kvr_artifact_meta(7, 1, 10)))
    for other in (kvr.make_desc(2, 4, 1, 64, 4096, model_id=8),   # another model
                  kvr.make_desc(3, 4, 1, 64, 4096, model_id=7),   # layers
                  kvr.make_desc(2, 8, 2, 64, 4096, model_id=7),   # KV heads
                  kvr.make_desc(2, 4, 1, 128, 4096, model_id=7)):  # head_dim
        with pytest.raises(kvr.KvrError) as e:
            kvr.kvr_artifact_read_header(other, bytes(h))
        assert e.value.status == kvr.KVR_ERR_META_MISMATCH
    bad_dtype = bytearray(h)
    bad_dtype[16] = 3  # neither the model's dtype nor its int8 encoding
    with pytest.raises(kvr.KvrError) as e:
        kvr.kvr_artifact_read_header(d, bytes(bad_dtype))
    assert e.value.status == kvr.KVR_ERR_META_MISMATCH
    for off, val in ((0, 0x58), (4, 2), (40, 3)):  # magic, version, payload size
        bad = bytearray(h)
        bad[off] = val
        with pytest.raises(kvr.KvrError) as e:
            kvr.kvr_artifact_read_header(d, bytes(bad))
        assert e.value.status == kvr.KVR_ERR_INVALID_ARG
    with pytest.raises(kvr.KvrError) as e:  # writing another model's metadata
        kvr.kvr_artifact_write_header(d, kvr.kvr_artifact_meta(8, 1, 10))
    assert e.value.status == kvr.KVR_ERR_INVALID_ARG


def test_layer_workspace_and_argument_checks(kvr):
    """Host-only parts of the whole-layer call: the workspace covers the
    activations of T tokens (the gate/up rows only at decode sizes: above 8
    tokens SwiGLU runs in the gate/up GEMM's epilogue) and the split-K
    partials; bad arguments are refused before anything is enqueued."""
    d = kvr.make_desc(36, 32, 8, 128, max_positions=4096)
    ld = kvr.kvr_layer_desc(2560, 9728)
    n1, n2 = kvr.kvr_layer_workspace_bytes(d, ld, 1), kvr.kvr_layer_workspace_bytes(d, ld, 3774)
    per_tok = 2 * (3 * 2560 + 3 * 4096 + 2 * 1024 + 9728)  # x, h1, x2; q, q', o; k, v; a
    split = 16 << 20  # fp32 split-K partials of one projection (short batches)
    assert n1 >= 2 * (per_tok // 2 + 2 * 9728)
    assert 3774 * per_tok + split <= n2 <= 3774 * per_tok + split + 12 * 256
    assert kvr.kvr_layer_workspace_bytes(d, ld, 8) >= 8 * (per_tok + 4 * 9728)  # decode sizes: gate/up rows too
    assert kvr.kvr_layer_workspace_bytes(d, kvr.kvr_layer_desc(2560, 9727), 8) == 0
    w = kvr.kvr_layer_weights()
    st = kvr.lib.kvr_layer_forward(None, 0, ctypes.byref(ld), ctypes.byref(w), 1, kvr._i32([0]), kvr._i32([0]),
                                   kvr._i32([0, 4]), None, None, None, 0, None)
    assert st == kvr.KVR_ERR_INVALID_ARG


def test_i32_arrays_are_reused_by_value_and_bounded(kvr):
    """The binding keeps the small const int32 arrays it passes by value: the
    same values give the same array with those contents, different values a
    different array, and the store stays bounded."""
    a = kvr._i32([3, 5, 7])
    b = kvr._i32(np.array([3, 5, 7], dtype=np.int64))
    assert a is b and list(a) == [3, 5, 7]
    c = kvr._i32([3, 5, 8])
    assert c is not a and list(c) == [3, 5, 8] and list(a) == [3, 5, 7]
    assert list(kvr._i32([])) == [0]  # a one-element array for an empty list
    for i in range(5000):
        kvr._i32([i, i + 1])
    assert len(kvr._I32_CACHE) <= 4096
    assert list(kvr._i32([3, 5, 7])) == [3, 5, 7]
