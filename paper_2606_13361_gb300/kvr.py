"""Python binding of libkvr (include/kvr.h): same call names, argument
marshalling only.  Every step of the path runs in the library's CUDA kernels;
there is no Python or CPU fallback, and importing this module fails loudly when
the compiled library is missing.

Tensors are torch tensors (bf16 as torch.bfloat16, device memory unless noted);
streams default to torch's current CUDA stream.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libkvr.so")

KVR_OK = 0
KVR_ERR_INVALID_ARG = 1
KVR_ERR_META_MISMATCH = 2
KVR_ERR_POSITION = 3
KVR_ERR_OOM = 4
KVR_ERR_UNSUPPORTED = 5
KVR_ERR_TIMEOUT = 6
KVR_ERR_CUDA = 7
KVR_ERR_DEVICE = 8
KVR_DTYPE_BF16 = 1
KVR_DTYPE_Q8 = 2
KVR_ARTIFACT_HEADER_BYTES = 64
KVR_PAGE_TOKENS = 128
KVR_MAX_BATCH = 512

# Every symbol include/kvr.h declares.
EXPORTED = (
    "kvr_artifact_bytes", "kvr_page_bytes", "kvr_pool_bytes", "kvr_status_string", "kvr_last_error",
    "kvr_version", "kvr_create", "kvr_destroy", "kvr_free_pages", "kvr_launch_count", "kvr_sync_status", "kvr_seq_open",
    "kvr_seq_fork", "kvr_seq_close", "kvr_seq_length", "kvr_seq_reserve", "kvr_seq_advance",
    "kvr_load_kv", "kvr_export_kv", "kvr_append_kv", "kvr_reuse_attn", "kvr_prefill_attn",
    "kvr_reuse_attn_noalloc", "kvr_decode_step", "kvr_artifact_write_header", "kvr_artifact_read_header",
    "kvr_artifact_bytes_q8", "kvr_export_kv_q8", "kvr_layer_workspace_bytes", "kvr_layer_forward",
    "kvr_selftest_wait_timeout", "kvr_load_kv_q8_resident", "kvr_linear", "kvr_linear_swiglu",
)


class kvr_model_desc(ctypes.Structure):
    _fields_ = [("layers", ctypes.c_uint32), ("n_q_heads", ctypes.c_uint32),
                ("n_kv_heads", ctypes.c_uint32), ("head_dim", ctypes.c_uint32),
                ("dtype", ctypes.c_uint32), ("max_positions", ctypes.c_uint32),
                ("rope_theta", ctypes.c_double), ("rms_eps", ctypes.c_double),
                ("model_id", ctypes.c_uint64)]


class kvr_artifact_meta(ctypes.Structure):
    _fields_ = [("model_id", ctypes.c_uint64), ("dtype", ctypes.c_uint32), ("L", ctypes.c_uint32)]


class kvr_layer_desc(ctypes.Structure):
    _fields_ = [("hidden", ctypes.c_uint32), ("intermediate", ctypes.c_uint32)]


LAYER_WEIGHT_NAMES = ("input_norm", "wq", "wk", "wv", "q_norm", "k_norm", "wo", "post_norm", "w_gate_up",
                      "w_down")


class kvr_layer_weights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in LAYER_WEIGHT_NAMES]


class kvr_attn_opts(ctypes.Structure):
    _fields_ = [("num_splits", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class KvrError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"kvr status {status}: {msg}")
        self.status = status


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libkvr.so is not built ({LIB_PATH}); run __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    P, I, U32, SZ = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint32, ctypes.c_size_t
    I32P = ctypes.POINTER(ctypes.c_int32)
    DESC = ctypes.POINTER(kvr_model_desc)
    sig = {
        "kvr_artifact_bytes": (SZ, [DESC, U32]),
        "kvr_artifact_bytes_q8": (SZ, [DESC, U32]),
        "kvr_page_bytes": (SZ, [DESC]),
        "kvr_pool_bytes": (SZ, [DESC, U32, U32, SZ]),
        "kvr_status_string": (ctypes.c_char_p, [I]),
        "kvr_last_error": (ctypes.c_char_p, []),
        "kvr_version": (I, []),
        "kvr_create": (I, [DESC, P, SZ, U32, SZ, P, ctypes.POINTER(P)]),
        "kvr_destroy": (I, [P]),
        "kvr_free_pages": (I, [P, ctypes.POINTER(U32)]),
        "kvr_launch_count": (I, [P, ctypes.POINTER(ctypes.c_uint64)]),
        "kvr_sync_status": (I, [P, P]),
        "kvr_selftest_wait_timeout": (I, [P, P]),
        "kvr_seq_open": (I, [P, I32P]),
        "kvr_seq_fork": (I, [P, ctypes.c_int32, P, I32P]),
        "kvr_seq_close": (I, [P, ctypes.c_int32]),
        "kvr_seq_length": (I, [P, ctypes.c_int32, ctypes.POINTER(U32)]),
        "kvr_seq_reserve": (I, [P, I, I32P, I32P, P]),
        "kvr_seq_advance": (I, [P, I, I32P, I32P]),
        "kvr_load_kv": (I, [P, ctypes.POINTER(kvr_artifact_meta), P, I, P, I32P]),
        "kvr_export_kv": (I, [P, ctypes.c_int32, P, I, P, ctypes.POINTER(kvr_artifact_meta)]),
        "kvr_export_kv_q8": (I, [P, ctypes.c_int32, P, I, P, ctypes.POINTER(kvr_artifact_meta)]),
        "kvr_load_kv_q8_resident": (I, [P, ctypes.POINTER(kvr_artifact_meta), P, I, P, I32P]),
        "kvr_layer_workspace_bytes": (SZ, [DESC, ctypes.POINTER(kvr_layer_desc), U32]),
        "kvr_linear": (I, [P, I, I, I, P, P, P, P, P, SZ, P]),
        "kvr_linear_swiglu": (I, [P, I, I, I, P, P, P, P, SZ, P]),
        "kvr_layer_forward": (I, [P, I, ctypes.POINTER(kvr_layer_desc), ctypes.POINTER(kvr_layer_weights), I, I32P,
                                  I32P, I32P, P, P, P, SZ, P]),
        "kvr_artifact_write_header": (I, [DESC, ctypes.POINTER(kvr_artifact_meta), P]),
        "kvr_artifact_read_header": (I, [DESC, P, ctypes.POINTER(kvr_artifact_meta),
                                         ctypes.POINTER(ctypes.c_uint64)]),
        "kvr_append_kv": (I, [P, I, I, I32P, I32P, I32P, P, P, P, P, P, P, P]),
        "kvr_reuse_attn": (I, [P, I, I, I32P, I32P, P, P, P, ctypes.POINTER(kvr_attn_opts), P]),
        "kvr_prefill_attn": (I, [P, I, ctypes.c_int32, I, P, P, P, ctypes.POINTER(kvr_attn_opts), P]),
        "kvr_reuse_attn_noalloc": (I, [P, I, I, I32P, I32P, P, P, P, ctypes.POINTER(kvr_attn_opts), P]),
        "kvr_decode_step": (I, [P, I, I, I32P, I32P, I32P, P, P, P, P, P, P, P, P,
                                ctypes.POINTER(kvr_attn_opts), P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype, f.argtypes = res, args
    return lib


lib = _load()


def _check(status: int) -> None:
    if status != KVR_OK:
        raise KvrError(status, lib.kvr_last_error().decode(errors="replace"))


def _ptr(t):
    """Address of a tensor / array / int for a c_void_p parameter (None: NULL);
    a plain int, which ctypes converts, costs less per call than a c_void_p."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


_raw_stream = None


def _current_raw_stream() -> int:
    """torch's current stream on the current device, as a cudaStream_t value.
    torch.cuda.current_stream() builds a Python Stream object (about 3 us, more
    than the library's own host work per call); torch's raw accessor does not."""
    global _raw_stream
    if _raw_stream is None:
        import torch
        get = getattr(torch._C, "_cuda_getCurrentRawStream", None)
        dev = getattr(torch._C, "_cuda_getDevice", None)
        if get is not None and dev is not None:
            _raw_stream = lambda: get(dev())
        else:
            _raw_stream = lambda: torch.cuda.current_stream().cuda_stream
    return _raw_stream()


def _stream(stream):
    if stream is None:
        return _current_raw_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


_I32_CACHE = {}


def _i32(xs):
    """A read-only int32 array for a const int32_t* parameter.  The few small
    arrays a serving loop passes (sequence ids, cu_q, and start positions that
    stay the same across a step's layers) repeat, so they are kept by value;
    the library only reads them during the call."""
    key = tuple(int(x) for x in xs)
    arr = _I32_CACHE.get(key)
    if arr is None:
        if len(_I32_CACHE) >= 4096:
            _I32_CACHE.clear()
        arr = (ctypes.c_int32 * max(1, len(key)))(*key)
        _I32_CACHE[key] = arr
    return arr


def make_desc(layers, n_q_heads, n_kv_heads, head_dim, max_positions, rope_theta=1.0e6,
              rms_eps=1.0e-6, model_id=0x5157454E33344200, dtype=KVR_DTYPE_BF16) -> kvr_model_desc:
    return kvr_model_desc(layers, n_q_heads, n_kv_heads, head_dim, dtype, max_positions,
                          rope_theta, rms_eps, model_id)


# ------------------------------------------------------------ size helpers ----

def kvr_artifact_bytes(desc: kvr_model_desc, L: int) -> int:
    return int(lib.kvr_artifact_bytes(ctypes.byref(desc), L))


def kvr_artifact_bytes_q8(desc: kvr_model_desc, L: int) -> int:
    return lib.kvr_artifact_bytes_q8(ctypes.byref(desc), L)


def kvr_page_bytes(desc: kvr_model_desc) -> int:
    return int(lib.kvr_page_bytes(ctypes.byref(desc)))


def kvr_pool_bytes(desc: kvr_model_desc, max_seqs: int, n_pages: int, workspace_bytes: int = 0) -> int:
    return int(lib.kvr_pool_bytes(ctypes.byref(desc), max_seqs, n_pages, workspace_bytes))


def kvr_status_string(status: int) -> str:
    return lib.kvr_status_string(status).decode()


def kvr_last_error() -> str:
    return lib.kvr_last_error().decode(errors="replace")


def kvr_version() -> int:
    return int(lib.kvr_version())


# ------------------------------------------------------------------ context ----

def kvr_create(desc: kvr_model_desc, pool, pool_bytes: int, max_seqs: int,
               workspace_bytes: int = 0, stream=None) -> ctypes.c_void_p:
    out = ctypes.c_void_p()
    _check(lib.kvr_create(ctypes.byref(desc), _ptr(pool), pool_bytes, max_seqs, workspace_bytes,
                          _stream(stream), ctypes.byref(out)))
    return out


def kvr_destroy(ctx) -> None:
    _check(lib.kvr_destroy(ctx))


def kvr_free_pages(ctx) -> int:
    n = ctypes.c_uint32()
    _check(lib.kvr_free_pages(ctx, ctypes.byref(n)))
    return n.value


def kvr_launch_count(ctx) -> int:
    n = ctypes.c_uint64()
    _check(lib.kvr_launch_count(ctx, ctypes.byref(n)))
    return n.value


def kvr_sync_status(ctx, stream=None) -> int:
    """Returns the status code (does not raise): KVR_OK, KVR_ERR_TIMEOUT, ..."""
    return int(lib.kvr_sync_status(ctx, _stream(stream)))


def kvr_selftest_wait_timeout(ctx, stream=None) -> None:
    _check(lib.kvr_selftest_wait_timeout(ctx, _stream(stream)))


def kvr_seq_open(ctx) -> int:
    s = ctypes.c_int32()
    _check(lib.kvr_seq_open(ctx, ctypes.byref(s)))
    return s.value


def kvr_seq_fork(ctx, parent: int, stream=None) -> int:
    s = ctypes.c_int32()
    _check(lib.kvr_seq_fork(ctx, parent, _stream(stream), ctypes.byref(s)))
    return s.value


def kvr_seq_close(ctx, seq: int) -> None:
    _check(lib.kvr_seq_close(ctx, seq))


def kvr_seq_length(ctx, seq: int) -> int:
    n = ctypes.c_uint32()
    _check(lib.kvr_seq_length(ctx, seq, ctypes.byref(n)))
    return n.value


def kvr_seq_reserve(ctx, seqs, n_tokens, stream=None) -> None:
    _check(lib.kvr_seq_reserve(ctx, len(seqs), _i32(seqs), _i32(n_tokens), _stream(stream)))


def kvr_seq_advance(ctx, seqs, n_tokens) -> None:
    _check(lib.kvr_seq_advance(ctx, len(seqs), _i32(seqs), _i32(n_tokens)))


# ----------------------------------------------------------- artifact I/O ----

def kvr_load_kv(ctx, meta: kvr_artifact_meta, artifact, on_device: bool, stream=None) -> int:
    s = ctypes.c_int32()
    _check(lib.kvr_load_kv(ctx, ctypes.byref(meta), _ptr(artifact), int(on_device), _stream(stream),
                           ctypes.byref(s)))
    return s.value


def kvr_load_kv_q8_resident(ctx, meta: kvr_artifact_meta, artifact, on_device: bool, stream=None) -> int:
    s = ctypes.c_int32()
    _check(lib.kvr_load_kv_q8_resident(ctx, ctypes.byref(meta), _ptr(artifact), int(on_device), _stream(stream),
                                       ctypes.byref(s)))
    return s.value


def kvr_export_kv(ctx, seq: int, artifact, on_device: bool, stream=None) -> kvr_artifact_meta:
    m = kvr_artifact_meta()
    _check(lib.kvr_export_kv(ctx, seq, _ptr(artifact), int(on_device), _stream(stream), ctypes.byref(m)))
    return m


def kvr_artifact_write_header(desc: kvr_model_desc, meta: kvr_artifact_meta) -> bytes:
    buf = ctypes.create_string_buffer(KVR_ARTIFACT_HEADER_BYTES)
    _check(lib.kvr_artifact_write_header(ctypes.byref(desc), ctypes.byref(meta), buf))
    return buf.raw


def kvr_artifact_read_header(desc: kvr_model_desc, header: bytes):
    """Returns (meta, payload_bytes) of a container header, or raises KvrError."""
    if len(header) < KVR_ARTIFACT_HEADER_BYTES:
        raise KvrError(KVR_ERR_INVALID_ARG, f"header shorter than {KVR_ARTIFACT_HEADER_BYTES} bytes")
    buf = ctypes.create_string_buffer(bytes(header[:KVR_ARTIFACT_HEADER_BYTES]), KVR_ARTIFACT_HEADER_BYTES)
    m, n = kvr_artifact_meta(), ctypes.c_uint64()
    _check(lib.kvr_artifact_read_header(ctypes.byref(desc), buf, ctypes.byref(m), ctypes.byref(n)))
    return m, n.value


def save_artifact(path, desc: kvr_model_desc, meta: kvr_artifact_meta, payload) -> None:
    """Writes a container file: the header, then the artifact bytes (a host
    numpy array or CPU tensor of exactly the header's payload size)."""
    header = kvr_artifact_write_header(desc, meta)
    view = memoryview(payload.numpy() if hasattr(payload, "numpy") else payload).cast("B")
    if len(view) != payload_bytes(desc, meta):
        raise KvrError(KVR_ERR_INVALID_ARG, f"payload is {len(view)} bytes, L = {meta.L} needs "
                                            f"{payload_bytes(desc, meta)}")
    with open(path, "wb") as f:
        f.write(header)
        f.write(view)


def read_artifact(path, desc: kvr_model_desc, out=None):
    """Reads a container file, checking its header against `desc` (Algorithm 2's
    metadata check happens here and again in kvr_load_kv).  The payload goes into
    `out` (a host buffer of at least the payload size, e.g. a pinned CPU tensor)
    or a new numpy array.  Returns (meta, payload)."""
    with open(path, "rb") as f:
        meta, n = kvr_artifact_read_header(desc, f.read(KVR_ARTIFACT_HEADER_BYTES))
        if out is None:
            out = np.empty(n, dtype=np.uint8)
        view = memoryview(out.numpy() if hasattr(out, "numpy") else out).cast("B")
        if len(view) < n:
            raise KvrError(KVR_ERR_INVALID_ARG, f"output buffer of {len(view)} bytes < payload {n}")
        got = f.readinto(view[:n])
        if got != n:
            raise KvrError(KVR_ERR_INVALID_ARG, f"file holds {got} payload bytes, header says {n}")
    return meta, out


def kvr_export_kv_q8(ctx, seq: int, artifact, on_device: bool, stream=None) -> kvr_artifact_meta:
    m = kvr_artifact_meta()
    _check(lib.kvr_export_kv_q8(ctx, seq, _ptr(artifact), int(on_device), _stream(stream), ctypes.byref(m)))
    return m


def payload_bytes(desc: kvr_model_desc, meta: kvr_artifact_meta) -> int:
    """Artifact bytes for meta's encoding (bf16 or int8) and length."""
    return (kvr_artifact_bytes_q8 if meta.dtype == KVR_DTYPE_Q8 else kvr_artifact_bytes)(desc, meta.L)


# ----------------------------------------------------------- whole layer ----

def kvr_layer_workspace_bytes(desc: kvr_model_desc, ldesc: kvr_layer_desc, max_tokens: int) -> int:
    return lib.kvr_layer_workspace_bytes(ctypes.byref(desc), ctypes.byref(ldesc), max_tokens)


def layer_weights(tensors: dict) -> kvr_layer_weights:
    """kvr_layer_weights from a dict of device tensors keyed by LAYER_WEIGHT_NAMES."""
    return kvr_layer_weights(*[tensors[n].data_ptr() for n in LAYER_WEIGHT_NAMES])


def kvr_layer_forward(ctx, layer: int, ldesc: kvr_layer_desc, weights: kvr_layer_weights, seqs, start_pos, cu_q,
                      h_in, h_out, workspace, stream=None) -> None:
    _check(lib.kvr_layer_forward(ctx, layer, ctypes.byref(ldesc), ctypes.byref(weights), len(seqs), _i32(seqs),
                                 _i32(start_pos), _i32(cu_q), _ptr(h_in), _ptr(h_out), _ptr(workspace),
                                 workspace.numel() * workspace.element_size(), _stream(stream)))


def _nbytes(t):
    return 0 if t is None else t.numel() * t.element_size()


def kvr_linear(ctx, x, w, out, c=None, workspace=None, stream=None) -> None:
    """out[T][N] = bf16(x[T][K] w[N][K]^T (+ c[T][N])) on the tcgen05 GEMM;
    workspace (optional device tensor) lets short batches split K."""
    T, K = x.shape
    _check(lib.kvr_linear(ctx, T, w.shape[0], K, _ptr(x), _ptr(w), _ptr(c), _ptr(out), _ptr(workspace),
                          _nbytes(workspace), _stream(stream)))


def kvr_linear_swiglu(ctx, x, w_gate_up, out, workspace=None, stream=None) -> None:
    """out[T][I] = bf16(silu(bf16(x Wg^T)) * bf16(x Wu^T)), w_gate_up = [Wg; Wu] ([2 I][K])."""
    T, K = x.shape
    _check(lib.kvr_linear_swiglu(ctx, T, w_gate_up.shape[0] // 2, K, _ptr(x), _ptr(w_gate_up), _ptr(out),
                                 _ptr(workspace), _nbytes(workspace), _stream(stream)))


# --------------------------------------------------------------- hot path ----

def kvr_append_kv(ctx, layer: int, seqs, start_pos, cu_q, q_pre, k_pre, v, q_norm_w, k_norm_w,
                  q_out, stream=None) -> None:
    _check(lib.kvr_append_kv(ctx, layer, len(seqs), _i32(seqs), _i32(start_pos), _i32(cu_q),
                             _ptr(q_pre), _ptr(k_pre), _ptr(v), _ptr(q_norm_w), _ptr(k_norm_w),
                             _ptr(q_out), _stream(stream)))


def _opts(num_splits):
    return None if num_splits is None else ctypes.byref(kvr_attn_opts(int(num_splits), 0))


def kvr_reuse_attn(ctx, layer: int, seqs, cu_q, q, out, lse=None, num_splits=None,
                   stream=None) -> None:
    _check(lib.kvr_reuse_attn(ctx, layer, len(seqs), _i32(seqs), _i32(cu_q), _ptr(q), _ptr(out),
                              _ptr(lse), _opts(num_splits), _stream(stream)))


def kvr_decode_step(ctx, layer: int, seqs, start_pos, cu_q, q_pre, k_pre, v, q_norm_w, k_norm_w,
                    q_out, out, lse=None, num_splits=None, stream=None) -> None:
    _check(lib.kvr_decode_step(ctx, layer, len(seqs), _i32(seqs), _i32(start_pos), _i32(cu_q),
                               _ptr(q_pre), _ptr(k_pre), _ptr(v), _ptr(q_norm_w), _ptr(k_norm_w),
                               _ptr(q_out), _ptr(out), _ptr(lse), _opts(num_splits), _stream(stream)))


def kvr_reuse_attn_noalloc(ctx, layer: int, seqs, cu_q, q, out, lse=None, num_splits=None,
                           stream=None) -> None:
    """kvr_reuse_attn for callers that cannot allocate device memory: the split
    partials live in the library's fixed device scratch
    (KVR_NOALLOC_SCRATCH_BYTES).  Make the first call on a device before any
    stream capture; do not overlap calls on the GPU (they share the scratch)."""
    _check(lib.kvr_reuse_attn_noalloc(ctx, layer, len(seqs), _i32(seqs), _i32(cu_q), _ptr(q),
                                      _ptr(out), _ptr(lse), _opts(num_splits), _stream(stream)))


KVR_NOALLOC_SCRATCH_BYTES = 16 << 20


def kvr_prefill_attn(ctx, layer: int, seq: int, n_tokens: int, q, out, lse=None,
                     num_splits=None, stream=None) -> None:
    _check(lib.kvr_prefill_attn(ctx, layer, seq, n_tokens, _ptr(q), _ptr(out), _ptr(lse),
                                _opts(num_splits), _stream(stream)))


class Context:
    """A kvr context over a pool tensor allocated with torch (the library never
    allocates device memory itself).  Holds the pool alive until close()."""

    def __init__(self, desc: kvr_model_desc, n_pages: int, max_seqs: int = 64,
                 workspace_bytes: int = 0, stream=None, fill: int | None = None):
        import torch
        self.desc = desc
        nbytes = kvr_pool_bytes(desc, max_seqs, n_pages, workspace_bytes)
        if nbytes == 0:
            raise KvrError(KVR_ERR_INVALID_ARG, "invalid model description")
        self.pool = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
        if fill is not None:  # e.g. stale bytes left by an earlier user of the memory
            self.pool.fill_(fill)
        self.ctx = kvr_create(desc, self.pool, nbytes, max_seqs, workspace_bytes, stream)

    def close(self) -> None:
        if self.ctx is not None:
            kvr_destroy(self.ctx)
            self.ctx = None
            self.pool = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
