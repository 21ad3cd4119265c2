"""CPU oracle for the KV-reuse attention path (fp64).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, by ``__graft_entry__.smoke()``
and by the CPU-baseline leg of ``bench.py``.  The product library never imports,
links or runs anything here, and this package imports nothing from the product
package.  Inputs arrive as numpy arrays (bf16 values as uint16 bit patterns).

Paper: "Can I Buy Your KV Cache?" (arXiv 2606.13361).
  - Sec. 3 setup: per-layer keys/values; position i depends on x_{1:i} only.
  - Sec. 3.1 / Algorithm 1: the artifact is the per-layer K, V tensors plus
    metadata m = (model id, dtype, L); Sec. 5 "Artifact size": linear in L.
  - Sec. 3.2 / Algorithm 2: continuation positions L, L+1, ...; mask over the
    whole L+|q| span.
  - Sec. 3.3, Claim 1: reuse rows == prefill rows of prefix||suffix.
  - Sec. 4, Eq. 1-3: per-call cost and break-even count N*.
  - Sec. 5 "Quantizing the artifact": per-tensor symmetric int8 artifact.

Pins for every function live in tests/test_oracle_pins.py.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "kvr_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the C oracle (gcc, -O2, OpenMP) into oracle/liboracle.so."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-std=c11",
           "-fno-fast-math", "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
    subprocess.check_call(cmd)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            P = ctypes.c_void_p
            i64, i32, f64 = ctypes.c_int64, ctypes.c_int, ctypes.c_double
            lib.kvro_bf16_encode.argtypes = [P, i64, P]
            lib.kvro_bf16_decode.argtypes = [P, i64, P]
            lib.kvro_rmsnorm.argtypes = [i64, i32, P, P, f64, P]
            lib.kvro_rope.argtypes = [i64, i32, P, f64, P]
            lib.kvro_qk_prep.argtypes = [i64, i32, i32, i32, P, P, P, P, P, f64, f64,
                                         P, P, P, P]
            lib.kvro_attention.argtypes = [i64, i32, i32, i32, P, P, i64, P, P, P, P]
            lib.kvro_num_threads.restype = ctypes.c_int
            _lib = lib
    return _lib


def _p(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def num_threads() -> int:
    """OpenMP threads the oracle uses."""
    return int(_load().kvro_num_threads())


# ---------------------------------------------------------------- bf16 ----

def bf16_decode(h: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> exact fp64 values."""
    h = np.ascontiguousarray(h, dtype=np.uint16)
    out = np.empty(h.shape, dtype=np.float64)
    _load().kvro_bf16_decode(_p(h), h.size, _p(out))
    return out


def bf16_encode(x: np.ndarray) -> np.ndarray:
    """fp64 -> bf16 bit patterns, round to nearest, ties to even."""
    x = _f64(x)
    out = np.empty(x.shape, dtype=np.uint16)
    _load().kvro_bf16_encode(_p(x), x.size, _p(out))
    return out


# --------------------------------------------------------- norm / rope ----

def rmsnorm(x: np.ndarray, w: np.ndarray, eps: float) -> np.ndarray:
    """Per-vector RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * w."""
    x = _f64(x)
    d = x.shape[-1]
    w = _f64(w)
    y = np.empty_like(x)
    _load().kvro_rmsnorm(x.size // d, d, _p(x), _p(w), float(eps), _p(y))
    return y


def rope(x: np.ndarray, pos, theta: float) -> np.ndarray:
    """Rotate-half RoPE over the last axis; ``pos`` broadcasts over the
    leading axes (one position per vector)."""
    y = _f64(x).copy()
    d = y.shape[-1]
    n = y.size // d
    p = np.ascontiguousarray(np.broadcast_to(np.asarray(pos, dtype=np.int64),
                                             y.shape[:-1]).reshape(-1))
    assert p.size == n
    _load().kvro_rope(n, d, _p(p), float(theta), _p(y))
    return y


def qk_prep(q_pre, k_pre, wq, wk, pos, theta: float, eps: float):
    """Append-step math for new tokens (Sec. 3.2, positions L, L+1, ...).

    q_pre [T,Hq,d], k_pre [T,Hkv,d] (fp64 values, e.g. decoded bf16), wq/wk [d],
    pos [T].  Returns (q_f64, k_f64, q_bf16, k_bf16): RoPE(RMSNorm(.)) unrounded,
    and rounded once to bf16 (the cached keys and the q that attention reads)."""
    q_pre, k_pre = _f64(q_pre), _f64(k_pre)
    T, Hq, d = q_pre.shape
    Hkv = k_pre.shape[1]
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    assert pos.shape == (T,)
    wq, wk = _f64(wq), _f64(wk)
    qf = np.empty_like(q_pre)
    kf = np.empty_like(k_pre)
    qb = np.empty(q_pre.shape, dtype=np.uint16)
    kb = np.empty(k_pre.shape, dtype=np.uint16)
    _load().kvro_qk_prep(T, Hq, Hkv, d, _p(pos), _p(q_pre), _p(k_pre), _p(wq), _p(wk),
                         float(theta), float(eps), _p(qf), _p(kf), _p(qb), _p(kb))
    return qf, kf, qb, kb


# ------------------------------------------------------------ attention ----

def attention(q, row_pos, k, v):
    """Causal GQA attention, plain definition in fp64.

    q [R,Hq,d] rows at positions row_pos [R]; k, v [N,Hkv,d], key c at position c.
    Row r sees keys c <= row_pos[r].  Returns (O [R,Hq,d], lse [R,Hq])."""
    q, k, v = _f64(q), _f64(k), _f64(v)
    R, Hq, d = q.shape
    N, Hkv, dk = k.shape
    assert dk == d and v.shape == k.shape and Hq % Hkv == 0
    row_pos = np.ascontiguousarray(row_pos, dtype=np.int64)
    assert row_pos.shape == (R,)
    o = np.empty((R, Hq, d), dtype=np.float64)
    lse = np.empty((R, Hq), dtype=np.float64)
    _load().kvro_attention(R, Hq, Hkv, d, _p(q), _p(row_pos), N, _p(k), _p(v), _p(o), _p(lse))
    return o, lse


def prefill(q, k, v, rows=None):
    """Prefill attention over one sequence of N tokens (rows at positions
    0..N-1, keys 0..N-1); ``rows`` selects a subset of row indices."""
    N = k.shape[0]
    if rows is None:
        rows = np.arange(q.shape[0], dtype=np.int64)
    rows = np.asarray(rows, dtype=np.int64)
    return attention(np.asarray(q)[rows], rows, k, v)


def reuse(q_suffix, L: int, k_all, v_all, rows=None):
    """Reuse attention for suffix rows j at positions L+j over the prefix keys
    0..L-1 plus the suffix keys (k_all/v_all hold prefix||suffix)."""
    n = q_suffix.shape[0]
    if rows is None:
        rows = np.arange(n, dtype=np.int64)
    rows = np.asarray(rows, dtype=np.int64)
    return attention(np.asarray(q_suffix)[rows], L + rows, k_all, v_all)


# --------------------------------------------------------- artifact / cost ----

def artifact_bytes(layers: int, n_kv_heads: int, head_dim: int, L: int,
                   elem_bytes: int = 2) -> int:
    """Size of the per-layer K and V tensors of L positions (Sec. 2 'Prefill
    and the KV cache', Sec. 5 'Artifact size': linear in L)."""
    return layers * 2 * n_kv_heads * head_dim * elem_bytes * L


def per_call_cost(c_prefill: float, c_load: float, n):
    """Eq. 1-2: per-call cost from scratch (flat) and with KV reuse."""
    n = np.asarray(n, dtype=np.float64)
    return np.full_like(n, c_prefill), c_prefill / n + c_load


def break_even(c_prefill: float, c_load: float) -> float:
    """Eq. 3: N* = C_prefill / (C_prefill - C_load)."""
    return c_prefill / (c_prefill - c_load)


# ------------------------------------------------------------ int8 artifact ----
# Sec. 5 "Quantizing the artifact" stores the context's K/V at per-tensor
# symmetric int8 and names nothing else.  Readings (shared with the library):
# a tensor is one layer's K or one layer's V (all KV heads, all positions), its
# scale is s = max|x| / 127, a code is round-half-even(x / s) clamped to
# [-127, 127] (0 everywhere when s = 0), and the dequantised cache value is
# code * s rounded once to bf16.  The integer decision follows the rule that
# both sides take it in one precision: s, x / s and code * s are fp32
# operations (IEEE, correctly rounded) here and in the kernels.

def q8_quantize(x_bits: np.ndarray):
    """One tensor of bf16 bit patterns -> (int8 codes of the same shape, fp32 scale s)."""
    x = bf16_decode(x_bits).astype(np.float32)  # exact: bf16 values are fp32 values
    amax = np.float32(np.max(np.abs(x))) if x.size else np.float32(0.0)
    s = np.float32(amax / np.float32(127.0))
    if s == 0:
        return np.zeros(x.shape, dtype=np.int8), s
    with np.errstate(over="ignore"):
        r = np.rint(x / s)
    return np.clip(r, -127, 127).astype(np.int8), s


def q8_dequantize(codes: np.ndarray, s) -> np.ndarray:
    """int8 codes and their tensor's scale -> bf16 bit patterns of code * s
    (fp32 product, one rounding to bf16)."""
    p = codes.astype(np.float32) * np.float32(s)
    return bf16_encode(p.astype(np.float64))


def q8_artifact(art_bits: np.ndarray):
    """A bf16 artifact [layers][2][Hkv][L][d] -> (scales [layers][2] fp32,
    codes int8 of the same shape), one scale per layer's K and V tensor."""
    layers = art_bits.shape[0]
    scales = np.zeros((layers, 2), dtype=np.float32)
    codes = np.empty(art_bits.shape, dtype=np.int8)
    for l in range(layers):
        for kv in range(2):
            codes[l, kv], scales[l, kv] = q8_quantize(art_bits[l, kv])
    return scales, codes


def q8_artifact_dequantize(scales: np.ndarray, codes: np.ndarray) -> np.ndarray:
    """Inverse of q8_artifact up to the quantisation error: bf16 bits [layers][2][Hkv][L][d]."""
    out = np.empty(codes.shape, dtype=np.uint16)
    for l in range(codes.shape[0]):
        for kv in range(2):
            out[l, kv] = q8_dequantize(codes[l, kv], scales[l, kv])
    return out


def q8_artifact_values(scales: np.ndarray, codes: np.ndarray) -> np.ndarray:
    """The int8 artifact's tensors as exact values code * s in fp64 (an integer
    of at most 7 bits times an fp32 scale fits a double exactly): the keys and
    values that attention over an int8-resident prefix uses, without the bf16
    rounding of q8_artifact_dequantize.  [layers][2][Hkv][L][d]."""
    s = np.asarray(scales, dtype=np.float64)
    return codes.astype(np.float64) * s[:, :, None, None, None]


def q8_artifact_bytes(layers: int, n_kv_heads: int, head_dim: int, L: int) -> int:
    """Bytes of an int8 artifact: the fp32 scales (2 per layer, padded to 16
    bytes) followed by one byte per cached element."""
    return ((8 * layers + 15) // 16) * 16 + artifact_bytes(layers, n_kv_heads, head_dim, L, elem_bytes=1)


# ----------------------------------------------------------- full layer ----
# The paper's costs (Sec. 5, Table 1) are whole-model forwards of Qwen3-4B;
# the paper names the model, not its layer.  Readings (shared with the
# library): the public Qwen3 decoder layer -- pre-norm RMSNorm, q/k/v
# projections without bias, per-head q/k RMSNorm + rotate-half RoPE, causal
# GQA attention, output projection with a residual add, pre-norm RMSNorm,
# SwiGLU MLP (silu(x Wg^T) * (x Wu^T)) Wd^T with a residual add.  The model
# runs in bf16, so every tensor between two operations is a bf16 tensor: each
# step is computed here in fp64 from bf16 inputs and rounded once to bf16.

LAYER_WEIGHTS = ("input_norm", "wq", "wk", "wv", "q_norm", "k_norm", "wo", "post_norm", "w_gate", "w_up",
                 "w_down")


def silu(x: np.ndarray) -> np.ndarray:
    """x * sigmoid(x) in fp64."""
    x = _f64(x)
    return x / (1.0 + np.exp(-x))


def layer_forward(h_bits, W: dict, pos, k_cache_bits, v_cache_bits, n_q_heads: int, n_kv_heads: int,
                  theta: float, eps: float):
    """One decoder layer over T new tokens at positions pos [T] (consecutive,
    continuing the cache), with cached keys/values of positions 0..P-1
    (k_cache_bits, v_cache_bits [P, Hkv, d], keys after norm and RoPE).
    h_bits [T, hidden] is the residual stream in; W maps LAYER_WEIGHTS to bf16
    bits (projections [out, in], norms [width]).  Returns bf16 bits
    (h_out [T, hidden], k_new [T, Hkv, d], v_new [T, Hkv, d], o [T, Hq, d])."""
    dec, enc = bf16_decode, bf16_encode
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    T, hidden = h_bits.shape
    Hq, Hkv = n_q_heads, n_kv_heads
    d = dec(W["q_norm"]).shape[0]
    h = dec(h_bits)
    x = enc(rmsnorm(h, dec(W["input_norm"]), eps))
    q_pre = enc(dec(x) @ dec(W["wq"]).T).reshape(T, Hq, d)
    k_pre = enc(dec(x) @ dec(W["wk"]).T).reshape(T, Hkv, d)
    v_new = enc(dec(x) @ dec(W["wv"]).T).reshape(T, Hkv, d)
    _, _, qb, kb = qk_prep(dec(q_pre), dec(k_pre), dec(W["q_norm"]), dec(W["k_norm"]), pos, theta, eps)
    k_all = np.concatenate([dec(k_cache_bits), dec(kb)])
    v_all = np.concatenate([dec(v_cache_bits), dec(v_new)])
    o, _ = attention(dec(qb), pos, k_all, v_all)
    ob = enc(o)
    h1 = enc(h + dec(ob).reshape(T, Hq * d) @ dec(W["wo"]).T)
    x2 = dec(enc(rmsnorm(dec(h1), dec(W["post_norm"]), eps)))
    g = dec(enc(x2 @ dec(W["w_gate"]).T))
    u = dec(enc(x2 @ dec(W["w_up"]).T))
    a = dec(enc(silu(g) * u))
    h_out = enc(dec(h1) + a @ dec(W["w_down"]).T)
    return h_out, kb, v_new, ob


def linear(x_bits, w_bits, c_bits=None):
    """One projection of the layer as the bf16 model computes it: bf16(x W^T
    (+ c)) from bf16 x [T, K], W [N, K] (a Linear layer's [out, in]) and c
    [T, N], the product and sum in fp64, one rounding (the projection steps
    of layer_forward)."""
    y = bf16_decode(x_bits) @ bf16_decode(w_bits).T
    if c_bits is not None:
        y = y + bf16_decode(c_bits)
    return bf16_encode(y)


def linear_swiglu(x_bits, w_gate_bits, w_up_bits):
    """The MLP's first half as the bf16 model computes it (the gate, up and
    SwiGLU steps of layer_forward): g = bf16(x Wg^T), u = bf16(x Wu^T),
    a = bf16(silu(g) * u), each in fp64 from bf16 inputs."""
    g = bf16_decode(linear(x_bits, w_gate_bits))
    u = bf16_decode(linear(x_bits, w_up_bits))
    return bf16_encode(silu(g) * u)


def layer_flops(T: int, keys_per_row_sum: int, hidden: int, inter: int, Hq: int, Hkv: int, d: int) -> int:
    """Multiply-adds x 2 of one layer for T new tokens: the projections and the
    MLP (2 T hidden (Hq d + 2 Hkv d + Hq d) + 6 T hidden inter) plus attention
    (4 Hq d per visible (row, key) pair, keys_per_row_sum pairs per head)."""
    proj = 2 * T * hidden * (2 * Hq * d + 2 * Hkv * d)
    mlp = 6 * T * hidden * inter
    return proj + mlp + 4 * Hq * d * keys_per_row_sum
