"""Seeded synthetic inputs shaped like the paper's Qwen3-4B workloads.

This module holds no arithmetic of the method: it only draws random numbers and
stores them as bf16 bit patterns.  Both the CUDA path (through the binding) and
the CPU oracle read what it returns.

Recipe (fixed order per draw, numpy PCG64 ``default_rng(seed)``):
  q_pre [T,Hq,d], k_pre [T,Hkv,d], v [T,Hkv,d] ~ N(0,1),
  q_norm_w [d], k_norm_w [d] = 1 + 0.1 N(0,1),
each drawn in fp64, rounded to fp32 by numpy, then to bf16 (ties to even).
Ragged suffix lengths are drawn first, from the same generator, when asked for.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp64/fp32 values -> bf16 bit patterns (uint16), via fp32, ties to even.
    Inputs are finite draws; NaN/Inf never occur here."""
    f = np.ascontiguousarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    r = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return r.astype(np.uint16)


def bf16_bits_to_f32(h: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> fp32 values (exact)."""
    return (np.ascontiguousarray(h, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


@dataclass
class LayerInputs:
    """Pre-norm projections of T new tokens for one layer (bf16 bit patterns)."""
    q_pre: np.ndarray   # [T, Hq, d]
    k_pre: np.ndarray   # [T, Hkv, d]
    v: np.ndarray       # [T, Hkv, d]
    q_norm_w: np.ndarray  # [d]
    k_norm_w: np.ndarray  # [d]


def layer_inputs(seed: int, T: int, Hq: int, Hkv: int, d: int) -> LayerInputs:
    rng = np.random.default_rng(seed)
    q = to_bf16_bits(rng.standard_normal((T, Hq, d)))
    k = to_bf16_bits(rng.standard_normal((T, Hkv, d)))
    v = to_bf16_bits(rng.standard_normal((T, Hkv, d)))
    wq = to_bf16_bits(1.0 + 0.1 * rng.standard_normal(d))
    wk = to_bf16_bits(1.0 + 0.1 * rng.standard_normal(d))
    return LayerInputs(q, k, v, wq, wk)


def ragged_lengths(seed: int, n: int, lo: int, hi: int) -> np.ndarray:
    """n suffix lengths uniform in [lo, hi] (inclusive), drawn before tensors."""
    rng = np.random.default_rng(seed)
    return rng.integers(lo, hi + 1, size=n).astype(np.int64)


def normal_bf16(seed: int, shape) -> np.ndarray:
    """N(0,1) draws as bf16 bit patterns (used for stand-in artifacts and for
    the synthetic greedy head's tables)."""
    rng = np.random.default_rng(seed)
    return to_bf16_bits(rng.standard_normal(shape))


def head_tables(seed: int, vocab: int, Hq: int, Hkv: int, d: int):
    """Synthetic greedy head: W_head [vocab, Hq*d] ~ N(0,1)/sqrt(Hq*d) and the
    token table E [vocab, (Hq+2Hkv)*d] ~ N(0,1) (the next token's pre-norm
    q/k/v rows).  Stand-ins for the LM head and embeddings, which need weights."""
    rng = np.random.default_rng(seed)
    W = to_bf16_bits(rng.standard_normal((vocab, Hq * d)) / np.sqrt(Hq * d))
    E = to_bf16_bits(rng.standard_normal((vocab, (Hq + 2 * Hkv) * d)))
    return W, E


# Workload shapes (Qwen3-4B attention: 36 layers, 32 query heads, 8 KV heads,
# head dim 128, RoPE theta 1e6, RMSNorm eps 1e-6).
TINY = dict(layers=1, Hq=4, Hkv=1, d=64, L=256, q=8, B=1)
QWEN_LAYER = dict(layers=1, Hq=32, Hkv=8, d=128, L=3774, q=64, B=1, decode_steps=24)
SERVING = dict(layers=36, Hq=32, Hkv=8, d=128, L=3774, q=128, B=64)
SWEEP_L = (1024, 2048, 4096, 8192, 16384, 32768)
HOT_DOC = dict(layers=36, Hq=32, Hkv=8, d=128, L=32768, B=256, q_lo=16, q_hi=512,
               decode_steps=24)
ROPE_THETA = 1.0e6
RMS_EPS = 1.0e-6
