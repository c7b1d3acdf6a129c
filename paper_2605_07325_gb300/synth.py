"""Seeded synthetic inputs shared by the tests, the benchmark and the oracle runs.

This module holds no arithmetic of the method: it only draws numbers and rounds
them to bfloat16.  The synthetic Q/K/V stand in for the projections of
Eq. (k), (v) of section III-A (the paper's model weights and prompts are not
available); they are i.i.d. N(0, 1), drawn in float32 with
``numpy.random.default_rng(seed)`` in the order Q [n][hq][d], K [n][hkv][d],
V [n][hkv][d], then rounded to bfloat16 (round to nearest, ties to even).
Chunk ``c`` of a session uses seed ``base_seed + 1 + c`` and the static prefix
uses ``base_seed``, so a chunk can be regenerated when the cache is rebuilt.
Suffix blocks use ``base_seed + 1_000_000 + step``.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bfloat16 bit patterns (uint16), round to nearest even."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """bfloat16 bit patterns -> float64 (exact)."""
    u = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


@dataclass
class Block:
    """One block of new tokens: bf16 bits and their exact float64 values."""
    q: np.ndarray   # uint16 [n][hq][d]
    k: np.ndarray   # uint16 [n][hkv][d]
    v: np.ndarray   # uint16 [n][hkv][d]

    @property
    def n(self) -> int:
        return self.q.shape[0]

    def f64(self):
        return bf16_to_f64(self.q), bf16_to_f64(self.k), bf16_to_f64(self.v)


def block(seed: int, n: int, hq: int, hkv: int, d: int, kind: str = "normal") -> Block:
    """Draw one block.  ``kind``: "normal" (N(0,1)), "ones_v" (V = 1),
    "zero_k" (K = 0), "const_q" (every query row equal), "peaked" (Q and K
    scaled by 12: scores spread over hundreds of units, so a softmax that
    used a wrong row maximum would overflow or lose every weight),
    "kv_only" (K then V are drawn from the seed and Q is all zero:
    fill-phase chunks of long caches whose outputs are not compared)."""
    rng = np.random.default_rng(seed)
    if kind == "kv_only":
        k = rng.standard_normal((n, hkv, d), dtype=np.float32)
        v = rng.standard_normal((n, hkv, d), dtype=np.float32)
        return Block(np.zeros((n, hq, d), np.uint16), bf16_bits(k), bf16_bits(v))
    q = rng.standard_normal((n, hq, d), dtype=np.float32)
    k = rng.standard_normal((n, hkv, d), dtype=np.float32)
    v = rng.standard_normal((n, hkv, d), dtype=np.float32)
    if kind == "ones_v":
        v[...] = 1.0
    elif kind == "zero_k":
        k[...] = 0.0
    elif kind == "const_q":
        q[...] = q[:1]
    elif kind == "peaked":
        q *= 12.0
        k *= 12.0
    elif kind != "normal":
        raise ValueError(kind)
    return Block(bf16_bits(q), bf16_bits(k), bf16_bits(v))


def prefix_seed(base_seed: int) -> int:
    return base_seed


def chunk_seed(base_seed: int, chunk_index: int) -> int:
    return base_seed + 1 + chunk_index


def suffix_seed(base_seed: int, step: int) -> int:
    return base_seed + 1_000_000 + step
