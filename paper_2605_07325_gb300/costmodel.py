"""Algorithmic work of one incremental-prefill call (host arithmetic only).

A call adds n tokens to a cache of L tokens.  The query of the token at
1-based position i attends to i keys, so the call covers

    sum_{i = L+1}^{L+n} i = n*L + n*(n+1)/2

query-key pairs: Eq. TTFT_derivation_2 with i* = L + 1 and |T_t| = L + n,
which the paper writes as (|T_t| - i* + 1)(|T_t| + i*) / 2.  Each pair costs
2*d flops for q.k and 2*d for the weighted sum of v, per query head:

    F = 4 * H_q * d * (n*L + n*(n+1)/2)      (masked work excluded)

Bytes the call must move at least once:

    B = (L + n) * H_kv * d * 2 * 2           keys and values read once
      + n * H_q * d * 2 * 2                  queries in, outputs out
      + n * H_kv * d * 2 * 2 * 2             new keys/values in and written

all bf16 (2 bytes).  The roofline floor of a call is max(F / peak_flops,
B / peak_bandwidth).
"""
from __future__ import annotations


def query_key_pairs(L: int, n: int) -> int:
    """sum_{i=L+1}^{L+n} i  (Eq. TTFT_derivation_2 with i* = L + 1)."""
    return n * L + n * (n + 1) // 2


def attention_flops(hq: int, d: int, L: int, n: int) -> float:
    return 4.0 * hq * d * query_key_pairs(L, n)


def call_bytes(hq: int, hkv: int, d: int, L: int, n: int) -> float:
    return 4.0 * (L + n) * hkv * d + 4.0 * n * hq * d + 8.0 * n * hkv * d


def attention_kernel_bytes(hq: int, hkv: int, d: int, L: int, n: int) -> float:
    """Bytes the attention kernel itself must move: K and V of L + n keys per
    kv head once, the packed rotated queries in and the outputs out."""
    return 4.0 * (L + n) * hkv * d + 4.0 * n * hq * d


def floor_seconds(flops: float, nbytes: float, peak_tflops: float, peak_gbs: float) -> float:
    return max(flops / (peak_tflops * 1e12), nbytes / (peak_gbs * 1e9))


def recon_extension_pairs(base_len: int, delta_n: int) -> int:
    """Pairs of extending a cache of base_len tokens by delta_n tokens:
    Delta N (2|T^E| + Delta N + 1) / 2 of App. D, Eq. recon_time."""
    return delta_n * (2 * base_len + delta_n + 1) // 2
