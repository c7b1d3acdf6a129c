"""Helpers of the GPU parity tests: drive libcsr (through the C-ABI binding)
and the fp64 oracle in lockstep on the same seeded inputs, and compare.

Tolerances (bf16 inputs, fp32 accumulation):
  attention outputs and rotated keys: max-abs <= 2e-2 and relative Frobenius
  error <= 5e-3; values, page tables, slot maps, free lists: bit-exact;
  log-sum-exp: max-abs <= 1e-2.  The lse tolerance follows from the cache
  holding bf16 rotated keys and the kernel reading bf16 rotated queries: each
  score s = scale * q.k moves by scale * sum_i (dq_i k_i + q_i dk_i) with
  |dx| <= 2^-9 |x| uniformly spread, i.e. a standard deviation of about
  scale * sqrt(2d) * 2^-9 / sqrt(3) = 1.6e-3 for N(0,1) inputs (d = 64 or 128,
  scale = 1/sqrt(d)); lse moves by a softmax-weighted mean of those shifts,
  at most their maximum, so 1e-2 is about six standard deviations.
"""
from __future__ import annotations

import math
from typing import List, Optional

import numpy as np
import torch

from oracle import oracle as orc
from paper_2605_07325_gb300 import synth

TOL_MAX_ABS = 2e-2
TOL_REL_FRO = 5e-3
TOL_LSE = 1e-2

C1 = dict(hq=8, hkv=2, d=64, P=16, base=1e4)      # tiny correctness shape
C2 = dict(hq=64, hkv=4, d=128, P=64, base=1e6)    # the 8K/120K head shape


def csr_mod():
    from paper_2605_07325_gb300 import csr
    return csr


def to_dev(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def to_f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def bits_of(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def err_stats(got: np.ndarray, exp: np.ndarray):
    diff = got - exp
    max_abs = float(np.max(np.abs(diff))) if diff.size else 0.0
    denom = float(np.linalg.norm(exp))
    rel = float(np.linalg.norm(diff)) / denom if denom > 0 else float(np.linalg.norm(diff))
    return max_abs, rel


def assert_close(got: np.ndarray, exp: np.ndarray, what: str):
    assert got.shape == exp.shape, f"{what}: shape {got.shape} vs {exp.shape}"
    assert np.all(np.isfinite(got)), f"{what}: non-finite values"
    max_abs, rel = err_stats(got, exp)
    assert max_abs <= TOL_MAX_ABS and rel <= TOL_REL_FRO, (
        f"{what}: max-abs {max_abs:.3e} (tol {TOL_MAX_ABS}), rel-fro {rel:.3e} (tol {TOL_REL_FRO})")


def assert_lse_close(got: np.ndarray, exp: np.ndarray, what: str):
    err = float(np.max(np.abs(got - exp))) if got.size else 0.0
    assert err <= TOL_LSE, f"{what}: lse max-abs {err:.3e}"


class Pair:
    """A GPU context and an oracle session fed the same calls."""

    def __init__(self, shape: dict, pool_pages: int, max_seq: int, max_new: int = 1024,
                 seed: int = 0, **cfg_kw):
        csr = csr_mod()
        self.shape = shape
        self.hq, self.hkv, self.d, self.P = shape["hq"], shape["hkv"], shape["d"], shape["P"]
        self.cfg = csr.make_config(self.hq, self.hkv, self.d, self.P, shape["base"], max_new,
                                   pool_pages, max_seq, **cfg_kw)
        self.ctx = csr.Context(self.cfg)
        oracle_kw = {k: cfg_kw[k] for k in ("cap_tokens", "evict_tokens", "n_catchup") if k in cfg_kw}
        self.orc = orc.OracleCSR(self.hq, self.hkv, self.d, self.P, shape["base"], pool_pages,
                                 **oracle_kw)
        self.seed = seed
        self.blocks = {}          # chunk id -> synth.Block (for rebuild providers)
        self.outputs: List = []

    def blk(self, seed, n, kind="normal"):
        return synth.block(seed, n, self.hq, self.hkv, self.d, kind)

    def _dev(self, b: synth.Block):
        return to_dev(b.q), to_dev(b.k), to_dev(b.v)

    def _check(self, what, got_out, got_lse, exp, compare: bool):
        if not compare or exp[0] is None:
            return
        assert_close(to_f64(got_out), exp[0], what + " out")
        assert_lse_close(got_lse.cpu().numpy().astype(np.float64), exp[1], what + " lse")

    def _lse(self, n):
        return torch.empty((self.hq, n), dtype=torch.float32, device="cuda")

    def init_static(self, b: synth.Block, compare=True):
        q, k, v = self._dev(b)
        lse = self._lse(b.n)
        out, _ = self.ctx.init_static(q, k, v, lse=lse)
        self.orc.attend = compare
        exp = self.orc.init_static(*b.f64())
        self.orc.attend = True
        torch.cuda.synchronize()
        self._check("init_static", out, lse, exp, compare)
        return out, lse

    def append(self, b: synth.Block, compare=True):
        q, k, v = self._dev(b)
        lse = self._lse(b.n)
        self.orc.attend = compare
        exp = self.orc.append_chunk(*b.f64())
        self.orc.attend = True
        self.blocks[exp[2]] = b          # before the call: it may start a rebuild
        out, _, cid = self.ctx.append_chunk(q, k, v, lse=lse)
        assert cid == exp[2]
        torch.cuda.synchronize()
        self._check(f"chunk {cid}", out, lse, exp, compare)
        return out, lse, cid

    def fused(self, b: synth.Block, n_chunk: int, compare=True):
        """csr_append_chunk_attend_suffix of b (chunk = its first n_chunk
        tokens) against the oracle's append_chunk + attend_suffix."""
        q, k, v = self._dev(b)
        lse = self._lse(b.n)
        chunk = synth.Block(b.q[:n_chunk], b.k[:n_chunk], b.v[:n_chunk])
        suffix = synth.Block(b.q[n_chunk:], b.k[n_chunk:], b.v[n_chunk:])
        self.orc.attend = compare
        exp_c = self.orc.append_chunk(*chunk.f64())
        self.orc.attend = True
        exp_s = self.orc.attend_suffix(*suffix.f64()) if compare else (None, None)
        if not compare:
            self.orc.attend = False
            self.orc.attend_suffix(*suffix.f64())
            self.orc.attend = True
        self.blocks[exp_c[2]] = chunk     # before the call: it may start a rebuild
        out, _, cid = self.ctx.append_chunk_attend_suffix(q, k, v, n_chunk, lse=lse)
        assert cid == exp_c[2]
        torch.cuda.synchronize()
        self._check(f"fused chunk {cid}", out[:n_chunk], lse[:, :n_chunk], exp_c, compare)
        self._check("fused suffix", out[n_chunk:], lse[:, n_chunk:], exp_s, compare)
        return out, lse, cid

    def suffix(self, b: synth.Block, compare=True):
        q, k, v = self._dev(b)
        lse = self._lse(b.n)
        out, _ = self.ctx.attend_suffix(q, k, v, lse=lse)
        exp = self.orc.attend_suffix(*b.f64())
        torch.cuda.synchronize()
        self._check("suffix", out, lse, exp, compare)
        return out, lse

    def truncate(self):
        self.ctx.truncate_suffix()
        self.orc.truncate_suffix()

    def check_layout(self):
        csr = csr_mod()
        pt, length = self.ctx.layout(csr.VERSION_ACTIVE)
        assert length == self.orc.length()
        assert pt == self.orc.page_table(), "host page table differs from the oracle allocator"
        dev = self.ctx.device_page_table(csr.VERSION_ACTIVE).tolist()
        assert dev == pt, "device page table differs from the host page table"
        assert self.ctx.free_pages() == self.orc.free_ids()

    def check_cache(self, positions: Optional[np.ndarray] = None):
        """Rotated keys within tolerance, values bit-exact, at every position."""
        csr = csr_mod()
        L = self.orc.length()
        k_dev, v_dev = self.ctx.gather_kv(csr.VERSION_ACTIVE, 0, L)
        torch.cuda.synchronize()
        pos, k_exp, v_exp = self.orc.cache()
        assert np.array_equal(pos, np.arange(L))
        k_got = to_f64(k_dev)
        if positions is not None:
            k_got, k_exp = k_got[positions], k_exp[positions]
        assert_close(k_got, k_exp, "cached rotated keys")
        v_got = to_f64(v_dev)
        assert np.array_equal(v_got, v_exp), "cached values are not bit-exact"

    def device_clean(self):
        flags = self.ctx.device_status()
        assert flags == 0, f"device error word {flags:#x}"
