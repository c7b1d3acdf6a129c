"""fp64 CPU oracle for CSR incremental-prefill attention over a paged cache.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
module.  It shares no code with the CUDA library: it never imports the product
package, and the product package never imports it.

Contents
--------
* ``rope`` / ``attention``: ctypes wrappers over ``oracle.c`` (fp64 RoPE and
  causal softmax attention, Eq. causal_attention_1..3 of section III-A).
* ``PageAllocatorModel``: a set of free physical page ids; every page request
  takes the smallest free id.  Independent of the library's allocator.
* ``Alg2Router``: the per-query routing state machine of Algorithm 2
  (sequence versions k, k_ready; continuation, bridging, swap, stragglers).
* ``OracleCSR``: the CSR cache lifecycle as a list of cached segments
  (section III-D: X_static = (X_pre, X_chunks), X_dyn = (X_suff, X_task)) with
  the operations of Algorithm 1: Increment (append a chunk, buffer it while a
  reconciliation runs), Evict (drop the oldest chunks, Eq. eviction_operation),
  Reconcile (rebuild the retained context at renumbered positions, catch up the
  buffered chunks) and the swap.  It produces the expected outputs, the
  expected page tables and the expected cache contents.

Readings where the paper is silent (kept identical in the library):
  R1 rotate-half RoPE, angle pos * base^(-2i/d);
  R2 query head h reads kv head h // (hq // hkv);
  R3 the suffix occupies positions len..len+m-1 and truncation releases the
     pages that hold only suffix slots;
  R4 the smallest free page id is taken for every page, in logical order; a
     call appending to the active version while a reconciliation runs reserves
     the active version's pages first, then the pages of the version being
     rebuilt;
  R5 eviction drops the oldest whole chunks until at least E tokens are gone;
     the prefix keeps its positions and its full pages are shared by both
     versions; a partly filled last prefix page is copied into a fresh page;
     retained chunks are renumbered contiguously after the prefix and their
     keys are rotated again from the pre-rotation inputs (a fresh prefill of
     the retained context, App. D step 3);
  R6 N_catchup chunks may be left to the swap, where they are computed on the
     foreground; page reservation does not depend on when that happens.
"""
from __future__ import annotations

import ctypes
import math
import os
from dataclasses import dataclass, field
from typing import Dict, List, Optional, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB = None


def _lib():
    global _LIB
    if _LIB is None:
        from . import build_oracle  # noqa: WPS433 (local import keeps import cheap)
        path = build_oracle.build()
        lib = ctypes.CDLL(path)
        d = ctypes.POINTER(ctypes.c_double)
        i64 = ctypes.POINTER(ctypes.c_int64)
        lib.oracle_rope.argtypes = [d, i64, ctypes.c_int64, ctypes.c_int32,
                                    ctypes.c_int32, ctypes.c_double, d]
        lib.oracle_rope.restype = None
        lib.oracle_attention.argtypes = [d, i64, ctypes.c_int64, d, d, i64,
                                         ctypes.c_int64, ctypes.c_int32,
                                         ctypes.c_int32, ctypes.c_int32,
                                         ctypes.c_double, d, d, ctypes.c_int32]
        lib.oracle_attention.restype = ctypes.c_int
        _LIB = lib
    return _LIB


def _dp(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def _ip(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int64))


def default_threads() -> int:
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:  # pragma: no cover
        return max(1, os.cpu_count() or 1)


def rope(x: np.ndarray, pos: np.ndarray, base: float) -> np.ndarray:
    """Rotate-half RoPE of x[n][h][d] at absolute positions pos[n] (reading R1)."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    n, h, d = x.shape
    assert pos.shape == (n,) and d % 2 == 0
    y = np.empty_like(x)
    _lib().oracle_rope(_dp(x), _ip(pos), n, h, d, float(base), _dp(y))
    return y


def attention(q: np.ndarray, qpos: np.ndarray, k: np.ndarray, v: np.ndarray,
              kpos: np.ndarray, scale: float,
              threads: Optional[int] = None) -> Tuple[np.ndarray, np.ndarray]:
    """Causal softmax attention (Eq. causal_attention_1..3), fp64.

    q[n][hq][d] and k[nk][hkv][d] are already rotated; key tau is visible to
    query t iff kpos[tau] <= qpos[t].  Returns out[n][hq][d] and lse[hq][n]
    (natural log of the softmax normaliser of the scaled scores).
    """
    q = np.ascontiguousarray(q, dtype=np.float64)
    k = np.ascontiguousarray(k, dtype=np.float64)
    v = np.ascontiguousarray(v, dtype=np.float64)
    qpos = np.ascontiguousarray(qpos, dtype=np.int64)
    kpos = np.ascontiguousarray(kpos, dtype=np.int64)
    n, hq, d = q.shape
    nk, hkv, d2 = k.shape
    assert d2 == d and v.shape == k.shape and qpos.shape == (n,) and kpos.shape == (nk,)
    out = np.zeros((n, hq, d), dtype=np.float64)
    lse = np.zeros((hq, n), dtype=np.float64)
    rc = _lib().oracle_attention(_dp(q), _ip(qpos), n, _dp(k), _dp(v), _ip(kpos),
                                 nk, hq, hkv, d, float(scale), _dp(out), _dp(lse),
                                 int(threads or default_threads()))
    if rc != 0:
        raise RuntimeError("oracle_attention failed")
    return out, lse


# --------------------------------------------------------------------------
# Page allocator model (reading R4)
# --------------------------------------------------------------------------
class OracleOutOfPages(RuntimeError):
    pass


class PageAllocatorModel:
    """Free physical page ids kept as a Python set; each request takes min()."""

    def __init__(self, pool_pages: int):
        self.pool_pages = pool_pages
        self.free = set(range(pool_pages))
        self.refs: Dict[int, int] = {}

    def take(self) -> int:
        if not self.free:
            raise OracleOutOfPages("pool exhausted")
        pid = min(self.free)
        self.free.remove(pid)
        self.refs[pid] = 1
        return pid

    def share(self, pid: int) -> None:
        self.refs[pid] += 1

    def release(self, pid: int) -> None:
        self.refs[pid] -= 1
        if self.refs[pid] == 0:
            del self.refs[pid]
            self.free.add(pid)


# --------------------------------------------------------------------------
# CSR cache lifecycle model
# --------------------------------------------------------------------------
@dataclass
class Segment:
    kind: str                          # "prefix" | "chunk" | "suffix"
    ident: int                         # chunk id (or -1)
    pos: np.ndarray                    # absolute positions [m]
    k_rot: Optional[np.ndarray] = None # [m][hkv][d] rotated keys (None: not yet rebuilt)
    v: Optional[np.ndarray] = None     # [m][hkv][d]


@dataclass
class Version:
    segments: List[Segment] = field(default_factory=list)
    pages: List[int] = field(default_factory=list)

    @property
    def length(self) -> int:
        return int(sum(len(s.pos) for s in self.segments))

    def concat(self):
        if not self.segments:
            return (np.zeros((0,), np.int64), None, None)
        pos = np.concatenate([s.pos for s in self.segments])
        k = np.concatenate([s.k_rot for s in self.segments])
        v = np.concatenate([s.v for s in self.segments])
        return pos, k, v


class OracleCSR:
    """Reference model of the CSR cache lifecycle (section III-D, Algorithm 1)."""

    def __init__(self, hq: int, hkv: int, d: int, page_size: int,
                 rope_base: float, pool_pages: int, scale: Optional[float] = None,
                 cap_tokens: int = 0, evict_tokens: int = 0, n_catchup: int = 0,
                 threads: Optional[int] = None):
        assert hq % hkv == 0 and d % 2 == 0
        self.hq, self.hkv, self.d, self.P = hq, hkv, d, page_size
        self.base = rope_base
        self.scale = scale if scale is not None else 1.0 / math.sqrt(d)
        self.cap_tokens, self.evict_tokens, self.n_catchup = cap_tokens, evict_tokens, n_catchup
        self.alloc = PageAllocatorModel(pool_pages)
        self.active = Version()
        self.pending: Optional[Version] = None   # version being reconciled
        self.buffer: List[int] = []              # Delta X_buffer (chunk ids)
        self.sources: Dict[int, Tuple[np.ndarray, np.ndarray, np.ndarray]] = {}
        self.next_chunk_id = 0
        self.prefix_len = 0
        self.has_static = False
        self.threads = threads
        self.attend = True   # False: cache bookkeeping only (fill phases)

    # ---- helpers ---------------------------------------------------------
    @property
    def is_reconciling(self) -> bool:
        return self.pending is not None

    def _pages_for(self, length: int) -> int:
        return (length + self.P - 1) // self.P

    def _grow(self, ver: Version, new_len: int) -> None:
        while len(ver.pages) < self._pages_for(new_len):
            ver.pages.append(self.alloc.take())

    def _attend_new(self, ver: Version, q_rot: np.ndarray, qpos: np.ndarray):
        kpos, k, v = ver.concat()
        return attention(q_rot, qpos, k, v, kpos, self.scale, self.threads)

    def _add(self, ver: Version, kind: str, ident: int, q, k, v):
        """Rotate the block at positions len..len+n-1, cache it, attend it
        (the attention is skipped while ``self.attend`` is False)."""
        n = q.shape[0]
        L = ver.length
        pos = np.arange(L, L + n, dtype=np.int64)
        self._grow(ver, L + n)
        k_rot = rope(k, pos, self.base)
        ver.segments.append(Segment(kind, ident, pos, k_rot, np.array(v, np.float64)))
        if not self.attend:
            return None, None
        q_rot = rope(q, pos, self.base)
        return self._attend_new(ver, q_rot, pos)

    # ---- operations --------------------------------------------------------
    def init_static(self, q, k, v):
        """X_pre: computed once (Eq. x_static)."""
        if self.has_static or q.shape[0] == 0:
            raise ValueError("static prefix already set or empty")
        self.has_static = True
        self.prefix_len = q.shape[0]
        return self._add(self.active, "prefix", -1, q, k, v)

    def append_chunk(self, q, k, v):
        """Algorithm 1, Increment: X_static <- X_static (+) Delta X_t."""
        if not self.has_static or self._live_suffix(self.active):
            raise ValueError("bad state for append")
        cid = self.next_chunk_id
        self.next_chunk_id += 1
        self.sources[cid] = (np.array(q, np.float64), np.array(k, np.float64),
                             np.array(v, np.float64))
        was_reconciling = self.is_reconciling
        out = self._add(self.active, "chunk", cid, q, k, v)
        if not self.attend:
            self.sources.pop(cid, None)   # fill-phase chunks are never rebuilt
        if was_reconciling:
            # reserve the rebuilt version's pages now (reading R4), buffer the chunk
            start = self.pending.length
            n = q.shape[0]
            self._grow(self.pending, start + n)
            self.pending.segments.append(
                Segment("chunk", cid, np.arange(start, start + n, dtype=np.int64)))
            self.buffer.append(cid)
        return out[0], out[1], cid

    def _live_suffix(self, ver: Version) -> bool:
        return bool(ver.segments) and ver.segments[-1].kind == "suffix"

    def attend_suffix(self, q, k, v):
        """X_dyn = (X_suff, X_task), recomputed per task (Eq. x_dynamic)."""
        if not self.has_static or self._live_suffix(self.active):
            raise ValueError("bad state for suffix")
        return self._add(self.active, "suffix", -1, q, k, v)

    def truncate_suffix(self):
        ver = self.active
        if not self._live_suffix(ver):
            raise ValueError("no suffix")
        ver.segments.pop()
        keep = self._pages_for(ver.length)
        while len(ver.pages) > keep:
            self.alloc.release(ver.pages.pop())

    def rewind(self, length: int) -> None:
        """Keep the first `length` tokens: the cache is valid up to the first
        differing token (Eq. first_differing_token); later chunks are dropped."""
        ver = self.active
        if self._live_suffix(ver) or self.is_reconciling:
            raise ValueError("suffix live or reconciling")
        at, keep = 0, 0
        while at < length and keep < len(ver.segments):
            at += len(ver.segments[keep].pos)
            keep += 1
        if at != length:
            raise ValueError("not a segment boundary")
        ver.segments = ver.segments[:keep]
        while len(ver.pages) > self._pages_for(length):
            self.alloc.release(ver.pages.pop())

    def chunk_ids(self) -> List[int]:
        return [s.ident for s in self.active.segments if s.kind == "chunk"]

    def evict(self, evict_tokens: int) -> None:
        """Eq. eviction_operation on a copy: T^E = E(T_t) (App. D steps 1-2).

        The rebuilt version is reserved here; its contents are produced by
        ``reconcile_outputs`` (warm-up) and ``swap`` (catch-up).
        """
        if self.is_reconciling or self._live_suffix(self.active):
            raise ValueError("busy or suffix live")
        chunks = [s for s in self.active.segments if s.kind == "chunk"]
        dropped, drop_ids = 0, []
        for s in chunks:
            if dropped >= evict_tokens:
                break
            drop_ids.append(s.ident)
            dropped += len(s.pos)
        retained = [s for s in chunks if s.ident not in drop_ids]
        P = self.P
        new = Version()
        full_prefix_pages = self.prefix_len // P
        for i in range(full_prefix_pages):
            pid = self.active.pages[i]
            self.alloc.share(pid)
            new.pages.append(pid)
        prefix_seg = self.active.segments[0]
        new.segments.append(prefix_seg)
        start = self.prefix_len
        for s in retained:   # renumbered contiguously after the prefix (R5)
            m = len(s.pos)
            new.segments.append(
                Segment("chunk", s.ident, np.arange(start, start + m, dtype=np.int64)))
            start += m
        self._grow(new, start)
        self.pending = new
        self.retained_ids = [s.ident for s in retained]
        self.dropped_ids = drop_ids
        self.buffer = []

    def _materialise(self, ver: Version, cid: int):
        """Re-prefill one chunk of ``ver`` at its renumbered position (R5)."""
        idx = [i for i, s in enumerate(ver.segments) if s.kind == "chunk" and s.ident == cid][0]
        pos = ver.segments[idx].pos
        if cid not in self.sources:      # bookkeeping-only session (attend False)
            return None, None
        q, k, v = self.sources[cid]
        q_rot = rope(q, pos, self.base)
        k_rot = rope(k, pos, self.base)
        ver.segments[idx] = Segment("chunk", cid, pos, k_rot, np.array(v, np.float64))
        # causal attention of this chunk over the version up to and including itself
        sub = Version(segments=ver.segments[: idx + 1])
        return self._attend_new(sub, q_rot, pos)

    def reconcile(self) -> Dict[int, Tuple[np.ndarray, np.ndarray]]:
        """Algorithm 1, Reconcile: warm-up on the retained chunks, then catch up
        every buffered chunk, then swap (N_catchup chunks may be left for the
        swap, which computes them too: the resulting state is the same)."""
        assert self.pending is not None
        outs = {}
        for cid in self.retained_ids + list(self.buffer):
            outs[cid] = self._materialise(self.pending, cid)
        self._swap()
        return outs

    def cancel(self) -> None:
        """Abandon the reconciliation (App. D: the swap never follows an
        unfinished rebuild): the rebuilt version's page references are
        released; the active version, including the chunks appended while
        reconciling, stays as it is."""
        assert self.pending is not None
        for pid in self.pending.pages:
            self.alloc.release(pid)
        self.pending = None
        self.buffer = []

    def _swap(self):
        old = self.active
        for pid in old.pages:
            self.alloc.release(pid)
        self.active = self.pending
        self.pending = None
        self.buffer = []

    # ---- inspection ----------------------------------------------------------
    def page_table(self, which: str = "active") -> List[int]:
        ver = self.active if which == "active" else self.pending
        return list(ver.pages)

    def free_ids(self) -> List[int]:
        return sorted(self.alloc.free)

    def length(self) -> int:
        return self.active.length

    def cache(self, which: str = "active"):
        """(pos[L], k_rot[L][hkv][d], v[L][hkv][d]) of the version."""
        ver = self.active if which == "active" else self.pending
        return ver.concat()

    def slot_of(self, position: int, which: str = "active") -> int:
        ver = self.active if which == "active" else self.pending
        return ver.pages[position // self.P] * self.P + position % self.P


# --------------------------------------------------------------------------
# Algorithm 2: asynchronous state reconciliation with concurrent request routing
# --------------------------------------------------------------------------
class Alg2Router:
    """Which resource serves a query, and with which context, while a
    reconciliation runs (Algorithm 2, procedures Inference and Reconcile).

    The states are text.  A query carries its static state ``x_static`` (the
    prefix and chunks, j_t = len(x_static) characters), its dynamic suffix
    ``x_dyn`` (suffix and task), the sequence version k_t it was built on, and,
    for a state of the sequence produced by an eviction, ``j_eps_t``: how many
    characters of x_static are old chunks kept from before the eviction (the
    chunks past it arrived afterwards).

    Router state, in the algorithm's names: j and k (static length and version
    of the active sequence), k_ready (highest version whose cache the
    secondary resource holds in full), j_eps (cursor into the rebuilt
    sequence: its chunks past j_eps have not been bridged yet; unset until the
    first query of that sequence), x_recon (the active sequence's static state
    extended with every chunk bridged since the eviction), buffer (Delta X_eps:
    the bridged chunks the secondary has still to catch up on), the two
    resource names, is_reconciling, and x_eps (the state whose cache the
    secondary is computing).

    ``inference`` returns (case, resource, context): the case ("continue",
    "bridge", "swap", "straggler_primary", "straggler_secondary"), the
    resource that runs the model, and the text it runs on.

    Reading of the cursor: j_eps_t is a property of states of the rebuilt
    sequence, so only a query of version k + 1 sets j_eps (a query of the
    active version that happens to arrive first leaves it unset), and every
    bridged range starts at or before its end."""

    def __init__(self):
        self.j = 0
        self.k = 0
        self.k_ready = 0
        self.j_eps = None
        self.x_recon = ""
        self.buffer: List[str] = []
        self.primary, self.secondary = "R1", "R2"
        self.is_reconciling = False
        self.x_eps = None

    # ---- procedure Reconcile ---------------------------------------------------
    def reconcile_start(self, x_eps: str, k_target: int) -> None:
        """First steps: close the secondary to stragglers, empty the catch-up
        buffer, and start computing the evicted state X_eps there."""
        self.is_reconciling = True
        self.buffer = []
        self.x_eps = x_eps

    def catch_up(self) -> str:
        """One pass of the catch-up loop: take the buffered chunks (the buffer
        is emptied for the queries that keep arriving) and extend the state
        the secondary computes.  Returns the text handed to the secondary."""
        taken = "".join(self.buffer)
        self.buffer = []
        self.x_eps = self.x_eps + taken
        return taken

    def reconcile_done(self, k_target: int) -> None:
        """Last steps: drop what is left in the buffer (the swap query
        computes it) and authorise the swap."""
        self.buffer = []
        self.k_ready = k_target

    # ---- procedure Inference ---------------------------------------------------
    def inference(self, x_static: str, x_dyn: str, k_t: int, j_eps_t=None):
        j_t = len(x_static)
        if k_t == self.k:
            # case 1: the active sequence continues
            if j_t > self.j:
                self.x_recon = x_static
                self.j = j_t
            return "continue", self.primary, x_static + x_dyn
        if k_t == self.k + 1:
            # case 2: a state of the sequence the secondary is rebuilding
            if self.j_eps is None:
                self.j_eps = j_eps_t
            if k_t > self.k_ready:
                # not rebuilt yet: serve it on the primary, on the active
                # sequence extended with the chunks that are new since the cursor
                if self.j_eps is None or not 0 <= self.j_eps <= j_t:
                    raise ValueError("bridged range must run forward from the eviction cursor")
                delta = x_static[self.j_eps:j_t]
                self.x_recon = self.x_recon + delta
                self.buffer.append(delta)
                self.j_eps = j_t
                return "bridge", self.primary, self.x_recon + x_dyn
            # k_t == k_ready: the secondary holds the rebuilt cache -> swap
            self.primary, self.secondary = self.secondary, self.primary
            self.is_reconciling = False
            self.x_recon = x_static
            self.j, self.k, self.j_eps = j_t, k_t, None
            return "swap", self.primary, x_static + x_dyn
        if k_t < self.k:
            # case 3: a straggler built on an older version
            if self.is_reconciling:
                # the secondary is being rebuilt: stitch the query onto x_recon
                return "straggler_primary", self.primary, self.x_recon + x_dyn
            return "straggler_secondary", self.secondary, x_static + x_dyn
        raise ValueError("query version is ahead of the sequence being rebuilt")
