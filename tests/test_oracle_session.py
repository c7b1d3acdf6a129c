"""The oracle's CSR lifecycle model against the paper's invariants (no GPU).

* prefix stability (section III-A, the cached states are not altered by later
  tokens; Theorem 1): outputs of every incremental call equal the rows of a
  one-shot causal attention over the concatenated sequence;
* the dynamic suffix is transient (Eq. x_dynamic): truncation restores the
  page table, the free set and the cache exactly, and a chunk appended after
  truncation matches a run that never had the suffix;
* reconciliation (App. D, step 5: T^E = E(T_t) (+) Delta X): after the swap
  the cache equals a fresh prefill of the prefix plus the retained and the
  caught-up chunks;
* the allocator model hands out the smallest free ids, never one slot twice.
"""
import math

import numpy as np
import pytest

from paper_2605_07325_gb300 import synth

HQ, HKV, D, P, BASE = 8, 2, 64, 16, 10000.0


def _blk(seed, n, kind="normal"):
    return synth.block(seed, n, HQ, HKV, D, kind).f64()


def _session(orc, pool=256, **kw):
    return orc.OracleCSR(HQ, HKV, D, P, BASE, pool, **kw)


def _one_shot(orc, blocks):
    """Full causal recompute of the concatenated sequence from scratch."""
    q = np.concatenate([b[0] for b in blocks])
    k = np.concatenate([b[1] for b in blocks])
    v = np.concatenate([b[2] for b in blocks])
    pos = np.arange(q.shape[0])
    qr = orc.rope(q, pos, BASE)
    kr = orc.rope(k, pos, BASE)
    return orc.attention(qr, pos, kr, v, pos, 1.0 / math.sqrt(D))


def test_prefix_stability_incremental_equals_full(oracle_mod):
    orc = oracle_mod
    s = _session(orc)
    blocks = [_blk(0, 40), _blk(1, 23), _blk(2, 17), _blk(3, 5)]
    outs = [s.init_static(*blocks[0])]
    outs += [s.append_chunk(*b)[:2] for b in blocks[1:3]]
    outs.append(s.attend_suffix(*blocks[3]))
    full_o, full_lse = _one_shot(orc, blocks)
    o = np.concatenate([x[0] for x in outs])
    lse = np.concatenate([x[1] for x in outs], axis=1)
    assert np.max(np.abs(o - full_o)) < 1e-10
    assert np.max(np.abs(lse - full_lse)) < 1e-10


def test_truncate_restores_exactly(oracle_mod):
    orc = oracle_mod
    s = _session(orc)
    s.init_static(*_blk(0, 35))
    s.append_chunk(*_blk(1, 20))
    before = (s.page_table(), s.free_ids(), s.length())
    pos0, k0, v0 = s.cache()
    s.attend_suffix(*_blk(99, 30))
    assert s.length() == 85 and len(s.page_table()) == math.ceil(85 / P)
    s.truncate_suffix()
    assert (s.page_table(), s.free_ids(), s.length()) == before
    pos1, k1, v1 = s.cache()
    assert np.array_equal(pos0, pos1) and np.array_equal(k0, k1) and np.array_equal(v0, v1)


def test_append_after_truncate_matches_no_suffix(oracle_mod):
    orc = oracle_mod
    a, b = _session(orc), _session(orc)
    for s in (a, b):
        s.init_static(*_blk(0, 33))
        s.append_chunk(*_blk(1, 16))
    a.attend_suffix(*_blk(50, 21))
    a.truncate_suffix()
    oa = a.append_chunk(*_blk(2, 19))
    ob = b.append_chunk(*_blk(2, 19))
    assert np.array_equal(oa[0], ob[0]) and np.array_equal(oa[1], ob[1])
    assert a.page_table() == b.page_table() and a.free_ids() == b.free_ids()


def test_allocator_lowest_free_and_unique_slots(oracle_mod):
    orc = oracle_mod
    s = _session(orc, pool=64)
    s.init_static(*_blk(0, 20))                 # 2 pages: 0, 1
    assert s.page_table() == [0, 1]
    s.append_chunk(*_blk(1, 12))                # 32 tokens: still 2 pages
    assert s.page_table() == [0, 1]
    s.append_chunk(*_blk(2, 1))                 # 33 tokens: page 2
    assert s.page_table() == [0, 1, 2]
    s.attend_suffix(*_blk(3, 40))               # 73 tokens: pages 3, 4
    assert s.page_table() == [0, 1, 2, 3, 4]
    s.truncate_suffix()
    assert s.free_ids()[:3] == [3, 4, 5]
    slots = [s.slot_of(p) for p in range(s.length())]
    assert len(set(slots)) == len(slots)
    assert all(0 <= x < 64 * P for x in slots)


def test_pool_exhaustion_raises(oracle_mod):
    orc = oracle_mod
    s = _session(orc, pool=3)
    s.init_static(*_blk(0, 40))
    with pytest.raises(orc.OracleOutOfPages):
        s.append_chunk(*_blk(1, 16))


@pytest.mark.parametrize("prefix_len", [32, 37])
def test_reconcile_equals_fresh_prefill(oracle_mod, prefix_len):
    """App. D: the rebuilt version equals E(T_t) (+) Delta X computed fresh."""
    orc = oracle_mod
    s = _session(orc)
    pre = _blk(0, prefix_len)
    chunks = [_blk(10 + i, 16) for i in range(6)]
    s.init_static(*pre)
    for c in chunks:
        s.append_chunk(*c)
    s.evict(40)                       # oldest 3 chunks (48 >= 40 tokens)
    assert s.dropped_ids == [0, 1, 2] and s.retained_ids == [3, 4, 5]
    late = [_blk(30, 16), _blk(31, 9)]
    for c in late:                    # Delta X appended during reconciliation
        s.append_chunk(*c)
    assert s.buffer == [6, 7]
    outs = s.reconcile()
    fresh = _session(orc)
    fresh.init_static(*pre)
    expect = {}
    for cid, c in zip([3, 4, 5, 6, 7], chunks[3:] + late):
        expect[cid] = fresh.append_chunk(*c)[:2]
    p1, k1, v1 = s.cache()
    p2, k2, v2 = fresh.cache()
    assert np.array_equal(p1, p2)
    assert np.max(np.abs(k1 - k2)) == 0 and np.max(np.abs(v1 - v2)) == 0
    for cid in expect:
        assert np.max(np.abs(outs[cid][0] - expect[cid][0])) < 1e-12
    assert s.length() == prefix_len + 16 * 3 + 25
    # shared full prefix pages keep their ids; the partial prefix page is fresh
    full = prefix_len // P
    pt = s.page_table()
    assert pt[:full] == list(range(full))
    slots = [s.slot_of(p) for p in range(s.length())]
    assert len(set(slots)) == len(slots)


def test_reconcile_page_reservation_order(oracle_mod):
    """Reading R4: while reconciling, the active version's page is taken first,
    then the rebuilt version's."""
    orc = oracle_mod
    s = _session(orc, pool=64)
    s.init_static(*_blk(0, 32))                      # pages 0,1
    for i in range(4):
        s.append_chunk(*_blk(1 + i, 16))             # pages 2..5
    s.evict(32)                                      # drop chunks 0,1; retained 2,3
    assert s.page_table("pending") == [0, 1, 6, 7]
    s.append_chunk(*_blk(9, 16))                     # active gets 8, pending gets 9
    assert s.page_table() == [0, 1, 2, 3, 4, 5, 8]
    assert s.page_table("pending") == [0, 1, 6, 7, 9]
    s.reconcile()
    assert s.page_table() == [0, 1, 6, 7, 9]
    assert s.free_ids()[:5] == [2, 3, 4, 5, 8]


def test_rewind_then_append_equals_never_appended(oracle_mod):
    """Eq. first_differing_token: after invalidating the cache past a chunk
    boundary, the next chunk sees exactly the cache it would have seen."""
    orc = oracle_mod
    a, b = _session(orc), _session(orc)
    for s in (a, b):
        s.init_static(*_blk(0, 33))
        s.append_chunk(*_blk(1, 16))
    a.append_chunk(*_blk(2, 40))
    a.rewind(49)
    oa = a.append_chunk(*_blk(3, 21))
    ob = b.append_chunk(*_blk(3, 21))
    assert np.array_equal(oa[0], ob[0]) and a.page_table() == b.page_table()
    assert a.free_ids() == b.free_ids()
