"""Schedule of the fused foreground launch (csr_foreground_schedule), on the CPU.

For every block shape the pieces must cover each unit's key tiles [0, K(u))
exactly once -- K(u) from the causal rule, key range [0, L + last token of the
pair) -- with at most one piece per unit and CTA level, whole units written
directly and split units given distinct partial slots; the work per CTA must
be balanced, and only units left over after the full rounds may be split."""
import itertools
import math

import pytest

C1 = dict(hq=8, hkv=2, d=64, P=16)
C2 = dict(hq=64, hkv=4, d=128, P=64)


def _cfg(libcsr, shape, chunk=0, max_new=8192):
    return libcsr.make_config(shape["hq"], shape["hkv"], shape["d"], shape["P"], 1e6, max_new, 4096,
                              1 << 20, flags=libcsr.FLAG_PLAN_ONLY, fg_chunk_tiles=chunk)


def _unit_tiles(shape, L, n):
    G = shape["hq"] // shape["hkv"]
    T = 128 // G
    n_tiles = -(-n * G // 128)
    pairs = -(-n_tiles // 2)
    K = {}
    for u in range(pairs * shape["hkv"]):
        pair = u // shape["hkv"]
        last = min((2 * pair + 2) * T, n)          # tokens of the pair's second tile, clamped
        K[u] = -(-(L + last) // 128)
    return K


def _check(pieces, slots, K, grid):
    cover = {u: [] for u in K}
    per_cta = {}
    used_slots = set()
    for cta, order, u, j0, j1, slot in pieces:
        assert 0 <= cta < grid and 0 <= j0 < j1 <= K[u]
        cover[u].append((j0, j1, slot))
        per_cta.setdefault(cta, []).append((order, j1 - j0))
        if slot >= 0:
            assert slot not in used_slots
            used_slots.add(slot)
    for u, segs in cover.items():
        segs.sort()
        assert segs[0][0] == 0 and segs[-1][1] == K[u], (u, segs)
        for a, b in zip(segs, segs[1:]):
            assert a[1] == b[0], (u, segs)       # contiguous, no overlap
        if len(segs) == 1:
            assert segs[0][2] == -1               # a whole unit is written directly
        else:
            assert all(s >= 0 for _, _, s in segs)
    assert len(used_slots) == slots or (slots > 0 and len(used_slots) <= slots)
    for cta, items in per_cta.items():
        assert sorted(o for o, _ in items) == list(range(len(items)))
    return {cta: sum(w for _, w in items) for cta, items in per_cta.items()}


CASES = [
    (C2, 122_880, 768, 152),      # the 120K fused step: 192 units on 152 CTAs
    (C2, 131_072, 16, 152),       # 4 units: every one split 38 ways
    (C2, 131_072, 64, 152),
    (C2, 131_072, 256, 152),
    (C2, 131_072, 1024, 152),
    (C2, 16_384, 4096, 152),
    (C2, 0, 4096, 152),           # a prefill: unit lengths from 1 to 32 tiles
    (C2, 6_144, 192, 152),        # the 8K step
    (C1, 1_024, 32, 152),         # tiny shape: fewer tiles than CTAs
    (C1, 0, 256, 152),
    (C2, 122_880, 768, 7),
    (C2, 122_880, 768, 1),
]


@pytest.mark.parametrize("shape,L,n,grid", CASES)
def test_pieces_cover_every_key_tile_once(libcsr, shape, L, n, grid):
    cfg = _cfg(libcsr, shape)
    pieces, slots = libcsr.foreground_schedule(cfg, L, n, grid)
    K = _unit_tiles(shape, L, n)
    load = _check(pieces, slots, K, grid)
    used = len(load)
    total = sum(K.values())
    ideal = total / min(grid, total)
    # a CTA's load: at most the ideal plus one piece's worth of rounding per tail level
    longest = max(K.values())
    assert max(load.values()) <= max(ideal * 1.06 + 6 * 2, longest), (max(load.values()), ideal)
    assert used <= grid


def test_only_leftover_units_split(libcsr):
    """The 120K step: 152 units run whole in the first round; only the 40
    left over are cut, so the partials are far fewer than a split of every
    unit would write."""
    pieces, slots = libcsr.foreground_schedule(_cfg(libcsr, C2), 122_880, 768, 152)
    whole = [p for p in pieces if p[5] == -1]
    split_units = {p[2] for p in pieces if p[5] >= 0}
    assert len(whole) == 152 and len(split_units) == 40
    assert slots == sum(1 for p in pieces if p[5] >= 0) <= 6 * 152
    # pieces of one tail level cover the same key section of different units
    by_cta = {}
    for p in pieces:
        by_cta.setdefault(p[0], []).append(p)
    first_tail = [sorted(v, key=lambda x: x[1])[1] for v in by_cta.values() if len(v) > 1]
    sections = {p[3] for p in first_tail}
    assert len(sections) <= 8


@pytest.mark.parametrize("chunk,n,L", [(1, 300, 1_000), (3, 77, 513), (5, 1024, 8_000)])
def test_forced_chunks_round_robin(libcsr, chunk, n, L):
    cfg = _cfg(libcsr, C2, chunk=chunk, max_new=2048)
    pieces, slots = libcsr.foreground_schedule(cfg, L, n, 19)
    K = _unit_tiles(C2, L, n)
    _check(pieces, slots, K, 19)
    # every piece is at most `chunk` tiles long unless the partial buffer forced longer ones
    longest = max(j1 - j0 for _, _, _, j0, j1, _ in pieces)
    assert longest >= min(chunk, max(K.values()))
