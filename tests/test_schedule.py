"""Schedule of the fused foreground launch (csr_foreground_schedule), on the CPU.

For every block shape the pieces must cover each unit's key tiles [0, K(u))
exactly once -- K(u) from the causal rule, key range [0, L + last token of the
pair).  A unit run as one piece is written directly; of a cut unit, every
piece but its last writes its own partial slot and the last merges them (or,
when several last pieces run at the same time, all write slots and each
merges a share of the rows).  Every CTA's load must be the optimum ceil(W / P)
tiles (within 1 % for the least-advanced-first steps), the merge waits must
not be able to deadlock (checked by running the schedule as the kernel would:
a CTA takes its pieces in order and a merging piece finishes only once the
others have raised their flags), and the keys in use at any time must stay
within the schedule's window."""
import pytest

C1 = dict(hq=8, hkv=2, d=64, P=16)
C2 = dict(hq=64, hkv=4, d=128, P=64)


def _cfg(libcsr, shape, chunk=0, max_new=8192, flags=0):
    return libcsr.make_config(shape["hq"], shape["hkv"], shape["d"], shape["P"], 1e6, max_new, 4096,
                              1 << 20, flags=libcsr.FLAG_PLAN_ONLY | flags, fg_chunk_tiles=chunk)


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


def _check(pieces, n_slots, K, grid):
    """Coverage, slot bookkeeping and per-CTA order; returns each CTA's load."""
    cover = {u: [] for u in K}
    per_cta = {}
    for cta, order, u, j0, j1, slot, merges, group, member in pieces:
        assert 0 <= cta < grid and 0 <= j0 < j1 <= K[u]
        cover[u].append((j0, j1, slot, merges, group, member))
        per_cta.setdefault(cta, []).append((order, j1 - j0))
    written = []
    for u, segs in cover.items():
        segs.sort()
        assert segs and segs[0][0] == 0 and segs[-1][1] == K[u], (u, segs)
        for a, b in zip(segs, segs[1:]):
            assert a[1] == b[0], (u, segs)       # contiguous, no overlap
        if len(segs) == 1:
            assert segs[0][2:] == (-1, 0, 0, 0)   # a whole unit is written directly
            continue
        last = [s for s in segs if s[3] > 0]
        rest = sorted(s[2] for s in segs if s[3] == 0)
        g = last[0][4]
        assert all(s[4] == g for s in last) and len(last) == g >= 1, (u, segs)
        assert sorted(s[5] for s in last) == list(range(g))
        if g == 1:
            # the last piece merges every other piece's slot into its own rows
            assert last[0][3] == len(segs) - 1
            assert rest == list(range(last[0][2], last[0][2] + len(segs) - 1)), (u, segs)
            written += rest
        else:
            # every piece writes a slot; the group's are the last g of the unit's
            assert all(s[3] == len(segs) for s in last) and len(segs) > 3
            s0 = rest[0] if rest else min(s[2] for s in last)
            assert rest == list(range(s0, s0 + len(segs) - g))
            assert all(s[2] == s0 + len(segs) - g + s[5] for s in last), (u, segs)
            written += rest + [s[2] for s in last]
    assert sorted(written) == list(range(n_slots))
    for cta, items in per_cta.items():
        assert sorted(o for o, _ in items) == list(range(len(items)))
    return {cta: sum(w for _, w in items) for cta, items in per_cta.items()}


def _run(pieces):
    """Execute the schedule as the kernel does; True if every piece finishes.
    A piece raises its flag when its attention is done (after any waits of
    earlier pieces on its CTA); a piece of a last group then waits for the
    flags of every other piece of its unit before its CTA moves on."""
    seq = {}
    for p in pieces:
        seq.setdefault(p[0], []).append(p)
    for v in seq.values():
        v.sort(key=lambda p: p[1])
    of_unit = {}
    for p in pieces:
        of_unit.setdefault(p[2], set()).add(p)
    flagged, pos = set(), {c: 0 for c in seq}
    progress = True
    while progress:
        progress = False
        for c, v in seq.items():
            while pos[c] < len(v):
                p = v[pos[c]]
                if p not in flagged:
                    flagged.add(p)
                    progress = True
                if p[6] > 0 and not (of_unit[p[2]] - {p}) <= flagged:
                    break                             # the merging piece waits
                pos[c] += 1
                progress = True
    return all(pos[c] == len(v) for c, v in seq.items())


CASES = [
    (C2, 122_880, 768, 152),      # the 120K step: 192 units on 152 CTAs
    (C2, 131_072, 16, 152),       # 4 units on 152 CTAs: every unit cut into segments
    (C2, 131_072, 64, 152),
    (C2, 131_072, 256, 152),
    (C2, 131_072, 512, 152),
    (C2, 131_072, 1024, 152),
    (C2, 16_384, 4096, 152),
    (C2, 6_144, 192, 152),        # the 8K step
    (C1, 1_024, 32, 152),         # tiny shape: fewer tiles than CTAs
    (C1, 0, 256, 152),
    (C2, 122_880, 768, 37),
    (C2, 122_880, 96, 7),
    (C2, 1_000, 300, 19),
    (C2, 122_880, 768, 1),
]


@pytest.mark.parametrize("shape,L,n,grid", CASES)
def test_pieces_cover_balance_and_finish(libcsr, shape, L, n, grid):
    cfg = _cfg(libcsr, shape)
    pieces, n_slots = libcsr.foreground_schedule(cfg, L, n, grid)
    K = _unit_tiles(shape, L, n)
    load = _check(pieces, n_slots, K, grid)
    W = sum(K.values())
    opt = max(-(-W // grid), 1)
    assert max(load.values()) <= opt             # the idle-interval construction: the optimum
    assert _run(pieces)
    local, n_local = libcsr.foreground_schedule(_cfg(libcsr, shape, flags=libcsr.FLAG_SCHEDULE_LOCAL), L, n, grid)
    load_l = _check(local, n_local, K, grid)
    # least-advanced-first steps only where they stay within 1 % of the optimum
    assert max(load_l.values()) <= opt * 1.01
    assert _run(local)


def _times(pieces):
    """Start time of every piece: CTAs run back to back from time 0."""
    seq = {}
    for p in pieces:
        seq.setdefault(p[0], []).append(p)
    out = []
    for v in seq.values():
        t = 0
        for p in sorted(v, key=lambda p: p[1]):
            out.append((t, p))
            t += p[4] - p[3]
    return out


def _spread(pieces):
    """Largest spread of the key positions the CTAs read at one time, over
    every tile-time (CTAs run back to back from time 0, one tile per
    tile-time), per kv head (units u with the same u % 4)."""
    events = []
    for t, p in _times(pieces):
        events.append((t, t + p[4] - p[3], p[2] % 4, p[3]))
    horizon = max(e[1] for e in events)
    worst = 0
    for t in range(0, horizon, 7):
        pos = {}
        for a, b, h, j0 in events:
            if a <= t < b:
                pos.setdefault(h, []).append(j0 + t - a)
        worst = max([worst] + [max(v) - min(v) for v in pos.values()])
    return worst


def test_step_120k_cuts_and_locality(libcsr):
    """The 120K step: 192 units of 960-966 tiles on 152 CTAs.  The default
    idle-interval schedule cuts at most P - 1 = 151 units (partials of 256
    rows of 512 + 4 bytes, written once and read once: under 15 % of the
    278.4 MB the step must move), runs at most three pieces per CTA and keeps
    the keys read at any time within one idle period (T - K, ~253 tiles, 16 MB
    of each head's cache).  With CSR_FLAG_SCHEDULE_LOCAL the least-advanced-
    first steps of 128 tiles keep them within about one step (8 MB per head)
    for at most twice the cuts, the load within 1 % of the optimum."""
    pieces, n_slots = libcsr.foreground_schedule(_cfg(libcsr, C2), 122_880, 768, 152)
    assert n_slots <= 151
    assert 2 * n_slots * 256 * (128 * 4 + 4) <= 0.15 * 278.4e6
    per_cta = {}
    for p in pieces:
        per_cta[p[0]] = per_cta.get(p[0], 0) + 1
    assert max(per_cta.values()) <= 3
    K = _unit_tiles(C2, 122_880, 768)
    T = -(-sum(K.values()) // 152)
    assert _spread(pieces) <= T - min(K.values()) + 2
    local, n_local = libcsr.foreground_schedule(_cfg(libcsr, C2, flags=libcsr.FLAG_SCHEDULE_LOCAL), 122_880, 768, 152)
    assert 151 < n_local <= 2 * 151 + 8
    assert _spread(local) <= 128 + 16


def test_short_units_run_whole(libcsr):
    """With fewer units than CTAs and units no longer than the balanced load,
    nothing is cut."""
    cfg = _cfg(libcsr, C2)
    pieces, n_slots = libcsr.foreground_schedule(cfg, 0, 1024, 152)   # 256 units of <= 8 tiles
    K = _unit_tiles(C2, 0, 1024)
    _check(pieces, n_slots, K, 152)
    assert _run(pieces)


@pytest.mark.parametrize("chunk,n,L,grid", [(1, 300, 1_000, 19), (3, 77, 513, 19), (5, 1024, 8_000, 152),
                                            (2, 512, 4_000, 64)])
def test_forced_piece_length(libcsr, chunk, n, L, grid):
    """fg_chunk_tiles caps the pieces' length (grown by halves only while the
    launch would hold more than 2,304 pieces)."""
    cfg = _cfg(libcsr, C2, chunk=chunk, max_new=2048)
    pieces, n_slots = libcsr.foreground_schedule(cfg, L, n, grid)
    K = _unit_tiles(C2, L, n)
    _check(pieces, n_slots, K, grid)
    assert _run(pieces)
    longest = max(p[4] - p[3] for p in pieces)
    # a longer piece only where the cap was grown: pieces at the cap would
    # have overflowed the table, so the grown schedule is still large
    assert len(pieces) <= 2304 and (longest <= chunk or len(pieces) > 2304 // 2)


def test_concurrent_pieces_share_the_merge(libcsr):
    """n = 16 at 128K: four units of 1,025 tiles, each cut into 38 pieces that
    run at the same time on 38 CTAs; all 38 write partials and the pieces that
    end last (37 of 27 tiles; one has 26) each merge 6 or 7 of the unit's 256
    rows, so no CTA reads all 38 partials."""
    pieces, n_slots = libcsr.foreground_schedule(_cfg(libcsr, C2), 131_072, 16, 152)
    assert len(pieces) == 152 and n_slots == 152
    group = [p for p in pieces if p[6] > 0]
    assert len(group) == 4 * 37 and all(p[7] == 37 and p[6] == 38 for p in group)
    assert _run(pieces)


def test_one_cta_runs_every_unit(libcsr):
    """192 units of 960-966 tiles on one CTA: every unit whole, once."""
    pieces, n_slots = libcsr.foreground_schedule(_cfg(libcsr, C2), 122_880, 768, 1)
    assert n_slots == 0 and len(pieces) == 192
    assert sorted(p[2] for p in pieces) == list(range(192))


def test_too_many_pieces_is_refused(libcsr):
    """A prefill of 16,384 tokens is 4,096 units, more pieces than one
    launch's table holds (2,304): the call reports it (a foreground call then
    takes the three-launch path)."""
    with pytest.raises(libcsr.CsrError):
        libcsr.foreground_schedule(_cfg(libcsr, C2, max_new=16384), 0, 16384, 152)
