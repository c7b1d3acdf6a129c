"""Algorithm 2 (concurrent request routing) on the CPU: the oracle's router
against a trace derived by hand from the algorithm, and the library's
csr_route / csr_get_versions (plan-only context) against the oracle router on
every (state, k_t) pair both define."""
import json
import os

import pytest

from oracle import oracle as orc

HERE = os.path.dirname(os.path.abspath(__file__))
HQ, HKV, D, P = 8, 2, 64, 16


def run_hand_trace(orc):
    """Replay the hand-derived trace on `orc.Alg2Router` (asserts on a mismatch)."""
    g = json.load(open(os.path.join(HERE, "golden", "alg2_routing.json")))
    r = orc.Alg2Router()
    for ev in g["events"]:
        if ev["op"] == "reconcile_start":
            r.reconcile_start(ev["x_eps"], ev["k_target"])
        elif ev["op"] == "catch_up":
            assert r.catch_up() == ev["expect_taken"], ev
            assert r.x_eps == ev["x_eps"], ev
        elif ev["op"] == "reconcile_done":
            r.reconcile_done(ev["k_target"])
        elif ev.get("expect_error"):
            try:
                r.inference(ev["x_static"], ev["x_dyn"], ev["k_t"], ev["j_eps_t"])
            except ValueError:
                pass
            else:
                raise AssertionError(f"query not rejected: {ev}")
        else:
            got = r.inference(ev["x_static"], ev["x_dyn"], ev["k_t"], ev["j_eps_t"])
            assert list(got) == ev["expect"], ev
            assert (r.k, r.k_ready) == (ev["k"], ev["k_ready"]), ev
            assert (r.j, r.j_eps) == (ev["j"], ev["j_eps"]), ev
            assert r.x_recon == ev["x_recon"], ev
            assert list(r.buffer) == ev["buffer"], ev
            assert r.is_reconciling == ev["is_reconciling"], ev


def test_oracle_router_matches_hand_trace():
    run_hand_trace(orc)


def _plan(libcsr, n_catchup):
    cfg = libcsr.make_config(HQ, HKV, D, P, 1e4, 512, 128, 4096, n_catchup=n_catchup,
                             flags=libcsr.FLAG_PLAN_ONLY)
    ctx = libcsr.Context(cfg)
    ctx.set_reconciler(lambda cid, n: None)
    ctx.init_static(None, None, None, n=32)
    for _ in range(4):
        ctx.append_chunk(None, None, None, n=16)
    return ctx


def test_library_routes_hand_trace(libcsr):
    """N_catchup = 1: the rebuild counts as ready once at most one chunk is
    buffered (a plan-only context has no device work to wait for)."""
    ctx = _plan(libcsr, n_catchup=1)
    assert ctx.versions() == (0, 0)
    assert ctx.route(0) == libcsr.ROUTE_CONTINUE
    with pytest.raises(libcsr.CsrError):            # no version 1 before an eviction
        ctx.route(1)
    ctx.evict_and_reconcile(16)
    for _ in range(2):                               # two chunks bridged: |buffer| > N_catchup
        ctx.append_chunk(None, None, None, n=16)
    assert ctx.route(1) == libcsr.ROUTE_BRIDGE       # catch-up handed to R_2, not ready
    assert ctx.versions() == (0, 0)
    assert ctx.route(0) == libcsr.ROUTE_CONTINUE     # a query on the old sequence
    ctx.attend_suffix(None, None, None, n=8)
    assert ctx.route(1) == libcsr.ROUTE_BRIDGE       # ready, but the swap waits for the suffix
    assert ctx.versions() == (0, 1)
    ctx.truncate_suffix()
    assert ctx.route(1) == libcsr.ROUTE_SWAPPED      # k_t = k_ready: resource swap
    assert ctx.versions() == (1, 1)
    assert ctx.route(0) == libcsr.ROUTE_STRAGGLER
    assert ctx.route(1) == libcsr.ROUTE_CONTINUE
    assert ctx.poll_swap() == libcsr.RECON_IDLE


_CASE = {"continue": "ROUTE_CONTINUE", "bridge": "ROUTE_BRIDGE", "swap": "ROUTE_SWAPPED",
         "straggler_primary": "ROUTE_STRAGGLER", "straggler_secondary": "ROUTE_STRAGGLER"}


@pytest.mark.parametrize("after_swap", [False, True])
@pytest.mark.parametrize("state", ["idle", "rebuilding", "ready"])
@pytest.mark.parametrize("dk", [-1, 0, 1])
def test_library_routes_match_oracle_router(libcsr, after_swap, state, dk):
    ctx = _plan(libcsr, n_catchup=1)
    r = orc.Alg2Router()
    k = 0
    if after_swap:                                   # bring both to version 1
        ctx.evict_and_reconcile(16)
        assert ctx.wait_reconcile(5.0) == libcsr.RECON_SWAPPED
        r.reconcile_start("ab", 1), r.reconcile_done(1), r.inference("abc", "?", 1, 2)
        k = 1
    if state != "idle":
        ctx.evict_and_reconcile(16)
        r.reconcile_start("ab", k + 1)
        if state == "rebuilding":
            for _ in range(2):
                ctx.append_chunk(None, None, None, n=16)
        else:
            r.reconcile_done(k + 1)
    k_t = k + dk
    if k_t < 0:
        pytest.skip("no version below 0")
    if dk == 1 and state == "idle":
        # the paper's client only sends k + 1 once Reconcile has started; the
        # library rejects a version it is not building
        with pytest.raises(libcsr.CsrError):
            ctx.route(k_t)
        return
    case, _, _ = r.inference("abcd", "?", k_t, 2 if k_t > k else None)
    assert ctx.route(k_t) == getattr(libcsr, _CASE[case])


def test_router_invariants_on_random_sessions():
    """Properties that hold for any interleaving the clients can produce
    (Algorithm 2): the bridged context is always the active sequence's static
    state followed by every chunk bridged since the eviction, in order; the
    secondary's state plus the buffered chunks is the rebuilt sequence up to
    the cursor; and the swap query's static state starts with what the
    secondary computed (only the remainder is computed at the swap)."""
    import random
    rng = random.Random(7)
    import itertools
    letters = (chr(0x4E00 + i) for i in itertools.count())   # a distinct character per chunk
    for trial in range(200):
        r = orc.Alg2Router()
        active = "ab" + "".join(next(letters) for _ in range(4))   # the active static state
        r.inference(active, "?", 0)
        k = 0
        rebuilt = None            # the static state of version k + 1, once evicted
        old = None                # old chunks kept by the eviction
        bridged = ""
        done = False              # Reconcile has authorised the swap
        for step in range(30):
            a = rng.random()
            if rebuilt is None and a < 0.2:
                keep = rng.randrange(2, len(active))
                old = active[:2] + active[keep:]
                rebuilt, bridged, done = old, "", False
                r.reconcile_start(old, k + 1)
            elif rebuilt is not None and a < 0.5:
                rebuilt += "".join(next(letters) for _ in range(rng.randrange(0, 3)))
                case, res, ctx = r.inference(rebuilt, "?", k + 1, len(old))
                if case == "bridge":
                    bridged = rebuilt[len(old):]
                    assert ctx == active + bridged + "?"
                    assert r.x_recon == active + bridged
                    assert not done and r.x_eps + "".join(r.buffer) == rebuilt[:r.j_eps]
                else:
                    assert done and case == "swap" and rebuilt.startswith(r.x_eps)
                    active, rebuilt, k = rebuilt, None, k + 1
            elif rebuilt is not None and not done and a < 0.6:
                r.catch_up()
                assert r.x_eps + "".join(r.buffer) == (rebuilt[:r.j_eps] if r.j_eps else old)
            elif rebuilt is not None and not done and a < 0.7:
                r.reconcile_done(k + 1)
                done = True
            elif rebuilt is None and a < 0.8:
                active += next(letters)
                assert r.inference(active, "?", k)[0] == "continue"
            elif k > 0:
                case, res, ctx = r.inference("stale", "?", k - 1)
                if r.is_reconciling:
                    assert (case, res, ctx) == ("straggler_primary", r.primary, r.x_recon + "?")
                else:
                    assert (case, res, ctx) == ("straggler_secondary", r.secondary, "stale?")
