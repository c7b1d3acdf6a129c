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
            r.reconcile_start(ev["k_target"])
        elif ev["op"] == "reconcile_done":
            r.reconcile_done(ev["k_target"])
        else:
            got = r.inference(ev["j_t"], ev["k_t"], ev["j_eps_t"])
            assert list(got) == ev["expect"], ev
            assert (r.k, r.k_ready) == (ev["k"], ev["k_ready"]), ev
            assert (r.j, r.j_eps) == (ev["j"], ev["j_eps"]), ev
            assert [list(x) for x in r.buffer] == ev["buffer"], ev


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
        r.reconcile_start(1), r.reconcile_done(1), r.inference(50, 1, 50)
        k = 1
    if state != "idle":
        ctx.evict_and_reconcile(16)
        r.reconcile_start(k + 1)
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
    case, _ = r.inference(100, k_t, 100)
    assert ctx.route(k_t) == getattr(libcsr, _CASE[case])
