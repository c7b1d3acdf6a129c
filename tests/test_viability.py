"""App. D viability check (csr_check_viability) on plan-only contexts (no GPU).

The expected times are built from their definitions, not from the library's
closed forms: the warm-up and reconciliation costs as explicit sums over the
query positions of the causal prefill (Eq. TTFT_derivation_2 with i* =
|X_pre| + 1 for the warm-up, Eq. recon_time for the extension), and N_buffer
by counting, token by token, the pages both versions would take."""
import math

import pytest

HQ, HKV, D, P = 8, 2, 64, 16


def _plan(libcsr, pool, max_seq=1 << 20, prefix=40, chunks=(32, 32, 48, 32, 32)):
    cfg = libcsr.make_config(HQ, HKV, D, P, 1e4, 512, pool, max_seq, flags=libcsr.FLAG_PLAN_ONLY)
    ctx = libcsr.Context(cfg)
    ctx.set_reconciler(lambda cid, n: None)
    ctx.init_static(None, None, None, n=prefix)
    for n in chunks:
        ctx.append_chunk(None, None, None, n=n)
    return ctx


def _brute_n_buffer(free, active, rebuilt, max_seq):
    pages = lambda L: -(-L // P)  # noqa: E731
    x = 0
    while active + x + 1 <= max_seq and \
            (pages(active + x + 1) - pages(active)) + (pages(rebuilt + x + 1) - pages(rebuilt)) <= free:
        x += 1
    return x


@pytest.mark.parametrize("evict", [1, 32, 64, 70])
def test_viability_terms_from_definitions(libcsr, evict):
    prefix, chunks = 40, (32, 32, 48, 32, 32)
    ctx = _plan(libcsr, pool=64, prefix=prefix, chunks=chunks)
    # the chunks an eviction of `evict` tokens drops: oldest whole chunks
    dropped, k = 0, 0
    while dropped < evict:
        dropped += chunks[k]
        k += 1
    rebuilt = prefix + sum(chunks[k:])
    active = prefix + sum(chunks)
    c = 2.5e-9
    warm_pairs = sum(i for i in range(prefix + 1, rebuilt + 1))
    t_warm = c * warm_pairs
    dn = 7                                   # choose the rate so that Delta N is a whole number
    rate = dn / t_warm
    recon_pairs = sum(i for i in range(rebuilt + 1, rebuilt + dn + 1))
    got = ctx.check_viability(evict, rate, c)
    assert got["rebuilt_tokens"] == rebuilt
    assert math.isclose(got["t_warm_s"], t_warm, rel_tol=1e-12)
    assert math.isclose(got["delta_n_tokens"], dn, rel_tol=1e-12)
    assert math.isclose(got["t_recon_s"], c * recon_pairs, rel_tol=1e-12)
    full_prefix_pages = prefix // P
    fresh = -(-rebuilt // P) - full_prefix_pages
    spare = len(ctx.free_pages()) - fresh
    n_buf = _brute_n_buffer(spare, active, rebuilt, 1 << 20)
    assert got["n_buffer_tokens"] == n_buf
    assert math.isclose(got["t_mem_s"], n_buf / rate, rel_tol=1e-12)
    assert got["viable"] == int(got["t_warm_s"] + got["t_recon_s"] <= got["t_mem_s"])
    assert got["measured"] == 0 and got["pair_seconds"] == c
    # the prediction names the same retained chunks the eviction keeps
    ctx.evict_and_reconcile(evict)
    _, pending_len = ctx.layout(libcsr.VERSION_PENDING)
    assert pending_len == rebuilt


def test_viability_flips_with_pool_headroom(libcsr):
    """The same context and append rate are viable with a roomy pool and not
    with one page of headroom once the rebuilt version is reserved; a pool
    that cannot hold the rebuilt version at all has no buffer."""
    # active: 40 + 176 = 216 tokens (14 pages); evicting 64 keeps 152 tokens
    # (10 pages, 2 of them the shared prefix): 8 fresh pages
    args = (64, 1e6, 1e-9)                  # Delta t_warm = 1e-9 * (41 + ... + 152) = 10.8 us
    roomy = _plan(libcsr, pool=4096).check_viability(*args)
    one_page = _plan(libcsr, pool=23).check_viability(*args)
    no_room = _plan(libcsr, pool=18).check_viability(*args)
    assert roomy["viable"] == 1
    # one spare page: both versions fill their last pages (8 slots each), the
    # ninth token needs a page in each
    assert one_page["n_buffer_tokens"] == 8 and one_page["viable"] == 0
    assert no_room["n_buffer_tokens"] == 0 and no_room["viable"] == 0


def test_viability_caps_at_max_seq_tokens(libcsr):
    active = 40 + 176
    ctx = _plan(libcsr, pool=4096, max_seq=active + 5)
    got = ctx.check_viability(32, 100.0, 1e-9)
    assert got["n_buffer_tokens"] == 5


def test_viability_errors(libcsr):
    ctx = _plan(libcsr, pool=64)
    with pytest.raises(libcsr.CsrError):
        ctx.check_viability(0, 100.0, 1e-9)          # evict_tokens < 1
    with pytest.raises(libcsr.CsrError):
        ctx.check_viability(32, 0.0, 1e-9)           # no append rate
    with pytest.raises(libcsr.CsrError):
        ctx.check_viability(32, 100.0, 0.0)          # nothing observed on a plan-only context
    ctx.attend_suffix(None, None, None, n=8)
    with pytest.raises(libcsr.CsrError):
        ctx.check_viability(32, 100.0, 1e-9)         # live suffix
    ctx.truncate_suffix()
    ctx.evict_and_reconcile(32)
    with pytest.raises(libcsr.CsrError):
        ctx.check_viability(32, 100.0, 1e-9)         # reconciliation running
    empty = libcsr.Context(libcsr.make_config(HQ, HKV, D, P, 1e4, 512, 64, 4096,
                                              flags=libcsr.FLAG_PLAN_ONLY))
    empty.init_static(None, None, None, n=40)
    with pytest.raises(libcsr.CsrError):
        empty.check_viability(32, 100.0, 1e-9)       # no chunk to evict
