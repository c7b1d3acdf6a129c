"""Host logic of libcsr on the CPU (plan-only contexts: no device memory, no
kernels): page tables, free lists and the Algorithm 1 state machine against
the oracle's independent allocator model, and every error code."""
import pytest

from oracle import oracle as orc

HQ, HKV, D, P = 8, 2, 64, 16


def _plan(libcsr, pool=64, max_seq=4096, max_new=512, **kw):
    cfg = libcsr.make_config(HQ, HKV, D, P, 1e4, max_new, pool, max_seq,
                             flags=libcsr.FLAG_PLAN_ONLY, **kw)
    return libcsr.Context(cfg)


class _Model:
    """Oracle session without attention (bookkeeping only)."""

    def __init__(self, pool, **kw):
        import numpy as np
        self.np = np
        self.o = orc.OracleCSR(HQ, HKV, D, P, 1e4, pool, **kw)
        self.o.attend = False

    def blk(self, n):
        z = self.np.zeros
        return z((n, HQ, D)), z((n, HKV, D)), z((n, HKV, D))


def _same(ctx, m, libcsr, which="active"):
    v = libcsr.VERSION_ACTIVE if which == "active" else libcsr.VERSION_PENDING
    pt, length = ctx.layout(v)
    assert pt == m.o.page_table(which)
    if which == "active":
        assert length == m.o.length()
    assert ctx.free_pages() == m.o.free_ids()


def test_layout_matches_oracle_allocator(libcsr):
    ctx, m = _plan(libcsr), _Model(64)
    for call, n in [("init", 70), ("chunk", 5), ("chunk", 27), ("suffix", 40), ("trunc", 0),
                    ("chunk", 16), ("suffix", 1), ("trunc", 0), ("chunk", 100)]:
        if call == "init":
            ctx.init_static(None, None, None, n=n)
            m.o.init_static(*m.blk(n))
        elif call == "chunk":
            ctx.append_chunk(None, None, None, n=n)
            m.o.append_chunk(*m.blk(n))
        elif call == "suffix":
            ctx.attend_suffix(None, None, None, n=n)
            m.o.attend_suffix(*m.blk(n))
        else:
            ctx.truncate_suffix()
            m.o.truncate_suffix()
        _same(ctx, m, libcsr)


@pytest.mark.parametrize("prefix", [32, 37])
@pytest.mark.parametrize("n_catchup", [0, 1])
def test_reconcile_state_machine_matches_oracle(libcsr, prefix, n_catchup):
    ctx, m = _plan(libcsr, pool=128, n_catchup=n_catchup), _Model(128, n_catchup=n_catchup)
    ctx.set_reconciler(lambda cid, n: None)
    ctx.init_static(None, None, None, n=prefix)
    m.o.init_static(*m.blk(prefix))
    for _ in range(6):
        ctx.append_chunk(None, None, None, n=20)
        m.o.append_chunk(*m.blk(20))
    ctx.evict_and_reconcile(45)
    m.o.evict(45)
    assert ctx.chunks(libcsr.VERSION_PENDING)[0] == m.o.retained_ids
    _same(ctx, m, libcsr, "pending")
    with pytest.raises(libcsr.CsrError) as e:
        ctx.evict_and_reconcile(10)
    assert e.value.status == libcsr.EBUSY
    for _ in range(2):                         # chunks arriving during the rebuild
        ctx.append_chunk(None, None, None, n=9)
        m.o.append_chunk(*m.blk(9))
        _same(ctx, m, libcsr)
        _same(ctx, m, libcsr, "pending")
    states = []
    while True:
        s = ctx.poll_swap()
        states.append(s)
        if s == libcsr.RECON_SWAPPED:
            break
        assert len(states) < 10
    m.o.reconcile()
    _same(ctx, m, libcsr)
    assert ctx.poll_swap() == libcsr.RECON_IDLE
    # n_catchup = 0 computes each arriving chunk at once, so the first poll swaps;
    # n_catchup = 1 first catches up the 2 buffered chunks, then swaps
    assert states == ([libcsr.RECON_SWAPPED] if n_catchup == 0
                      else [libcsr.RECON_RUNNING, libcsr.RECON_SWAPPED])


def test_swap_waits_for_live_suffix(libcsr):
    ctx = _plan(libcsr, pool=128)
    ctx.set_reconciler(lambda cid, n: None)
    ctx.init_static(None, None, None, n=32)
    for _ in range(4):
        ctx.append_chunk(None, None, None, n=16)
    ctx.evict_and_reconcile(16)
    ctx.attend_suffix(None, None, None, n=8)
    assert ctx.poll_swap() == libcsr.RECON_RUNNING
    ctx.truncate_suffix()
    assert ctx.poll_swap() == libcsr.RECON_SWAPPED
    assert ctx.layout()[1] == 32 + 3 * 16


def test_automatic_eviction_at_tau_mem(libcsr):
    """Algorithm 1, Increment: reaching cap_tokens starts the eviction."""
    ctx = _plan(libcsr, pool=128, cap_tokens=100, evict_tokens=40)
    m = _Model(128)
    ctx.set_reconciler(lambda cid, n: None)
    ctx.init_static(None, None, None, n=20)
    m.o.init_static(*m.blk(20))
    for i in range(3):
        ctx.append_chunk(None, None, None, n=20)
        m.o.append_chunk(*m.blk(20))
    assert ctx.poll_swap() == libcsr.RECON_IDLE     # 80 < 100 tokens
    ctx.append_chunk(None, None, None, n=20)        # 100 = tau_mem: eviction starts
    m.o.append_chunk(*m.blk(20))
    m.o.evict(40)
    _same(ctx, m, libcsr, "pending")
    ctx.wait_reconcile(5.0)
    m.o.reconcile()
    _same(ctx, m, libcsr)


def _err(libcsr, fn, code):
    with pytest.raises(libcsr.CsrError) as e:
        fn()
    assert e.value.status == code, str(e.value)


def test_error_codes_and_no_state_change(libcsr):
    ctx = _plan(libcsr, pool=8, max_seq=200, max_new=100)
    _err(libcsr, lambda: ctx.append_chunk(None, None, None, n=4), libcsr.ESTATE)
    _err(libcsr, lambda: ctx.attend_suffix(None, None, None, n=4), libcsr.ESTATE)
    _err(libcsr, lambda: ctx.init_static(None, None, None, n=0), libcsr.EINVAL)
    _err(libcsr, lambda: ctx.init_static(None, None, None, n=101), libcsr.EINVAL)
    ctx.init_static(None, None, None, n=50)
    _err(libcsr, lambda: ctx.init_static(None, None, None, n=5), libcsr.ESTATE)
    _err(libcsr, ctx.truncate_suffix, libcsr.ESTATE)
    _err(libcsr, lambda: ctx.evict_and_reconcile(10), libcsr.ESTATE)   # no reconciler
    ctx.append_chunk(None, None, None, n=60)                            # 110 tokens, 7 pages
    before = (ctx.layout(), ctx.free_pages())
    _err(libcsr, lambda: ctx.append_chunk(None, None, None, n=40), libcsr.ENOMEM)  # pool: 8 pages
    assert (ctx.layout(), ctx.free_pages()) == before
    ctx.attend_suffix(None, None, None, n=3)
    _err(libcsr, lambda: ctx.attend_suffix(None, None, None, n=3), libcsr.ESTATE)
    _err(libcsr, lambda: ctx.append_chunk(None, None, None, n=3), libcsr.ESTATE)
    ctx.set_reconciler(lambda cid, n: None)
    _err(libcsr, lambda: ctx.evict_and_reconcile(10), libcsr.ESTATE)   # suffix live
    ctx.truncate_suffix()
    _err(libcsr, lambda: ctx.evict_and_reconcile(0), libcsr.EINVAL)
    assert (ctx.layout(), ctx.free_pages()) == before
    full = _plan(libcsr, pool=10, max_seq=400, max_new=100)
    full.set_reconciler(lambda cid, n: None)
    full.init_static(None, None, None, n=16)
    for _ in range(4):
        full.append_chunk(None, None, None, n=32)      # 9 of 10 pages used
    snap = (full.layout(), full.free_pages())
    _err(libcsr, lambda: full.evict_and_reconcile(32), libcsr.ENOMEM)  # rebuild needs 6 pages
    assert (full.layout(), full.free_pages()) == snap
    assert full.poll_swap() == libcsr.RECON_IDLE
    big = _plan(libcsr, pool=64, max_seq=120, max_new=100)
    big.init_static(None, None, None, n=100)
    _err(libcsr, lambda: big.append_chunk(None, None, None, n=21), libcsr.ENOMEM)  # max_seq


@pytest.mark.parametrize("bad", [dict(head_dim=96), dict(page_size=48), dict(num_q_heads=12),
                                 dict(num_kv_heads=3), dict(max_new_tokens=0),
                                 dict(pool_pages=0), dict(pool_pages=70000),
                                 dict(cap_tokens=10, evict_tokens=0), dict(rebuild_duty=-0.5),
                                 dict(rebuild_duty=float("nan")), dict(fg_chunk_tiles=-1)])
def test_invalid_configs_rejected(libcsr, bad):
    kw = dict(num_q_heads=8, num_kv_heads=2, head_dim=64, page_size=16, rope_base=1e4,
              max_new_tokens=64, pool_pages=16, max_seq_tokens=256,
              flags=libcsr.FLAG_PLAN_ONLY)
    kw.update(bad)
    cfg = libcsr.make_config(**kw)
    with pytest.raises(libcsr.CsrError) as e:
        libcsr.Context(cfg)
    assert e.value.status == libcsr.EINVAL


def test_rewind_matches_oracle(libcsr):
    ctx, m = _plan(libcsr), _Model(64)
    ctx.init_static(None, None, None, n=40)
    m.o.init_static(*m.blk(40))
    for n in (10, 30, 7):
        ctx.append_chunk(None, None, None, n=n)
        m.o.append_chunk(*m.blk(n))
    for bad in (41, 45, 200, 39):
        _err(libcsr, lambda: ctx.rewind(bad), libcsr.EINVAL)
    ctx.rewind(80)
    m.o.rewind(80)
    _same(ctx, m, libcsr)
    ctx.rewind(40)
    m.o.rewind(40)
    _same(ctx, m, libcsr)
    assert ctx.chunks()[0] == []
    ctx.append_chunk(None, None, None, n=25)
    m.o.append_chunk(*m.blk(25))
    _same(ctx, m, libcsr)
    ctx.attend_suffix(None, None, None, n=3)
    _err(libcsr, lambda: ctx.rewind(40), libcsr.ESTATE)


def test_fused_step_layout_matches_separate_calls(libcsr):
    """csr_append_chunk_attend_suffix = csr_append_chunk + csr_attend_suffix:
    the same page tables, free lists and chunk ids, against the oracle."""
    fused, sep, m = _plan(libcsr, pool=128), _plan(libcsr, pool=128), _Model(128)
    for c in (fused, sep):
        c.init_static(None, None, None, n=37)
    m.o.init_static(*m.blk(37))
    for n_chunk, n_suffix in [(5, 40), (16, 16), (27, 1), (100, 29), (1, 63), (64, 64)]:
        _, _, cid = fused.append_chunk_attend_suffix(None, None, None, n_chunk, n=n_chunk + n_suffix)
        _, _, cid2 = sep.append_chunk(None, None, None, n=n_chunk)
        sep.attend_suffix(None, None, None, n=n_suffix)
        _, _, cid3 = m.o.append_chunk(*m.blk(n_chunk))
        m.o.attend_suffix(*m.blk(n_suffix))
        assert cid == cid2 == cid3
        _same(fused, m, libcsr)
        assert fused.layout() == sep.layout() and fused.free_pages() == sep.free_pages()
        for c in (fused, sep):
            c.truncate_suffix()
        m.o.truncate_suffix()
        _same(fused, m, libcsr)
    assert fused.chunks() == sep.chunks()


def test_fused_step_eviction_starts_at_truncate(libcsr):
    """tau_mem reached by a fused step: the eviction waits for the truncation
    (it needs no live suffix), then matches the oracle; a fused step during the
    reconciliation forks only its chunk into the rebuilt version."""
    ctx = _plan(libcsr, pool=128, cap_tokens=100, evict_tokens=40)
    m = _Model(128)
    ctx.set_reconciler(lambda cid, n: None)
    ctx.init_static(None, None, None, n=20)
    m.o.init_static(*m.blk(20))
    for i in range(4):
        ctx.append_chunk_attend_suffix(None, None, None, 20, n=33)
        m.o.append_chunk(*m.blk(20))
        m.o.attend_suffix(*m.blk(13))
        if i == 3:                                  # 100 = tau_mem, suffix still live
            assert ctx.poll_swap() == libcsr.RECON_IDLE
        ctx.truncate_suffix()
        m.o.truncate_suffix()
    m.o.evict(40)
    _same(ctx, m, libcsr, "pending")
    ctx.append_chunk_attend_suffix(None, None, None, 12, n=30)   # forked: 12 tokens
    m.o.append_chunk(*m.blk(12))
    m.o.attend_suffix(*m.blk(18))
    _same(ctx, m, libcsr, "pending")
    assert ctx.poll_swap() == libcsr.RECON_RUNNING  # swap waits for the live suffix
    ctx.truncate_suffix()
    m.o.truncate_suffix()
    assert ctx.wait_reconcile(5.0) == libcsr.RECON_SWAPPED
    m.o.reconcile()
    _same(ctx, m, libcsr)


def test_fused_step_errors(libcsr):
    ctx = _plan(libcsr, pool=64, max_new=64)
    _err(libcsr, lambda: ctx.append_chunk_attend_suffix(None, None, None, 4, n=8), libcsr.ESTATE)
    ctx.init_static(None, None, None, n=16)
    before = (ctx.layout(), ctx.free_pages())
    _err(libcsr, lambda: ctx.append_chunk_attend_suffix(None, None, None, 0, n=8), libcsr.EINVAL)
    _err(libcsr, lambda: ctx.append_chunk_attend_suffix(None, None, None, 8, n=8), libcsr.EINVAL)
    _err(libcsr, lambda: ctx.append_chunk_attend_suffix(None, None, None, 40, n=65), libcsr.EINVAL)
    assert (ctx.layout(), ctx.free_pages()) == before
    ctx.append_chunk_attend_suffix(None, None, None, 4, n=8)
    _err(libcsr, lambda: ctx.append_chunk_attend_suffix(None, None, None, 4, n=8), libcsr.ESTATE)
    _err(libcsr, lambda: ctx.append_chunk(None, None, None, n=4), libcsr.ESTATE)
    ctx.truncate_suffix()
    assert ctx.layout()[1] == 20


def test_cancel_reconcile_restores_layout(libcsr):
    """csr_cancel_reconcile: the rebuilt version's pages return to the pool and
    the active version keeps every chunk appended meanwhile (its page ids as
    reserved while the rebuild ran); a later eviction runs normally."""
    ctx = _plan(libcsr, pool=128)
    m = _Model(128)
    ctx.set_reconciler(lambda cid, n: None)
    ctx.init_static(None, None, None, n=37)
    m.o.init_static(*m.blk(37))
    for _ in range(5):
        ctx.append_chunk(None, None, None, n=21)
        m.o.append_chunk(*m.blk(21))
    ctx.evict_and_reconcile(40)
    m.o.evict(40)
    for _ in range(2):                       # forked into the rebuild, then abandoned
        ctx.append_chunk(None, None, None, n=13)
        m.o.append_chunk(*m.blk(13))
    ctx.cancel_reconcile()
    m.o.cancel()
    _same(ctx, m, libcsr)
    assert ctx.poll_swap() == libcsr.RECON_IDLE
    _err(libcsr, lambda: ctx.cancel_reconcile(), libcsr.ESTATE)
    ctx.evict_and_reconcile(40)
    m.o.evict(40)
    _same(ctx, m, libcsr, "pending")
    assert ctx.wait_reconcile(5.0) == libcsr.RECON_SWAPPED
    m.o.reconcile()
    _same(ctx, m, libcsr)
