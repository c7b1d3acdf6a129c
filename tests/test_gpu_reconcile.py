"""Eviction + asynchronous state reconciliation on the GPU (Algorithm 1, App. D).

After the swap the active cache must equal a fresh prefill of the prefix plus
the retained and caught-up chunks (App. D step 5): page table, free list and
slot mapping bit-exact against the oracle allocator, cached values bit-exact,
rotated keys within tolerance of the oracle and bit-exact against a second GPU
context built fresh from the same chunks; the rebuilt attention outputs and
every later output within tolerance of the oracle.
"""
import numpy as np
import pytest
import torch

from gpu_util import C1, C2, Pair, assert_close, bits_of, csr_mod, to_dev, to_f64

pytestmark = pytest.mark.gpu


def _provider(p: Pair, outs: dict):
    def prov(cid, n):
        b = p.blocks[cid]
        out = torch.empty((n, p.hq, p.d), dtype=torch.bfloat16, device="cuda")
        outs[cid] = out
        return to_dev(b.q), to_dev(b.k), to_dev(b.v), out
    return prov


def _fresh_copy(p: Pair, prefix_block, chunk_ids):
    q = Pair(p.shape, pool_pages=p.cfg.pool_pages, max_seq=p.cfg.max_seq_tokens,
             max_new=p.cfg.max_new_tokens)
    q.init_static(prefix_block, compare=False)
    for cid in chunk_ids:
        q.append(p.blocks[cid], compare=False)
    return q


@pytest.mark.parametrize("shape,prefix,chunk,evict,n_catchup", [
    (C1, 64, 40, 100, 0),    # aligned prefix, unaligned chunks
    (C1, 70, 48, 100, 0),    # partly filled prefix page: copied by the compaction kernel
    (C1, 70, 48, 100, 2),    # both buffered chunks left for the swap (foreground)
    (C2, 192, 96, 200, 0),   # 64/4/128 head shape, page 64
])
def test_evict_reconcile_swap(libcsr, shape, prefix, chunk, evict, n_catchup):
    csr = csr_mod()
    p = Pair(shape, pool_pages=256, max_seq=8192, max_new=512, n_catchup=n_catchup,
             rebuild_tiles_per_cta=2)   # short rebuild items: exercises the split merge
    lo = torch.cuda.Stream(priority=0)
    outs = {}
    p.ctx.set_reconciler(_provider(p, outs), lo)
    pre = p.blk(500, prefix)
    p.init_static(pre)
    for i in range(8):
        p.append(p.blk(501 + i, chunk))
    p.ctx.evict_and_reconcile(evict)
    p.orc.evict(evict)
    pt_pend, len_pend = p.ctx.layout(csr.VERSION_PENDING)
    assert pt_pend == p.orc.page_table("pending")
    assert p.ctx.chunks(csr.VERSION_PENDING)[0] == p.orc.retained_ids
    # the foreground keeps serving the old version while the rebuild runs
    for i in range(2):
        p.append(p.blk(600 + i, chunk // 2 + 3))
        p.suffix(p.blk(700 + i, 19))
        p.truncate()
    state = p.ctx.wait_reconcile(60.0)
    assert state == csr.RECON_SWAPPED
    expect = p.orc.reconcile()
    torch.cuda.synchronize()
    for cid, (eo, _) in expect.items():
        assert_close(to_f64(outs[cid]), eo, f"rebuilt chunk {cid}")
    p.check_layout()
    p.check_cache()
    # bit-exact against a context built from scratch on the same chunks
    ids, lens, pre_len = p.ctx.chunks(csr.VERSION_ACTIVE)
    fresh = _fresh_copy(p, pre, ids)
    L = p.orc.length()
    k1, v1 = p.ctx.gather_kv(csr.VERSION_ACTIVE, 0, L)
    k2, v2 = fresh.ctx.gather_kv(csr.VERSION_ACTIVE, 0, L)
    torch.cuda.synchronize()
    assert np.array_equal(bits_of(k1), bits_of(k2)) and np.array_equal(bits_of(v1), bits_of(v2))
    # and later calls on the swapped version match the oracle
    p.append(p.blk(800, chunk))
    p.suffix(p.blk(801, 33))
    p.check_layout()
    p.truncate()
    p.device_clean()


def test_automatic_eviction_and_repeated_cycles(libcsr):
    """cap_tokens = tau_mem triggers the eviction from csr_append_chunk; three
    eviction cycles in a row keep matching the oracle."""
    csr = csr_mod()
    p = Pair(C1, pool_pages=256, max_seq=4096, max_new=256, cap_tokens=400, evict_tokens=128)
    lo = torch.cuda.Stream(priority=0)
    outs = {}
    p.ctx.set_reconciler(_provider(p, outs), lo)
    p.init_static(p.blk(900, 64))
    seed, cycles = 901, 0
    while cycles < 3:
        p.append(p.blk(seed, 32))
        seed += 1
        if p.orc.length() >= 400 and not p.orc.is_reconciling:
            p.orc.evict(128)            # the library started it inside append_chunk
            assert p.ctx.layout(csr.VERSION_PENDING)[0] == p.orc.page_table("pending")
            assert p.ctx.wait_reconcile(60.0) == csr.RECON_SWAPPED
            expect = p.orc.reconcile()
            torch.cuda.synchronize()
            for cid, (eo, _) in expect.items():
                assert_close(to_f64(outs[cid]), eo, f"cycle {cycles} chunk {cid}")
            p.check_layout()
            cycles += 1
    p.check_cache()
    p.device_clean()


@pytest.mark.parametrize("pacing", ["paced", "unpaced", "duty"])
def test_fused_steps_through_eviction_cycles(libcsr, pacing):
    """Fused chunk + suffix steps: tau_mem reached by a fused step starts the
    eviction at its truncation; fused steps during the reconciliation fork
    only their chunk; two cycles against the oracle -- with the rebuild paced
    (one task in flight after the foreground work, the default), unpaced
    (CSR_FLAG_UNPACED_REBUILD) and held to half of the wall time."""
    csr = csr_mod()
    kw = {"paced": {}, "unpaced": {"flags": csr.FLAG_UNPACED_REBUILD},
          "duty": {"rebuild_duty": 0.5}}[pacing]
    p = Pair(C1, pool_pages=256, max_seq=4096, max_new=256, cap_tokens=400, evict_tokens=128, **kw)
    lo = torch.cuda.Stream(priority=0)
    outs = {}
    p.ctx.set_reconciler(_provider(p, outs), lo)
    p.init_static(p.blk(950, 70))
    seed, cycles, steps = 951, 0, 0
    while cycles < 2:
        assert steps < 100
        if p.orc.is_reconciling and p.ctx.poll_swap() == csr.RECON_SWAPPED:
            expect = p.orc.reconcile()
            torch.cuda.synchronize()
            for cid, (eo, _) in expect.items():
                assert_close(to_f64(outs[cid]), eo, f"cycle {cycles} chunk {cid}")
            p.check_layout()
            p.check_cache()
            cycles += 1
        p.fused(p.blk(seed, 45), 30)
        trigger = not p.orc.is_reconciling and p.orc.length() - 15 >= 400
        p.truncate()
        if trigger:
            p.orc.evict(128)            # the library started it at the truncation
            assert p.ctx.layout(csr.VERSION_PENDING)[0] == p.orc.page_table("pending")
        seed += 1
        steps += 1
    p.device_clean()


def test_routing_swaps_on_first_query_of_rebuilt_version(libcsr):
    """Algorithm 2 on the GPU: queries of the evicted sequence (k_t = k + 1)
    are bridged on the active version until the rebuild is ready, and the
    first one after that swaps; the swapped cache matches the oracle."""
    csr = csr_mod()
    p = Pair(C2, pool_pages=256, max_seq=8192, max_new=512)
    lo = torch.cuda.Stream(priority=0)
    outs = {}
    p.ctx.set_reconciler(_provider(p, outs), lo)
    p.init_static(p.blk(970, 300))
    for i in range(12):
        p.append(p.blk(971 + i, 200))
    assert p.ctx.route(0) == csr.ROUTE_CONTINUE
    p.ctx.evict_and_reconcile(600)
    p.orc.evict(600)
    routes, seed = [], 990
    while True:
        r = p.ctx.route(1)
        routes.append(r)
        if r == csr.ROUTE_SWAPPED:
            break
        assert r == csr.ROUTE_BRIDGE and len(routes) < 10000
        if len(routes) <= 3:            # bridged tasks: their chunks join the rebuild
            p.append(p.blk(seed, 64))
            p.suffix(p.blk(seed + 100, 16))
            p.truncate()
            seed += 1
    assert p.ctx.versions() == (1, 1)
    p.orc.reconcile()
    torch.cuda.synchronize()
    p.check_layout()
    p.check_cache()
    assert p.ctx.route(0) == csr.ROUTE_STRAGGLER
    p.suffix(p.blk(999, 33))
    p.truncate()
    p.device_clean()


def test_deadline_and_cancel(libcsr):
    """csr_wait_reconcile with a deadline the rebuild cannot meet returns
    CSR_ETIMEOUT and leaves it running; csr_cancel_reconcile abandons it (the
    active version keeps serving, the pending pages return to the pool); a
    second eviction then runs to the swap and matches the oracle."""
    csr = csr_mod()
    p = Pair(C2, pool_pages=256, max_seq=8192, max_new=1024)
    lo = torch.cuda.Stream(priority=0)
    outs = {}
    p.ctx.set_reconciler(_provider(p, outs), lo)
    p.init_static(p.blk(1100, 300))
    for i in range(6):
        p.append(p.blk(1101 + i, 300))
    free_before = p.ctx.free_pages()
    p.ctx.evict_and_reconcile(600)
    with pytest.raises(csr.CsrError) as e:
        p.ctx.wait_reconcile(1e-6)
    assert e.value.status == csr.ETIMEOUT
    p.ctx.cancel_reconcile()
    assert p.ctx.free_pages() == free_before
    assert p.ctx.poll_swap() == csr.RECON_IDLE
    p.check_layout()
    p.suffix(p.blk(1120, 40))               # the active version still serves
    p.truncate()
    p.ctx.evict_and_reconcile(600)
    p.orc.evict(600)
    assert p.ctx.wait_reconcile(60.0) == csr.RECON_SWAPPED
    p.orc.reconcile()
    torch.cuda.synchronize()
    p.check_layout()
    p.check_cache()
    p.device_clean()


def test_provider_failure_keeps_old_version(libcsr):
    csr = csr_mod()
    p = Pair(C1, pool_pages=128, max_seq=4096, max_new=256)
    lo = torch.cuda.Stream(priority=0)

    def bad(cid, n):
        raise RuntimeError("layer below unavailable")

    p.ctx.set_reconciler(bad, lo)
    p.init_static(p.blk(950, 32))
    for i in range(4):
        p.append(p.blk(951 + i, 32))
    snap = (p.ctx.layout(), p.ctx.free_pages())
    # the call returns before the provider runs (on the reconciliation
    # thread); the failure surfaces at the next wait/poll, which aborts
    p.ctx.evict_and_reconcile(32)
    with pytest.raises(csr.CsrError) as e:
        p.ctx.wait_reconcile(30.0)
    assert e.value.status == csr.ESTATE
    assert "provider" in str(e.value)
    assert (p.ctx.layout(), p.ctx.free_pages()) == snap
    assert p.ctx.poll_swap() == csr.RECON_IDLE
    p.suffix(p.blk(960, 9))
    p.truncate()
    p.device_clean()
