"""The asynchronous state reconciliation cycle (Algorithm 1) as the paper runs
it, on the GPU, against the oracle.

* The paper's ASR setting (section IV: 100-token state chunks, the oldest half
  of the chunks evicted when tau_mem is reached), scaled down so the fp64
  oracle attends every call: an unaligned prefix (1,000 tokens, page 64),
  100-token chunks, a 37-token suffix truncated every step (partial pages),
  tau_mem = 3,000 tokens, three eviction cycles.  Every output, every post-swap
  page table and free list, and the whole rebuilt cache match the oracle.
* The full-size cycle of the 120K head shape (cap 131,072 tokens, 4,096-token
  prefix, 256-token chunks, 32,768 tokens evicted per cycle): two cycles with
  the page tables and free lists bit-exact against the oracle's allocator and
  256 sampled cache rows per swap checked one by one (rotated keys against the
  oracle's RoPE at the renumbered position, values bit-exact).
"""
import time

import numpy as np
import pytest
import torch

from gpu_util import C2, Pair, assert_close, csr_mod, to_dev, to_f64
from oracle import oracle as orc

pytestmark = pytest.mark.gpu


def _provider(p: Pair, outs: dict):
    def prov(cid, n):
        b = p.blocks[cid]
        out = torch.empty((n, p.hq, p.d), dtype=torch.bfloat16, device="cuda")
        outs[cid] = out
        return to_dev(b.q), to_dev(b.k), to_dev(b.v), out
    return prov


def test_paper_asr_setting_scaled(libcsr):
    csr = csr_mod()
    cap, prefix, chunk, suffix = 3000, 1000, 100, 37
    evict = (cap - prefix) // 2        # the oldest half of the chunk tokens at tau_mem
    p = Pair(C2, pool_pages=256, max_seq=8192, max_new=1024, cap_tokens=cap, evict_tokens=evict)
    lo = torch.cuda.Stream(priority=0)
    outs = {}
    p.ctx.set_reconciler(_provider(p, outs), lo)
    p.init_static(p.blk(1000, prefix))
    seed, cycles, steps = 1001, 0, 0
    while cycles < 3:
        assert steps < 200, "the reconciliation never swapped"
        # a task starts by polling: the swap happens between tasks
        if p.orc.is_reconciling and p.ctx.poll_swap() == csr.RECON_SWAPPED:
            expect = p.orc.reconcile()
            torch.cuda.synchronize()
            for cid, (eo, _) in expect.items():
                assert_close(to_f64(outs[cid]), eo, f"cycle {cycles}: rebuilt chunk {cid}")
            p.check_layout()
            p.check_cache()
            cycles += 1
        p.append(p.blk(seed, chunk))
        if not p.orc.is_reconciling and p.orc.length() >= cap:
            p.orc.evict(evict)              # the library started it inside append_chunk
            assert p.ctx.layout(csr.VERSION_PENDING)[0] == p.orc.page_table("pending")
            assert p.ctx.chunks(csr.VERSION_PENDING)[0] == p.orc.retained_ids
        p.suffix(p.blk(seed + 5000, suffix))
        p.truncate()
        seed += 1
        steps += 1
    p.device_clean()


def test_asr_full_size_cycles(libcsr):
    csr = csr_mod()
    hq, hkv, d, P, base = 64, 4, 128, 64, 1e6
    cap, prefix, chunk, suffix, evict = 131072, 4096, 256, 512, 32768
    n_max = cap + evict
    pool_pages = 2 * n_max // P + 64
    cfg = csr.make_config(hq, hkv, d, P, base, max_new_tokens=prefix, pool_pages=pool_pages,
                          max_seq_tokens=n_max, cap_tokens=cap, evict_tokens=evict)
    fg = torch.cuda.Stream(priority=-1)
    lo = torch.cuda.Stream(priority=0)
    gen = torch.Generator(device="cuda").manual_seed(77)

    def rnd(n, h):
        return torch.randn((n, h, d), generator=gen, device="cuda").to(torch.bfloat16)

    chunks = {}                            # chunk id -> (q, k, v) pre-RoPE device tensors
    ctx = csr.Context(cfg, stream=fg)
    ctx.set_reconciler(lambda cid, n: (*chunks[cid], None), lo)
    # the oracle's allocator on the same operations (bookkeeping only)
    model = orc.OracleCSR(1, 1, 2, P, base, pool_pages)
    model.attend = False
    z = lambda n: (np.zeros((n, 1, 2)), np.zeros((n, 1, 2)), np.zeros((n, 1, 2)))
    with torch.cuda.stream(fg):
        ctx.init_static(rnd(prefix, hq), rnd(prefix, hkv), rnd(prefix, hkv), stream=fg)
        model.init_static(*z(prefix))
        fill = 4096
        while model.length() + fill < cap - chunk:
            cid = len(chunks)
            chunks[cid] = (rnd(fill, hq), rnd(fill, hkv), rnd(fill, hkv))
            assert ctx.append_chunk(*chunks[cid], stream=fg)[2] == cid
            model.append_chunk(*z(fill))
        sq, sk, sv = rnd(suffix, hq), rnd(suffix, hkv), rnd(suffix, hkv)
    fg.synchronize()
    rng = np.random.default_rng(5)
    cycles, steps = 0, 0
    while cycles < 2:
        assert steps < 2000, "the reconciliation never swapped"
        if model.is_reconciling and ctx.poll_swap(fg) == csr.RECON_SWAPPED:
            model.reconcile()
            pt, length = ctx.layout()
            assert pt == model.page_table(), f"cycle {cycles}: page table"
            assert ctx.free_pages() == model.free_ids(), f"cycle {cycles}: free list"
            assert length == model.length()
            # sampled rows of the rebuilt cache, one by one against the oracle's RoPE
            ids, lens, pre_len = ctx.chunks(csr.VERSION_ACTIVE)
            starts = pre_len + np.concatenate([[0], np.cumsum(lens)[:-1]])
            rows = np.sort(rng.choice(np.arange(pre_len, length), size=256, replace=False))
            for pos in rows:
                i = int(np.searchsorted(starts, pos, side="right") - 1)
                off = int(pos - starts[i])
                _, k_pre, v_pre = chunks[ids[i]]
                k_got, v_got = ctx.gather_kv(csr.VERSION_ACTIVE, int(pos), 1, stream=fg)
                fg.synchronize()
                k_exp = orc.rope(to_f64(k_pre[off:off + 1]), np.array([pos]), base)
                assert_close(to_f64(k_got), k_exp, f"cycle {cycles}: rotated key at {pos}")
                assert torch.equal(v_got.view(torch.int16), v_pre[off:off + 1].view(torch.int16)), \
                    f"cycle {cycles}: value at {pos}"
            cycles += 1
        with torch.cuda.stream(fg):
            cid = len(chunks)
            chunks[cid] = (rnd(chunk, hq), rnd(chunk, hkv), rnd(chunk, hkv))
            assert ctx.append_chunk(*chunks[cid], stream=fg)[2] == cid
            model.append_chunk(*z(chunk))
            if not model.is_reconciling and model.length() >= cap:
                model.evict(evict)
                assert ctx.layout(csr.VERSION_PENDING)[0] == model.page_table("pending")
            ctx.attend_suffix(sq, sk, sv, stream=fg)
            ctx.truncate_suffix()
        fg.synchronize()
        if model.is_reconciling:
            time.sleep(0.005)   # a task cadence: leaves the low-priority rebuild room to run
        steps += 1
    assert ctx.device_status() == 0
    ctx.close()
