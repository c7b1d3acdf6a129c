"""Seeded random sessions on the GPU in lockstep with the oracle: every
operation of the C ABI that changes the cache (appends of random lengths,
suffixes, fused chunk + suffix steps, truncations, rewinds, evictions with a
rebuild and swap, cancelled rebuilds, routing by sequence version), with every
attention output compared with the oracle, the layout after every call and
the whole cache at the end."""
import numpy as np
import pytest
import torch

from gpu_util import C1, Pair, assert_close, csr_mod, to_dev, to_f64

pytestmark = pytest.mark.gpu


def _provider(p, outs):
    def prov(cid, n):
        b = p.blocks[cid]
        out = torch.empty((n, p.hq, p.d), dtype=torch.bfloat16, device="cuda")
        outs[cid] = out
        return to_dev(b.q), to_dev(b.k), to_dev(b.v), out
    return prov


@pytest.mark.parametrize("seed", [1, 2, 3, 4])
def test_random_session_matches_oracle(libcsr, seed):
    csr = csr_mod()
    rng = np.random.default_rng(seed)
    p = Pair(C1, pool_pages=512, max_seq=6000, max_new=300, fg_chunk_tiles=int(rng.integers(0, 4)))
    lo = torch.cuda.Stream(priority=0)
    outs = {}
    p.ctx.set_reconciler(_provider(p, outs), lo)
    p.init_static(p.blk(seed * 1000, int(rng.integers(1, 200))))
    bseed = seed * 1000 + 1
    version = 0
    done = {"evict": 0, "cancel": 0, "swap": 0, "rewind": 0, "fused": 0}
    for _ in range(80):
        op = rng.choice(["chunk", "chunk", "step", "fused", "evict", "rewind", "poll"])
        if op == "chunk":
            p.append(p.blk(bseed, int(rng.integers(1, 150))))
        elif op in ("step", "fused"):
            nc, ns = int(rng.integers(1, 100)), int(rng.integers(1, 150))
            if op == "fused":
                p.fused(p.blk(bseed, nc + ns), nc)
                done["fused"] += 1
            else:
                p.append(p.blk(bseed, nc))
                p.suffix(p.blk(bseed + 50000, ns))
            if p.orc.is_reconciling and p.ctx.route(version + 1) == csr.ROUTE_SWAPPED:
                raise AssertionError("swapped while a suffix was live")
            p.truncate()
        elif op == "evict" and not p.orc.is_reconciling and len(p.orc.chunk_ids()) >= 2:
            e = int(rng.integers(1, 400))
            p.ctx.evict_and_reconcile(e)
            p.orc.evict(e)
            done["evict"] += 1
            assert p.ctx.layout(csr.VERSION_PENDING)[0] == p.orc.page_table("pending")
            if rng.random() < 0.25:
                p.ctx.cancel_reconcile()
                p.orc.cancel()
                done["cancel"] += 1
        elif op == "rewind" and p.orc.chunk_ids():
            if p.orc.is_reconciling:
                # a rewind needs a settled cache: finish the rebuild first (how
                # many steps it spans depends on the GPU's pace)
                assert p.ctx.wait_reconcile(60.0) == csr.RECON_SWAPPED
                expect = p.orc.reconcile()
                torch.cuda.synchronize()
                for cid, (eo, _) in expect.items():
                    assert_close(to_f64(outs[cid]), eo, f"rebuilt chunk {cid}")
                version += 1
                done["swap"] += 1
                assert p.ctx.versions() == (version, version)
                if not p.orc.chunk_ids():
                    bseed += 1
                    p.check_layout()
                    continue
            ids, lens, pre = p.ctx.chunks(csr.VERSION_ACTIVE)
            keep = int(rng.integers(0, len(ids) + 1))
            length = pre + int(sum(lens[:keep]))
            p.ctx.rewind(length)
            p.orc.rewind(length)
            done["rewind"] += 1
        elif op == "poll" and p.orc.is_reconciling:
            r = p.ctx.route(version + 1)
            assert r in (csr.ROUTE_BRIDGE, csr.ROUTE_SWAPPED)
            if r == csr.ROUTE_SWAPPED:
                expect = p.orc.reconcile()
                torch.cuda.synchronize()
                for cid, (eo, _) in expect.items():
                    assert_close(to_f64(outs[cid]), eo, f"rebuilt chunk {cid}")
                version += 1
                done["swap"] += 1
                assert p.ctx.versions() == (version, version)
        bseed += 1
        p.check_layout()
    if p.orc.is_reconciling:
        assert p.ctx.wait_reconcile(60.0) == csr.RECON_SWAPPED
        p.orc.reconcile()
    torch.cuda.synchronize()
    p.check_layout()
    p.check_cache()
    p.device_clean()
    assert done["evict"] >= 2 and done["swap"] >= 1 and done["rewind"] >= 1 and done["fused"] >= 1, done
