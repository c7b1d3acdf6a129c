"""The 120K-context step at full size, in the launch configuration the
benchmark times, against the fp64 oracle on sampled query rows.

A 122,880-token cache (4,096-token static prefix + 4,096-token chunks) of the
64 q / 4 kv head, head_dim 128, page 64 shape; then the step -- a 256-token
chunk and a 512-token suffix -- once fused (csr_append_chunk_attend_suffix,
the benchmark's default) and once as two calls.  For 71 sampled query tokens
the oracle computes the attention of all 64 heads over every cached key one
row at a time (inputs are the bf16 values the library received, keys rotated by
the oracle's RoPE at their absolute positions); outputs and log-sum-exps must
be within the parity tolerances, and the page table must equal the oracle
allocator's.
"""
import math

import numpy as np
import pytest
import torch

from gpu_util import assert_close, assert_lse_close, csr_mod, to_dev, to_f64
from oracle import oracle as orc
from paper_2605_07325_gb300 import synth

pytestmark = pytest.mark.gpu

HQ, HKV, D, P, BASE = 64, 4, 128, 64, 1e6
PREFIX, FILL, L0, CHUNK, SUFFIX = 4096, 4096, 122880, 256, 512
# Sampled token offsets in the 768-token step (8 tokens per 128-row tile at
# 16 query heads per kv head, 16 per pair of tiles): both sides of tile and
# tile-pair boundaries, the chunk/suffix boundary (255 | 256), the first and
# last token, and one token of every one of the 48 pairs (each pair is four
# units, one per kv head, most of them cut into pieces by the fused schedule).
_EDGES = [0, 1, 7, 8, 15, 16, 17, 31, 32, 127, 128, 247, 248, 255, 256, 257, 263, 264, 271, 272,
          511, 512, 759, 760, 766, 767]
SAMPLE = np.array(sorted(set(_EDGES) | {16 * p + (5 * p) % 16 for p in range(48)}))
assert len(SAMPLE) >= 64


@pytest.fixture(scope="module")
def cache():
    csr = csr_mod()
    cfg = csr.make_config(HQ, HKV, D, P, BASE, max_new_tokens=FILL,
                          pool_pages=(L0 + CHUNK + SUFFIX) // P + 16,
                          max_seq_tokens=L0 + CHUNK + SUFFIX + P)
    ctx = csr.Context(cfg)
    model = orc.OracleCSR(1, 1, 2, P, BASE, cfg.pool_pages)     # the allocator, bookkeeping only
    model.attend = False
    z = lambda n: (np.zeros((n, 1, 2)), np.zeros((n, 1, 2)), np.zeros((n, 1, 2)))
    ks, vs = [], []
    for i in range(L0 // FILL):
        b = synth.block(5000 + i, FILL, HQ, HKV, D, "kv_only")   # queries zero: outputs unused
        q, k, v = to_dev(b.q), to_dev(b.k), to_dev(b.v)
        if i == 0:
            ctx.init_static(q, k, v)
            model.init_static(*z(FILL))
        else:
            ctx.append_chunk(q, k, v)
            model.append_chunk(*z(FILL))
        ks.append(synth.bf16_to_f64(b.k))
        vs.append(synth.bf16_to_f64(b.v))
    torch.cuda.synchronize()
    assert ctx.layout()[1] == L0
    k_rot = orc.rope(np.concatenate(ks), np.arange(L0), BASE)
    v = np.concatenate(vs)
    yield ctx, model, k_rot, v
    ctx.close()


def _expected(block, k_rot, v):
    """Oracle outputs of the sampled step tokens over the cache + the step block."""
    q, k, vn = block.f64()
    pos = L0 + np.arange(CHUNK + SUFFIX)
    k_all = np.concatenate([k_rot, orc.rope(k, pos, BASE)])
    v_all = np.concatenate([v, vn])
    kpos = np.arange(L0 + CHUNK + SUFFIX)
    q_rot = orc.rope(q[SAMPLE], pos[SAMPLE], BASE)
    return orc.attention(q_rot, pos[SAMPLE], k_all, v_all, kpos, 1.0 / math.sqrt(D))


@pytest.mark.parametrize("fused", [True, False], ids=["fused", "separate"])
def test_120k_step_sampled_rows_match_oracle(cache, fused):
    csr = csr_mod()
    ctx, model, k_rot, v = cache
    block = synth.block(6000 + int(fused), CHUNK + SUFFIX, HQ, HKV, D)
    q, k, vv = to_dev(block.q), to_dev(block.k), to_dev(block.v)
    out = torch.empty((CHUNK + SUFFIX, HQ, D), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((HQ, CHUNK + SUFFIX), dtype=torch.float32, device="cuda")
    if fused:
        ctx.append_chunk_attend_suffix(q, k, vv, CHUNK, out=out, lse=lse)
    else:
        c, s = slice(0, CHUNK), slice(CHUNK, CHUNK + SUFFIX)
        lse_c = torch.empty((HQ, CHUNK), dtype=torch.float32, device="cuda")
        lse_s = torch.empty((HQ, SUFFIX), dtype=torch.float32, device="cuda")
        ctx.append_chunk(q[c], k[c], vv[c], out=out[c], lse=lse_c)
        ctx.attend_suffix(q[s], k[s], vv[s], out=out[s], lse=lse_s)
        lse = torch.cat([lse_c, lse_s], dim=1)
    torch.cuda.synchronize()
    model.append_chunk(*[np.zeros((CHUNK, 1, 2))] * 3)
    model.attend_suffix(*[np.zeros((SUFFIX, 1, 2))] * 3)
    assert ctx.layout()[0] == model.page_table()
    exp_out, exp_lse = _expected(block, k_rot, v)
    assert_close(to_f64(out)[SAMPLE], exp_out, "120K step, sampled rows")
    assert_lse_close(lse.cpu().numpy().astype(np.float64)[:, SAMPLE], exp_lse, "120K step lse")
    ctx.truncate_suffix()
    ctx.rewind(L0)
    model.truncate_suffix()
    model.rewind(L0)
    assert ctx.layout()[0] == model.page_table() and ctx.free_pages() == model.free_ids()
    assert ctx.device_status() == 0
