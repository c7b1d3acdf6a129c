"""GPU path (through the C-ABI) against the fp64 oracle, element by element.

Covers the tiny correctness configuration in full, the 64/4/128 head shape
with ragged sizes, split-KV partial merging under forced CTA counts, edge
cases (one token, n = max_new_tokens, special inputs, scores spread over
hundreds of units) and run-to-run bitwise determinism.
"""
import math

import numpy as np
import pytest
import torch

from gpu_util import (C1, C2, TOL_LSE, TOL_MAX_ABS, TOL_REL_FRO, Pair, assert_close, bits_of,
                      csr_mod, err_stats, to_dev, to_f64)
from oracle import oracle as orc
from paper_2605_07325_gb300 import synth

pytestmark = pytest.mark.gpu


def test_tiny_config_full_session(libcsr):
    """8 q heads / 2 kv heads, d=64, page 16, base 1e4: 256-token prefix,
    3 chunks of 256, a 32-token suffix, truncate, one more chunk, suffix again."""
    p = Pair(C1, pool_pages=256, max_seq=4096, max_new=512, fg_chunk_tiles=3)
    p.init_static(p.blk(0, 256))
    for i in range(3):
        p.append(p.blk(1 + i, 256))
    p.check_layout()
    p.suffix(p.blk(1_000_000, 32))
    p.check_layout()
    p.truncate()
    p.check_layout()
    p.append(p.blk(4, 256))
    p.suffix(p.blk(1_000_001, 32))
    p.check_layout()
    p.check_cache()
    p.truncate()
    p.check_layout()
    p.device_clean()


def test_single_token_prefix_returns_v(libcsr):
    """L=0, n=1: the only visible key is the token itself, so out = V exactly."""
    p = Pair(C2, pool_pages=16, max_seq=1024, max_new=256)
    b = p.blk(5, 1)
    out, lse = p.init_static(b)
    v = b.f64()[2]                                    # [1][hkv][d]
    expect = np.repeat(v, p.hq // p.hkv, axis=1)
    assert np.array_equal(to_f64(out), expect)
    p.device_clean()


# Foreground paths: one cooperative launch of the fused kernel, or three
# chained launches (the library picks by the call's work; the flags force).
PATHS = {"fused": 0x2, "three": 0x4}


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("shape", [C1, C2], ids=["d64_p16_g4", "d128_p64_g16"])
@pytest.mark.parametrize("chunk_tiles", [0, 2])
def test_ragged_sizes(libcsr, shape, chunk_tiles, path):
    p = Pair(shape, pool_pages=128, max_seq=4096, max_new=512, fg_chunk_tiles=chunk_tiles,
             flags=PATHS[path])
    p.init_static(p.blk(10, 37))
    for i, n in enumerate([1, 129, 64, 300, 17]):
        p.append(p.blk(11 + i, n))
    p.suffix(p.blk(20, 7))
    p.check_layout()
    p.truncate()
    p.append(p.blk(21, 5))
    p.suffix(p.blk(22, 250))
    p.check_layout()
    p.check_cache()
    p.device_clean()


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("num_ctas,chunk_tiles", [(1, 0), (3, 1), (7, 2), (19, 3), (64, 5),
                                                   (152, 1), (0, 4), (0, 0), (5, 0)])
def test_split_kv_partials_any_grid(libcsr, num_ctas, chunk_tiles, path):
    """Forced CTA counts and piece lengths: every cut of a unit into pieces
    (down to one 128-key tile) must merge back to the oracle, on both paths
    (the fused kernel's last pieces merge the others' partials; the
    three-launch path's merge kernel combines chunk partials)."""
    sizes = (700, 1000, 33, 200)
    p = Pair(C2, pool_pages=256, max_seq=8192, max_new=1024, num_ctas=num_ctas,
             fg_chunk_tiles=chunk_tiles, flags=PATHS[path])
    p.init_static(p.blk(30, sizes[0]))
    p.append(p.blk(31, sizes[1]))
    p.append(p.blk(32, sizes[2]))
    p.suffix(p.blk(33, sizes[3]))
    p.truncate()
    p.device_clean()


def test_max_new_tokens_call(libcsr):
    p = Pair(C2, pool_pages=128, max_seq=8192, max_new=1024)
    p.init_static(p.blk(40, 1024))
    p.append(p.blk(41, 1024))
    p.check_layout()
    p.device_clean()


def test_special_inputs(libcsr):
    """V = 1 gives outputs of 1 (the weights sum to one); K = 0 gives the
    causal mean of V (within the bf16 rounding of the weights)."""
    p = Pair(C2, pool_pages=64, max_seq=4096, max_new=512)
    out, _ = p.init_static(p.blk(50, 300, "ones_v"))
    got = to_f64(out)
    assert np.max(np.abs(got - 1.0)) <= 2e-2
    p2 = Pair(C1, pool_pages=64, max_seq=4096, max_new=512)
    p2.init_static(p2.blk(51, 200, "zero_k"))
    p2.append(p2.blk(52, 100, "zero_k"))
    p.device_clean()
    p2.device_clean()


@pytest.mark.parametrize("shape", [C1, C2], ids=["d64_p16_g4", "d128_p64_g16"])
def test_large_scores_match_oracle(libcsr, shape):
    """Scores spread over hundreds of units (Q and K scaled by 12): the softmax
    must take each row's true maximum -- from the reducing TMEM load on whole
    key tiles, recomputed after masking on a row's diagonal tile -- and rescale
    O when it jumps; a wrong maximum overflows (non-finite outputs) or flushes
    every weight (zero rows).  At this scale the bf16 rounding of the rotated
    queries and keys alone moves scores by ~0.2 and near-ties by as much, so
    the bound is three times the difference the oracle itself shows between
    exact and bf16-rounded rotated operands on the same inputs."""
    csr = csr_mod()
    hq, hkv, d, P, base = shape["hq"], shape["hkv"], shape["d"], shape["P"], shape["base"]
    ctx = csr.Context(csr.make_config(hq, hkv, d, P, base, max_new_tokens=512, pool_pages=128,
                                      max_seq_tokens=4096))
    blocks = [synth.block(90 + i, n, hq, hkv, d, "peaked") for i, n in enumerate((300, 200, 50))]
    ctx.init_static(*(to_dev(x) for x in (blocks[0].q, blocks[0].k, blocks[0].v)))
    lse_c = torch.empty((hq, 200), dtype=torch.float32, device="cuda")
    lse_s = torch.empty((hq, 50), dtype=torch.float32, device="cuda")
    out_c, _, _ = ctx.append_chunk(*(to_dev(x) for x in (blocks[1].q, blocks[1].k, blocks[1].v)), lse=lse_c)
    out_s, _ = ctx.attend_suffix(*(to_dev(x) for x in (blocks[2].q, blocks[2].k, blocks[2].v)), lse=lse_s)
    torch.cuda.synchronize()
    f64 = [b.f64() for b in blocks]
    k = np.concatenate([x[1] for x in f64])
    v = np.concatenate([x[2] for x in f64])
    pos = np.arange(len(k))
    k_rot = orc.rope(k, pos, base)

    def rounded(x):
        return synth.bf16_to_f64(synth.bf16_bits(x.astype(np.float32)))

    scale = 1.0 / math.sqrt(d)
    for (q, _, _), p0, out, lse in ((f64[1], 300, out_c, lse_c), (f64[2], 500, out_s, lse_s)):
        qp = pos[p0:p0 + len(q)]
        q_rot = orc.rope(q, qp, base)
        exp_o, exp_l = orc.attention(q_rot, qp, k_rot[:qp[-1] + 1], v[:qp[-1] + 1], pos[:qp[-1] + 1], scale)
        rnd_o, rnd_l = orc.attention(rounded(q_rot), qp, rounded(k_rot[:qp[-1] + 1]), v[:qp[-1] + 1],
                                     pos[:qp[-1] + 1], scale)
        got_o = to_f64(out)
        got_l = lse.cpu().numpy().astype(np.float64)
        assert np.all(np.isfinite(got_o)) and np.all(np.isfinite(got_l))
        assert np.all(np.abs(got_o).reshape(len(q), -1).max(axis=1) > 0), "a row lost every weight"
        base_abs, base_rel = err_stats(rnd_o, exp_o)
        got_abs, got_rel = err_stats(got_o, exp_o)
        assert got_rel <= 3 * base_rel + TOL_REL_FRO, (got_rel, base_rel)
        assert got_abs <= 3 * base_abs + TOL_MAX_ABS, (got_abs, base_abs)
        assert np.max(np.abs(got_l - exp_l)) <= 3 * np.max(np.abs(rnd_l - exp_l)) + TOL_LSE
    assert ctx.device_status() == 0
    ctx.close()


def test_bitwise_deterministic(libcsr):
    outs = []
    for _ in range(2):
        p = Pair(C2, pool_pages=128, max_seq=8192, max_new=1024)
        p.init_static(p.blk(60, 500), compare=False)
        o1, _, _ = p.append(p.blk(61, 700), compare=False)
        o2, _ = p.suffix(p.blk(62, 100), compare=False)
        torch.cuda.synchronize()
        outs.append((bits_of(o1), bits_of(o2)))
    assert np.array_equal(outs[0][0], outs[1][0]) and np.array_equal(outs[0][1], outs[1][1])


def test_8k_context_step(libcsr):
    """64 q heads / 4 kv heads, d=128, page 64, base 1e6: 2048-token prefix plus
    48 chunks of 128 (8192 cached); a step appends a 128-token chunk, attends a
    64-token suffix over the whole cache, then truncates."""
    p = Pair(C2, pool_pages=512, max_seq=16384, max_new=2048)
    p.init_static(p.blk(100, 2048), compare=False)
    for i in range(48):
        p.append(p.blk(101 + i, 128, "kv_only"), compare=False)
    assert p.orc.length() == 8192
    for step in range(2):
        p.append(p.blk(200 + step, 128))
        p.suffix(p.blk(1_000_000 + step, 64))
        p.check_layout()
        p.truncate()
    p.check_layout()
    p.check_cache(positions=np.arange(0, p.orc.length(), 7))
    p.device_clean()


def test_launch_count_reported(libcsr):
    """A fused foreground call is one launch (RoPE + append, attention, merge),
    split or not; the three-launch path runs RoPE/append and attention, plus
    the merge when the keys were split."""
    p = Pair(C1, pool_pages=64, max_seq=2048, max_new=256, flags=PATHS["fused"])
    before = p.ctx.kernel_launches()
    p.init_static(p.blk(70, 100))
    assert p.ctx.kernel_launches() - before == 1
    p.append(p.blk(71, 37))
    assert p.ctx.kernel_launches() - before == 2
    p.device_clean()
    q = Pair(C1, pool_pages=64, max_seq=2048, max_new=256, flags=PATHS["three"])
    before = q.ctx.kernel_launches()
    q.init_static(q.blk(70, 100))
    assert 2 <= q.ctx.kernel_launches() - before <= 3
    q.device_clean()


def test_rewind_then_append_matches_never_appended(libcsr):
    """Cache invalidation after a chunk boundary (Eq. first_differing_token):
    the next chunk's output and layout equal a run that never had the dropped
    chunk, bit for bit."""
    a = Pair(C2, pool_pages=128, max_seq=8192, max_new=512)
    b = Pair(C2, pool_pages=128, max_seq=8192, max_new=512)
    for p in (a, b):
        p.init_static(p.blk(80, 300), compare=False)
        p.append(p.blk(81, 100), compare=False)
    a.append(a.blk(82, 200), compare=False)
    a.ctx.rewind(400)
    a.orc.rewind(400)
    oa, _, _ = a.append(a.blk(83, 150))
    ob, _, _ = b.append(b.blk(83, 150))
    torch.cuda.synchronize()
    assert np.array_equal(bits_of(oa), bits_of(ob))
    assert a.ctx.layout() == b.ctx.layout()
    a.check_layout()
    a.device_clean()


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("shape", [C1, C2], ids=["d64_p16_g4", "d128_p64_g16"])
@pytest.mark.parametrize("chunk_tiles", [0, 2])
def test_fused_step_matches_oracle(libcsr, shape, chunk_tiles, path):
    """csr_append_chunk_attend_suffix: the chunk's outputs equal those of
    append_chunk and the suffix's those of attend_suffix on the same cache;
    the layout after the truncation equals the two-call layout."""
    p = Pair(shape, pool_pages=160, max_seq=4096, max_new=1024, fg_chunk_tiles=chunk_tiles,
             flags=PATHS[path])
    p.init_static(p.blk(40, 77))
    for i, (nc, ns) in enumerate([(1, 1), (37, 100), (129, 300), (256, 512)]):
        p.fused(p.blk(41 + i, nc + ns), nc)
        p.check_layout()
        p.truncate()
        p.check_layout()
    p.append(p.blk(60, 50))
    p.check_cache()
    p.device_clean()


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("shape", [C1, C2], ids=["d64_p16_g4", "d128_p64_g16"])
@pytest.mark.parametrize("chunk_tiles", [1, 2, 3, 9])
def test_merge_many_chunks_per_row(libcsr, shape, chunk_tiles, path):
    """Long context, short blocks, short key chunks: rows merged from up to 67
    partials (the merge spreads such rows over several lane groups, and above
    64 partials takes its general path)."""
    pages = 16384 // shape["P"] + 64
    p = Pair(shape, pool_pages=pages, max_seq=16384, max_new=4096, fg_chunk_tiles=chunk_tiles,
             flags=PATHS[path])
    p.init_static(p.blk(70, 4000), compare=False)
    p.append(p.blk(71, 4000), compare=False)
    p.append(p.blk(72, 500))
    p.suffix(p.blk(73, 16))
    p.truncate()
    p.suffix(p.blk(74, 100))
    p.truncate()
    p.device_clean()


@pytest.mark.parametrize("num_ctas", [7, 19])
def test_local_schedule_matches_oracle(libcsr, num_ctas):
    """CSR_FLAG_SCHEDULE_LOCAL: the least-advanced-first pieces (taken on
    these shapes: 300-token suffixes over 2,000-8,000 cached tokens on 7 or 19
    CTAs, where they stay within 1 % of the optimum load) merge back to the
    oracle like the default idle-interval pieces."""
    csr = csr_mod()
    p = Pair(C2, pool_pages=256, max_seq=12000, max_new=4096, num_ctas=num_ctas,
             flags=PATHS["fused"] | csr.FLAG_SCHEDULE_LOCAL)
    p.init_static(p.blk(80, 2000), compare=False)
    p.suffix(p.blk(81, 300))
    p.truncate()
    p.append(p.blk(82, 2000), compare=False)
    p.suffix(p.blk(83, 300))
    p.truncate()
    p.append(p.blk(84, 4000), compare=False)
    p.suffix(p.blk(85, 300))
    p.truncate()
    p.check_layout()
    p.device_clean()


def _scale_v(b, shift):
    """The block with V multiplied by 2^shift, exactly (bf16 exponent field)."""
    v = b.v.copy()
    nz = (v & 0x7FFF) != 0
    v[nz] = v[nz] + np.uint16(shift << 7)
    return synth.Block(b.q, b.k, v)


@pytest.mark.parametrize("path", ["fused", "three"])
def test_split_partials_scale_exactly(libcsr, path):
    """Split partials are stored as fp16 rows scaled by their largest
    magnitude.  Values 2^20 times larger (outputs, averages of V, and the
    partial rows well past 65,504, the largest fp16 value) must give exactly
    2^20 times the outputs: every step of the path, the partials and their
    merge included, scales exactly by a power of two.  Short key chunks make
    every unit split on both paths."""
    outs = []
    for shift in (0, 20):
        p = Pair(C2, pool_pages=128, max_seq=8192, max_new=1024, fg_chunk_tiles=2, flags=PATHS[path])
        b0, b1 = p.blk(90, 1000), p.blk(91, 300)
        if shift:
            b0, b1 = _scale_v(b0, shift), _scale_v(b1, shift)
        p.init_static(b0, compare=False)
        q, k, v = p._dev(b1)
        out, _ = p.ctx.attend_suffix(q, k, v)
        torch.cuda.synchronize()
        outs.append(to_f64(out))
        p.ctx.truncate_suffix()
        p.device_clean()
    assert np.max(np.abs(outs[0])) > 0.1
    assert np.max(np.abs(outs[1])) > 65504.0
    assert np.array_equal(outs[1], outs[0] * 2.0 ** 20)
