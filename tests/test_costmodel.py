"""FLOP accounting of the benchmark against the paper's closed forms (no GPU)."""
import json
import os

from paper_2605_07325_gb300 import costmodel

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "cost_model.json")


def test_pairs_match_eq_ttft_derivation_2():
    g = json.load(open(GOLDEN))
    for c in g["cases"]:
        T, i_star, L, n = c["T"], c["i_star"], c["L"], c["n"]
        closed = (T - i_star + 1) * (T + i_star) // 2          # the paper's form
        assert costmodel.query_key_pairs(L, n) == closed
        assert closed == sum(range(i_star, T + 1))              # brute force


def test_recon_time_closed_form():
    for a, dn in [(0, 1), (98304, 256), (7, 13)]:
        assert costmodel.recon_extension_pairs(a, dn) == sum(range(a + 1, a + dn + 1))


def test_prefix_stability_flop_ratio_order():
    """App. A: full recompute of |T| tokens vs an increment of Delta tokens is
    O(|T| / Delta) more work (1e5 / 1e3 ~ 1e2)."""
    g = json.load(open(GOLDEN))["ratio_case"]
    T, delta = g["T"], g["delta"]
    full = costmodel.query_key_pairs(0, T)
    inc = costmodel.query_key_pairs(T - delta, delta)
    ratio = full / inc
    assert g["ratio_order"] / 3 < ratio < g["ratio_order"] * 3


def test_flops_and_bytes_of_the_120k_step():
    # 256-token chunk over 122,880 cached tokens, then a 512-token suffix
    f = costmodel.attention_flops(64, 128, 122880, 256) + costmodel.attention_flops(64, 128, 123136, 512)
    assert abs(f / 1e12 - 3.10) < 0.01
    b = costmodel.call_bytes(64, 4, 128, 122880, 256)
    assert b == 4 * (122880 + 256) * 4 * 128 + 4 * 256 * 64 * 128 + 8 * 256 * 4 * 128
