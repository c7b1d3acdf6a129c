"""Pins of the fp64 oracle to facts that do not come from the oracle itself.

Each pin returns a list of failure messages (empty when it holds).  The same
pins run against the real oracle (tests/test_oracle_pins.py, all must hold)
and against copies of oracle.c with a planted mistake
(tests/test_oracle_mutations.py, at least one must fail for every mistake).

Sources of truth used here:
  * closed forms and hand computations (golden files under tests/golden/);
  * a different formulation of the same mathematics (RoPE as complex
    multiplication; the attention of a block as rows of the one-shot
    attention over the whole sequence);
  * special cases that reduce to textbook results (V = 1 gives rows that sum
    to one; K = 0 gives the causal mean of V; one key gives V);
  * a library routine: torch.nn.functional.scaled_dot_product_attention and
    torch.logsumexp in float64 on the CPU.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _close(a, b, tol):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    if a.shape != b.shape:
        return False
    return bool(np.all(np.abs(a - b) <= tol))


# ---------------------------------------------------------------- RoPE pins
def pin_rope_identity_at_zero(orc):
    rng = np.random.default_rng(1)
    x = rng.standard_normal((3, 2, 8))
    y = orc.rope(x, np.zeros(3, np.int64), 10000.0)
    return [] if np.array_equal(x, y) else ["rope(x, 0) != x"]


def pin_rope_golden_unit_pair(orc):
    g = _load("rope_unit_pair.json")
    fails = []
    for case in g["cases"]:
        x = np.array(case["x"], np.float64).reshape(1, 1, -1)
        y = orc.rope(x, np.array([case["pos"]], np.int64), g["base"])
        if not _close(y.ravel(), case["y"], 1e-15):
            fails.append(f"rope golden {case}: got {y.ravel().tolist()}")
    return fails


def pin_rope_complex_form(orc):
    """Pair (i, i + d/2) as the complex number x_i + j x_{i+d/2}; RoPE
    multiplies it by exp(j * pos * base^(-2i/d))."""
    rng = np.random.default_rng(2)
    n, h, d, base = 5, 3, 16, 10000.0
    x = rng.standard_normal((n, h, d))
    pos = np.array([0, 1, 7, 1000, 131071], np.int64)
    y = orc.rope(x, pos, base)
    half = d // 2
    z = x[..., :half] + 1j * x[..., half:]
    freq = base ** (-(np.arange(half) * 2.0) / d)
    rot = np.exp(1j * pos[:, None, None] * freq[None, None, :])
    w = z * rot
    expect = np.concatenate([w.real, w.imag], axis=-1)
    err = np.max(np.abs(expect - y))
    return [] if err <= 1e-9 else [f"rope complex form max err {err}"]


def pin_rope_relative(orc):
    """<rope(q, p), rope(k, p')> depends only on p - p'."""
    rng = np.random.default_rng(3)
    d = 32
    q = rng.standard_normal((1, 1, d))
    k = rng.standard_normal((1, 1, d))
    fails = []
    for p, pp, s in [(5, 2, 11), (100, 0, 977), (3, 40, 50000)]:
        a = float(np.sum(orc.rope(q, np.array([p]), 1e6) * orc.rope(k, np.array([pp]), 1e6)))
        b = float(np.sum(orc.rope(q, np.array([p + s]), 1e6) * orc.rope(k, np.array([pp + s]), 1e6)))
        if abs(a - b) > 1e-9 * max(1.0, abs(a)):
            fails.append(f"relative property {p},{pp},{s}: {a} vs {b}")
    return fails


def pin_rope_norm(orc):
    rng = np.random.default_rng(4)
    x = rng.standard_normal((4, 2, 64))
    y = orc.rope(x, np.array([3, 99, 4096, 122879]), 1e6)
    half = 32
    nx = x[..., :half] ** 2 + x[..., half:] ** 2
    ny = y[..., :half] ** 2 + y[..., half:] ** 2
    err = np.max(np.abs(nx - ny))
    return [] if err < 1e-12 else [f"pair norm changed by {err}"]


# ----------------------------------------------------------- attention pins
def _sdpa(q, qpos, k, v, kpos, scale):
    import torch
    G = q.shape[1] // k.shape[1]
    qt = torch.from_numpy(q).permute(1, 0, 2)            # [hq][n][d]
    kt = torch.from_numpy(k).permute(1, 0, 2).repeat_interleave(G, 0)
    vt = torch.from_numpy(v).permute(1, 0, 2).repeat_interleave(G, 0)
    mask = torch.from_numpy(kpos[None, :] <= qpos[:, None])  # [n][nk]
    out = torch.nn.functional.scaled_dot_product_attention(
        qt, kt, vt, attn_mask=mask, scale=scale)
    s = torch.einsum("hnd,hmd->hnm", qt, kt) * scale
    s = s.masked_fill(~mask, float("-inf"))
    lse = torch.logsumexp(s, dim=-1)                      # [hq][n]
    return out.permute(1, 0, 2).numpy(), lse.numpy()


def pin_attention_vs_library(orc):
    rng = np.random.default_rng(5)
    fails = []
    for (n, nk0, hq, hkv, d) in [(7, 0, 4, 2, 8), (5, 11, 8, 2, 16), (9, 20, 6, 3, 4)]:
        nk = nk0 + n
        q = rng.standard_normal((n, hq, d))
        k = rng.standard_normal((nk, hkv, d))
        v = rng.standard_normal((nk, hkv, d))
        kpos = np.arange(nk, dtype=np.int64)
        qpos = kpos[nk0:]
        scale = 1.0 / math.sqrt(d)
        o, lse = orc.attention(q, qpos, k, v, kpos, scale, threads=2)
        eo, e_lse = _sdpa(q, qpos, k, v, kpos, scale)
        if not _close(o, eo, 1e-12):
            fails.append(f"attention vs sdpa max err {np.max(np.abs(o - eo))}")
        if not _close(lse, e_lse, 1e-12):
            fails.append(f"lse vs logsumexp max err {np.max(np.abs(lse - e_lse))}")
    return fails


def pin_attention_ones_v(orc):
    """V = 1: every output is 1 (the softmax weights sum to one)."""
    rng = np.random.default_rng(6)
    n, nk, hq, hkv, d = 6, 10, 4, 2, 8
    q = rng.standard_normal((n, hq, d)) * 3
    k = rng.standard_normal((nk, hkv, d)) * 3
    v = np.ones((nk, hkv, d))
    kpos = np.arange(nk)
    o, _ = orc.attention(q, kpos[nk - n:], k, v, kpos, 0.5, threads=1)
    err = np.max(np.abs(o - 1.0))
    return [] if err < 1e-12 else [f"V=1 gives {err} off 1"]


def pin_attention_zero_k(orc):
    """K = 0: uniform weights, out = mean of the visible V, lse = log(count)."""
    rng = np.random.default_rng(7)
    n, nk, hq, hkv, d = 5, 9, 4, 2, 8
    q = rng.standard_normal((n, hq, d))
    k = np.zeros((nk, hkv, d))
    v = rng.standard_normal((nk, hkv, d))
    kpos = np.arange(nk)
    qpos = kpos[nk - n:]
    o, lse = orc.attention(q, qpos, k, v, kpos, 0.3, threads=1)
    fails = []
    G = hq // hkv
    for t in range(n):
        cnt = qpos[t] + 1
        for h in range(hq):
            mean = v[:cnt, h // G, :].mean(axis=0)
            if not _close(o[t, h], mean, 1e-12):
                fails.append(f"K=0 mean mismatch t={t} h={h}")
            if abs(lse[h, t] - math.log(cnt)) > 1e-12:
                fails.append(f"K=0 lse mismatch t={t} h={h}")
    return fails[:3]


def pin_attention_single_key(orc):
    """One visible key: out = V of that key, whatever q and k are."""
    rng = np.random.default_rng(8)
    q = rng.standard_normal((1, 4, 8))
    k = rng.standard_normal((1, 2, 8))
    v = rng.standard_normal((1, 2, 8))
    o, lse = orc.attention(q, np.array([0]), k, v, np.array([0]), 0.25, threads=1)
    expect = np.repeat(v, 2, axis=1)  # heads 0,1 -> kv 0; heads 2,3 -> kv 1
    return [] if _close(o, expect, 0.0) else ["single key out != V"]


def pin_attention_gqa_grouping(orc):
    """Each kv head carries a constant V equal to its index: q head h must
    return h // (hq / hkv) (contiguous grouping, reading R2)."""
    hq, hkv, d, nk = 8, 4, 4, 5
    rng = np.random.default_rng(9)
    q = rng.standard_normal((2, hq, d))
    k = rng.standard_normal((nk, hkv, d))
    v = np.zeros((nk, hkv, d))
    for j in range(hkv):
        v[:, j, :] = j
    kpos = np.arange(nk)
    o, _ = orc.attention(q, np.array([3, 4]), k, v, kpos, 0.5, threads=1)
    expect = np.array([h // (hq // hkv) for h in range(hq)], np.float64)
    got = o[:, :, 0]
    return [] if np.allclose(got, expect[None, :], atol=1e-12) else [f"grouping {got}"]


def pin_attention_golden_hand_case(orc):
    g = _load("attention_hand_case.json")
    q = np.array(g["q"], np.float64).reshape(1, 1, -1)
    k = np.array(g["k"], np.float64).reshape(-1, 1, len(g["q"]))
    v = np.array(g["v"], np.float64).reshape(-1, 1, len(g["q"]))
    kpos = np.zeros(k.shape[0], np.int64)
    o, lse = orc.attention(q, np.array([0]), k, v, kpos, g["scale"], threads=1)
    fails = []
    if not _close(o.ravel(), g["out"], 1e-12):
        fails.append(f"hand case out {o.ravel()}")
    if abs(lse[0, 0] - g["lse"]) > 1e-12:
        fails.append(f"hand case lse {lse[0, 0]}")
    return fails


def pin_attention_causal_future_invisible(orc):
    """Changing keys/values at positions after the query leaves its output
    unchanged (section III-A: cached states are not altered by later tokens)."""
    rng = np.random.default_rng(10)
    n, hq, hkv, d = 6, 2, 1, 8
    q = rng.standard_normal((n, hq, d))
    k = rng.standard_normal((n, hkv, d))
    v = rng.standard_normal((n, hkv, d))
    pos = np.arange(n)
    o1, _ = orc.attention(q, pos, k, v, pos, 0.4, threads=1)
    k2, v2 = k.copy(), v.copy()
    k2[4:] += 5.0
    v2[4:] -= 3.0
    o2, _ = orc.attention(q, pos, k2, v2, pos, 0.4, threads=1)
    ok = np.array_equal(o1[:4], o2[:4]) and not np.allclose(o1[4:], o2[4:])
    return [] if ok else ["future keys changed a past output (or were ignored)"]


ROPE_PINS = [pin_rope_identity_at_zero, pin_rope_golden_unit_pair, pin_rope_complex_form,
             pin_rope_relative, pin_rope_norm]
ATTENTION_PINS = [pin_attention_vs_library, pin_attention_ones_v, pin_attention_zero_k,
                  pin_attention_single_key, pin_attention_gqa_grouping,
                  pin_attention_golden_hand_case, pin_attention_causal_future_invisible]
ALL_PINS = ROPE_PINS + ATTENTION_PINS


def run_all(orc):
    fails = []
    for p in ALL_PINS:
        try:
            fails += [f"{p.__name__}: {m}" for m in p(orc)]
        except Exception as e:  # a crash is a failed pin too
            fails.append(f"{p.__name__}: raised {e!r}")
    return fails
