"""Plant plausible mistakes in copies of oracle.c and check that the pins
catch every one of them (no GPU).

Each mutation is a text substitution in a temporary copy of the oracle's C
source; the copy is compiled with gcc into a temporary directory and swapped
into the oracle module for the duration of the check.
"""
import ctypes
import os
import subprocess
import tempfile

import pytest

import oracle_pins

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "oracle.c")

MUTATIONS = {
    "rope_sign": ("yr[i] = a * c - b * s;", "yr[i] = a * c + b * s;"),
    "rope_freq_exponent": ("pow(base, -2.0 * (double)i / (double)d)",
                           "pow(base, -1.0 * (double)i / (double)d)"),
    "rope_pairing_index": ("double a = xr[i], b = xr[i + half];",
                           "double a = xr[i], b = xr[(i + 1) % half + half];"),
    "causal_excludes_diagonal": ("if (j->kpos[tau] > j->qpos[t]) continue;",
                                 "if (j->kpos[tau] >= j->qpos[t]) continue;"),
    "gqa_strided_grouping": ("int32_t kvh = h / group;", "int32_t kvh = h % j->hkv;"),
    "dropped_normaliser": ("double w = scores[a] / z;", "double w = scores[a];"),
    "dropped_scale": ("scores[m_count] = dot * j->scale;", "scores[m_count] = dot;"),
    "v_reads_k": ("const double *vv = j->v +", "const double *vv = j->k +"),
    "lse_drops_max": ("j->lse[(size_t)h * j->n + t] = mx + log(z);",
                      "j->lse[(size_t)h * j->n + t] = log(z);"),
    "lse_transposed": ("j->lse[(size_t)h * j->n + t] = mx + log(z);",
                       "j->lse[(size_t)t * j->hq + h] = mx + log(z);"),
}


def _compile(src_text, tmpdir, name):
    c = os.path.join(tmpdir, name + ".c")
    so = os.path.join(tmpdir, name + ".so")
    with open(c, "w") as f:
        f.write(src_text)
    subprocess.check_call(["gcc", "-O1", "-fPIC", "-shared", "-std=c11", c, "-o", so,
                           "-lm", "-lpthread"])
    return so


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_is_caught(oracle_mod, name):
    old, new = MUTATIONS[name]
    text = open(SRC).read()
    assert text.count(old) == 1, f"mutation anchor for {name} not found exactly once"
    mutated = text.replace(old, new)
    saved = oracle_mod._LIB
    with tempfile.TemporaryDirectory() as tmp:
        so = _compile(mutated, tmp, name)
        lib = ctypes.CDLL(so)
        lib.oracle_rope.argtypes = saved.oracle_rope.argtypes
        lib.oracle_rope.restype = None
        lib.oracle_attention.argtypes = saved.oracle_attention.argtypes
        lib.oracle_attention.restype = ctypes.c_int
        oracle_mod._LIB = lib
        try:
            fails = oracle_pins.run_all(oracle_mod)
        finally:
            oracle_mod._LIB = saved
    assert fails, f"no pin caught the planted mistake {name}"
