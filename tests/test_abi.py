"""The C-ABI library loads and exports every function include/csr.h declares
(no GPU, no compute call)."""
import ctypes
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    inc = os.path.join(ROOT, "include")
    for fn in os.listdir(inc):
        if not fn.endswith(".h"):
            continue
        text = open(os.path.join(inc, fn)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        text = re.sub(r"//[^\n]*", "", text)
        for m in re.finditer(r"\b(csr_\w+)\s*\(", text):
            names.add(m.group(1))
    return names


def test_header_declares_the_boundary():
    names = _declared()
    for required in ["csr_init_static", "csr_append_chunk", "csr_attend_suffix",
                     "csr_truncate_suffix", "csr_evict_and_reconcile", "csr_create",
                     "csr_destroy", "csr_poll_swap"]:
        assert required in names


def test_library_exports_every_declared_symbol(libcsr):
    lib = ctypes.CDLL(libcsr.LIB_PATH)
    missing = [n for n in sorted(_declared()) if not hasattr(lib, n)]
    assert not missing, f"not exported: {missing}"


def test_size_queries_without_gpu(libcsr):
    cfg = libcsr.make_config(64, 4, 128, 64, 1e6, 4096, 4096, 131072)
    assert libcsr.pool_bytes(cfg) == 4096 * 4 * 64 * 128 * 2
    assert libcsr.workspace_bytes(cfg) > 0
    bad = libcsr.make_config(64, 4, 96, 64, 1e6, 4096, 4096, 131072)
    assert libcsr.pool_bytes(bad) == 0 and libcsr.workspace_bytes(bad) == 0
