"""csr_attend_block_noalloc, the entry point for callers that cannot allocate
device memory (a real-time loop that must not wait on the allocator, or a
process whose device memory belongs to another allocator), must give the same
attention as the workspace-based entry point on the same inputs.

It is called through the C ABI (ctypes) on three blocks in a row (up to the
largest n its static scratch holds), each right after csr_append_chunk has
placed the same block in a context's cache; the no-alloc call rewrites the
block's keys/values into the same slots (identical values) and its output
must match the oracle's and csr_append_chunk's within the parity tolerance.
Kept in a file pytest collects last.
"""
import ctypes

import numpy as np
import pytest
import torch

from gpu_util import C1, C2, Pair, TOL_LSE, assert_close, assert_lse_close, csr_mod, to_dev, to_f64

pytestmark = pytest.mark.gpu


class BlockArgs(ctypes.Structure):
    _fields_ = [
        ("q", ctypes.c_void_p), ("k", ctypes.c_void_p), ("v", ctypes.c_void_p),
        ("k_pool", ctypes.c_void_p), ("v_pool", ctypes.c_void_p),
        ("page_table", ctypes.c_void_p),
        ("out", ctypes.c_void_p), ("lse", ctypes.c_void_p),
        ("L", ctypes.c_int64), ("n", ctypes.c_int32),
        ("num_q_heads", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32), ("page_size", ctypes.c_int32),
        ("pool_pages", ctypes.c_int32),
        ("rope_base", ctypes.c_double), ("softmax_scale", ctypes.c_float),
    ]


def _noalloc():
    csr = csr_mod()
    lib = ctypes.CDLL(csr.LIB_PATH)
    fn = lib.csr_attend_block_noalloc
    fn.argtypes = [ctypes.POINTER(BlockArgs), ctypes.c_void_p]
    fn.restype = ctypes.c_int
    return csr, lib, fn


@pytest.mark.parametrize("shape,calls", [(C2, [(1301, 300), (1302, 77), (1303, 512)]),
                                         (C1, [(1311, 200), (1312, 33), (1313, 512)])],
                         ids=["d128_g16_up_to_n512", "d64_g4"])
def test_noalloc_block_matches_oracle_and_workspace_entry_point(libcsr, shape, calls):
    """Each block is appended through csr_append_chunk (checked against the
    oracle by the same call), then the no-alloc call repeats it over the same
    page table: its output and lse must match the oracle's within the parity
    tolerance and csr_append_chunk's.  n = 512 is the largest block the static
    scratch holds at 64 query heads of 128 dims."""
    csr, lib, fn = _noalloc()
    p = Pair(shape, pool_pages=256, max_seq=8192, max_new=512)
    p.init_static(p.blk(1300, 500), compare=False)
    p.append(p.blk(1299, 211), compare=False)
    stream = torch.cuda.current_stream()
    for call, (seed, n) in enumerate(calls):
        L = p.ctx.layout()[1]
        b = p.blk(seed, n)
        exp_out, exp_lse, cid = p.orc.append_chunk(*b.f64())
        q, k, v = to_dev(b.q), to_dev(b.k), to_dev(b.v)
        ref_lse = torch.empty((p.hq, n), dtype=torch.float32, device="cuda")
        ref_out, _, got_cid = p.ctx.append_chunk(q, k, v, lse=ref_lse)
        assert got_cid == cid
        pt = ctypes.c_void_p()
        assert lib.csr_device_page_table(ctypes.c_void_p(p.ctx._h.value), 0, ctypes.byref(pt)) == 0
        out = torch.empty_like(ref_out)
        lse = torch.empty_like(ref_lse)
        args = BlockArgs(q.data_ptr(), k.data_ptr(), v.data_ptr(),
                         p.ctx.k_pool.data_ptr(), p.ctx.v_pool.data_ptr(), pt.value,
                         out.data_ptr(), lse.data_ptr(), L, n, p.hq, p.hkv, p.d, p.P,
                         p.cfg.pool_pages, p.shape["base"], 0.0)
        assert fn(ctypes.byref(args), stream.cuda_stream) == 0, f"call {call}"
        torch.cuda.synchronize()
        got_lse = lse.cpu().numpy().astype(np.float64)
        assert_close(to_f64(out), exp_out, f"no-alloc block {call} (n={n}) vs oracle")
        assert_lse_close(got_lse, exp_lse, f"no-alloc lse {call} vs oracle")
        assert_close(to_f64(out), to_f64(ref_out), f"no-alloc block {call} vs csr_append_chunk")
        assert_lse_close(got_lse, ref_lse.cpu().numpy().astype(np.float64), f"no-alloc lse {call}")
    p.device_clean()


def test_noalloc_rejects_blocks_beyond_its_scratch(libcsr):
    """n = 513 at 64 query heads of 128 dims needs 8208 packed rows, more than
    the 8 MiB of query scratch (8192): CSR_EINVAL, nothing launched.  So are a
    NULL argument block and a misaligned query pointer."""
    csr, lib, fn = _noalloc()
    p = Pair(C2, pool_pages=64, max_seq=4096, max_new=512)
    p.init_static(p.blk(1320, 100), compare=False)
    stream = torch.cuda.current_stream()
    q = torch.zeros((520, p.hq, p.d), dtype=torch.bfloat16, device="cuda")
    kv = torch.zeros((520, p.hkv, p.d), dtype=torch.bfloat16, device="cuda")
    out = torch.empty_like(q)
    pt = ctypes.c_void_p()
    assert lib.csr_device_page_table(ctypes.c_void_p(p.ctx._h.value), 0, ctypes.byref(pt)) == 0

    def args(n, qptr=None):
        return BlockArgs(qptr if qptr is not None else q.data_ptr(), kv.data_ptr(), kv.data_ptr(),
                         p.ctx.k_pool.data_ptr(), p.ctx.v_pool.data_ptr(), pt.value, out.data_ptr(),
                         None, 0, n, p.hq, p.hkv, p.d, p.P, p.cfg.pool_pages, p.shape["base"], 0.0)
    assert fn(ctypes.byref(args(513)), stream.cuda_stream) == csr.EINVAL
    assert fn(ctypes.byref(args(4096)), stream.cuda_stream) == csr.EINVAL
    assert fn(ctypes.byref(args(16, q.data_ptr() + 2)), stream.cuda_stream) == csr.EINVAL
    assert fn(None, stream.cuda_stream) == csr.EINVAL
    torch.cuda.synchronize()
    p.device_clean()
