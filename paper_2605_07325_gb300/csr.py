"""Thin Python binding of libcsr (include/csr.h): argument marshalling only.

Every step of the attention path runs in the library's CUDA kernels; this
module allocates the caller-owned device buffers with PyTorch, passes raw
pointers and streams, and turns status codes into exceptions.  Importing it
fails loudly when libcsr.so has not been built (``python -m
paper_2605_07325_gb300.build``); there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
from typing import Callable, Dict, List, Optional, Tuple

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_lib", "libcsr.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"libcsr.so is not built ({LIB_PATH}); run "
                      "`python -m paper_2605_07325_gb300.build` (needs nvcc)")

_lib = ctypes.CDLL(LIB_PATH)

# status codes
OK, EINVAL, ENOMEM, ESTATE, EBUSY, ECUDA, ETIMEOUT, EDEVICE = range(8)
STATUS_NAMES = {0: "CSR_OK", 1: "CSR_EINVAL", 2: "CSR_ENOMEM", 3: "CSR_ESTATE", 4: "CSR_EBUSY",
                5: "CSR_ECUDA", 6: "CSR_ETIMEOUT", 7: "CSR_EDEVICE"}
DEVERR_WAIT_TIMEOUT, DEVERR_BAD_PAGE, DEVERR_ALLOC = 0x1, 0x2, 0x4
FLAG_PLAN_ONLY = 0x1
FLAG_FUSED_ALWAYS = 0x2
FLAG_FUSED_NEVER = 0x4
FLAG_UNPACED_REBUILD = 0x8
FLAG_SCHEDULE_LOCAL = 0x10
RECON_IDLE, RECON_RUNNING, RECON_SWAPPED = 0, 1, 2
ROUTE_CONTINUE, ROUTE_BRIDGE, ROUTE_SWAPPED, ROUTE_STRAGGLER = 0, 1, 2, 3
VERSION_ACTIVE, VERSION_PENDING = 0, 1


class Config(ctypes.Structure):
    _fields_ = [
        ("num_q_heads", ctypes.c_int32),
        ("num_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("page_size", ctypes.c_int32),
        ("rope_base", ctypes.c_double),
        ("softmax_scale", ctypes.c_float),
        ("max_new_tokens", ctypes.c_int32),
        ("pool_pages", ctypes.c_int32),
        ("max_seq_tokens", ctypes.c_int32),
        ("cap_tokens", ctypes.c_int32),
        ("evict_tokens", ctypes.c_int32),
        ("n_catchup", ctypes.c_int32),
        ("num_ctas", ctypes.c_int32),
        ("rebuild_tiles_per_cta", ctypes.c_int32),
        ("flags", ctypes.c_int32),
        ("fg_chunk_tiles", ctypes.c_int32),
        ("rebuild_duty", ctypes.c_float),
    ]


KERNEL_KINDS = ("rope_append", "attention", "merge", "evict_compact")


class Timing(ctypes.Structure):
    _fields_ = [("ms", ctypes.c_double * 4), ("launches", ctypes.c_int64 * 4)]


class Piece(ctypes.Structure):
    _fields_ = [("cta", ctypes.c_int32), ("order", ctypes.c_int32), ("unit", ctypes.c_int32),
                ("j0", ctypes.c_int32), ("j1", ctypes.c_int32), ("slot", ctypes.c_int32),
                ("merges", ctypes.c_int32), ("group", ctypes.c_int32), ("member", ctypes.c_int32)]


class Viability(ctypes.Structure):
    _fields_ = [("t_warm_s", ctypes.c_double), ("delta_n_tokens", ctypes.c_double),
                ("t_recon_s", ctypes.c_double), ("t_mem_s", ctypes.c_double),
                ("n_buffer_tokens", ctypes.c_double), ("rebuilt_tokens", ctypes.c_double),
                ("pair_seconds", ctypes.c_double), ("viable", ctypes.c_int32),
                ("measured", ctypes.c_int32)]


PROVIDER = ctypes.CFUNCTYPE(ctypes.c_int, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32,
                            ctypes.POINTER(ctypes.c_void_p), ctypes.POINTER(ctypes.c_void_p),
                            ctypes.POINTER(ctypes.c_void_p), ctypes.POINTER(ctypes.c_void_p))

_vp, _i32, _i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
_P32, _P64, _Pu32 = (ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int64),
                     ctypes.POINTER(ctypes.c_uint32))
_SIGS = {
    "csr_pool_bytes": ([ctypes.POINTER(Config)], ctypes.c_size_t),
    "csr_workspace_bytes": ([ctypes.POINTER(Config)], ctypes.c_size_t),
    "csr_create": ([ctypes.POINTER(Config), _vp, _vp, _vp, _vp, ctypes.POINTER(_vp)], ctypes.c_int),
    "csr_destroy": ([_vp], None),
    "csr_init_static": ([_vp, _vp, _vp, _vp, _i32, _vp, _vp, _vp], ctypes.c_int),
    "csr_append_chunk": ([_vp, _vp, _vp, _vp, _i32, _vp, _vp, _vp, _P64], ctypes.c_int),
    "csr_append_chunk_attend_suffix": ([_vp, _vp, _vp, _vp, _i32, _i32, _vp, _vp, _vp, _P64],
                                       ctypes.c_int),
    "csr_get_versions": ([_vp, _P64, _P64], ctypes.c_int),
    "csr_cancel_reconcile": ([_vp], ctypes.c_int),
    "csr_foreground_schedule": ([ctypes.POINTER(Config), _i64, _i32, _i32, ctypes.POINTER(Piece), _i32,
                                 _P32, _P32], ctypes.c_int),
    "csr_check_viability": ([_vp, _i32, ctypes.c_double, ctypes.c_double, ctypes.POINTER(Viability)],
                            ctypes.c_int),
    "csr_route": ([_vp, ctypes.c_int64, _vp, ctypes.POINTER(ctypes.c_int)], ctypes.c_int),
    "csr_attend_suffix": ([_vp, _vp, _vp, _vp, _i32, _vp, _vp, _vp], ctypes.c_int),
    "csr_truncate_suffix": ([_vp], ctypes.c_int),
    "csr_rewind": ([_vp, _i64], ctypes.c_int),
    "csr_set_reconciler": ([_vp, PROVIDER, _vp, _vp], ctypes.c_int),
    "csr_evict_and_reconcile": ([_vp, _i32, _vp], ctypes.c_int),
    "csr_poll_swap": ([_vp, _vp, ctypes.POINTER(ctypes.c_int)], ctypes.c_int),
    "csr_wait_reconcile": ([_vp, _vp, _i64, ctypes.POINTER(ctypes.c_int)], ctypes.c_int),
    "csr_get_layout": ([_vp, ctypes.c_int, _P32, _i32, _P32, _P64], ctypes.c_int),
    "csr_get_free_pages": ([_vp, _P32, _i32, _P32], ctypes.c_int),
    "csr_get_chunks": ([_vp, ctypes.c_int, _P64, _P32, _i32, _P32, _P64], ctypes.c_int),
    "csr_device_page_table": ([_vp, ctypes.c_int, ctypes.POINTER(_vp)], ctypes.c_int),
    "csr_gather_kv": ([_vp, ctypes.c_int, _i64, _i32, _vp, _vp, _vp], ctypes.c_int),
    "csr_device_status": ([_vp, _Pu32], ctypes.c_int),
    "csr_kernel_launches": ([_vp], ctypes.c_int64),
    "csr_last_error": ([_vp], ctypes.c_char_p),
    "csr_set_timing": ([_vp, ctypes.c_int], ctypes.c_int),
    "csr_get_timing": ([_vp, ctypes.POINTER(Timing)], ctypes.c_int),
}
for _name, (_args, _res) in _SIGS.items():
    _fn = getattr(_lib, _name)
    _fn.argtypes = _args
    _fn.restype = _res


class CsrError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


def make_config(num_q_heads, num_kv_heads, head_dim, page_size, rope_base, max_new_tokens,
                pool_pages, max_seq_tokens, softmax_scale=0.0, cap_tokens=0, evict_tokens=0,
                n_catchup=0, num_ctas=0, rebuild_tiles_per_cta=0, flags=0,
                fg_chunk_tiles=0, rebuild_duty=0.0) -> Config:
    return Config(num_q_heads, num_kv_heads, head_dim, page_size, float(rope_base),
                  float(softmax_scale), max_new_tokens, pool_pages, max_seq_tokens, cap_tokens,
                  evict_tokens, n_catchup, num_ctas, rebuild_tiles_per_cta, flags, fg_chunk_tiles,
                  float(rebuild_duty))


def foreground_schedule(cfg: Config, L: int, n: int, grid: int = 0):
    """Pieces (cta, order, unit, j0, j1, slot, merges, group, member) of a
    fused foreground call of n tokens over L cached, and the number of partial
    slots written."""
    cnt, slots = ctypes.c_int32(0), ctypes.c_int32(0)
    st = _lib.csr_foreground_schedule(ctypes.byref(cfg), int(L), int(n), int(grid), None, 0,
                                      ctypes.byref(cnt), ctypes.byref(slots))
    if st != 0:
        raise CsrError(st, "csr_foreground_schedule failed")
    arr = (Piece * max(1, cnt.value))()
    st = _lib.csr_foreground_schedule(ctypes.byref(cfg), int(L), int(n), int(grid), arr, cnt.value,
                                      ctypes.byref(cnt), ctypes.byref(slots))
    if st != 0:
        raise CsrError(st, "csr_foreground_schedule failed")
    return [tuple(getattr(arr[i], f) for f, _ in Piece._fields_) for i in range(cnt.value)], slots.value


def pool_bytes(cfg: Config) -> int:
    return int(_lib.csr_pool_bytes(ctypes.byref(cfg)))


def workspace_bytes(cfg: Config) -> int:
    return int(_lib.csr_workspace_bytes(ctypes.byref(cfg)))


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream_ptr(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


class Context:
    """One layer's CSR cache on the current CUDA device (see include/csr.h)."""

    def __init__(self, cfg: Config, device: str = "cuda", stream=None):
        self.cfg = cfg
        self.plan_only = bool(cfg.flags & FLAG_PLAN_ONLY)
        self._h = ctypes.c_void_p()
        self._keep: Dict[int, tuple] = {}
        self._provider_cb = None
        if self.plan_only:
            self.k_pool = self.v_pool = self.workspace = None
            st = _lib.csr_create(ctypes.byref(cfg), None, None, None, None, ctypes.byref(self._h))
        else:
            pb, wb = pool_bytes(cfg), workspace_bytes(cfg)
            if pb == 0 or wb == 0:
                raise CsrError(EINVAL, "invalid configuration")
            self.device = torch.device(device)
            self.k_pool = torch.empty(pb, dtype=torch.uint8, device=self.device)
            self.v_pool = torch.empty(pb, dtype=torch.uint8, device=self.device)
            self.workspace = torch.empty(wb, dtype=torch.uint8, device=self.device)
            with torch.cuda.device(self.device):
                st = _lib.csr_create(ctypes.byref(cfg), self.k_pool.data_ptr(),
                                     self.v_pool.data_ptr(), self.workspace.data_ptr(),
                                     _stream_ptr(stream), ctypes.byref(self._h))
        if st != OK:
            raise CsrError(st, "csr_create failed")

    # ------------------------------------------------------------------ util
    def _check(self, st: int) -> None:
        if st != OK:
            raise CsrError(st, _lib.csr_last_error(self._h).decode())

    def close(self) -> None:
        if self._h:
            _lib.csr_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):  # pragma: no cover
        try:
            self.close()
        except Exception:
            pass

    def _io(self, q, k, v, out, lse):
        c = self.cfg
        if self.plan_only:
            return q, out, lse
        n = q.shape[0]
        for t, h in ((q, c.num_q_heads), (k, c.num_kv_heads), (v, c.num_kv_heads)):
            if (t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous()
                    or tuple(t.shape) != (n, h, c.head_dim)):
                raise CsrError(EINVAL, "q/k/v must be contiguous CUDA bf16 [n][heads][head_dim]")
        if out is None:
            out = torch.empty((n, c.num_q_heads, c.head_dim), dtype=torch.bfloat16, device=q.device)
        return q, out, lse

    # ---------------------------------------------------------- compute calls
    def init_static(self, q, k, v, out=None, lse=None, stream=None, n=None):
        q, out, lse = self._io(q, k, v, out, lse)
        n = q.shape[0] if n is None else n
        self._check(_lib.csr_init_static(self._h, _ptr(q), _ptr(k), _ptr(v), n, _ptr(out),
                                         _ptr(lse), _stream_ptr_opt(self, stream)))
        return out, lse

    def append_chunk(self, q, k, v, out=None, lse=None, stream=None, n=None):
        q, out, lse = self._io(q, k, v, out, lse)
        n = q.shape[0] if n is None else n
        cid = ctypes.c_int64(-1)
        self._check(_lib.csr_append_chunk(self._h, _ptr(q), _ptr(k), _ptr(v), n, _ptr(out),
                                          _ptr(lse), _stream_ptr_opt(self, stream),
                                          ctypes.byref(cid)))
        return out, lse, cid.value

    def append_chunk_attend_suffix(self, q, k, v, n_chunk, out=None, lse=None, stream=None,
                                   n=None):
        """One step: the first n_chunk tokens join the cache as a chunk, the rest
        are a live suffix (truncate it with truncate_suffix)."""
        q, out, lse = self._io(q, k, v, out, lse)
        n = q.shape[0] if n is None else n
        cid = ctypes.c_int64(-1)
        self._check(_lib.csr_append_chunk_attend_suffix(
            self._h, _ptr(q), _ptr(k), _ptr(v), int(n_chunk), int(n - n_chunk), _ptr(out),
            _ptr(lse), _stream_ptr_opt(self, stream), ctypes.byref(cid)))
        return out, lse, cid.value

    def attend_suffix(self, q, k, v, out=None, lse=None, stream=None, n=None):
        q, out, lse = self._io(q, k, v, out, lse)
        n = q.shape[0] if n is None else n
        self._check(_lib.csr_attend_suffix(self._h, _ptr(q), _ptr(k), _ptr(v), n, _ptr(out),
                                           _ptr(lse), _stream_ptr_opt(self, stream)))
        return out, lse

    def truncate_suffix(self) -> None:
        self._check(_lib.csr_truncate_suffix(self._h))

    def rewind(self, length: int) -> None:
        """Keep the first `length` tokens (a prefix or chunk boundary)."""
        self._check(_lib.csr_rewind(self._h, int(length)))

    # -------------------------------------------------------- reconciliation
    def set_reconciler(self, provider: Callable[[int, int], tuple], lo_stream=None) -> None:
        """provider(chunk_id, n_tokens) -> (q, k, v, out_or_None) device tensors."""
        keep = self._keep

        def _cb(user, chunk_id, n_tokens, pq, pk, pv, pout):
            try:
                res = provider(int(chunk_id), int(n_tokens))
                q, k, v = res[0], res[1], res[2]
                out = res[3] if len(res) > 3 else None
                keep[int(chunk_id)] = (q, k, v, out)
                pq[0], pk[0], pv[0] = _ptr(q), _ptr(k), _ptr(v)
                pout[0] = _ptr(out)
                return 0
            except Exception:  # any failure aborts the reconciliation
                return 1

        self._provider_cb = PROVIDER(_cb)
        lo = None if self.plan_only else _stream_ptr(lo_stream)
        self._check(_lib.csr_set_reconciler(self._h, self._provider_cb, None, lo))

    def evict_and_reconcile(self, evict_tokens: int, stream=None) -> None:
        self._check(_lib.csr_evict_and_reconcile(self._h, evict_tokens,
                                                 _stream_ptr_opt(self, stream)))

    def poll_swap(self, stream=None) -> int:
        st = ctypes.c_int(0)
        self._check(_lib.csr_poll_swap(self._h, _stream_ptr_opt(self, stream), ctypes.byref(st)))
        if st.value == RECON_SWAPPED:
            self._keep.clear()
        return st.value

    def wait_reconcile(self, timeout_s: float = 60.0, stream=None) -> int:
        st = ctypes.c_int(0)
        self._check(_lib.csr_wait_reconcile(self._h, _stream_ptr_opt(self, stream),
                                            int(timeout_s * 1e6), ctypes.byref(st)))
        if st.value == RECON_SWAPPED:
            self._keep.clear()
        return st.value

    def cancel_reconcile(self) -> None:
        """Abandon the running reconciliation; the active version stays."""
        self._check(_lib.csr_cancel_reconcile(self._h))
        self._keep.clear()

    def check_viability(self, evict_tokens: int, append_tokens_per_s: float,
                        pair_seconds: float = 0.0) -> Dict[str, float]:
        """App. D viability of an eviction of evict_tokens started now
        (csr_check_viability); pair_seconds <= 0 uses the observed rebuild pace."""
        v = Viability()
        self._check(_lib.csr_check_viability(self._h, int(evict_tokens), float(append_tokens_per_s),
                                             float(pair_seconds), ctypes.byref(v)))
        return {name: getattr(v, name) for name, _ in Viability._fields_}

    def versions(self) -> Tuple[int, int]:
        """(k, k_ready) of Algorithm 2."""
        k, kr = ctypes.c_int64(0), ctypes.c_int64(0)
        self._check(_lib.csr_get_versions(self._h, ctypes.byref(k), ctypes.byref(kr)))
        return k.value, kr.value

    def route(self, k_t: int, stream=None) -> int:
        """Algorithm 2's routing of a query built on version k_t (ROUTE_*)."""
        r = ctypes.c_int(0)
        self._check(_lib.csr_route(self._h, int(k_t), _stream_ptr_opt(self, stream), ctypes.byref(r)))
        if r.value == ROUTE_SWAPPED:
            self._keep.clear()
        return r.value

    # ------------------------------------------------------------ inspection
    def layout(self, which: int = VERSION_ACTIVE) -> Tuple[List[int], int]:
        npg, length = ctypes.c_int32(0), ctypes.c_int64(0)
        self._check(_lib.csr_get_layout(self._h, which, None, 0, ctypes.byref(npg),
                                        ctypes.byref(length)))
        arr = (ctypes.c_int32 * max(1, npg.value))()
        self._check(_lib.csr_get_layout(self._h, which, arr, npg.value, ctypes.byref(npg),
                                        ctypes.byref(length)))
        return list(arr[:npg.value]), int(length.value)

    def free_pages(self) -> List[int]:
        cnt = ctypes.c_int32(0)
        self._check(_lib.csr_get_free_pages(self._h, None, 0, ctypes.byref(cnt)))
        arr = (ctypes.c_int32 * max(1, cnt.value))()
        self._check(_lib.csr_get_free_pages(self._h, arr, cnt.value, ctypes.byref(cnt)))
        return list(arr[:cnt.value])

    def chunks(self, which: int = VERSION_ACTIVE):
        cnt, pre = ctypes.c_int32(0), ctypes.c_int64(0)
        self._check(_lib.csr_get_chunks(self._h, which, None, None, 0, ctypes.byref(cnt),
                                        ctypes.byref(pre)))
        ids = (ctypes.c_int64 * max(1, cnt.value))()
        lens = (ctypes.c_int32 * max(1, cnt.value))()
        self._check(_lib.csr_get_chunks(self._h, which, ids, lens, cnt.value, ctypes.byref(cnt),
                                        ctypes.byref(pre)))
        return list(ids[:cnt.value]), list(lens[:cnt.value]), int(pre.value)

    def device_page_table(self, which: int = VERSION_ACTIVE) -> torch.Tensor:
        """Host copy of the version's device page table (synchronises)."""
        pt, _ = self.layout(which)
        p = ctypes.c_void_p()
        self._check(_lib.csr_device_page_table(self._h, which, ctypes.byref(p)))
        torch.cuda.synchronize()
        if not pt:
            return torch.empty(0, dtype=torch.int32)
        return _alias_int32(p.value, len(pt), self.device).cpu().clone()

    def gather_kv(self, which: int, pos0: int, n: int, stream=None):
        c = self.cfg
        k = torch.empty((n, c.num_kv_heads, c.head_dim), dtype=torch.bfloat16, device=self.device)
        v = torch.empty_like(k)
        self._check(_lib.csr_gather_kv(self._h, which, pos0, n, k.data_ptr(), v.data_ptr(),
                                       _stream_ptr(stream)))
        return k, v

    def device_status(self) -> int:
        flags = ctypes.c_uint32(0)
        st = _lib.csr_device_status(self._h, ctypes.byref(flags))
        if st not in (OK, EDEVICE):
            self._check(st)
        return int(flags.value)

    def kernel_launches(self) -> int:
        return int(_lib.csr_kernel_launches(self._h))

    def set_timing(self, enable: bool) -> None:
        self._check(_lib.csr_set_timing(self._h, 1 if enable else 0))

    def get_timing(self) -> Dict[str, Tuple[float, int]]:
        """{kernel: (summed ms, launches)} of the foreground launches timed so far."""
        t = Timing()
        self._check(_lib.csr_get_timing(self._h, ctypes.byref(t)))
        return {k: (t.ms[i], int(t.launches[i])) for i, k in enumerate(KERNEL_KINDS)}

    def last_error(self) -> str:
        return _lib.csr_last_error(self._h).decode()


def _stream_ptr_opt(ctx: Context, stream):
    return None if ctx.plan_only else _stream_ptr(stream)


def _alias_int32(ptr: int, n: int, device) -> torch.Tensor:
    """An int32 CUDA tensor viewing n entries of raw device memory (no ownership)."""

    class _Holder:
        __cuda_array_interface__ = {"shape": (n,), "typestr": "<i4", "data": (ptr, False),
                                    "version": 3, "strides": None}
    return torch.as_tensor(_Holder(), device=device)
