"""Thin ctypes binding of libdge.so (include/dge.h), with the same call names.

Argument marshalling only: every step of the pass runs in the library's CUDA
kernels.  PyTorch supplies device memory and the current stream.  The library
must have been built (``paper_2609_33334_gb300._build.build()``); loading fails
loudly otherwise -- there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
import threading
from ctypes import POINTER, c_float, c_int, c_int32, c_int64, c_size_t, c_void_p

from . import _build

DGE_OK = 0
DGE_ERR_INVALID_ARG = 1
DGE_ERR_UNSUPPORTED = 2
DGE_ERR_WORKSPACE_TOO_SMALL = 3
DGE_ERR_CUDA = 4
DGE_ERR_DEVICE_TIMEOUT = 5

DGE_VARIANT_SCORED, DGE_VARIANT_H2O, DGE_VARIANT_STREAMING = 0, 1, 2
DGE_POOL_NONE, DGE_POOL_MAX, DGE_POOL_AVG = 0, 1, 2


class dge_problem(ctypes.Structure):
    _fields_ = [("num_layers", c_int32), ("batch", c_int32), ("num_q_heads", c_int32),
                ("num_kv_heads", c_int32), ("head_dim", c_int32), ("obs_rows", c_int32),
                ("seq_len", c_int64), ("tail", c_int32), ("sinks", c_int32),
                ("variant", c_int32), ("pool", c_int32), ("pool_kernel", c_int32),
                ("scale", c_float), ("select_block", c_int32), ("budgets", POINTER(c_int32))]


class dge_tensor(ctypes.Structure):
    _fields_ = [("data", c_void_p), ("stride_layer", c_int64), ("stride_batch", c_int64),
                ("stride_head", c_int64), ("stride_pos", c_int64)]


class dge_paging(ctypes.Structure):
    _fields_ = [("block_table", c_void_p), ("page_size", c_int32), ("pages_per_seq", c_int32),
                ("num_pages", c_int32), ("reserved", c_int32), ("stride_page", c_int64)]


class dge_buffers(ctypes.Structure):
    _fields_ = [("K", dge_tensor), ("V", dge_tensor), ("Q", dge_tensor), ("scores", c_void_p),
                ("idx", c_void_p), ("Kc", c_void_p), ("Vc", c_void_p), ("lse_in", c_void_p),
                ("lse_out", c_void_p), ("paging", POINTER(dge_paging))]


class dge_diag(ctypes.Structure):
    _fields_ = [("evicted_mass", c_void_p), ("l_match", c_void_p), ("run_length", c_void_p),
                ("heldout_q", dge_tensor), ("heldout_mass", c_void_p), ("heldout_err", c_void_p),
                ("heldout_gap", c_void_p)]


class dge_kernel_time(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 48), ("launches", c_int64), ("total_ms", ctypes.c_double)]


class DgeError(RuntimeError):
    def __init__(self, call: str, code: int):
        lib = _lib()
        text = lib.dge_status_string(code).decode()
        detail = lib.dge_last_error().decode() if code == DGE_ERR_CUDA else ""
        super().__init__(f"{call} -> {code} ({text}){': ' + detail if detail else ''}")
        self.code = code


_LOCK = threading.Lock()
_LIB = None

_P = POINTER(dge_problem)
_B = POINTER(dge_buffers)
_T = POINTER(dge_tensor)
_G = POINTER(dge_paging)
_SIGS = {
    "dge_workspace_size": [_P, POINTER(c_size_t)],
    "dge_packed_rows": [_P, POINTER(c_int64)],
    "dge_score": [_P, _B, c_void_p, c_size_t, c_void_p],
    "dge_score_noalloc": [_P, _B, c_void_p],
    "dge_noalloc_status": [c_void_p],
    "dge_select": [_P, c_void_p, c_void_p, c_void_p],
    "dge_compact": [_P, c_void_p, _T, _T, c_void_p, c_void_p, c_void_p, c_void_p],
    "dge_evict": [_P, _B, c_void_p, c_size_t, c_void_p],
    "dge_evict_inplace": [_P, _B, c_void_p, c_size_t, c_void_p],
    "dge_diagnostics": [_P, _B, ctypes.POINTER(dge_diag), c_void_p, c_size_t, c_void_p],
    "dge_compact_inplace": [_P, c_void_p, _T, _T, c_void_p, c_void_p],
    "dge_compact_paged": [_P, _G, c_void_p, _T, _T, c_void_p, c_void_p, c_void_p, c_void_p],
    "dge_compact_inplace_paged": [_P, _G, c_void_p, _T, _T, c_void_p, c_void_p],
    "dge_pyramid_budgets": [c_int32, c_int32, c_int32, POINTER(c_int32)],
    "dge_get_device_status": [c_void_p, c_void_p],
    "dge_status_string": [c_int],
    "dge_last_error": [],
    "dge_profile_begin": [],
    "dge_trace_set": [c_void_p, c_size_t, c_int],
    "dge_debug_set_waits": [ctypes.c_uint64, c_int32],
    "dge_profile_end": [POINTER(dge_kernel_time), c_int, POINTER(c_int)],
}


def library_path() -> str:
    return _build.LIB


def _lib():
    global _LIB
    with _LOCK:
        if _LIB is None:
            path = library_path()
            if not os.path.exists(path):
                raise RuntimeError(
                    f"libdge.so not built at {path}: run paper_2609_33334_gb300._build.build()")
            lib = ctypes.CDLL(path)
            for name, args in _SIGS.items():
                fn = getattr(lib, name)
                fn.argtypes = args
                fn.restype = ctypes.c_char_p if name in ("dge_status_string",
                                                          "dge_last_error") else c_int
            _LIB = lib
    return _LIB


def _check(call: str, rc: int) -> None:
    if rc != DGE_OK:
        raise DgeError(call, rc)


# --- the ABI calls, one wrapper each -------------------------------------------------

def dge_workspace_size(p: dge_problem) -> int:
    out = c_size_t(0)
    _check("dge_workspace_size", _lib().dge_workspace_size(ctypes.byref(p), ctypes.byref(out)))
    return out.value


def dge_packed_rows(p: dge_problem) -> int:
    out = c_int64(0)
    _check("dge_packed_rows", _lib().dge_packed_rows(ctypes.byref(p), ctypes.byref(out)))
    return out.value


def dge_score(p: dge_problem, bufs: dge_buffers, ws: int, ws_bytes: int, stream: int) -> None:
    _check("dge_score", _lib().dge_score(ctypes.byref(p), ctypes.byref(bufs), ws, ws_bytes,
                                         stream))


def dge_score_noalloc(p: dge_problem, bufs: dge_buffers, stream: int) -> None:
    """dge_score with the library's built-in scratch (no workspace, nothing allocated)."""
    _check("dge_score_noalloc", _lib().dge_score_noalloc(ctypes.byref(p), ctypes.byref(bufs),
                                                         stream))


def dge_noalloc_status(stream: int) -> int:
    """Reads and clears the status word of dge_score_noalloc's built-in scratch."""
    return _lib().dge_noalloc_status(stream)


def dge_select(p: dge_problem, scores: int, idx: int, stream: int) -> None:
    _check("dge_select", _lib().dge_select(ctypes.byref(p), scores, idx, stream))


def dge_compact(p: dge_problem, idx: int, K: dge_tensor, V: dge_tensor, Kc: int, Vc: int,
                ws: int, stream: int) -> None:
    _check("dge_compact", _lib().dge_compact(ctypes.byref(p), idx, ctypes.byref(K),
                                             ctypes.byref(V), Kc, Vc, ws, stream))


def dge_diagnostics(p: dge_problem, bufs: dge_buffers, out: dge_diag, ws: int, ws_bytes: int,
                    stream: int) -> None:
    _check("dge_diagnostics", _lib().dge_diagnostics(ctypes.byref(p), ctypes.byref(bufs),
                                                     ctypes.byref(out), ws, ws_bytes, stream))


def dge_evict_inplace(p: dge_problem, bufs: dge_buffers, ws: int, ws_bytes: int,
                      stream: int) -> None:
    _check("dge_evict_inplace", _lib().dge_evict_inplace(ctypes.byref(p), ctypes.byref(bufs), ws,
                                                         ws_bytes, stream))


def dge_compact_inplace(p: dge_problem, idx: int, K: dge_tensor, V: dge_tensor, ws: int,
                        stream: int) -> None:
    _check("dge_compact_inplace", _lib().dge_compact_inplace(ctypes.byref(p), idx,
                                                             ctypes.byref(K), ctypes.byref(V),
                                                             ws, stream))


def dge_compact_paged(p: dge_problem, paging: dge_paging, idx: int, K: dge_tensor,
                      V: dge_tensor, Kc: int, Vc: int, ws: int, stream: int) -> None:
    _check("dge_compact_paged", _lib().dge_compact_paged(ctypes.byref(p), ctypes.byref(paging),
                                                         idx, ctypes.byref(K), ctypes.byref(V),
                                                         Kc, Vc, ws, stream))


def dge_compact_inplace_paged(p: dge_problem, paging: dge_paging, idx: int, K: dge_tensor,
                              V: dge_tensor, ws: int, stream: int) -> None:
    _check("dge_compact_inplace_paged",
           _lib().dge_compact_inplace_paged(ctypes.byref(p), ctypes.byref(paging), idx,
                                            ctypes.byref(K), ctypes.byref(V), ws, stream))


def dge_evict(p: dge_problem, bufs: dge_buffers, ws: int, ws_bytes: int, stream: int) -> None:
    _check("dge_evict", _lib().dge_evict(ctypes.byref(p), ctypes.byref(bufs), ws, ws_bytes,
                                         stream))


def dge_pyramid_budgets(B: int, w: int, L: int) -> list:
    out = (c_int32 * L)()
    _check("dge_pyramid_budgets", _lib().dge_pyramid_budgets(B, w, L, out))
    return list(out)


def dge_get_device_status(ws: int, stream: int) -> int:
    return _lib().dge_get_device_status(ws, stream)


def dge_status_string(code: int) -> str:
    return _lib().dge_status_string(code).decode()


def dge_last_error() -> str:
    return _lib().dge_last_error().decode()


def dge_profile_begin() -> None:
    _check("dge_profile_begin", _lib().dge_profile_begin())


def dge_profile_end(capacity: int = 32) -> list:
    """[(kernel name, launches, total device ms)] since dge_profile_begin()."""
    arr = (dge_kernel_time * capacity)()
    count = c_int(0)
    _check("dge_profile_end", _lib().dge_profile_end(arr, capacity, ctypes.byref(count)))
    return [(arr[i].name.decode(), arr[i].launches, arr[i].total_ms)
            for i in range(min(count.value, capacity))]


TRACE_SLOTS, TRACE_LEN = 24, 4096


def dge_debug_set_waits(limit_ns: int = 0, extra_chunks: int = 0) -> None:
    """Test hook: bound of the tcgen05 kernels' device-side waits (0 = default) and extra
    chunks the scoring kernel's unit-count wait expects (> 0: that wait runs out)."""
    _check("dge_debug_set_waits", _lib().dge_debug_set_waits(limit_ns, extra_chunks))


def dge_trace_set(buffer: int, nbytes: int, cta: int = 0) -> None:
    """Record per-tile clock stamps of one CTA of the tensor-core scoring kernel."""
    _check("dge_trace_set", _lib().dge_trace_set(buffer, nbytes, cta))


# --- marshalling helpers --------------------------------------------------------------

def make_problem(*, L, b, Hq, Hkv, d, n, m=0, tail=0, sinks=0, variant=DGE_VARIANT_SCORED,
                 pool=DGE_POOL_NONE, pool_kernel=1, scale=0.0, select_block=0,
                 budgets) -> dge_problem:
    """A dge_problem; keeps the budgets array alive on the returned object."""
    arr = (c_int32 * len(budgets))(*[int(x) for x in budgets])
    p = dge_problem(num_layers=L, batch=b, num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d,
                    obs_rows=m, seq_len=n, tail=tail, sinks=sinks, variant=variant, pool=pool,
                    pool_kernel=pool_kernel, scale=scale, select_block=select_block,
                    budgets=ctypes.cast(arr, POINTER(c_int32)))
    p._budgets_keepalive = arr
    return p


def tensor_desc(t) -> dge_tensor:
    """dge_tensor of a 5-D [layer][batch][head][pos][d] bf16 tensor (d contiguous)."""
    if t is None:
        return dge_tensor()
    if t.dim() != 5 or t.stride(-1) != 1:
        raise ValueError("expected a 5-D tensor with a contiguous last dim")
    s = t.stride()
    return dge_tensor(data=t.data_ptr(), stride_layer=s[0], stride_batch=s[1],
                      stride_head=s[2], stride_pos=s[3])


def ptr(t) -> int:
    return 0 if t is None else t.data_ptr()
