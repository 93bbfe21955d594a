"""The C ABI on a machine without a GPU: exports, host-only calls, validation.

Validation errors are returned before anything is enqueued, so every call
here is safe without a device.
"""
import ctypes
import os
import re

import pytest

from paper_2609_33334_gb300 import _build, binding as B
from paper_2609_33334_gb300 import inputs
from paper_2609_33334_gb300.api import problem_from_workload

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "dge.h")


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return B._lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(dge_\w+)\s*\(", text, re.M)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for want in ("dge_score", "dge_select", "dge_compact", "dge_evict", "dge_workspace_size",
                 "dge_pyramid_budgets", "dge_get_device_status", "dge_status_string"):
        assert want in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert name in B._SIGS, f"binding lacks {name}"


def declared_signature(name):
    """Parameter names of `name` as include/dge.h declares it."""
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    m = re.search(r"\b" + name + r"\s*\(([^)]*)\)\s*;", text)
    assert m, name
    params = [x.strip() for x in m.group(1).split(",") if x.strip() and x.strip() != "void"]
    return [re.findall(r"(\w+)\s*$", x)[0] for x in params]


# The boundary's calls with their parameters.  The scope table's boundary row lists
# dge_select(p, scores, idx, ws, ws_bytes, stream) and dge_compact(p, idx, K, V, Kc, Vc,
# stream); the library departs from it in two places, on purpose: dge_select takes no
# workspace (the selection needs no device scratch and reports no device status), and
# dge_compact takes an optional workspace whose status word receives out-of-range index
# reports (NULL skips them).  Every other call matches the table.
BOUNDARY = {
    "dge_workspace_size": ["p", "bytes"],
    "dge_score": ["p", "bufs", "ws", "ws_bytes", "stream"],
    "dge_select": ["p", "scores", "idx", "stream"],
    "dge_compact": ["p", "idx", "K", "V", "Kc", "Vc", "ws", "stream"],
    "dge_evict": ["p", "bufs", "ws", "ws_bytes", "stream"],
    "dge_pyramid_budgets": ["B", "w", "L", "out"],
    "dge_get_device_status": ["ws", "stream"],
    "dge_status_string": ["code"],
}


@pytest.mark.parametrize("name", sorted(BOUNDARY))
def test_boundary_signatures(name):
    assert declared_signature(name) == BOUNDARY[name]
    assert len(B._SIGS[name]) == len(BOUNDARY[name])


def test_struct_layout_matches_c():
    # int32 x6, int64, int32 x5, float, int32, pointer
    assert ctypes.sizeof(B.dge_problem) == 72
    assert B.dge_problem.seq_len.offset == 24
    assert B.dge_problem.select_block.offset == 56
    assert B.dge_problem.budgets.offset == 64
    assert ctypes.sizeof(B.dge_tensor) == 40
    assert ctypes.sizeof(B.dge_buffers) == 3 * 40 + 7 * 8
    assert B.dge_buffers.lse_in.offset == 3 * 40 + 4 * 8
    assert B.dge_buffers.lse_out.offset == 3 * 40 + 5 * 8
    assert B.dge_buffers.paging.offset == 3 * 40 + 6 * 8
    assert ctypes.sizeof(B.dge_paging) == 32
    assert B.dge_paging.stride_page.offset == 24


def test_pyramid_budgets_paper_examples(lib):
    """App. L worked examples, through the library's own host routine."""
    assert B.dge_pyramid_budgets(64, 8, 28)[-4:] == [14, 10, 6, 2]
    assert B.dge_pyramid_budgets(32, 8, 28)[-4:] == [23, 22, 21, 20]
    assert set(B.dge_pyramid_budgets(32, 8, 48)) == {47}
    assert B.dge_pyramid_budgets(64, 8, 48)[-1] == 16
    assert B.dge_pyramid_budgets(64, 8, 32)[-1] == 17
    with pytest.raises(B.DgeError):
        B.dge_pyramid_budgets(8, 8, 32)


def test_status_strings(lib):
    for code in range(6):
        assert B.dge_status_string(code)
    assert "unknown" in B.dge_status_string(99)


@pytest.mark.parametrize("name", list(inputs.WORKLOADS))
def test_packed_rows_and_workspace(lib, name):
    wl = inputs.WORKLOADS[name]
    p = problem_from_workload(wl)
    assert p.packed_rows() == wl.b * wl.Hkv * sum(wl.budgets)
    ws = p.workspace_bytes()
    assert ws >= 256 and ws % 256 == 0
    if wl.variant != inputs.STREAMING:
        # at least the raw scores of every unit
        assert ws >= p.U * p.P * 4


@pytest.mark.parametrize("n", [80, 127, 128, 129, 1000, 3000, 5000, 8192, 32768, 131072])
@pytest.mark.parametrize("G,m", [(4, 34), (8, 66)])   # whole units (R = 136); 4 row blocks
def test_workspace_for_cache_lengths_and_row_blocks(lib, n, G, m):
    """The scoring plan (key chunks of the tensor-core kernel, row blocks) is computed on the
    host for every problem: every cache length from below one key tile up to 128K keys gives a
    valid workspace size, with room for the raw scores and the fixed-point row-block sums."""
    p = _problem(Hq=8 * G, Hkv=8, d=128, n=n, m=m, tail=m, budgets=[min(n, 2 * m)])
    ws = ctypes.c_size_t(0)
    assert lib.dge_workspace_size(ctypes.byref(p), ctypes.byref(ws)) == 0
    U, P = 8, n - m
    need = U * P * 4 * (3 if G == 8 else 1)   # raw scores (+ 8-byte fixed-point sums)
    assert ws.value >= need and ws.value % 256 == 0


def _problem(**kw):
    base = dict(L=1, b=1, Hq=8, Hkv=2, d=64, n=1024, m=10, tail=10, sinks=0,
                variant=B.DGE_VARIANT_SCORED, pool=B.DGE_POOL_MAX, pool_kernel=7,
                budgets=[128])
    base.update(kw)
    return B.make_problem(**base)


@pytest.mark.parametrize("kw,code", [
    (dict(Hq=6, Hkv=4), B.DGE_ERR_INVALID_ARG),             # Hq % Hkv != 0
    (dict(d=96), B.DGE_ERR_UNSUPPORTED),                     # head_dim
    (dict(n=0), B.DGE_ERR_INVALID_ARG),
    (dict(m=0), B.DGE_ERR_INVALID_ARG),
    (dict(pool_kernel=6), B.DGE_ERR_INVALID_ARG),            # even pooling kernel
    (dict(pool=7), B.DGE_ERR_INVALID_ARG),
    (dict(budgets=[9]), B.DGE_ERR_INVALID_ARG),              # B < tail
    (dict(budgets=[2000]), B.DGE_ERR_INVALID_ARG),           # B > n
    (dict(tail=1025), B.DGE_ERR_INVALID_ARG),
    (dict(m=100, Hq=64, Hkv=8), B.DGE_ERR_UNSUPPORTED),      # R = 800 rows > on-chip limit
    (dict(variant=5), B.DGE_ERR_INVALID_ARG),
    (dict(select_block=65), B.DGE_ERR_INVALID_ARG),
    (dict(select_block=-1), B.DGE_ERR_INVALID_ARG),
    (dict(n=100000, select_block=2, budgets=[128]), B.DGE_ERR_UNSUPPORTED),   # > 16384 blocks
    (dict(L=300, budgets=[128] * 300), B.DGE_ERR_INVALID_ARG),
])
def test_problem_validation(lib, kw, code):
    p = _problem(**kw)
    n = ctypes.c_size_t(0)
    assert lib.dge_workspace_size(ctypes.byref(p), ctypes.byref(n)) == code


def test_null_and_misaligned_arguments_rejected_before_launch(lib):
    p = _problem()
    assert lib.dge_evict(None, None, None, 0, None) == B.DGE_ERR_INVALID_ARG
    assert lib.dge_evict(ctypes.byref(p), None, None, 0, None) == B.DGE_ERR_INVALID_ARG
    t = B.dge_tensor(data=0x1000, stride_layer=1024 * 64 * 2, stride_batch=1024 * 64 * 2,
                     stride_head=1024 * 64, stride_pos=64)
    bad = B.dge_tensor(data=0x1008, stride_layer=0, stride_batch=0, stride_head=0, stride_pos=64)
    bufs = B.dge_buffers(K=t, V=t, Q=t, scores=0, idx=0x2000, Kc=0x3000, Vc=0x4000)
    need = ctypes.c_size_t(0)
    assert lib.dge_workspace_size(ctypes.byref(p), ctypes.byref(need)) == 0
    # workspace missing / misaligned / too small
    assert lib.dge_evict(ctypes.byref(p), ctypes.byref(bufs), None, 0, None) == \
        B.DGE_ERR_INVALID_ARG
    assert lib.dge_evict(ctypes.byref(p), ctypes.byref(bufs), 0x10010, need.value, None) == \
        B.DGE_ERR_UNSUPPORTED
    assert lib.dge_evict(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value - 1, None) == \
        B.DGE_ERR_WORKSPACE_TOO_SMALL
    # misaligned K
    bufs.K = bad
    assert lib.dge_evict(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value, None) == \
        B.DGE_ERR_UNSUPPORTED
    # stride not a multiple of 8 elements
    bufs.K = B.dge_tensor(data=0x1000, stride_layer=0, stride_batch=0, stride_head=0,
                          stride_pos=60)
    assert lib.dge_evict(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value, None) == \
        B.DGE_ERR_UNSUPPORTED
    # dge_score needs a scores buffer; STREAMING has no scores
    bufs.K = t
    assert lib.dge_score(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value, None) == \
        B.DGE_ERR_INVALID_ARG
    ps = _problem(variant=B.DGE_VARIANT_STREAMING, sinks=4)
    bufs.scores = 0x5000
    assert lib.dge_score(ctypes.byref(ps), ctypes.byref(bufs), 0x10000, need.value, None) == \
        B.DGE_ERR_INVALID_ARG
    # misaligned row normalisers (supplied or requested)
    bufs.lse_in = 0x6002
    assert lib.dge_score(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value, None) == \
        B.DGE_ERR_UNSUPPORTED
    assert lib.dge_evict(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value, None) == \
        B.DGE_ERR_UNSUPPORTED
    bufs.lse_in = 0
    bufs.lse_out = 0x6001
    assert lib.dge_evict(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value, None) == \
        B.DGE_ERR_UNSUPPORTED
    bufs.lse_out = 0
    assert lib.dge_select(ctypes.byref(p), None, 0x2000, None) == B.DGE_ERR_INVALID_ARG
    assert lib.dge_compact(ctypes.byref(p), None, None, None, 0, 0, None, None) == \
        B.DGE_ERR_INVALID_ARG
    assert lib.dge_get_device_status(None, None) == B.DGE_ERR_INVALID_ARG
    # in place: no Kc / Vc needed, idx still required and aligned
    bufs.Kc = bufs.Vc = 0
    assert lib.dge_evict(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value, None) == \
        B.DGE_ERR_INVALID_ARG
    bufs.idx = 0
    assert lib.dge_evict_inplace(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value,
                                 None) == B.DGE_ERR_INVALID_ARG
    bufs.idx = 0x2002
    assert lib.dge_evict_inplace(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value,
                                 None) == B.DGE_ERR_UNSUPPORTED
    assert lib.dge_compact_inplace(ctypes.byref(p), None, ctypes.byref(t), ctypes.byref(t), None,
                                   None) == B.DGE_ERR_INVALID_ARG
    assert lib.dge_compact_inplace(ctypes.byref(p), 0x2002, ctypes.byref(t), ctypes.byref(t),
                                   None, None) == B.DGE_ERR_UNSUPPORTED


@pytest.mark.parametrize("kw,code", [
    (dict(block_table=0), B.DGE_ERR_INVALID_ARG),
    (dict(page_size=8), B.DGE_ERR_UNSUPPORTED),            # a 128-key tile would span 16 pages
    (dict(page_size=48), B.DGE_ERR_UNSUPPORTED),
    (dict(page_size=192), B.DGE_ERR_UNSUPPORTED),
    (dict(pages_per_seq=63), B.DGE_ERR_INVALID_ARG),       # 63 * 16 < n = 1024
    (dict(num_pages=0), B.DGE_ERR_INVALID_ARG),
    (dict(reserved=1), B.DGE_ERR_INVALID_ARG),
    (dict(stride_page=0), B.DGE_ERR_INVALID_ARG),
    (dict(stride_page=12), B.DGE_ERR_UNSUPPORTED),
    (dict(block_table=0x7002), B.DGE_ERR_UNSUPPORTED),     # misaligned table
])
def test_paging_validation(lib, kw, code):
    """Bad paged-cache geometry is rejected before anything is enqueued, by every call that
    takes K / V."""
    p = _problem()
    base = dict(block_table=0x7000, page_size=16, pages_per_seq=64, num_pages=200,
                reserved=0, stride_page=16 * 2 * 64)
    base.update(kw)
    pg = B.dge_paging(**base)
    t = B.dge_tensor(data=0x1000, stride_layer=200 * 16 * 2 * 64, stride_batch=0,
                     stride_head=64, stride_pos=2 * 64)
    bufs = B.dge_buffers(K=t, V=t, Q=t, scores=0x5000, idx=0x2000, Kc=0x3000, Vc=0x4000,
                         paging=ctypes.pointer(pg))
    need = ctypes.c_size_t(0)
    assert lib.dge_workspace_size(ctypes.byref(p), ctypes.byref(need)) == 0
    assert lib.dge_evict(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value, None) == code
    assert lib.dge_evict_inplace(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value,
                                 None) == code
    assert lib.dge_score(ctypes.byref(p), ctypes.byref(bufs), 0x10000, need.value, None) == code
    assert lib.dge_compact_paged(ctypes.byref(p), ctypes.byref(pg), 0x2000, ctypes.byref(t),
                                 ctypes.byref(t), 0x3000, 0x4000, None, None) == code
    assert lib.dge_compact_inplace_paged(ctypes.byref(p), ctypes.byref(pg), 0x2000,
                                         ctypes.byref(t), ctypes.byref(t), None, None) == code
