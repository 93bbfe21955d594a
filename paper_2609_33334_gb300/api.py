"""Public Python entry points: allocate outputs with PyTorch, call the C ABI.

Every function here marshals arguments and calls libdge; the computation runs
in the library's CUDA kernels on the tensors' device and the current stream.
"""
from __future__ import annotations

import ctypes
import dataclasses
from typing import Optional, Sequence

import torch

from . import binding as B


@dataclasses.dataclass
class Problem:
    """Shape and policy of one eviction pass (mirrors dge_problem)."""

    L: int
    b: int
    Hq: int
    Hkv: int
    d: int
    n: int
    budgets: Sequence[int]
    m: int = 0
    tail: int = 0
    sinks: int = 0
    variant: int = B.DGE_VARIANT_SCORED
    pool: int = B.DGE_POOL_NONE
    pool_kernel: int = 1
    scale: float = 0.0
    select_block: int = 0

    def c(self) -> B.dge_problem:
        return B.make_problem(L=self.L, b=self.b, Hq=self.Hq, Hkv=self.Hkv, d=self.d, n=self.n,
                              m=self.m, tail=self.tail, sinks=self.sinks, variant=self.variant,
                              pool=self.pool, pool_kernel=self.pool_kernel, scale=self.scale,
                              select_block=self.select_block, budgets=self.budgets)

    @property
    def U(self) -> int:
        return self.L * self.b * self.Hkv

    @property
    def P(self) -> int:
        return self.n if self.variant == B.DGE_VARIANT_STREAMING else self.n - self.tail

    def packed_rows(self) -> int:
        return B.dge_packed_rows(self.c())

    @property
    def lse_shape(self) -> tuple:
        """Layout of the row normalisers (dge_buffers.lse_in / lse_out): [L][b][Hq][rows]."""
        rows = self.n if self.variant == B.DGE_VARIANT_H2O else self.m
        return (self.L, self.b, self.Hq, rows)

    def workspace_bytes(self) -> int:
        return B.dge_workspace_size(self.c())

    def unit_row_offsets(self) -> list:
        """First packed row of every unit, in unit order (layer, batch, kv head)."""
        offs, acc = [], 0
        for l in range(self.L):
            for _ in range(self.b * self.Hkv):
                offs.append(acc)
                acc += self.budgets[l]
        return offs


@dataclasses.dataclass
class Paging:
    """A paged cache (dge_paging): K and V are then pools [L][num_pages][page_size][Hkv][d]
    (``head_major``: [L][num_pages][Hkv][page_size][d]) and position p of sequence b lives in
    slot p % page_size of page block_table[b, p // page_size] (int32 [b][pages_per_seq] on the
    device)."""

    block_table: torch.Tensor
    page_size: int
    head_major: bool = False

    def c(self, pool: torch.Tensor) -> B.dge_paging:
        bt = self.block_table
        if bt.dtype != torch.int32 or not bt.is_contiguous() or bt.dim() != 2:
            raise ValueError("block_table must be a contiguous int32 [b][pages_per_seq] tensor")
        if pool.dim() != 5 or pool.shape[3 if self.head_major else 2] != self.page_size:
            raise ValueError("paged K / V must be [L][num_pages][page_size][Hkv][d] "
                             "([L][num_pages][Hkv][page_size][d] when head_major)")
        return B.dge_paging(block_table=bt.data_ptr(), page_size=self.page_size,
                            pages_per_seq=bt.shape[1], num_pages=pool.shape[1],
                            stride_page=pool.stride(1))


def _kv_desc(t: torch.Tensor, paging: Optional[Paging]) -> B.dge_tensor:
    if paging is None:
        return B.tensor_desc(t)
    if t.dim() != 5 or t.stride(-1) != 1:
        raise ValueError("expected a 5-D pool with a contiguous last dim")
    s = t.stride()   # [L][page][slot][head][d], or [L][page][head][slot][d] when head-major
    head, slot = (s[2], s[3]) if paging.head_major else (s[3], s[2])
    return B.dge_tensor(data=t.data_ptr(), stride_layer=s[0], stride_batch=0,
                        stride_head=head, stride_pos=slot)


def _paging_ptr(paging: Optional[Paging], pool: torch.Tensor):
    if paging is None:
        return None, None
    c = paging.c(pool)
    return c, ctypes.pointer(c)


def problem_from_workload(wl) -> Problem:
    """The Problem of a synthetic workload (``inputs.Workload``)."""
    return Problem(L=wl.L, b=wl.b, Hq=wl.Hq, Hkv=wl.Hkv, d=wl.d, n=wl.n, budgets=wl.budgets,
                   m=wl.m, tail=wl.tail, sinks=wl.sinks, variant=wl.variant, pool=wl.pool,
                   pool_kernel=wl.pool_kernel)


def _stream(stream: Optional[torch.cuda.Stream]) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def workspace(p: Problem, device) -> torch.Tensor:
    """A device workspace of dge_workspace_size() bytes (256-byte aligned)."""
    nbytes = max(p.workspace_bytes(), 256)
    ws = torch.empty(nbytes + 256, dtype=torch.uint8, device=device)
    off = (-ws.data_ptr()) % 256
    return ws[off:off + nbytes]


def _check_cache(t: torch.Tensor, name: str) -> None:
    if t.dtype != torch.bfloat16 or not t.is_cuda:
        raise ValueError(f"{name} must be a bf16 CUDA tensor")


def _lse_arg(p: Problem, lse_in: Optional[torch.Tensor]) -> int:
    if lse_in is None:
        return 0
    if lse_in.dtype != torch.float32 or not lse_in.is_contiguous() or \
            tuple(lse_in.shape) != p.lse_shape:
        raise ValueError(f"lse_in must be contiguous float32 of shape {p.lse_shape}")
    return lse_in.data_ptr()


def evict(p: Problem, K: torch.Tensor, V: torch.Tensor, Q: Optional[torch.Tensor] = None, *,
          want_scores: bool = False, lse_in: Optional[torch.Tensor] = None,
          want_lse: bool = False, ws: Optional[torch.Tensor] = None,
          out: Optional[dict] = None, paging: Optional[Paging] = None, stream=None) -> dict:
    """dge_evict: the fused score -> pool -> select -> compact pass.

    Returns {"idx", "Kc", "Vc", "scores", "lse"} (scores / lse are None unless requested).
    ``lse_in``: the rows' natural-log normalisers [L][b][Hq][rows] (Problem.lse_shape), so the
    scoring reads K once; ``want_lse``: return the normalisers the scoring computed.
    ``out`` may hold preallocated outputs with those keys.  ``paging``: K and V are the pools
    of a paged cache (see Paging).
    """
    _check_cache(K, "K")
    _check_cache(V, "V")
    dev = K.device
    rows = p.packed_rows()
    o = dict(out or {})
    if o.get("idx") is None:
        o["idx"] = torch.empty(rows, dtype=torch.int32, device=dev)
    if o.get("Kc") is None:
        o["Kc"] = torch.empty((rows, p.d), dtype=torch.bfloat16, device=dev)
    if o.get("Vc") is None:
        o["Vc"] = torch.empty((rows, p.d), dtype=torch.bfloat16, device=dev)
    if want_scores and o.get("scores") is None:
        o["scores"] = torch.empty((p.U, p.P), dtype=torch.float32, device=dev)
    o.setdefault("scores", None)
    if want_lse and lse_in is None and o.get("lse") is None:
        o["lse"] = torch.empty(p.lse_shape, dtype=torch.float32, device=dev)
    o.setdefault("lse", None)
    if ws is None:
        ws = workspace(p, dev)
    pg, pg_ptr = _paging_ptr(paging, K)
    bufs = B.dge_buffers(K=_kv_desc(K, paging), V=_kv_desc(V, paging), Q=B.tensor_desc(Q),
                         scores=B.ptr(o["scores"]), idx=B.ptr(o["idx"]), Kc=B.ptr(o["Kc"]),
                         Vc=B.ptr(o["Vc"]), lse_in=_lse_arg(p, lse_in),
                         lse_out=B.ptr(o["lse"]) if want_lse and lse_in is None else 0,
                         paging=pg_ptr)
    B.dge_evict(p.c(), bufs, ws.data_ptr(), ws.numel(), _stream(stream))
    return o


def score(p: Problem, K: torch.Tensor, Q: torch.Tensor, *, lse_in=None, want_lse=False,
          ws=None, paging: Optional[Paging] = None, stream=None):
    """dge_score: final (pooled) scores [unit][P] in float32.

    With ``want_lse`` returns (scores, lse); ``lse_in`` as for evict()."""
    _check_cache(K, "K")
    _check_cache(Q, "Q")
    scores = torch.empty((p.U, p.P), dtype=torch.float32, device=K.device)
    lse = torch.empty(p.lse_shape, dtype=torch.float32, device=K.device) \
        if want_lse and lse_in is None else None
    if ws is None:
        ws = workspace(p, K.device)
    pg, pg_ptr = _paging_ptr(paging, K)
    bufs = B.dge_buffers(K=_kv_desc(K, paging), Q=B.tensor_desc(Q), scores=scores.data_ptr(),
                         lse_in=_lse_arg(p, lse_in), lse_out=B.ptr(lse), paging=pg_ptr)
    B.dge_score(p.c(), bufs, ws.data_ptr(), ws.numel(), _stream(stream))
    return (scores, lse) if want_lse else scores


def select(p: Problem, scores: Optional[torch.Tensor], *, stream=None) -> torch.Tensor:
    """dge_select: packed ascending kept positions (int32)."""
    dev = scores.device if scores is not None else torch.device("cuda")
    idx = torch.empty(p.packed_rows(), dtype=torch.int32, device=dev)
    B.dge_select(p.c(), B.ptr(scores), idx.data_ptr(), _stream(stream))
    return idx


def compact(p: Problem, idx: torch.Tensor, K: torch.Tensor, V: torch.Tensor, *, ws=None,
            paging: Optional[Paging] = None, stream=None) -> tuple:
    """dge_compact (dge_compact_paged with ``paging``): packed Kc, Vc gathered at idx."""
    _check_cache(K, "K")
    _check_cache(V, "V")
    rows = p.packed_rows()
    Kc = torch.empty((rows, p.d), dtype=torch.bfloat16, device=K.device)
    Vc = torch.empty_like(Kc)
    kd, vd = _kv_desc(K, paging), _kv_desc(V, paging)
    if paging is None:
        B.dge_compact(p.c(), idx.data_ptr(), kd, vd, Kc.data_ptr(), Vc.data_ptr(),
                      B.ptr(ws), _stream(stream))
    else:
        B.dge_compact_paged(p.c(), paging.c(K), idx.data_ptr(), kd, vd, Kc.data_ptr(),
                            Vc.data_ptr(), B.ptr(ws), _stream(stream))
    return Kc, Vc


def compact_inplace(p: Problem, idx: torch.Tensor, K: torch.Tensor, V: torch.Tensor, *,
                    ws=None, paging: Optional[Paging] = None, stream=None) -> None:
    """dge_compact_inplace: rows [0, B_l) of every unit of K and V become the kept rows (with
    ``paging``: positions [0, B_l) of every sequence's pages)."""
    _check_cache(K, "K")
    _check_cache(V, "V")
    if paging is None:
        B.dge_compact_inplace(p.c(), idx.data_ptr(), B.tensor_desc(K), B.tensor_desc(V),
                              B.ptr(ws), _stream(stream))
    else:
        B.dge_compact_inplace_paged(p.c(), paging.c(K), idx.data_ptr(), _kv_desc(K, paging),
                                    _kv_desc(V, paging), B.ptr(ws), _stream(stream))


def evict_inplace(p: Problem, K: torch.Tensor, V: torch.Tensor, Q: Optional[torch.Tensor] = None,
                  *, want_scores: bool = False, lse_in: Optional[torch.Tensor] = None,
                  want_lse: bool = False, ws: Optional[torch.Tensor] = None,
                  out: Optional[dict] = None, paging: Optional[Paging] = None,
                  stream=None) -> dict:
    """dge_evict_inplace: score -> pool -> select, then the kept rows move to the front of
    every unit of K and V (written in place; with ``paging``, to the first positions of every
    sequence's pages).  Returns {"idx", "scores", "lse"}."""
    _check_cache(K, "K")
    _check_cache(V, "V")
    dev = K.device
    o = dict(out or {})
    if o.get("idx") is None:
        o["idx"] = torch.empty(p.packed_rows(), dtype=torch.int32, device=dev)
    if want_scores and o.get("scores") is None:
        o["scores"] = torch.empty((p.U, p.P), dtype=torch.float32, device=dev)
    o.setdefault("scores", None)
    if want_lse and lse_in is None and o.get("lse") is None:
        o["lse"] = torch.empty(p.lse_shape, dtype=torch.float32, device=dev)
    o.setdefault("lse", None)
    if ws is None:
        ws = workspace(p, dev)
    pg, pg_ptr = _paging_ptr(paging, K)
    bufs = B.dge_buffers(K=_kv_desc(K, paging), V=_kv_desc(V, paging), Q=B.tensor_desc(Q),
                         scores=B.ptr(o["scores"]), idx=B.ptr(o["idx"]),
                         lse_in=_lse_arg(p, lse_in),
                         lse_out=B.ptr(o["lse"]) if want_lse and lse_in is None else 0,
                         paging=pg_ptr)
    B.dge_evict_inplace(p.c(), bufs, ws.data_ptr(), ws.numel(), _stream(stream))
    return o


def diagnostics(p: Problem, Q: torch.Tensor, evicted: dict, lse: torch.Tensor, *, ws=None,
                heldout_q: Optional[torch.Tensor] = None, K: Optional[torch.Tensor] = None,
                V: Optional[torch.Tensor] = None, paging: Optional[Paging] = None,
                stream=None) -> dict:
    """dge_diagnostics: per-row evicted mass (Problem.lse_shape), and per unit the
    attention-matching loss and the mean run of retained positions, for an eviction whose
    outputs (``evicted["Kc"]``, ``evicted["idx"]``) came from evict(); ``lse`` = the rows'
    full-cache normalisers (evict(..., want_lse=True)["lse"]).  With ``heldout_q`` (bf16
    [L][b][Hq][d]) and the full cache K, V: per query head the held-out evicted mass,
    |o - o~| and m |mu_E - mu_R| (Eq. evict-mass)."""
    dev = Q.device
    rho = torch.empty(p.lse_shape, dtype=torch.float32, device=dev)
    lm = torch.empty(p.U, dtype=torch.float32, device=dev)
    rl = torch.empty(p.U, dtype=torch.float32, device=dev)
    if ws is None:
        ws = workspace(p, dev)
    bufs = B.dge_buffers(Q=B.tensor_desc(Q), Kc=B.ptr(evicted["Kc"]), idx=B.ptr(evicted["idx"]),
                         lse_in=_lse_arg(p, lse))
    out = B.dge_diag(evicted_mass=rho.data_ptr(), l_match=lm.data_ptr(), run_length=rl.data_ptr())
    res = {"evicted_mass": rho, "l_match": lm, "run_length": rl}
    if heldout_q is not None:
        if heldout_q.dtype != torch.bfloat16 or heldout_q.dim() != 4 or \
                tuple(heldout_q.shape) != (p.L, p.b, p.Hq, p.d) or heldout_q.stride(3) != 1:
            raise ValueError(f"heldout_q must be bf16 [{p.L}][{p.b}][{p.Hq}][{p.d}]")
        _check_cache(K, "K")
        _check_cache(V, "V")
        hq = heldout_q.unsqueeze(3)                      # [L][b][Hq][1][d] for the descriptor
        for k in ("heldout_mass", "heldout_err", "heldout_gap"):
            res[k] = torch.empty((p.L, p.b, p.Hq), dtype=torch.float32, device=dev)
        out.heldout_q = B.tensor_desc(hq)
        out.heldout_mass = res["heldout_mass"].data_ptr()
        out.heldout_err = res["heldout_err"].data_ptr()
        out.heldout_gap = res["heldout_gap"].data_ptr()
        bufs.K = _kv_desc(K, paging)
        bufs.V = _kv_desc(V, paging)
        if paging is not None:
            pg, bufs.paging = _paging_ptr(paging, K)
    B.dge_diagnostics(p.c(), bufs, out, ws.data_ptr(), ws.numel(), _stream(stream))
    return res


def device_status(ws: torch.Tensor, stream=None) -> int:
    """dge_get_device_status: sync the stream and read/clear the status word."""
    return B.dge_get_device_status(ws.data_ptr(), _stream(stream))


def pyramid_budgets(B_: int, w: int, L: int) -> list:
    """PyramidKV per-layer past budgets (App. L)."""
    return B.dge_pyramid_budgets(B_, w, L)
