"""Seeded synthetic inputs for the DGE score-select-compact pass.

This module only makes input bytes: shapes, seeds, random tensors, the sink and
the planted spans. It holds none of the method's arithmetic (no softmax, no
pooling, no selection) and is the one module that both the CUDA path's tests
and the fp64 oracle's tests read.

Workload shapes follow the paper's setting: a GQA cache [L][b][Hkv][n][d] of
post-RoPE keys/values (App. E, implementation notes; App. G, the native
``kv_head`` layout), observation queries = the last w prompt rows plus the k
draft rows (Alg. 1 line B and its DGE-W alternative), per-head budget B that
includes the protected window (Sec. 3, notation), SnapKV max-pool kernel 7
(App. A, compression settings), PyramidKV per-layer budgets (App. L), H2O's
all-prompt-query accumulator (Table "complexity", note a) and StreamingLLM's
sinks + recency window (App. L, composition).

Synthetic recipe (stand-in for LongBench-scale caches, which are not available):
Q, K, V ~ N(0, 1) drawn in fp32 and rounded to bf16 (round-to-nearest-even);
position 0 of K and V is scaled by 8 before rounding (an attention sink); and
``n_spans`` spans of ``span_len`` consecutive keys are planted so that each key
has cosine 0.5 with one draft query row of one query head of the group.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np
import torch

SCORED, H2O, STREAMING = 0, 1, 2
POOL_NONE, POOL_MAX, POOL_AVG = 0, 1, 2


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic eviction problem (all sizes in tokens / heads / elements)."""

    name: str
    L: int            # layers
    b: int            # sequences (batch)
    Hq: int           # query heads
    Hkv: int          # KV heads
    d: int            # head dim
    n: int            # cache length at eviction time (prompt + draft rows)
    w: int            # observation window rows
    k: int            # draft rows
    variant: int      # SCORED / H2O / STREAMING
    pool: int         # POOL_*
    pool_kernel: int
    budgets: tuple    # per-layer budget, incl. every protected position
    sinks: int = 0    # protected head [0, sinks)
    recent: int = 0   # H2O protected recent tail
    n_spans: int = 0
    span_len: int = 0
    seed: int = 0
    sink_scale: float = 8.0
    span_cos: float = 0.5  # cosine between a span key and its draft query row

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    @property
    def m(self) -> int:
        """Observation rows per query head (window + draft)."""
        return self.w + self.k

    @property
    def tail(self) -> int:
        """Protected tail length: the observation rows (SCORED) or H2O's recent window."""
        if self.variant == SCORED:
            return self.m
        if self.variant == H2O:
            return self.recent
        return 0

    @property
    def q_rows(self) -> int:
        """Query rows per query head that the scorer reads."""
        if self.variant == H2O:
            return self.n
        if self.variant == STREAMING:
            return 0
        return self.m

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


def literal_ramp(L: int, first: int, last: int) -> tuple:
    """Per-layer budgets on a straight line from ``first`` (layer 0) to ``last`` (layer L-1)."""
    return tuple(first - ((first - last) * l) // (L - 1) for l in range(L))


WORKLOADS = {
    # 1 layer, 8 Q / 2 KV heads, d=64, n=1024, w=8 + k=2, SnapKV max-pool 7, B=128.
    "c1_tiny": Workload("c1_tiny", L=1, b=1, Hq=8, Hkv=2, d=64, n=1024, w=8, k=2,
                        variant=SCORED, pool=POOL_MAX, pool_kernel=7, budgets=(128,),
                        n_spans=4, span_len=16, seed=0),
    # Llama-3.1-8B shape, n=8192, w=32 + k=2, max-pool 7, B=1024.
    "c2_8b_8k": Workload("c2_8b_8k", L=32, b=1, Hq=32, Hkv=8, d=128, n=8192, w=32, k=2,
                         variant=SCORED, pool=POOL_MAX, pool_kernel=7, budgets=(1024,) * 32,
                         n_spans=16, span_len=32, seed=1),
    # 8B shape, batch 4, n=32768, PyramidKV-style ramp 2048 -> 256, avg-pool 7.
    "c3_8b_32k_pyramid": Workload("c3_8b_32k_pyramid", L=32, b=4, Hq=32, Hkv=8, d=128,
                                  n=32768, w=32, k=2, variant=SCORED, pool=POOL_AVG,
                                  pool_kernel=7, budgets=literal_ramp(32, 2048, 256),
                                  n_spans=64, span_len=32, seed=2),
    # H2O accumulator: all prompt rows + 2 draft rows, 512 heavy + 64 recent + 4 sinks.
    "c4_h2o_8k": Workload("c4_h2o_8k", L=32, b=8, Hq=32, Hkv=8, d=128, n=8192, w=0, k=2,
                          variant=H2O, pool=POOL_NONE, pool_kernel=1, budgets=(580,) * 32,
                          sinks=4, recent=64, seed=3),
    # 70B shape at 128K, w=64 + k=2, max-pool 7, B=4096.
    "c5_70b_128k": Workload("c5_70b_128k", L=80, b=1, Hq=64, Hkv=8, d=128, n=131072, w=64,
                            k=2, variant=SCORED, pool=POOL_MAX, pool_kernel=7,
                            budgets=(4096,) * 80, n_spans=256, span_len=64, seed=4),
    # StreamingLLM gather floor on the same cache: 4 sinks + 4092 recent.
    "c5_slm": Workload("c5_slm", L=80, b=1, Hq=64, Hkv=8, d=128, n=131072, w=0, k=0,
                       variant=STREAMING, pool=POOL_NONE, pool_kernel=1,
                       budgets=(4096,) * 80, sinks=4, n_spans=256, span_len=64, seed=4),
}


def span_positions(wl: Workload, seq: int) -> np.ndarray:
    """Start positions of the planted spans of sequence ``seq`` (shared by all layers/heads).

    Non-overlapping, at least 7 positions apart (so a kernel-7 pooling halo
    never joins two spans), inside [8, n - tail - span_len - 8).
    """
    if wl.n_spans == 0:
        return np.zeros(0, dtype=np.int64)
    rng = np.random.default_rng(1_000_003 * wl.seed + seq)
    lo, hi = 8, wl.n - max(wl.tail, wl.m) - wl.span_len - 8
    slot = wl.span_len + 7
    n_slots = (hi - lo) // slot
    if n_slots < wl.n_spans:
        raise ValueError(f"{wl.name}: cache too short for {wl.n_spans} spans")
    slots = np.sort(rng.choice(n_slots, size=wl.n_spans, replace=False))
    jitter = rng.integers(0, 7, size=wl.n_spans)  # stays inside the slot's 7-gap
    return lo + slots * slot + jitter


def _gen(device, seed):
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def make_inputs(wl: Workload, device="cpu", layers: Optional[range] = None,
                batches: Optional[range] = None) -> dict:
    """Build Q, K, V (bf16 tensors) for ``wl`` on ``device``.

    Shapes: K, V [L'][b'][Hkv][n][d]; Q [L'][b'][Hq][rows][d] where rows = m
    (SCORED), n (H2O) or 0 (STREAMING). ``layers``/``batches`` select a
    sub-range; every (layer, sequence) slice is drawn from its own seeded
    stream, so a sub-range has the same bytes as the full tensor's slice.
    """
    layers = range(wl.L) if layers is None else layers
    batches = range(wl.b) if batches is None else batches
    Lp, bp = len(layers), len(batches)
    rows = wl.q_rows
    K = torch.empty((Lp, bp, wl.Hkv, wl.n, wl.d), dtype=torch.bfloat16, device=device)
    V = torch.empty_like(K)
    Q = torch.empty((Lp, bp, wl.Hq, rows, wl.d), dtype=torch.bfloat16, device=device)
    for li, l in enumerate(layers):
        for bi, s in enumerate(batches):
            g = _gen(device, (wl.seed * 7919 + l) * 104729 + s)
            q = torch.randn((wl.Hq, rows, wl.d), generator=g, device=device, dtype=torch.float32)
            k = torch.randn((wl.Hkv, wl.n, wl.d), generator=g, device=device, dtype=torch.float32)
            v = torch.randn((wl.Hkv, wl.n, wl.d), generator=g, device=device, dtype=torch.float32)
            if wl.sink_scale != 1.0:
                k[:, 0, :] *= wl.sink_scale
                v[:, 0, :] *= wl.sink_scale
            Q[li, bi] = q.to(torch.bfloat16)
            if wl.n_spans and rows:
                _plant_spans(wl, s, Q[li, bi].float(), k, g)
            K[li, bi] = k.to(torch.bfloat16)
            V[li, bi] = v.to(torch.bfloat16)
    return {"Q": Q, "K": K, "V": V}


def _plant_spans(wl: Workload, seq: int, q: torch.Tensor, k: torch.Tensor, g) -> None:
    """Overwrite span keys so each has cosine ``span_cos`` with one draft query row.

    Span s uses query head (h*G + s mod G) of KV head h and draft row
    w + (s mod k); its keys have norm sqrt(d) and a fresh random direction
    orthogonal to that query.
    """
    starts = span_positions(wl, seq)
    G, d = wl.G, wl.d
    kdraft = max(wl.k, 1)
    for s, p0 in enumerate(starts.tolist()):
        heads = torch.arange(wl.Hkv, device=k.device) * G + (s % G)
        row = wl.w + (s % kdraft) if wl.k else wl.m - 1
        u = q[heads, row, :]                                    # [Hkv, d]
        u = u / u.norm(dim=-1, keepdim=True)
        r = torch.randn((wl.Hkv, wl.span_len, d), generator=g, device=k.device)
        r = r - (r * u[:, None, :]).sum(-1, keepdim=True) * u[:, None, :]
        r = r / r.norm(dim=-1, keepdim=True)
        c = wl.span_cos
        kk = math.sqrt(d) * (c * u[:, None, :] + math.sqrt(1.0 - c * c) * r)
        k[:, p0:p0 + wl.span_len, :] = kk


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """Raw bf16 bit patterns of a (CPU or CUDA) tensor as a contiguous uint16 array."""
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def paged_layout(cache: torch.Tensor, page_size: int, seed: int = 0, spare_pages: int = 3,
                 extra_table_pages: int = 1, head_major: bool = False,
                 order: str = "random") -> tuple:
    """Lay a contiguous cache [L][b][Hkv][n][d] out as a paged one, the way a paged-attention
    server keeps it: returns the pool [L][num_pages][page_size][Hkv][d] (``head_major``:
    [L][num_pages][Hkv][page_size][d]) and the block table, int32 [b][pages_per_seq].
    Sequences get pages in a seeded random order shared by all layers (``order=
    "sequential"``: each sequence's pages one after another, as a fresh allocator hands them
    out; ``"runs"``: sequential with one page in eight swapped with a random other).  The pool
    has ``spare_pages`` pages no sequence uses, and the table ``extra_table_pages`` entries per
    sequence past the cache (set to -1).  Every slot that holds no cache position is NaN, so a
    read of one shows in the results.  Pure layout: no arithmetic of the method."""
    L, b, Hkv, n, d = cache.shape
    used = (n + page_size - 1) // page_size
    pps = used + extra_table_pages
    num_pages = b * used + spare_pages
    rng = np.random.default_rng(seed)
    if order == "random":
        flat = rng.permutation(num_pages)
    else:
        flat = np.arange(num_pages)
        if order == "runs":
            for i in rng.choice(num_pages, num_pages // 8, replace=False):
                j = rng.integers(num_pages)
                flat[i], flat[j] = flat[j], flat[i]
        elif order != "sequential":
            raise ValueError(order)
    perm = flat[:b * used].reshape(b, used)
    table = np.full((b, pps), -1, dtype=np.int32)
    table[:, :used] = perm
    shape = (L, num_pages, Hkv, page_size, d) if head_major else (L, num_pages, page_size, Hkv, d)
    pool = torch.full(shape, float("nan"), dtype=cache.dtype, device=cache.device)
    for s in range(b):
        for j in range(used):
            lo, hi = j * page_size, min((j + 1) * page_size, n)
            if head_major:
                pool[:, int(perm[s, j]), :, :hi - lo] = cache[:, s, :, lo:hi]
            else:
                # [L][Hkv][rows][d] -> [L][rows][Hkv][d]
                pool[:, int(perm[s, j]), :hi - lo] = cache[:, s, :, lo:hi].permute(0, 2, 1, 3)
    return pool, torch.from_numpy(table).to(cache.device)


def unpaged(pool: torch.Tensor, block_table: torch.Tensor, n: int,
            head_major: bool = False) -> torch.Tensor:
    """The contiguous cache [L][b][Hkv][n][d] that a paged one holds (inverse of paged_layout
    on positions [0, n))."""
    if head_major:
        L, _, Hkv, page_size, d = pool.shape
    else:
        L, _, page_size, Hkv, d = pool.shape
    b = block_table.shape[0]
    out = torch.empty((L, b, Hkv, n, d), dtype=pool.dtype, device=pool.device)
    table = block_table.cpu().numpy()
    for s in range(b):
        for j in range((n + page_size - 1) // page_size):
            lo, hi = j * page_size, min((j + 1) * page_size, n)
            page = pool[:, int(table[s, j])]
            out[:, s, :, lo:hi] = page[:, :, :hi - lo] if head_major else \
                page[:, :hi - lo].permute(0, 2, 1, 3)
    return out
