"""fp64 CPU oracle for the DGE score -> select -> compact pass.

TEST INFRASTRUCTURE ONLY: tests/, ``__graft_entry__.smoke()`` and bench.py's
CPU-baseline leg may import this package; the product path never does.  It
shares no code with the CUDA library (``paper_2609_33334_gb300``) and imports
nothing from it.

The arithmetic lives in ``dge_oracle.c`` (plain C, double precision, loops
only); this module compiles it with gcc and marshals numpy arrays.  Each
function names the paper passage it follows:

* :func:`scores`   -- Alg. 1 line B, App. B (softmax per observation row, sum
  over rows and over the query heads of one KV group, App. G).
* :func:`pool`     -- App. B, max-pool kernel 7 (avg-pool for the PyramidKV
  workload).
* :func:`select`   -- Alg. 1 retention rule R_E(s, B - w) + App. E (sorted,
  temporal order), with protected head (sinks) and protected tail.
* :func:`streaming_indices` -- App. L (StreamingLLM: 4 sinks + recency).
* :func:`gather`   -- App. E (gather [retained past] || [window + draft tail]).
* :func:`pyramid_budgets` -- App. L, PyramidKV's discrete schedule.

Readings where the paper is silent: rows are causal (row at position p sees
keys <= p); SCORED observation rows of every head sit at n - m .. n - 1 (the
window, then the draft rows); H2O row i sits at position i; scores are sums
(not means) over rows and group heads; pooling runs over the scored range
only; ties go to the lower position; every budget counts the protected
positions.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dge_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

POOL_NONE, POOL_MAX, POOL_AVG = 0, 1, 2

_i64p = ctypes.POINTER(ctypes.c_int64)
_f64p = ctypes.POINTER(ctypes.c_double)
_u16p = ctypes.POINTER(ctypes.c_uint16)
_i32p = ctypes.POINTER(ctypes.c_int32)
_u8p = ctypes.POINTER(ctypes.c_uint8)


def build(force: bool = False) -> str:
    """Compile ``dge_oracle.c`` into ``liboracle.so`` (gcc, -O2, OpenMP)."""
    if not force and os.path.exists(_LIB_PATH) and \
            os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    tmp = _LIB_PATH + f".{os.getpid()}.tmp"
    cmd = ["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            lib.dgeo_scores.argtypes = [_u16p, _u16p, _i64p, ctypes.c_int64, ctypes.c_int64,
                                        ctypes.c_int64, ctypes.c_int64, ctypes.c_double,
                                        ctypes.c_int64, _f64p, _f64p]
            lib.dgeo_pool.argtypes = [_f64p, ctypes.c_int64, ctypes.c_int, ctypes.c_int, _f64p]
            lib.dgeo_select.argtypes = [_f64p, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                        ctypes.c_int64, _i32p]
            lib.dgeo_select_blocks.argtypes = [_f64p, ctypes.c_int64, ctypes.c_int64,
                                               ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                               _i32p]
            lib.dgeo_streaming_indices.argtypes = [ctypes.c_int64, ctypes.c_int64,
                                                   ctypes.c_int64, _i32p]
            lib.dgeo_gather.argtypes = [_u8p, ctypes.c_int64, _i32p, ctypes.c_int64, _u8p]
            lib.dgeo_gather.restype = None
            lib.dgeo_pyramid_budgets.argtypes = [ctypes.c_int64, ctypes.c_int64,
                                                 ctypes.c_int64, _i64p]
            _lib = lib
    return _lib


def _ptr(a: np.ndarray, t):
    return a.ctypes.data_as(t)


def scored_positions(n: int, m: int, G: int) -> np.ndarray:
    """Positions of the stacked observation rows (head-major): n-m .. n-1 per head."""
    return np.tile(np.arange(n - m, n, dtype=np.int64), G)


def h2o_positions(n: int, G: int) -> np.ndarray:
    """Positions of H2O's stacked rows: row i of every head sits at position i."""
    return np.tile(np.arange(n, dtype=np.int64), G)


def scores(Q: np.ndarray, K: np.ndarray, pos: np.ndarray, P: int, scale: float | None = None,
           want_lse: bool = False):
    """Raw attention scores of U KV heads (Alg. 1 line B; App. B; App. G).

    Q: uint16 bf16 bits [U][R][d] (stacked rows of the group's query heads);
    K: uint16 bf16 bits [U][n][d]; pos: int64 [R] row positions; P: positions
    scored.  Returns raw [U][P] (and lse [U][R] when ``want_lse``) in float64.
    """
    Q = np.ascontiguousarray(Q, dtype=np.uint16)
    K = np.ascontiguousarray(K, dtype=np.uint16)
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    U, R, d = Q.shape
    n = K.shape[1]
    if K.shape != (U, n, d) or pos.shape != (R,) or not (0 <= P <= n):
        raise ValueError("shape mismatch")
    if scale is None:
        scale = 1.0 / math.sqrt(d)
    raw = np.zeros((U, P), dtype=np.float64)
    lse = np.zeros((U, R), dtype=np.float64) if want_lse else None
    rc = _load().dgeo_scores(_ptr(Q, _u16p), _ptr(K, _u16p), _ptr(pos, _i64p), U, R, d, n,
                             float(scale), P, _ptr(raw, _f64p),
                             _ptr(lse, _f64p) if want_lse else None)
    if rc != 0:
        raise MemoryError("oracle scratch allocation failed")
    return (raw, lse) if want_lse else raw


def pool(raw: np.ndarray, pool_kind: int, kernel: int) -> np.ndarray:
    """Pooling along positions (App. B); works on the last axis."""
    raw = np.ascontiguousarray(raw, dtype=np.float64)
    out = np.empty_like(raw)
    flat_in, flat_out = raw.reshape(-1, raw.shape[-1]), out.reshape(-1, raw.shape[-1])
    lib = _load()
    for i in range(flat_in.shape[0]):
        row_in = np.ascontiguousarray(flat_in[i])
        row_out = np.empty_like(row_in)
        if lib.dgeo_pool(_ptr(row_in, _f64p), row_in.shape[0], pool_kind, kernel,
                         _ptr(row_out, _f64p)) != 0:
            raise ValueError("bad pooling arguments")
        flat_out[i] = row_out
    return out


def select(scores_by_pos: np.ndarray, n: int, s0: int, tail: int, budget: int) -> np.ndarray:
    """Kept positions of one head, ascending (Alg. 1 retention + App. E ordering).

    ``scores_by_pos`` holds the (pooled) score of positions [0, P), P = n - tail.
    Keeps [0, s0), the budget - s0 - tail best of [s0, P), and [P, n).
    """
    P = n - tail
    keep = budget - s0 - tail
    s = np.ascontiguousarray(scores_by_pos[:P], dtype=np.float64)
    idx = np.empty(budget, dtype=np.int32)
    if _load().dgeo_select(_ptr(s, _f64p), P, n, s0, keep, _ptr(idx, _i32p)) != 0:
        raise ValueError("bad selection arguments")
    return idx


def select_blocks(scores_by_pos: np.ndarray, n: int, s0: int, tail: int, budget: int,
                  bs: int) -> np.ndarray:
    """Block-granular kept positions of one head, ascending (the "fixed b-blocks" rung;
    the rule as read in dge_oracle.c): whole blocks of ``bs`` candidates by block-score sum,
    the first block that does not fit contributing its lowest positions."""
    P = n - tail
    keep = budget - s0 - tail
    s = np.ascontiguousarray(scores_by_pos[:P], dtype=np.float64)
    idx = np.empty(budget, dtype=np.int32)
    if _load().dgeo_select_blocks(_ptr(s, _f64p), P, n, s0, keep, bs, _ptr(idx, _i32p)) != 0:
        raise ValueError("bad selection arguments")
    return idx


def streaming_indices(n: int, sinks: int, budget: int) -> np.ndarray:
    """StreamingLLM kept positions: [0, sinks) then the last budget - sinks (App. L)."""
    idx = np.empty(budget, dtype=np.int32)
    if _load().dgeo_streaming_indices(n, sinks, budget, _ptr(idx, _i32p)) != 0:
        raise ValueError("bad streaming arguments")
    return idx


def gather(rows: np.ndarray, idx: np.ndarray) -> np.ndarray:
    """Byte copy of rows[idx[r]] for every r (App. E); rows is [n][...]."""
    rows = np.ascontiguousarray(rows)
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    if idx.size and (idx.min() < 0 or idx.max() >= rows.shape[0]):
        raise IndexError("index out of range")
    out = np.empty((idx.shape[0],) + rows.shape[1:], dtype=rows.dtype)
    row_bytes = rows[0].nbytes if rows.shape[0] else 0
    _load().dgeo_gather(_ptr(rows.view(np.uint8), _u8p), row_bytes, _ptr(idx, _i32p),
                        idx.shape[0], _ptr(out.view(np.uint8), _u8p))
    return out


def pyramid_budgets(B: int, w: int, L: int) -> np.ndarray:
    """PyramidKV per-layer past budgets (App. L, discrete schedule)."""
    out = np.empty(L, dtype=np.int64)
    if _load().dgeo_pyramid_budgets(B, w, L, _ptr(out, _i64p)) != 0:
        raise ValueError("bad pyramid arguments")
    return out


def evict_unit(Qg: np.ndarray, K: np.ndarray, V: np.ndarray, *, variant: int, m: int,
               tail: int, sinks: int, budget: int, pool_kind: int, kernel: int,
               select_block: int = 0,
               scale: float | None = None) -> dict:
    """The whole pass for one KV head: scores -> pool -> select -> gather.

    Qg: uint16 [G][rows][d] (the group's query heads); K, V: uint16 [n][d].
    variant 0 = SCORED (rows at n-m..n-1), 1 = H2O (row i at i, no pooling),
    2 = STREAMING (no scores).  Returns raw, pooled, idx, Kc, Vc.
    """
    n = K.shape[0]
    if variant == 2:
        idx = streaming_indices(n, sinks, budget)
        return {"raw": None, "pooled": None, "idx": idx, "Kc": gather(K, idx),
                "Vc": gather(V, idx)}
    G, rows, d = Qg.shape
    pos = h2o_positions(n, G) if variant == 1 else scored_positions(n, m, G)
    P = n - tail
    raw = scores(Qg.reshape(1, G * rows, d), K[None], pos, P, scale)[0]
    pooled = pool(raw, pool_kind, kernel) if variant == 0 else raw.copy()
    idx = select_blocks(pooled, n, sinks, tail, budget, select_block) if select_block > 1 \
        else select(pooled, n, sinks, tail, budget)
    return {"raw": raw, "pooled": pooled, "idx": idx, "Kc": gather(K, idx),
            "Vc": gather(V, idx)}
