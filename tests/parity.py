"""Comparison helpers: the CUDA path against the fp64 oracle (test code only).

Tolerances:
  * scores: |gpu - ref| <= 1e-3 * max(|ref|, 1e-6 * max_j ref_j of the unit)
    (fp32 accumulation and fp32 exponentials against an fp64 reference);
  * kept positions: exactly budget of them, strictly ascending, sinks and the
    protected tail present, and identical to the oracle's set except at
    positions whose oracle score lies within 1e-4 (relative) of the oracle's
    keep-th largest candidate score (a near-tie that fp32 may order either
    way);
  * Kc / Vc: bit-exact rows of K / V at the GPU's own indices.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2609_33334_gb300 import inputs

SCORE_RTOL = 1e-3
SCORE_FLOOR = 1e-6
TIE_RTOL = 1e-4


def unit_list(wl, units=None):
    """(layer, batch, kv_head) of every unit, or of the given unit numbers."""
    allu = [(l, b, h) for l in range(wl.L) for b in range(wl.b) for h in range(wl.Hkv)]
    return allu if units is None else [allu[u] for u in units]


def unit_index(wl, l, b, h):
    return (l * wl.b + b) * wl.Hkv + h


def assert_scores_close(gpu: np.ndarray, ref: np.ndarray, what: str = "scores"):
    gpu = np.asarray(gpu, dtype=np.float64)
    top = np.max(np.abs(ref)) if ref.size else 0.0
    tol = SCORE_RTOL * np.maximum(np.abs(ref), SCORE_FLOOR * top)
    err = np.abs(gpu - ref)
    bad = np.nonzero(~(err <= tol))[0]
    if bad.size:
        j = bad[np.argmax(err[bad] / np.maximum(tol[bad], 1e-300))]
        raise AssertionError(f"{what}: {bad.size} of {ref.size} out of tolerance; worst at {j}: "
                             f"gpu={gpu[j]!r} ref={ref[j]!r} tol={tol[j]:.3g}")


def check_kept(idx: np.ndarray, ref_scores: np.ndarray, ref_idx: np.ndarray, *, n, sinks, tail,
               budget, what="idx"):
    idx = np.asarray(idx, dtype=np.int64)
    assert idx.shape == (budget,), f"{what}: {idx.shape} rows, expected {budget}"
    assert np.all(np.diff(idx) > 0), f"{what}: not strictly ascending"
    assert idx.min() >= 0 and idx.max() < n
    s = set(idx.tolist())
    assert set(range(sinks)) <= s, f"{what}: sinks missing"
    assert set(range(n - tail, n)) <= s, f"{what}: protected tail missing"
    diff = s ^ set(ref_idx.tolist())
    if not diff:
        return 0
    P = n - tail
    keep = budget - sinks - tail
    cand = np.asarray(ref_scores[sinks:P], dtype=np.float64)
    T = np.sort(cand)[::-1][keep - 1]
    for j in diff:
        assert sinks <= j < P, f"{what}: differs at protected position {j}"
        assert abs(ref_scores[j] - T) <= TIE_RTOL * abs(T), \
            f"{what}: position {j} (score {ref_scores[j]!r}) differs, threshold {T!r}"
    return len(diff)


def oracle_units(wl, tens, units, want_lse=False):
    """Oracle results for several units, the scores of all of them in one
    multi-threaded oracle call; returns {(l, b, h): evict_unit-style dict} (with the
    unit's row normalisers [R], natural log, under "lse" when ``want_lse``)."""
    refs = {}
    if wl.variant == inputs.STREAMING:
        for (l, b, h) in units:
            refs[(l, b, h)] = oracle.evict_unit(None, unit_bits(tens["K"], l, b, h),
                                                unit_bits(tens["V"], l, b, h), variant=wl.variant,
                                                m=wl.m, tail=wl.tail, sinks=wl.sinks,
                                                budget=wl.budgets[l], pool_kind=wl.pool,
                                                kernel=wl.pool_kernel)
        return refs
    G = wl.G
    Q = np.stack([inputs.bf16_bits(tens["Q"][l, b, h * G:(h + 1) * G]).reshape(-1, wl.d)
                  for (l, b, h) in units])
    K = np.stack([unit_bits(tens["K"], l, b, h) for (l, b, h) in units])
    pos = oracle.h2o_positions(wl.n, G) if wl.variant == inputs.H2O else \
        oracle.scored_positions(wl.n, wl.m, G)
    if want_lse:
        raw, lse = oracle.scores(Q, K, pos, wl.n - wl.tail, want_lse=True)
    else:
        raw, lse = oracle.scores(Q, K, pos, wl.n - wl.tail), None
    for i, (l, b, h) in enumerate(units):
        pooled = oracle.pool(raw[i], wl.pool, wl.pool_kernel) if wl.variant == inputs.SCORED \
            else raw[i].copy()
        idx = oracle.select(pooled, wl.n, wl.sinks, wl.tail, wl.budgets[l])
        refs[(l, b, h)] = {"raw": raw[i], "pooled": pooled, "idx": idx}
        if lse is not None:
            refs[(l, b, h)]["lse"] = lse[i]
    return refs


def unit_rows(wl, l, b, h):
    """[start, stop) of a unit's rows in the packed outputs."""
    base = sum(wl.b * wl.Hkv * wl.budgets[i] for i in range(l))
    start = base + (b * wl.Hkv + h) * wl.budgets[l]
    return start, start + wl.budgets[l]


def unit_bits(t: torch.Tensor, l, b, h):
    return inputs.bf16_bits(t[l, b, h])


def compare_unit(wl, out, tens, l, b, h, ref=None):
    """Check one unit of a dge_evict result against the oracle; returns #near-tie diffs."""
    if ref is None:
        Qg = inputs.bf16_bits(tens["Q"][l, b, h * wl.G:(h + 1) * wl.G]) \
            if wl.variant != inputs.STREAMING else None
        ref = oracle.evict_unit(Qg, unit_bits(tens["K"], l, b, h), unit_bits(tens["V"], l, b, h),
                                variant=wl.variant, m=wl.m, tail=wl.tail, sinks=wl.sinks,
                                budget=wl.budgets[l], pool_kind=wl.pool, kernel=wl.pool_kernel)
    r0, r1 = unit_rows(wl, l, b, h)
    idx = out["idx"][r0:r1].cpu().numpy()
    u = unit_index(wl, l, b, h)
    diffs = 0
    if wl.variant == inputs.STREAMING:
        np.testing.assert_array_equal(idx, ref["idx"])
    else:
        if out.get("scores") is not None:
            assert_scores_close(out["scores"][u].cpu().numpy(), ref["pooled"],
                                f"scores unit {(l, b, h)}")
        diffs = check_kept(idx, ref["pooled"], ref["idx"], n=wl.n, sinks=wl.sinks,
                           tail=wl.tail, budget=wl.budgets[l], what=f"idx unit {(l, b, h)}")
    Kb = unit_bits(tens["K"], l, b, h)
    Vb = unit_bits(tens["V"], l, b, h)
    np.testing.assert_array_equal(inputs.bf16_bits(out["Kc"][r0:r1]), oracle.gather(Kb, idx))
    np.testing.assert_array_equal(inputs.bf16_bits(out["Vc"][r0:r1]), oracle.gather(Vb, idx))
    if "Kc" in ref:
        # the oracle's own gather at its own indices agrees wherever the indices agree
        same = idx == ref["idx"]
        np.testing.assert_array_equal(inputs.bf16_bits(out["Kc"][r0:r1])[same], ref["Kc"][same])
    return diffs
