"""Paged caches (dge_paging): K and V in page pools behind a block table.

A paged cache holds the same rows as the contiguous one, read in the same tile order, so
every output (scores, kept positions, gathered rows, normalisers) must equal the
contiguous run's bit for bit.  The pools put pages in a seeded random order, keep spare
pages, and fill every slot outside the cache with NaN: a read of a position past the cache
would show in the results.
"""
import os

import pytest
import torch

from paper_2609_33334_gb300 import _build, api, inputs

pytestmark = pytest.mark.gpu
WL = inputs.WORKLOADS

CASES = {
    "c2_small": WL["c2_8b_8k"].with_(L=2, n=3000),                              # tensor cores
    "c1_tiny_d64": WL["c1_tiny"],                                                # d = 64
    "c5_small": WL["c5_70b_128k"].with_(L=1, n=3000, budgets=(700,), n_spans=8),  # row blocks
    "c4_small": WL["c4_h2o_8k"].with_(L=1, b=2, n=1000, budgets=(200,)),         # H2O
    "slm_small": WL["c5_slm"].with_(L=2, n=5000, budgets=(700, 300), n_spans=0),  # gather only
}
PAGE_SIZES = [16, 64, 128, 256]


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    _build.build()


def _paged(tens, page_size, seed=0, head_major=False, order="random"):
    K, bt = inputs.paged_layout(tens["K"], page_size, seed=seed, head_major=head_major,
                                order=order)
    V, bt2 = inputs.paged_layout(tens["V"], page_size, seed=seed, head_major=head_major,
                                 order=order)
    assert torch.equal(bt, bt2)
    return K, V, api.Paging(block_table=bt, page_size=page_size, head_major=head_major)


def _q(wl, tens):
    return tens["Q"] if wl.variant != inputs.STREAMING else None


@pytest.mark.parametrize("page_size", PAGE_SIZES)
@pytest.mark.parametrize("name", sorted(CASES))
def test_paged_evict_equals_contiguous(name, page_size):
    wl = CASES[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    want = wl.variant != inputs.STREAMING
    ref = api.evict(p, tens["K"], tens["V"], _q(wl, tens), want_scores=want)
    K, V, pg = _paged(tens, page_size, seed=page_size)
    got = api.evict(p, K, V, _q(wl, tens), want_scores=want, paging=pg)
    torch.cuda.synchronize()
    for k in ("idx", "Kc", "Vc") + (("scores",) if want else ()):
        assert torch.equal(got[k], ref[k]), k


@pytest.mark.parametrize("name", ["c2_small", "c4_small"])
def test_paged_warp_level_path(monkeypatch, name):
    """The warp-level kernels (range recompute, DGE_SCORE_KERNEL=mma) read pages too."""
    monkeypatch.setenv("DGE_SCORE_KERNEL", "mma")
    wl = CASES[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    ref = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True)
    K, V, pg = _paged(tens, 32)
    got = api.evict(p, K, V, tens["Q"], want_scores=True, paging=pg)
    torch.cuda.synchronize()
    for k in ("idx", "Kc", "Vc", "scores"):
        assert torch.equal(got[k], ref[k]), k


def test_paged_large_logits_recompute():
    """Units flagged out of range on the tensor cores are recomputed from the pages."""
    wl = WL["c1_tiny"].with_(L=1, budgets=(128,))
    tens = inputs.make_inputs(wl, device="cuda")
    tens["Q"] = (tens["Q"].float() * 24.0).to(torch.bfloat16)
    p = api.problem_from_workload(wl)
    ref = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True)
    K, V, pg = _paged(tens, 16)
    got = api.evict(p, K, V, tens["Q"], want_scores=True, paging=pg)
    torch.cuda.synchronize()
    for k in ("idx", "Kc", "Vc", "scores"):
        assert torch.equal(got[k], ref[k]), k


@pytest.mark.parametrize("page_size", [16, 128])
def test_paged_separate_calls_and_lse(page_size):
    """dge_score / dge_compact_paged on pages, and one-pass scoring from supplied normalisers."""
    wl = CASES["c2_small"]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    ref = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True, want_lse=True)
    K, V, pg = _paged(tens, page_size)
    s = api.score(p, K, tens["Q"], paging=pg)
    idx = api.select(p, s)
    Kc, Vc = api.compact(p, idx, K, V, paging=pg)
    one = api.evict(p, K, V, tens["Q"], want_scores=True, lse_in=ref["lse"], paging=pg)
    ref1 = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True, lse_in=ref["lse"])
    torch.cuda.synchronize()
    assert torch.equal(s, ref["scores"])
    assert torch.equal(idx, ref["idx"])
    assert torch.equal(Kc, ref["Kc"]) and torch.equal(Vc, ref["Vc"])
    for k in ("idx", "Kc", "Vc", "scores"):
        assert torch.equal(one[k], ref1[k]), k


@pytest.mark.parametrize("page_size", [16, 64, 256])
@pytest.mark.parametrize("name", ["c2_small", "slm_small"])
def test_paged_inplace(name, page_size):
    """In place on pages: positions [0, B) of every sequence become the kept rows (the
    packed gather's rows), positions [B, n) keep their contents, pages outside the cache
    stay untouched."""
    wl = CASES[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    ref = api.evict(p, tens["K"], tens["V"], _q(wl, tens))
    K, V, pg = _paged(tens, page_size)
    K0, V0 = K.clone(), V.clone()
    got = api.evict_inplace(p, K, V, _q(wl, tens), paging=pg)
    torch.cuda.synchronize()
    assert torch.equal(got["idx"], ref["idx"])
    Kn = inputs.unpaged(K, pg.block_table, wl.n)
    Vn = inputs.unpaged(V, pg.block_table, wl.n)
    Korig = inputs.unpaged(K0, pg.block_table, wl.n)
    offs = p.unit_row_offsets()
    u = 0
    for l in range(wl.L):
        B = wl.budgets[l]
        for b in range(wl.b):
            for h in range(wl.Hkv):
                r0 = offs[u]
                assert torch.equal(Kn[l, b, h, :B], ref["Kc"][r0:r0 + B])
                assert torch.equal(Vn[l, b, h, :B], ref["Vc"][r0:r0 + B])
                assert torch.equal(Kn[l, b, h, B:], Korig[l, b, h, B:])
                u += 1
    # NaN slots (outside every sequence) are untouched: the same count as before
    assert torch.isnan(K.float()).sum() == torch.isnan(K0.float()).sum()


def test_paged_diagnostics_heldout():
    """The held-out evicted-mass check reads the full cache from the pages."""
    wl = CASES["c2_small"].with_(L=1)
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    ev = api.evict(p, tens["K"], tens["V"], tens["Q"], want_lse=True)
    g = torch.Generator(device="cuda").manual_seed(5)
    hq = torch.randn((wl.L, wl.b, wl.Hq, wl.d), generator=g, device="cuda").to(torch.bfloat16)
    a = api.diagnostics(p, tens["Q"], ev, ev["lse"], heldout_q=hq, K=tens["K"], V=tens["V"])
    K, V, pg = _paged(tens, 64)
    b = api.diagnostics(p, tens["Q"], ev, ev["lse"], heldout_q=hq, K=K, V=V, paging=pg)
    torch.cuda.synchronize()
    for k in a:
        assert torch.equal(a[k], b[k]), k


@pytest.mark.parametrize("page_size", [16, 128])
@pytest.mark.parametrize("name", ["c2_small", "c4_small", "slm_small"])
def test_head_major_pages(name, page_size):
    """Pools laid out [page][head][slot][d] (each head's page contiguous) through the same
    strides: identical outputs, and the in-place gather writes the right slots."""
    wl = CASES[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    want = wl.variant != inputs.STREAMING
    ref = api.evict(p, tens["K"], tens["V"], _q(wl, tens), want_scores=want)
    K, V, pg = _paged(tens, page_size, seed=3, head_major=True)
    got = api.evict(p, K, V, _q(wl, tens), want_scores=want, paging=pg)
    torch.cuda.synchronize()
    for k in ("idx", "Kc", "Vc") + (("scores",) if want else ()):
        assert torch.equal(got[k], ref[k]), k
    api.evict_inplace(p, K, V, _q(wl, tens), paging=pg)
    torch.cuda.synchronize()
    Kn = inputs.unpaged(K, pg.block_table, wl.n, head_major=True)
    offs = p.unit_row_offsets()
    u = 0
    for l in range(wl.L):
        B = wl.budgets[l]
        for b in range(wl.b):
            for h in range(wl.Hkv):
                assert torch.equal(Kn[l, b, h, :B], ref["Kc"][offs[u]:offs[u] + B])
                u += 1


@pytest.mark.parametrize("order", ["sequential", "runs"])
@pytest.mark.parametrize("page_size", [16, 64])
@pytest.mark.parametrize("name", ["c2_small", "c5_small", "c4_small"])
def test_consecutive_pages(name, page_size, order):
    """Pages handed out in order (and in order with some swapped): tiles whose pages follow
    each other in the pool load as one box of the merged map, the others page by page; the
    outputs are the contiguous run's either way."""
    wl = CASES[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    ref = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True)
    K, V, pg = _paged(tens, page_size, seed=7, order=order)
    got = api.evict(p, K, V, tens["Q"], want_scores=True, paging=pg)
    torch.cuda.synchronize()
    for k in ("idx", "Kc", "Vc", "scores"):
        assert torch.equal(got[k], ref[k]), k


# --- paged runs against the oracle -------------------------------------------------------
# The equality checks above tie a paged run to the contiguous run; these tie it to the fp64
# oracle directly (scores, kept sets, gathered rows), so that a fault shared by both layouts,
# or one only the paged producer has (per-page boxes, page clamping), cannot hide.

@pytest.mark.parametrize("page_size", [16, 128])
@pytest.mark.parametrize("name", ["c2_small", "c5_small", "c4_small", "slm_small"])
def test_paged_evict_matches_oracle(name, page_size):
    import oracle
    from parity import compare_unit, oracle_units, unit_list
    oracle.build()
    wl = CASES[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    want = wl.variant != inputs.STREAMING
    K, V, pg = _paged(tens, page_size, seed=11 + page_size)
    got = api.evict(p, K, V, _q(wl, tens), want_scores=want, paging=pg)
    torch.cuda.synchronize()
    units = unit_list(wl)
    refs = oracle_units(wl, tens, units)
    for (l, b, h) in units:
        compare_unit(wl, got, tens, l, b, h, ref=refs[(l, b, h)])


@pytest.mark.parametrize("page_size,order", [(16, "sequential"), (16, "runs"), (16, "random"),
                                             (32, "sequential"), (128, "random")])
def test_paged_tasks_span_page_windows(page_size, order):
    """Key chunks longer than the producer's page-id window (32 tiles): 128 units of 32768
    positions take chunks of 64 tiles, so each task reads two windows, the second one's ids
    fetched while the first is in use, and the consecutive-pages check runs per window.  The
    outputs equal the contiguous run's."""
    wl = WL["c3_8b_32k_pyramid"].with_(L=4, b=4, budgets=(2048, 1024, 512, 256), n_spans=16)
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    ref = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True)
    K, V, pg = _paged(tens, page_size, seed=5, order=order)
    got = api.evict(p, K, V, tens["Q"], want_scores=True, paging=pg)
    torch.cuda.synchronize()
    for k in ("idx", "Kc", "Vc", "scores"):
        assert torch.equal(got[k], ref[k]), k
