"""Parity of the CUDA path (through the C ABI) with the fp64 oracle.

Small cases compare every unit element by element; the full-size workloads
run in the launch configuration bench.py times and are checked on sampled
units that the oracle computes one by one.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_33334_gb300 import _build, api, inputs
from parity import compare_unit, oracle_units, unit_list, unit_rows

pytestmark = pytest.mark.gpu

WL = inputs.WORKLOADS


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    _build.build()
    oracle.build()


def run(wl, want_scores=True, tens=None, **kw):
    tens = tens or inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    Q = tens["Q"] if wl.variant != inputs.STREAMING else None
    out = api.evict(p, tens["K"], tens["V"], Q, want_scores=want_scores and
                    wl.variant != inputs.STREAMING, **kw)
    torch.cuda.synchronize()
    return tens, out


def check_all(wl, tens, out, units=None):
    units = unit_list(wl) if units is None else units
    refs = oracle_units(wl, tens, units)
    diffs = 0
    for (l, b, h) in units:
        diffs += compare_unit(wl, out, tens, l, b, h, ref=refs[(l, b, h)])
    return diffs


# --- small cases: every unit ------------------------------------------------------------

def test_tiny_workload_matches_oracle():
    wl = WL["c1_tiny"]
    tens, out = run(wl)
    check_all(wl, tens, out)


SMALL = {
    # reduced-n / reduced-L variants of the larger workloads (ragged tails included)
    "c2_small": WL["c2_8b_8k"].with_(L=2, n=3000),
    "c3_small": WL["c3_8b_32k_pyramid"].with_(L=3, b=2, n=4500, budgets=(900, 610, 301),
                                              n_spans=8),
    "c4_small": WL["c4_h2o_8k"].with_(L=1, b=2, n=1000, budgets=(200,)),
    "c5_small": WL["c5_70b_128k"].with_(L=1, n=5000, budgets=(700,), n_spans=16),
    "slm_small": WL["c5_slm"].with_(L=2, n=5000, budgets=(700, 300), n_spans=0),
    # edge cases
    "keep_none": WL["c1_tiny"].with_(budgets=(10,)),                   # B == tail
    "keep_all": WL["c1_tiny"].with_(budgets=(1024,)),                  # B == n
    "one_row": WL["c1_tiny"].with_(Hq=2, Hkv=2, w=1, k=0, budgets=(40,), n_spans=0),
    "short_cache": WL["c1_tiny"].with_(n=37, budgets=(20,), n_spans=0),
    "sinks_scored": WL["c1_tiny"].with_(sinks=4, budgets=(100,)),
    "no_pool": WL["c1_tiny"].with_(pool=inputs.POOL_NONE, pool_kernel=1),
    "long_p": WL["c1_tiny"].with_(n=33500, budgets=(600,), n_spans=0),  # P > 32768
    # longer rows pool tile by tile (32768 positions a tile): avg-7 over two tiles, and max-5
    # (radius known only at run time) over three
    "long_p_avg": WL["c1_tiny"].with_(n=33500, budgets=(600,), n_spans=0, pool=inputs.POOL_AVG),
    "long_p_max5": WL["c1_tiny"].with_(n=70000, budgets=(2000,), n_spans=0, pool_kernel=5),
    # the fused pooling reads whole 128-position chunks: P = 32768 exactly (the largest fused
    # row, no partial chunk) and P = 129 (one chunk and one position)
    "p_32768": WL["c1_tiny"].with_(n=32778, budgets=(700,), n_spans=0),
    "p_129": WL["c1_tiny"].with_(n=139, budgets=(60,), n_spans=0),
    "p_32768_avg": WL["c1_tiny"].with_(n=32778, budgets=(700,), n_spans=0,
                                       pool=inputs.POOL_AVG),
    "avg_pool_31": WL["c1_tiny"].with_(pool=inputs.POOL_AVG, pool_kernel=31),
    "max_pool_3_d128": WL["c1_tiny"].with_(d=128, pool_kernel=3),
    "gqa8_ragged": WL["c1_tiny"].with_(Hq=16, Hkv=2, n=2117, budgets=(333,)),
    "h2o_tiny": WL["c4_h2o_8k"].with_(L=1, b=1, Hq=4, Hkv=2, d=64, n=300, budgets=(100,)),
    # H2O query blocks (phase 1 / phase 2): G = 5 gives 25 / 28 positions x 5 heads = 125 / 140
    # rows (3 / 4 padded columns), G = 8 gives 16 / 18 positions, G = 1 single-head blocks of
    # 128 / 144 positions
    "h2o_g5_padded": WL["c4_h2o_8k"].with_(L=1, b=1, Hq=10, Hkv=2, d=64, n=777, budgets=(200,)),
    "h2o_g8": WL["c4_h2o_8k"].with_(L=1, b=1, Hq=16, Hkv=2, n=500, budgets=(150,)),
    "h2o_g1": WL["c4_h2o_8k"].with_(L=2, b=1, Hq=2, Hkv=2, n=403, budgets=(120, 90)),
    # G = 9: fewer than 16 positions per 128-row block, so the warp-level kernels score it
    "h2o_g9": WL["c4_h2o_8k"].with_(L=1, b=1, Hq=18, Hkv=2, d=64, n=300, budgets=(100,)),
    "slm_keep_all": WL["c5_slm"].with_(L=1, n=300, Hq=8, Hkv=2, budgets=(300,), n_spans=0),
}


@pytest.mark.parametrize("name", list(SMALL))
def test_small_cases_match_oracle(name):
    wl = SMALL[name]
    tens, out = run(wl)
    check_all(wl, tens, out)


def test_strided_views_match_contiguous():
    """K/V/Q as strided views of larger buffers give the same result."""
    wl = WL["c1_tiny"].with_(L=2, b=2, budgets=(128, 64))
    tens = inputs.make_inputs(wl, device="cuda")
    big = {}
    for k, t in tens.items():
        shape = list(t.shape)
        shape[3] += 24          # extra positions / rows per head
        buf = torch.zeros(shape[:4] + [shape[4] + 64], dtype=t.dtype, device="cuda")
        view = buf[:, :, :, 5:5 + t.shape[3], 32:32 + t.shape[4]]
        view.copy_(t)
        big[k] = view
    p = api.problem_from_workload(wl)
    a = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True)
    b = api.evict(p, big["K"], big["V"], big["Q"], want_scores=True)
    torch.cuda.synchronize()
    for k in ("idx", "Kc", "Vc", "scores"):
        assert torch.equal(a[k], b[k]), k


def test_runs_are_bit_identical():
    """Re-runs reproduce every output byte (deterministic reductions)."""
    wl = SMALL["c3_small"]
    tens, a = run(wl)
    _, b = run(wl, tens=tens)
    for k in ("idx", "Kc", "Vc", "scores"):
        assert torch.equal(a[k], b[k]), k


@pytest.mark.parametrize("name", ["c2_small", "c3_small", "no_pool", "keep_none", "keep_all",
                                  "long_p", "long_p_avg", "long_p_max5", "p_32768",
                                  "p_32768_avg", "p_129"])
def test_separate_calls_match_fused(name):
    """dge_score -> dge_select -> dge_compact equals dge_evict, bit for bit.

    dge_evict pools and selects in one kernel (one for P <= 32768, one for longer rows) while
    the separate calls run the pooling and selection kernels; max-, avg- and no pooling, the
    degenerate budgets, and rows longer than 32768 positions."""
    wl = SMALL[name]
    tens, fused = run(wl)
    p = api.problem_from_workload(wl)
    s = api.score(p, tens["K"], tens["Q"])
    idx = api.select(p, s)
    Kc, Vc = api.compact(p, idx, tens["K"], tens["V"])
    torch.cuda.synchronize()
    assert torch.equal(s, fused["scores"])
    assert torch.equal(idx, fused["idx"])
    assert torch.equal(Kc, fused["Kc"]) and torch.equal(Vc, fused["Vc"])


def test_select_on_oracle_scores_is_exact():
    """With identical float32 scores on both sides, the kept set is identical."""
    wl = WL["c1_tiny"].with_(L=2, budgets=(128, 200))
    rng = np.random.default_rng(3)
    p = api.problem_from_workload(wl)
    # plateaus of equal values (as max-pooling makes) plus random values
    base = rng.random((p.U, p.P)).astype(np.float32)
    base[:, 100:140] = 0.75
    base[:, 500:520] = base[:, 500:501]
    scores = torch.from_numpy(base).cuda()
    idx = api.select(p, scores).cpu().numpy()
    for (l, b, h) in unit_list(wl):
        u = (l * wl.b + b) * wl.Hkv + h
        want = oracle.select(base[u].astype(np.float64), wl.n, wl.sinks, wl.tail, wl.budgets[l])
        r0, r1 = unit_rows(wl, l, b, h)
        np.testing.assert_array_equal(idx[r0:r1], want)


def test_compact_out_of_range_index_reports_status():
    """A bad index is skipped and reported through the status word, not a fault."""
    wl = WL["c1_tiny"]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    idx = torch.arange(p.packed_rows(), dtype=torch.int32, device="cuda")
    idx[5] = wl.n + 3
    ws = api.workspace(p, "cuda")
    ws.zero_()
    Kc, Vc = api.compact(p, idx, tens["K"], tens["V"], ws=ws)
    assert api.device_status(ws) == 1
    assert api.device_status(ws) == 0          # reading clears it
    good = idx.clone()
    good[5] = 5
    Kc2, _ = api.compact(p, good, tens["K"], tens["V"])
    torch.cuda.synchronize()
    assert torch.equal(Kc[:5], Kc2[:5]) and torch.equal(Kc[6:], Kc2[6:])


# --- full-size workloads, sampled units --------------------------------------------------

FULL = ["c2_8b_8k", "c3_8b_32k_pyramid", "c4_h2o_8k", "c5_70b_128k", "c5_slm"]


def sample_units(wl, k=3, seed=0):
    U = wl.L * wl.b * wl.Hkv
    rng = np.random.default_rng(seed)
    picks = {0, U - 1} | set(rng.choice(U, size=min(k, U), replace=False).tolist())
    return sorted(picks)


@pytest.mark.parametrize("name", FULL)
def test_full_size_sampled_units(name):
    wl = WL[name]
    tens, out = run(wl)
    units = unit_list(wl, sample_units(wl, k=2 if name in ("c4_h2o_8k", "c5_70b_128k") else 3))
    check_all(wl, tens, out, units)
    # properties over every unit: ascending, exact length, tail kept
    idx = out["idx"].cpu().numpy()
    start = 0
    for l in range(wl.L):
        B = wl.budgets[l]
        blk = idx[start:start + wl.b * wl.Hkv * B].reshape(-1, B)
        start += wl.b * wl.Hkv * B
        assert np.all(np.diff(blk, axis=1) > 0)
        if wl.tail:
            assert np.all(blk[:, -wl.tail:] == np.arange(wl.n - wl.tail, wl.n))
    del tens, out
    torch.cuda.empty_cache()


# --- the two scoring kernel families ----------------------------------------------------

@pytest.fixture
def mma_path(monkeypatch):
    """Force the warp-level (mma.sync) scoring kernels for the duration of a test."""
    monkeypatch.setenv("DGE_SCORE_KERNEL", "mma")
    yield


@pytest.mark.parametrize("name", ["c2_small", "c3_small", "gqa8_ragged", "short_cache"])
def test_warp_level_path_matches_oracle(mma_path, name):
    wl = SMALL[name]
    tens, out = run(wl)
    check_all(wl, tens, out)


def _kernels_run(fn):
    from paper_2609_33334_gb300 import binding as B
    B.dge_profile_begin()
    fn()
    torch.cuda.synchronize()
    return {name for name, _, _ in B.dge_profile_end()}


@pytest.mark.parametrize("name,kernel", [("c2_small", "score_tc"), ("c1_tiny", "score_tc"),
                                         ("c5_small", "score_tc"), ("c4_small", "h2o_tc_colsum"),
                                         ("h2o_g8", "h2o_tc_colsum")])
def test_tensor_core_path_is_taken_where_eligible(name, kernel):
    wl = SMALL.get(name) or WL[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    names = _kernels_run(lambda: api.evict(p, tens["K"], tens["V"], tens["Q"]))
    assert kernel in names, names
    assert "colsum_rows" not in names and "colsum_keys" not in names, names


def test_h2o_large_groups_take_the_warp_level_kernels():
    """H2O with G = 9 cannot form 16-position query blocks: it is scored by the warp-level
    kernels (and matches the oracle in test_small_cases_match_oracle)."""
    wl = SMALL["h2o_g9"]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    names = _kernels_run(lambda: api.evict(p, tens["K"], tens["V"], tens["Q"]))
    assert "colsum_keys" in names and not any(n.startswith("h2o_tc") for n in names), names


def test_paths_agree_closely():
    """tcgen05 and mma.sync scores agree far inside the oracle tolerance."""
    import os
    wl = SMALL["c3_small"]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    a = api.score(p, tens["K"], tens["Q"])
    os.environ["DGE_SCORE_KERNEL"] = "mma"
    try:
        b = api.score(p, tens["K"], tens["Q"])
    finally:
        del os.environ["DGE_SCORE_KERNEL"]
    torch.cuda.synchronize()
    rel = ((a - b).abs() / b.abs().clamp_min(1e-30)).max().item()
    assert rel < 1e-4, rel


def test_row_blocks_are_deterministic_and_agree_with_warp_level_path():
    """R = 528 rows (8 query heads x 66) run as 4 row blocks of 2 heads on the tensor cores,
    their column sums added in fixed point: byte-identical across runs, and within 1e-4 of
    the warp-level path that takes all 528 rows at once."""
    import os
    wl = SMALL["c5_small"]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    a = api.score(p, tens["K"], tens["Q"])
    a2 = api.score(p, tens["K"], tens["Q"])
    os.environ["DGE_SCORE_KERNEL"] = "mma"
    try:
        b = api.score(p, tens["K"], tens["Q"])
    finally:
        del os.environ["DGE_SCORE_KERNEL"]
    torch.cuda.synchronize()
    assert torch.equal(a, a2)
    rel = ((a - b).abs() / b.abs().clamp_min(1e-6 * b.abs().max())).max().item()
    assert rel < 1e-4, rel


def test_h2o_paths_agree_and_repeat():
    """H2O on tcgen05 (query blocks, fp32 sums without a running maximum) agrees with the
    warp-level kernels far inside the oracle tolerance, and re-runs are byte-identical."""
    import os
    wl = SMALL["c4_small"]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    a = api.score(p, tens["K"], tens["Q"])
    a2 = api.score(p, tens["K"], tens["Q"])
    os.environ["DGE_SCORE_KERNEL"] = "mma"
    try:
        b = api.score(p, tens["K"], tens["Q"])
    finally:
        del os.environ["DGE_SCORE_KERNEL"]
    torch.cuda.synchronize()
    assert torch.equal(a, a2)
    rel = ((a - b).abs() / b.abs().clamp_min(1e-6 * b.abs().max())).max().item()
    assert rel < 1e-4, rel


def test_h2o_large_logits_are_recomputed_exactly():
    """H2O units whose fp32 row sums leave range are flagged by the tensor-core kernel and
    recomputed by the warp-level kernels (which carry a running maximum)."""
    wl = SMALL["c4_small"].with_(b=1)
    tens = inputs.make_inputs(wl, device="cuda")
    tens["Q"] = (tens["Q"].float() * 24.0).to(torch.bfloat16)
    tens, out = run(wl, tens=tens)
    check_all(wl, tens, out)


def test_large_logits_are_recomputed_exactly():
    """Logits far beyond fp32's unshifted exponent range take the recompute path."""
    wl = WL["c1_tiny"].with_(L=1, budgets=(128,))
    tens = inputs.make_inputs(wl, device="cuda")
    tens["Q"] = (tens["Q"].float() * 24.0).to(torch.bfloat16)   # logits ~ 100+ nats
    tens, out = run(wl, tens=tens)
    check_all(wl, tens, out)


def test_tail_shorter_than_observation_rows():
    """tail < m: observation rows see only their causal prefix of the scored range."""
    wl = WL["c1_tiny"].with_(n=700, n_spans=0)
    tens = inputs.make_inputs(wl, device="cuda")
    tail = 3
    p = api.problem_from_workload(wl)
    p.tail = tail
    out = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True)
    torch.cuda.synchronize()
    for h in range(wl.Hkv):
        Qg = inputs.bf16_bits(tens["Q"][0, 0, h * wl.G:(h + 1) * wl.G])
        ref = oracle.evict_unit(Qg, inputs.bf16_bits(tens["K"][0, 0, h]),
                                inputs.bf16_bits(tens["V"][0, 0, h]), variant=0, m=wl.m,
                                tail=tail, sinks=0, budget=wl.budgets[0], pool_kind=wl.pool,
                                kernel=wl.pool_kernel)
        from parity import assert_scores_close, check_kept
        assert_scores_close(out["scores"][h].cpu().numpy(), ref["pooled"])
        r0 = h * wl.budgets[0]
        check_kept(out["idx"][r0:r0 + wl.budgets[0]].cpu().numpy(), ref["pooled"], ref["idx"],
                   n=wl.n, sinks=0, tail=tail, budget=wl.budgets[0])
