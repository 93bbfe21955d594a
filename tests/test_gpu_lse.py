"""Row normalisers in and out of the scoring (dge_buffers.lse_in / lse_out).

lse_out: the normalisers the two-pass scoring computes, checked against the
oracle's fp64 log-sum-exp.  lse_in: scores computed in one pass from normalisers
the caller supplies (here the oracle's, rounded to fp32, as an attention pass
would hand them over), checked against the oracle's scores and kept sets, on the
tensor-core path, the warp-level path and H2O.
"""
import numpy as np
import pytest
import torch

from paper_2609_33334_gb300 import _build, api, inputs
from parity import check_kept, compare_unit, oracle_units, unit_list, unit_index, unit_rows

pytestmark = pytest.mark.gpu
WL = inputs.WORKLOADS

CASES = {
    "c2_small": WL["c2_8b_8k"].with_(L=2, n=3000),                     # tensor-core path
    "c3_small": WL["c3_8b_32k_pyramid"].with_(L=2, b=2, n=4500, budgets=(900, 610),
                                              n_spans=8),
    "c1_tiny": WL["c1_tiny"],
    "c4_small": WL["c4_h2o_8k"].with_(L=1, b=2, n=1000, budgets=(200,)),   # H2O
    "c5_small": WL["c5_70b_128k"].with_(L=1, n=3000, budgets=(700,), n_spans=8),  # R = 528
}


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    _build.build()


@pytest.fixture(params=["auto", "mma"])
def kernel_choice(request, monkeypatch):
    if request.param == "mma":
        monkeypatch.setenv("DGE_SCORE_KERNEL", "mma")
    return request.param


def _oracle(wl, tens):
    units = unit_list(wl)
    return units, oracle_units(wl, tens, units, want_lse=True)


@pytest.mark.parametrize("name", sorted(CASES))
def test_lse_out_matches_oracle(name, kernel_choice):
    wl = CASES[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    out = api.evict(p, tens["K"], tens["V"], tens["Q"], want_lse=True)
    torch.cuda.synchronize()
    assert tuple(out["lse"].shape) == p.lse_shape
    got = out["lse"].reshape(p.U, -1).double().cpu().numpy()
    units, refs = _oracle(wl, tens)
    for (l, b, h) in units:
        ref = refs[(l, b, h)]["lse"]
        g = got[unit_index(wl, l, b, h)]
        np.testing.assert_allclose(g, ref, rtol=1e-6, atol=2e-5,
                                   err_msg=f"{name} lse unit {(l, b, h)}")


@pytest.mark.parametrize("name", sorted(CASES))
def test_supplied_lse_scores_match_oracle(name, kernel_choice):
    wl = CASES[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    units, refs = _oracle(wl, tens)
    lse = np.zeros((p.U, int(np.prod(p.lse_shape)) // p.U), dtype=np.float32)
    for (l, b, h) in units:
        lse[unit_index(wl, l, b, h)] = refs[(l, b, h)]["lse"]
    lse_in = torch.from_numpy(lse).reshape(p.lse_shape).cuda()
    out = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True, lse_in=lse_in)
    torch.cuda.synchronize()
    assert out["lse"] is None
    for (l, b, h) in units:
        compare_unit(wl, out, tens, l, b, h, ref=refs[(l, b, h)])


def test_supplied_lse_round_trip_matches_two_pass():
    """Scores from the normalisers the two-pass scoring returned equal its own scores."""
    wl = CASES["c3_small"]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    two = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True, want_lse=True)
    one = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True,
                    lse_in=two["lse"].clone())
    torch.cuda.synchronize()
    a, b = two["scores"].double(), one["scores"].double()
    rel = ((a - b).abs() / a.abs().clamp_min(1e-6 * a.abs().max())).max().item()
    assert rel < 1e-4, rel
    refs = None
    for (l, bb, h) in unit_list(wl):
        r0, r1 = unit_rows(wl, l, bb, h)
        sa = set(two["idx"][r0:r1].tolist())
        sb = set(one["idx"][r0:r1].tolist())
        if sa != sb:   # only near-ties may differ
            u = unit_index(wl, l, bb, h)
            sc = a[u].cpu().numpy()
            keep = wl.budgets[l] - wl.sinks - wl.tail
            T = np.sort(sc[wl.sinks:p.P])[::-1][keep - 1]
            for j in sa ^ sb:
                assert abs(sc[j] - T) <= 1e-4 * abs(T)


def test_supplied_lse_full_size_sampled():
    """c3 at full size with supplied normalisers: sampled units against the oracle."""
    wl = WL["c3_8b_32k_pyramid"]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    two = api.evict(p, tens["K"], tens["V"], tens["Q"], want_lse=True)
    one = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True,
                    lse_in=two["lse"].clone())
    torch.cuda.synchronize()
    units = [(0, 0, 0), (13, 2, 5), (31, 3, 7)]
    refs = oracle_units(wl, tens, units, want_lse=True)
    got = two["lse"].reshape(p.U, -1).double().cpu().numpy()
    for (l, b, h) in units:
        np.testing.assert_allclose(got[unit_index(wl, l, b, h)], refs[(l, b, h)]["lse"],
                                   rtol=1e-6, atol=2e-5)
        compare_unit(wl, one, tens, l, b, h, ref=refs[(l, b, h)])
