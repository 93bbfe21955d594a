"""Block-granular selection (dge_problem.select_block), the selection ladder's fixed-block rung.

On scores whose fp32 block sums are exact (small multiples of 1/64) the GPU's kept set equals
the oracle's bit for bit, ties included; through dge_evict on real scores it equals the
oracle's applied to the GPU's own pooled scores except for blocks whose sums tie within fp32
rounding at the cut.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_33334_gb300 import _build, api, inputs
from parity import unit_index, unit_list, unit_rows

pytestmark = pytest.mark.gpu
WL = inputs.WORKLOADS


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    _build.build()


def _structure(idx, n, s0, tail, budget, bs):
    P = n - tail
    assert len(idx) == budget and np.all(np.diff(idx) > 0)
    assert set(range(s0)) <= set(idx.tolist()) and set(range(P, n)) <= set(idx.tolist())
    blocks = {}
    for j in idx.tolist():
        if s0 <= j < P:
            blocks.setdefault((j - s0) // bs, []).append(j)
    partial = [k for k, js in blocks.items() if len(js) < min(bs, P - (s0 + k * bs))]
    assert len(partial) <= 1
    for k in partial:
        assert blocks[k] == list(range(s0 + k * bs, s0 + k * bs + len(blocks[k])))


@pytest.mark.parametrize("bs", [2, 8, 16, 32])
def test_block_select_exact_on_given_scores(bs):
    wl = WL["c1_tiny"].with_(L=2, budgets=(128, 300))
    p = api.problem_from_workload(wl)
    p.select_block = bs
    rng = np.random.default_rng(bs)
    base = (rng.integers(0, 8, size=(p.U, p.P)) / 64.0).astype(np.float32)   # exact sums, ties
    idx = api.select(p, torch.from_numpy(base).cuda()).cpu().numpy()
    for (l, b, h) in unit_list(wl):
        u = unit_index(wl, l, b, h)
        r0, r1 = unit_rows(wl, l, b, h)
        want = oracle.select_blocks(base[u].astype(np.float64), wl.n, wl.sinks, wl.tail,
                                    wl.budgets[l], bs)
        np.testing.assert_array_equal(idx[r0:r1], want)
        _structure(idx[r0:r1], wl.n, wl.sinks, wl.tail, wl.budgets[l], bs)


@pytest.mark.parametrize("name,bs", [("c2_small", 8), ("c3_small", 32), ("c4_small", 16)])
def test_block_select_through_evict(name, bs):
    wls = {"c2_small": WL["c2_8b_8k"].with_(L=2, n=3000),
           "c3_small": WL["c3_8b_32k_pyramid"].with_(L=3, b=2, n=4500, budgets=(900, 610, 301),
                                                     n_spans=8),
           "c4_small": WL["c4_h2o_8k"].with_(L=1, b=2, n=1000, budgets=(200,))}
    wl = wls[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    p.select_block = bs
    out = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True)
    torch.cuda.synchronize()
    sc = out["scores"].double().cpu().numpy()
    for (l, b, h) in unit_list(wl):
        u = unit_index(wl, l, b, h)
        r0, r1 = unit_rows(wl, l, b, h)
        got = out["idx"][r0:r1].cpu().numpy()
        _structure(got, wl.n, wl.sinks, wl.tail, wl.budgets[l], bs)
        want = oracle.select_blocks(sc[u], wl.n, wl.sinks, wl.tail, wl.budgets[l], bs)
        diff = set(got.tolist()) ^ set(want.tolist())
        if diff:                       # only blocks tied within fp32 rounding at the cut
            P = wl.n - wl.tail
            sums = {}
            for k, lo in enumerate(range(wl.sinks, P, bs)):
                t = 0.0
                for j in range(lo, min(lo + bs, P)):
                    t += sc[u][j]
                sums[k] = t
            cut = [sums[(j - wl.sinks) // bs] for j in diff]
            assert max(cut) - min(cut) <= 1e-5 * max(cut), (name, (l, b, h), sorted(diff))
        assert torch.equal(out["Kc"][r0:r1], tens["K"][l, b, h][torch.from_numpy(got).long().cuda()])
