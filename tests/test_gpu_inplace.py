"""In-place compaction (dge_compact_inplace, dge_evict_inplace).

The kept rows of every unit move to the front of that unit's K and V rows, in ascending
position order; rows [B, n) keep their old contents.  Checked bit for bit against the
out-of-place gather (itself checked against the oracle in test_gpu_parity.py) and against the
original cache at the GPU's own indices.
"""
import numpy as np
import pytest
import torch

from paper_2609_33334_gb300 import _build, api, inputs
from paper_2609_33334_gb300 import binding as B
from parity import compare_unit, unit_list, unit_rows

pytestmark = pytest.mark.gpu
WL = inputs.WORKLOADS

CASES = {
    "c2_small": WL["c2_8b_8k"].with_(L=2, n=3000),
    "c3_small": WL["c3_8b_32k_pyramid"].with_(L=3, b=2, n=4500, budgets=(900, 610, 301),
                                              n_spans=8),
    "c4_small": WL["c4_h2o_8k"].with_(L=1, b=2, n=1000, budgets=(200,)),
    "slm_small": WL["c5_slm"].with_(L=2, n=5000, budgets=(700, 300), n_spans=0),
    "keep_all": WL["c1_tiny"].with_(budgets=(1024,)),
    "keep_none": WL["c1_tiny"].with_(budgets=(10,)),
}


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    _build.build()


@pytest.mark.parametrize("name", sorted(CASES))
def test_evict_inplace_matches_out_of_place(name):
    wl = CASES[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    Q = tens["Q"] if wl.variant != inputs.STREAMING else None
    ref = api.evict(p, tens["K"], tens["V"], Q, want_scores=wl.variant != inputs.STREAMING)
    K, V = tens["K"].clone(), tens["V"].clone()
    ws = api.workspace(p, "cuda")
    got = api.evict_inplace(p, K, V, Q, want_scores=wl.variant != inputs.STREAMING, ws=ws)
    torch.cuda.synchronize()
    assert api.device_status(ws) == 0
    assert torch.equal(got["idx"], ref["idx"])
    if ref["scores"] is not None:
        assert torch.equal(got["scores"], ref["scores"])
    for (l, b, h) in unit_list(wl):
        r0, r1 = unit_rows(wl, l, b, h)
        Bl = r1 - r0
        assert torch.equal(K[l, b, h, :Bl], ref["Kc"][r0:r1])
        assert torch.equal(V[l, b, h, :Bl], ref["Vc"][r0:r1])
        assert torch.equal(K[l, b, h, Bl:], tens["K"][l, b, h, Bl:])   # untouched tail
        assert torch.equal(V[l, b, h, Bl:], tens["V"][l, b, h, Bl:])


def test_compact_inplace_with_given_indices_and_oracle():
    """Selection out of place, then the in-place gather; the front rows against the oracle."""
    wl = CASES["c3_small"]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    out = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True)
    K, V = tens["K"].clone(), tens["V"].clone()
    api.compact_inplace(p, out["idx"], K, V)
    torch.cuda.synchronize()
    for (l, b, h) in unit_list(wl)[:4]:
        compare_unit(wl, out, tens, l, b, h)
        r0, r1 = unit_rows(wl, l, b, h)
        idx = out["idx"][r0:r1].long()
        assert torch.equal(K[l, b, h, :r1 - r0], tens["K"][l, b, h][idx])
        assert torch.equal(V[l, b, h, :r1 - r0], tens["V"][l, b, h][idx])


def test_compact_inplace_rejects_positions_before_their_row():
    """A descending index (position < its row) is reported and skipped, not copied."""
    wl = WL["c1_tiny"].with_(budgets=(64,))
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    idx = torch.arange(p.packed_rows(), dtype=torch.int32, device="cuda") % 64
    idx[5] = 2                                   # row 5 <- position 2: unsafe in place
    K, V = tens["K"].clone(), tens["V"].clone()
    ws = api.workspace(p, "cuda")
    ws.zero_()                                   # compaction calls report into the word as is
    api.compact_inplace(p, idx, K, V, ws=ws)
    assert api.device_status(ws) == B.DGE_ERR_INVALID_ARG
    assert torch.equal(K[0, 0, 0, 5], tens["K"][0, 0, 0, 5])       # skipped
    assert torch.equal(K, tens["K"])          # every other row maps to itself
