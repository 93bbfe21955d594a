"""The workspace needs no initialisation: garbage left in it cannot reach the results.

include/dge.h promises that a workspace's contents need no initialisation.  Every call must
therefore clear or overwrite, before it reads them, the cross-CTA chunk counters, the range
flags and the recompute list, the fixed-point column sums of row blocks and the partial sums.
Each case runs dge_evict once on a zeroed workspace and then on workspaces filled with 0xFF
bytes and with NaN; the outputs must be byte-identical.
"""
import pytest
import torch

from paper_2609_33334_gb300 import _build, api, inputs

pytestmark = pytest.mark.gpu
WL = inputs.WORKLOADS

CASES = {
    "c3_small": WL["c3_8b_32k_pyramid"].with_(L=3, b=2, n=4500, budgets=(900, 610, 301),
                                              n_spans=8),
    "c5_small": WL["c5_70b_128k"].with_(L=1, n=5000, budgets=(700,), n_spans=16),  # row blocks
    "c4_small": WL["c4_h2o_8k"].with_(L=1, b=2, n=1000, budgets=(200,)),           # H2O
    "long_p": WL["c1_tiny"].with_(n=33500, budgets=(600,), n_spans=0),            # P > 32768
}


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    _build.build()


def _fill(ws, how):
    if how == "zero":
        ws.zero_()
    elif how == "ones":
        ws.fill_(0xFF)
    else:
        n = ws.numel() // 4 * 4
        ws[:n].view(torch.float32).fill_(float("nan"))


@pytest.mark.parametrize("name", sorted(CASES))
def test_poisoned_workspace_gives_identical_outputs(name):
    wl = CASES[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    ws = api.workspace(p, "cuda")
    outs = {}
    for how in ("zero", "ones", "nan"):
        _fill(ws, how)
        outs[how] = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True,
                              want_lse=True, ws=ws)
        torch.cuda.synchronize()
        assert api.device_status(ws) == 0, how
    for how in ("ones", "nan"):
        for k in ("idx", "Kc", "Vc", "scores", "lse"):
            assert torch.equal(outs[how][k].view(torch.uint8), outs["zero"][k].view(torch.uint8)), \
                (how, k)


def test_poisoned_workspace_large_logits():
    """Units whose row sums leave fp32's range (queries x24) go through the recompute list,
    which the call must clear too."""
    wl = WL["c2_8b_8k"].with_(L=1, n=2000)
    tens = inputs.make_inputs(wl, device="cuda")
    tens["Q"] = (tens["Q"].float() * 24).to(torch.bfloat16)
    p = api.problem_from_workload(wl)
    ws = api.workspace(p, "cuda")
    outs = {}
    for how in ("zero", "ones", "nan"):
        _fill(ws, how)
        outs[how] = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True,
                              want_lse=True, ws=ws)
        torch.cuda.synchronize()
    for how in ("ones", "nan"):
        for k in ("idx", "Kc", "Vc", "scores", "lse"):
            assert torch.equal(outs[how][k].view(torch.uint8), outs["zero"][k].view(torch.uint8)), \
                (how, k)
