"""dge_score_noalloc: scoring with the library's own fixed scratch array.

This entry point exists for callers that may not allocate device memory -- a
serving runtime that owns the whole device-memory plan, or code that must not
call cudaMalloc/cudaFree because they can synchronise the device while other
streams run.  It runs the same plan and kernels on the same bytes as dge_score
with a caller workspace, so its scores must equal those bit for bit, also when
consecutive calls reuse the array holding the previous call's data; and its
device-side reports must reach the caller through dge_noalloc_status.

Kept in a file of its own that pytest collects last, so that a run stopping at
the first failure has already run every other test.
"""
import ctypes

import pytest
import torch

from paper_2609_33334_gb300 import _build, api, inputs
from paper_2609_33334_gb300 import binding as B
from parity import assert_scores_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    _build.build()


def _scores_noalloc(p, K, Q):
    scores = torch.full((p.U, p.P), float("nan"), dtype=torch.float32, device=K.device)
    bufs = B.dge_buffers(K=B.tensor_desc(K), Q=B.tensor_desc(Q), scores=scores.data_ptr())
    B.dge_score_noalloc(p.c(), bufs, torch.cuda.current_stream().cuda_stream)
    return scores


def test_noalloc_scores_match_workspace_entry_point():
    cases = [
        inputs.WORKLOADS["c1_tiny"],
        inputs.WORKLOADS["c2_8b_8k"].with_(L=2, n=3000),
        inputs.WORKLOADS["c4_h2o_8k"].with_(L=1, b=1, n=700, budgets=(200,)),
        inputs.WORKLOADS["c1_tiny"],            # back to the first shape: stale scratch
    ]
    for wl in cases:
        tens = inputs.make_inputs(wl, device="cuda")
        p = api.problem_from_workload(wl)
        assert p.workspace_bytes() <= (32 << 20)
        ref = api.score(p, tens["K"], tens["Q"])          # caller-allocated workspace
        for _ in range(2):                                  # two calls in a row
            got = _scores_noalloc(p, tens["K"], tens["Q"])
            stream = torch.cuda.current_stream().cuda_stream
            assert B.dge_noalloc_status(stream) == B.DGE_OK
            assert torch.equal(got, ref), wl.name
            for u in range(p.U):
                assert_scores_close(got[u].cpu().numpy(), ref[u].double().cpu().numpy(),
                                    f"{wl.name} unit {u}")


def test_noalloc_reports_device_timeout():
    """A device-side wait that gives up inside dge_score_noalloc is reported by
    dge_noalloc_status (the status word lives in the built-in array), and the next call is
    correct again."""
    wl = inputs.WORKLOADS["c1_tiny"]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    ref = api.score(p, tens["K"], tens["Q"])
    stream = torch.cuda.current_stream().cuda_stream
    _scores_noalloc(p, tens["K"], tens["Q"])
    assert B.dge_noalloc_status(stream) == B.DGE_OK
    B.dge_debug_set_waits(50_000_000, 1)
    try:
        _scores_noalloc(p, tens["K"], tens["Q"])
        status = B.dge_noalloc_status(stream)
    finally:
        B.dge_debug_set_waits(0, 0)
    assert status == B.DGE_ERR_DEVICE_TIMEOUT
    got = _scores_noalloc(p, tens["K"], tens["Q"])
    assert B.dge_noalloc_status(stream) == B.DGE_OK
    assert torch.equal(got, ref)


def test_noalloc_rejects_problems_larger_than_its_buffer():
    wl = inputs.WORKLOADS["c3_8b_32k_pyramid"]
    p = api.problem_from_workload(wl)
    assert p.workspace_bytes() > (32 << 20)
    bufs = B.dge_buffers(scores=0x1000)
    rc = B._lib().dge_score_noalloc(ctypes.byref(p.c()), ctypes.byref(bufs), None)
    assert rc == B.DGE_ERR_WORKSPACE_TOO_SMALL
    assert "built-in buffer" in B.dge_last_error()
