"""Device-side failure detection on the GPU, with no fault: a bounded wait made to run out.

The tensor-core scoring kernel waits, for every phase-2 task, until all key chunks of the
task's unit have counted in their row sums.  The test hook dge_debug_set_waits shortens every
device-side wait to 50 ms and makes that count wait expect one chunk more than exists, so it
can only give up.  The kernel must then record DGE_ERR_DEVICE_TIMEOUT in the workspace status
word, stop, drain its copies and MMAs, free its tensor memory and return; the host reads the
status, and the next normal call in the same process must match the oracle.
"""
import time

import pytest
import torch

import oracle
from paper_2609_33334_gb300 import _build, api, inputs
from paper_2609_33334_gb300 import binding as B
from parity import compare_unit, oracle_units, unit_list

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    _build.build()
    oracle.build()


def _evict(wl, tens, ws):
    p = api.problem_from_workload(wl)
    return api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True, ws=ws)


@pytest.mark.parametrize("name", ["c1_tiny", "c2_small"])
def test_count_wait_runs_out_and_reports_timeout(name):
    wl = inputs.WORKLOADS["c1_tiny"] if name == "c1_tiny" else \
        inputs.WORKLOADS["c2_8b_8k"].with_(L=2, n=3000)
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    ws = api.workspace(p, "cuda")
    _evict(wl, tens, ws)                       # warm: the kernels are loaded
    assert api.device_status(ws) == B.DGE_OK
    B.dge_debug_set_waits(50_000_000, 1)
    try:
        t0 = time.perf_counter()
        _evict(wl, tens, ws)
        status = api.device_status(ws)         # synchronises the stream
        elapsed = time.perf_counter() - t0
    finally:
        B.dge_debug_set_waits(0, 0)
    assert status == B.DGE_ERR_DEVICE_TIMEOUT
    assert elapsed < 2.0, f"the wait gave up only after {elapsed:.3f} s"
    assert torch.cuda.is_available()
    # The context is intact: a normal call right after matches the oracle.
    out = _evict(wl, tens, ws)
    assert api.device_status(ws) == B.DGE_OK
    units = unit_list(wl)
    refs = oracle_units(wl, tens, units)
    for (l, b, h) in units:
        compare_unit(wl, out, tens, l, b, h, ref=refs[(l, b, h)])


def test_wait_limit_alone_changes_nothing():
    """A short limit that no wait reaches leaves the results bit-identical."""
    wl = inputs.WORKLOADS["c2_8b_8k"].with_(L=2, n=3000)
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    ws = api.workspace(p, "cuda")
    ref = _evict(wl, tens, ws)
    B.dge_debug_set_waits(200_000_000, 0)
    try:
        got = _evict(wl, tens, ws)
        status = api.device_status(ws)
    finally:
        B.dge_debug_set_waits(0, 0)
    assert status == B.DGE_OK
    for k in ("idx", "Kc", "Vc", "scores"):
        assert torch.equal(got[k], ref[k]), k


def test_negative_extra_chunks_rejected():
    with pytest.raises(B.DgeError):
        B.dge_debug_set_waits(0, -1)
