"""Exact selection on crafted score distributions, on both selection kernels.

The radix search starts at the highest bit in which a unit's smallest and largest key
differ, so the distributions here cover every way that bit can fall: all keys equal (no
pass at all), keys that differ only in the lowest bit, keys spanning the whole float range
(bit 31 differs through +0.0 / negative zero), ties across the threshold, and plateaus.
The expected kept set is computed here from its definition: the budget - sinks - tail
largest candidates, equal values broken by the lower position, plus sinks and tail,
ascending.  dge_select runs the separate selection kernel (shared-memory keys up to 53248
candidates, global-memory keys above); dge_evict without pooling runs the fused one.
"""
import numpy as np
import pytest
import torch

from paper_2609_33334_gb300 import _build, api, inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    _build.build()


def expected(scores, n, sinks, tail, budget):
    P = n - tail
    cand = np.arange(sinks, P)
    keep = budget - sinks - tail
    # larger value first, then lower position (stable sort on the negated value)
    order = cand[np.argsort(-scores[sinks:P].astype(np.float64), kind="stable")]
    kept = np.sort(order[:keep])
    return np.concatenate([np.arange(sinks), kept, np.arange(P, n)]).astype(np.int32)


def crafted(kind, P, rng):
    if kind == "all_equal":
        return np.full(P, 0.37, np.float32)
    if kind == "lowest_bit":
        base = np.float32(0.5).view(np.uint32)
        return (base + rng.integers(0, 2, P).astype(np.uint32)).view(np.float32)
    if kind == "two_values":
        return np.where(rng.random(P) < 0.3, 2.0, 1.0).astype(np.float32)
    if kind == "full_range":
        v = (10.0 ** rng.uniform(-38, 38, P)).astype(np.float32)
        v[rng.random(P) < 0.05] = 0.0
        v[rng.random(P) < 0.05] = -0.0
        return v
    if kind == "plateaus":
        v = rng.random(P).astype(np.float32)
        for s in range(0, P, 97):
            v[s:s + 40] = v[s]
        return v
    if kind == "tie_at_threshold":
        v = rng.random(P).astype(np.float32) * 0.5
        v[rng.choice(P, P // 4, replace=False)] = 0.75      # far more 0.75s than the budget
        return v
    raise ValueError(kind)


KINDS = ["all_equal", "lowest_bit", "two_values", "full_range", "plateaus", "tie_at_threshold"]


@pytest.mark.parametrize("n", [3000, 40000, 70000])   # shared-memory / larger-P paths
@pytest.mark.parametrize("kind", KINDS)
def test_select_crafted(kind, n):
    wl = inputs.WORKLOADS["c1_tiny"].with_(L=1, b=1, Hq=4, Hkv=2, n=n, budgets=(n // 7,),
                                           sinks=4)
    p = api.problem_from_workload(wl)
    rng = np.random.default_rng(len(kind) * 1000 + n)
    base = np.stack([crafted(kind, p.P, rng) for _ in range(p.U)])
    idx = api.select(p, torch.from_numpy(base).cuda()).cpu().numpy()
    B = wl.budgets[0]
    for u in range(p.U):
        np.testing.assert_array_equal(idx[u * B:(u + 1) * B],
                                      expected(base[u], n, wl.sinks, wl.tail, B), err_msg=kind)


@pytest.mark.parametrize("kind", ["all_equal", "tie_at_threshold"])
def test_fused_select_crafted(kind):
    """The fused pooling + selection kernel of dge_evict, pooling off, on crafted raw scores:
    scores enter through the library's own scoring, so craft them through K instead --
    identical key rows give identical (all-equal) raw scores."""
    wl = inputs.WORKLOADS["c1_tiny"].with_(L=1, b=1, Hq=4, Hkv=2, n=2000, budgets=(300,),
                                           pool=inputs.POOL_NONE, pool_kernel=1, n_spans=0)
    tens = inputs.make_inputs(wl, device="cuda")
    if kind == "all_equal":
        tens["K"][:] = tens["K"][:, :, :, :1, :]
    else:                                   # every third key the same: plateaus of ties
        tens["K"][:, :, :, ::3, :] = tens["K"][:, :, :, :1, :]
    p = api.problem_from_workload(wl)
    out = api.evict(p, tens["K"], tens["V"], tens["Q"], want_scores=True)
    torch.cuda.synchronize()
    scores = out["scores"].cpu().numpy()
    B = wl.budgets[0]
    idx = out["idx"].cpu().numpy()
    for u in range(p.U):
        np.testing.assert_array_equal(idx[u * B:(u + 1) * B],
                                      expected(scores[u], wl.n, wl.sinks, wl.tail, B))


@pytest.mark.parametrize("n", [3000, 40000, 70000])
@pytest.mark.parametrize("extra", [0, 1, -1])
def test_select_whole_bin(n, extra):
    """keep + extra large candidates (1000 plus less than 0.5, so they share exponent and top
    mantissa bits) among small ones.  With extra = 0 the first radix pass selects a bin that
    is kept whole, several distinct keys in it, and the passes stop there with the bin's
    lowest possible key as the threshold; with extra = +1 the threshold falls inside that bin,
    with extra = -1 among the small keys."""
    wl = inputs.WORKLOADS["c1_tiny"].with_(L=1, b=1, Hq=4, Hkv=2, n=n, budgets=(n // 7,),
                                           sinks=4)
    p = api.problem_from_workload(wl)
    B = wl.budgets[0]
    keep = B - wl.sinks - wl.tail
    rng = np.random.default_rng(n * 10 + extra + 1)
    base = rng.uniform(1e-4, 2e-4, (p.U, p.P)).astype(np.float32)
    for u in range(p.U):
        pos = rng.choice(np.arange(wl.sinks, p.P), keep + extra, replace=False)
        base[u, pos] = (1000.0 + 0.5 * rng.random(keep + extra)).astype(np.float32)
    idx = api.select(p, torch.from_numpy(base).cuda()).cpu().numpy()
    for u in range(p.U):
        np.testing.assert_array_equal(idx[u * B:(u + 1) * B],
                                      expected(base[u], n, wl.sinks, wl.tail, B),
                                      err_msg=f"extra {extra}")
