"""Eviction diagnostics (dge_diagnostics): per-row evicted mass, per-unit attention-matching
loss and retained-run length, against the oracle.

The reference evicted mass of a row is 1 - exp(lse_hat - lse), lse from the oracle over the
whole cache and lse_hat from the oracle over the unit's kept keys (the GPU's own indices) as a
cache of length B -- the composition pinned against the definition in test_oracle.py.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_33334_gb300 import _build, api, inputs
from paper_2609_33334_gb300 import binding as B
from parity import oracle_units, unit_bits, unit_index, unit_list, unit_rows

pytestmark = pytest.mark.gpu
WL = inputs.WORKLOADS

CASES = {
    "c1_tiny": WL["c1_tiny"],
    "c2_small": WL["c2_8b_8k"].with_(L=2, n=3000),
    "c3_small": WL["c3_8b_32k_pyramid"].with_(L=3, b=2, n=4500, budgets=(900, 610, 301),
                                              n_spans=8),
    "keep_all": WL["c1_tiny"].with_(budgets=(1024,)),
}


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    _build.build()


@pytest.mark.parametrize("name", sorted(CASES))
def test_diagnostics_match_oracle(name):
    wl = CASES[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    out = api.evict(p, tens["K"], tens["V"], tens["Q"], want_lse=True)
    diag = api.diagnostics(p, tens["Q"], out, out["lse"])
    torch.cuda.synchronize()
    rho = diag["evicted_mass"].reshape(p.U, -1).double().cpu().numpy()
    lm = diag["l_match"].double().cpu().numpy()
    rl = diag["run_length"].double().cpu().numpy()
    units = unit_list(wl)
    refs = oracle_units(wl, tens, units, want_lse=True)
    G, m = wl.G, wl.m
    for (l, b, h) in units:
        u = unit_index(wl, l, b, h)
        r0, r1 = unit_rows(wl, l, b, h)
        idx = out["idx"][r0:r1].cpu().numpy().astype(np.int64)
        Bl = r1 - r0
        Qg = inputs.bf16_bits(tens["Q"][l, b, h * G:(h + 1) * G]).reshape(-1, wl.d)
        Kk = oracle.gather(unit_bits(tens["K"], l, b, h), idx)
        _, lse_hat = oracle.scores(Qg[None], Kk[None], oracle.scored_positions(Bl, m, G),
                                   Bl - wl.tail, want_lse=True)
        d_ref = refs[(l, b, h)]["lse"] - lse_hat[0]
        rho_ref = -np.expm1(-d_ref)
        np.testing.assert_allclose(rho[u], rho_ref, rtol=1e-3, atol=2e-5,
                                   err_msg=f"{name} evicted mass unit {(l, b, h)}")
        assert lm[u] == pytest.approx(d_ref.mean(), rel=1e-3, abs=2e-5)
        runs = 1 + int(np.count_nonzero(np.diff(idx) != 1))
        assert rl[u] == pytest.approx(Bl / runs, rel=1e-6)
    if name == "keep_all":
        assert np.all(np.abs(rho) <= 2e-5) and np.all(rl == wl.n)


def test_diagnostics_need_observation_rows_in_the_tail():
    wl = WL["c1_tiny"].with_(budgets=(60,))
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    p.tail = 4                                              # m = 10 > tail
    out = api.evict(p, tens["K"], tens["V"], tens["Q"], want_lse=True)
    with pytest.raises(B.DgeError) as e:
        api.diagnostics(p, tens["Q"], out, out["lse"])
    assert "UNSUPPORTED" in str(e.value).upper() or f"-> {B.DGE_ERR_UNSUPPORTED}" in str(e.value)


@pytest.mark.parametrize("name", ["c1_tiny", "c3_small"])
def test_heldout_query_evicted_mass_identity(name):
    """Eq. evict-mass on held-out decode queries: |o - o~| = m(E) |mu_E - mu_R|, and each of
    m(E), |o - o~| against a float64 evaluation of the definitions."""
    wl = CASES[name]
    tens = inputs.make_inputs(wl, device="cuda")
    p = api.problem_from_workload(wl)
    out = api.evict(p, tens["K"], tens["V"], tens["Q"], want_lse=True)
    g = torch.Generator(device="cuda").manual_seed(7)
    hq = torch.randn((wl.L, wl.b, wl.Hq, wl.d), generator=g, device="cuda").to(torch.bfloat16)
    diag = api.diagnostics(p, tens["Q"], out, out["lse"], heldout_q=hq, K=tens["K"],
                           V=tens["V"])
    torch.cuda.synchronize()
    mass, err, gap = (diag[k].double().cpu().numpy() for k in
                      ("heldout_mass", "heldout_err", "heldout_gap"))
    np.testing.assert_allclose(err, gap, rtol=2e-3, atol=1e-5)
    scale = 1.0 / np.sqrt(wl.d)
    Hf = hq.double().cpu().numpy()
    for (l, b, hq_i) in [(0, 0, 0), (wl.L - 1, wl.b - 1, wl.Hq - 1), (0, wl.b - 1, wl.G)]:
        h = hq_i // wl.G
        r0, r1 = unit_rows(wl, l, b, h)
        keep = np.zeros(wl.n, bool)
        keep[out["idx"][r0:r1].cpu().numpy()] = True
        Kf = tens["K"][l, b, h].double().cpu().numpy()
        Vf = tens["V"][l, b, h].double().cpu().numpy()
        s = Kf @ Hf[l, b, hq_i] * scale
        a = np.exp(s - s.max())
        a /= a.sum()
        m = a[~keep].sum()
        o = a @ Vf
        mu_r = (a[keep] @ Vf[keep]) / (1 - m)
        assert mass[l, b, hq_i] == pytest.approx(m, rel=1e-4, abs=1e-7)
        assert err[l, b, hq_i] == pytest.approx(np.linalg.norm(o - mu_r), rel=2e-3, abs=1e-5)
