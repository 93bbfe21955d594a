"""Pins of the fp64 oracle against facts fixed by the paper and by mathematics.

None of these compare the oracle with itself: each check uses brute force in
pure Python, a library routine (numpy / scipy / torch), a closed form, an
invariant, or a number printed in the paper (tests/golden/).
"""
import math
import os

import numpy as np
import pytest
import scipy.special
import torch

import oracle
from oracle import brute
from paper_2609_33334_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _bf16_bits(a):
    return inputs.bf16_bits(torch.as_tensor(np.asarray(a, dtype=np.float32)).to(torch.bfloat16))


def _bits_to_f64(bits):
    return (np.asarray(bits, dtype=np.uint32) << 16).view(np.float32).astype(np.float64)


def _rand_case(rng, U, R, n, d, spread=1.5):
    Q = _bf16_bits(rng.normal(0, spread, size=(U, R, d)))
    K = _bf16_bits(rng.normal(0, spread, size=(U, n, d)))
    return Q, K


@pytest.mark.parametrize("n,m,G,d,tail,h2o", [
    (1, 1, 1, 4, 0, False), (5, 2, 1, 4, 2, False), (17, 3, 2, 8, 3, False),
    (64, 4, 2, 8, 4, False), (64, 4, 2, 8, 1, False), (33, 1, 2, 4, 0, True),
    (64, 1, 1, 8, 5, True),
])
def test_oracle_matches_pure_python_brute_force(oracle_lib, n, m, G, d, tail, h2o):
    """Brute force (math.fsum over softmax rows) agrees with the C oracle to 1e-12."""
    rng = np.random.default_rng(n * 131 + m * 7 + G)
    rows = n if h2o else m
    R = G * rows
    pos = oracle.h2o_positions(n, G) if h2o else oracle.scored_positions(n, m, G)
    P = n - tail
    Q, K = _rand_case(rng, 2, R, n, d)
    raw = oracle.scores(Q, K, pos, P)
    for u in range(2):
        qf = _bits_to_f64(Q[u]).tolist()
        kf = _bits_to_f64(K[u]).tolist()
        ref = brute.scores(qf, kf, pos.tolist(), P, 1.0 / math.sqrt(d))
        np.testing.assert_allclose(raw[u], ref, rtol=1e-12, atol=1e-15)
        for kern in (1, 3, 7):
            np.testing.assert_allclose(oracle.pool(raw[u], oracle.POOL_MAX, kern),
                                       brute.max_pool(ref, kern), rtol=1e-12, atol=1e-15)
            np.testing.assert_allclose(oracle.pool(raw[u], oracle.POOL_AVG, kern),
                                       brute.avg_pool(ref, kern), rtol=1e-12, atol=1e-15)


def test_single_row_is_numpy_softmax(oracle_lib):
    """One row, one head, no pooling: raw scores are scipy's softmax of the logits."""
    rng = np.random.default_rng(5)
    n, d = 300, 16
    Q, K = _rand_case(rng, 1, 1, n, d)
    pos = oracle.scored_positions(n, 1, 1)           # the row sits at position n-1
    raw = oracle.scores(Q, K, pos, n)
    logits = _bits_to_f64(K[0]) @ _bits_to_f64(Q[0, 0]) / math.sqrt(d)
    np.testing.assert_allclose(raw[0], scipy.special.softmax(logits), rtol=1e-12, atol=1e-18)


def test_lse_is_logsumexp_and_rows_sum_to_one(oracle_lib):
    """lse matches scipy logsumexp; with every position scored the total is R."""
    rng = np.random.default_rng(6)
    n, m, G, d = 200, 5, 3, 8
    Q, K = _rand_case(rng, 2, G * m, n, d, spread=2.0)
    pos = oracle.scored_positions(n, m, G)
    raw, lse = oracle.scores(Q, K, pos, n, want_lse=True)
    for u in range(2):
        for r in range(G * m):
            vis = _bits_to_f64(K[u][:pos[r] + 1]) @ _bits_to_f64(Q[u, r]) / math.sqrt(d)
            assert lse[u, r] == pytest.approx(scipy.special.logsumexp(vis), rel=1e-13)
        assert raw[u].sum() == pytest.approx(G * m, rel=1e-12)


def test_uniform_keys_closed_form(oracle_lib):
    """All keys equal: each row is uniform over its visible keys, raw_j = sum_r 1/(p_r+1)."""
    n, m, G, d, tail = 97, 6, 2, 8, 6
    rng = np.random.default_rng(7)
    Q = _bf16_bits(rng.normal(size=(1, G * m, d)))
    K = np.tile(_bf16_bits(rng.normal(size=(1, 1, d))), (1, n, 1))
    pos = oracle.scored_positions(n, m, G)
    raw = oracle.scores(Q, K, pos, n - tail)
    expect = sum(1.0 / (p + 1) for p in pos)
    np.testing.assert_allclose(raw[0], expect, rtol=1e-12)


def test_h2o_uniform_harmonic_closed_form(oracle_lib):
    """H2O with zero queries: raw_j = G * (H_n - H_j), H_k the k-th harmonic number."""
    n, G, d = 150, 3, 4
    Q = np.zeros((1, G * n, d), dtype=np.uint16)     # bf16 zero
    K = _bf16_bits(np.random.default_rng(8).normal(size=(1, n, d)))
    raw = oracle.scores(Q, K, oracle.h2o_positions(n, G), n)
    H = np.concatenate([[0.0], np.cumsum(1.0 / np.arange(1, n + 1))])
    np.testing.assert_allclose(raw[0], G * (H[n] - H[np.arange(n)]), rtol=1e-12)


def test_selection_reduces_to_argsort_of_logits(oracle_lib):
    """m=1, G=1, no pooling: softmax is monotone, so the kept set is the top logits."""
    rng = np.random.default_rng(9)
    n, d, tail, budget = 500, 16, 1, 60
    Q, K = _rand_case(rng, 1, 1, n, d)
    raw = oracle.scores(Q, K, oracle.scored_positions(n, 1, 1), n - tail)[0]
    idx = oracle.select(raw, n, 0, tail, budget)
    logits = _bits_to_f64(K[0][:n - tail]) @ _bits_to_f64(Q[0, 0])
    order = np.lexsort((np.arange(n - tail), -logits))[:budget - tail]
    expect = np.concatenate([np.sort(order), np.arange(n - tail, n)])
    np.testing.assert_array_equal(idx, expect)


@pytest.mark.parametrize("kernel", [1, 3, 7, 9])
def test_pooling_matches_torch(oracle_lib, kernel):
    """MAX = torch max_pool1d (-inf padding); AVG = avg_pool1d with count_include_pad."""
    raw = np.random.default_rng(kernel).random(113)
    t = torch.from_numpy(raw)[None, None]
    mx = torch.nn.functional.max_pool1d(t, kernel, 1, kernel // 2)[0, 0].numpy()
    av = torch.nn.functional.avg_pool1d(t, kernel, 1, kernel // 2, count_include_pad=True)[0, 0]
    np.testing.assert_allclose(oracle.pool(raw, oracle.POOL_MAX, kernel), mx, rtol=0, atol=0)
    np.testing.assert_allclose(oracle.pool(raw, oracle.POOL_AVG, kernel), av.numpy(), rtol=1e-14)


def test_ties_go_to_lower_position(oracle_lib):
    """Equal scores at the threshold: the lowest positions are kept."""
    s = np.array([5.0, 1.0, 3.0, 3.0, 3.0, 3.0, 0.5, 3.0, 7.0, 0.0, 0.0])
    # n = 11, tail 2 -> candidates [0, 9); keep 4 = {8 (7.0), 0 (5.0), 2, 3 (first two 3.0s)}
    idx = oracle.select(s, 11, 0, 2, 6)
    np.testing.assert_array_equal(idx, [0, 2, 3, 8, 9, 10])
    # one protected sink: position 0 no longer competes, keep 4 of [1, 9) = {8, 2, 3, 4}
    idx = oracle.select(s, 11, 1, 2, 7)
    np.testing.assert_array_equal(idx, [0, 2, 3, 4, 8, 9, 10])


def test_select_invariants_and_degenerate_budgets(oracle_lib):
    rng = np.random.default_rng(10)
    n, tail, s0 = 257, 9, 4
    s = rng.random(n)
    for budget in (s0 + tail, s0 + tail + 1, 100, n):
        idx = oracle.select(s, n, s0, tail, budget)
        assert idx.shape == (budget,)
        assert np.all(np.diff(idx) > 0)
        assert set(range(s0)) <= set(idx.tolist())
        assert set(range(n - tail, n)) <= set(idx.tolist())
    np.testing.assert_array_equal(oracle.select(s, n, s0, tail, n), np.arange(n))
    with pytest.raises(ValueError):
        oracle.select(s, n, s0, tail, s0 + tail - 1)


def test_streaming_indices(oracle_lib):
    np.testing.assert_array_equal(oracle.streaming_indices(20, 4, 9),
                                  [0, 1, 2, 3, 15, 16, 17, 18, 19])
    np.testing.assert_array_equal(oracle.streaming_indices(9, 4, 9), np.arange(9))


def _read_golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]


def test_pyramid_budgets_reproduce_paper_examples(oracle_lib):
    """App. L's five worked PyramidKV schedules."""
    for row in _read_golden("pyramidkv_examples.txt"):
        B, w, L, which = int(row[0]), int(row[1]), int(row[2]), row[3]
        got = oracle.pyramid_budgets(B, w, L)
        want = [int(x) for x in row[4:]]
        if which == "all":
            assert set(got.tolist()) == set(want)
        else:
            k = int(which[4:])
            assert got[-k:].tolist() == want


def test_missed_mass_identity_on_gathered_cache(oracle_lib):
    """Sec. 3 identity / App. E Eq. evict-mass: o = (1 - beta) o_keep + beta mu_evict.

    o_keep is attention renormalised over the gathered (Kc, Vc); this fails if
    the gather copies any row other than the one its index names.
    """
    rng = np.random.default_rng(11)
    n, d, budget = 400, 16, 70
    K = _bf16_bits(rng.normal(size=(n, d)))
    V = _bf16_bits(rng.normal(size=(n, d)))
    idx = oracle.select(rng.random(n), n, 0, 5, budget)
    Kc, Vc = oracle.gather(K, idx), oracle.gather(V, idx)
    q = rng.normal(size=d)
    a = scipy.special.softmax(_bits_to_f64(K) @ q)
    o = a @ _bits_to_f64(V)
    keep = np.zeros(n, bool)
    keep[idx] = True
    beta = a[~keep].sum()
    mu_e = (a[~keep] @ _bits_to_f64(V)[~keep]) / beta
    o_keep = scipy.special.softmax(_bits_to_f64(Kc) @ q) @ _bits_to_f64(Vc)
    np.testing.assert_allclose((1 - beta) * o_keep + beta * mu_e, o, rtol=1e-10, atol=1e-12)
    # and the per-step error equals beta * |mu_E - mu_R| <= 2 beta rho_v
    vf = _bits_to_f64(V)
    rho = np.linalg.norm(vf - vf.mean(0), axis=1).max()
    err = np.linalg.norm(o - o_keep)
    assert err == pytest.approx(beta * np.linalg.norm(mu_e - o_keep), rel=1e-9)
    assert err <= 2 * beta * rho + 1e-12


def test_evicted_mass_from_kept_cache_normaliser(oracle_lib):
    """Eq. match: rho_q = sum over evicted visible keys of the row's softmax weights.

    The diagnostics compute it as 1 - exp(lse_hat - lse), with lse_hat the normaliser of the
    kept keys taken as a cache of length B (the observation rows in the kept tail keep their
    relative positions).  Pinned against the definition, summed by brute force (pure Python,
    math.fsum) over the evicted keys each row sees.
    """
    from oracle import brute
    rng = np.random.default_rng(12)
    n, d, m, G, budget = 90, 8, 3, 2, 30
    K = _bf16_bits(rng.normal(size=(n, d)))
    Q = _bf16_bits(rng.normal(size=(G * m, d)))
    pos = oracle.scored_positions(n, m, G)
    scale = 1.0 / np.sqrt(d)
    idx = oracle.select(rng.random(n - m), n, 0, m, budget)      # tail [n-m, n) kept
    _, lse = oracle.scores(Q[None], K[None], pos, n - m, scale, want_lse=True)
    _, lse_hat = oracle.scores(Q[None], oracle.gather(K, idx)[None],
                               oracle.scored_positions(budget, m, G), budget - m, scale,
                               want_lse=True)
    rho = -np.expm1(lse_hat[0] - lse[0])
    Kf = [[brute.bf16_to_float(x) for x in row] for row in K]
    kept = set(idx.tolist())
    for r in range(G * m):
        q = [brute.bf16_to_float(x) for x in Q[r]]
        a = brute.attention_row(q, Kf[:pos[r] + 1], scale)
        want = math.fsum(a[j] for j in range(pos[r] + 1) if j not in kept)
        assert rho[r] == pytest.approx(want, rel=1e-9, abs=1e-13)
    assert np.all((rho > 0) & (rho < 1))


def _blocks_brute(scores, n, s0, tail, budget, bs):
    """The block rule written out plainly: rank blocks by (sum desc, index asc) with a Python
    sort, take whole blocks while they fit, then a prefix of the first that does not."""
    P = n - tail
    keep = budget - s0 - tail
    blocks = []
    for k, lo in enumerate(range(s0, P, bs)):
        pos = list(range(lo, min(lo + bs, P)))
        total = 0.0                  # left to right, as the rule adds (not Python's sum())
        for j in pos:
            total += scores[j]
        blocks.append((-total, k, pos))
    blocks.sort(key=lambda t: (t[0], t[1]))
    kept, left = [], keep
    for _, _, pos in blocks:
        if left == 0:
            break
        take = pos if len(pos) <= left else pos[:left]
        kept += take
        left -= len(take)
    return sorted(range(s0)) + sorted(kept) + list(range(P, n))


def test_block_selection(oracle_lib):
    """The block-granular rule: bs = 1 is token selection exactly; a hand-worked case; a plain
    Python version of the rule on random scores with ties; whole blocks plus at most one
    prefix, exactly `budget` positions, ascending."""
    rng = np.random.default_rng(13)
    for trial in range(20):
        n, s0, tail = int(rng.integers(20, 300)), int(rng.integers(0, 5)), int(rng.integers(1, 12))
        P = n - tail
        budget = int(rng.integers(s0 + tail, n + 1))
        sc = rng.random(P).round(1)                  # many ties
        np.testing.assert_array_equal(oracle.select_blocks(sc, n, s0, tail, budget, 1),
                                      oracle.select(sc, n, s0, tail, budget))
        for bs in (2, 8, 16, 32):
            got = oracle.select_blocks(sc, n, s0, tail, budget, bs)
            assert got.tolist() == _blocks_brute(sc.tolist(), n, s0, tail, budget, bs)
            assert len(got) == budget and np.all(np.diff(got) > 0)
            cand = [j for j in got.tolist() if s0 <= j < P]
            blocks = {}
            for j in cand:
                blocks.setdefault((j - s0) // bs, []).append(j)
            partial = [k for k, js in blocks.items()
                       if len(js) < min(bs, P - (s0 + k * bs))]
            assert len(partial) <= 1
            for k in partial:                        # a prefix of its block
                assert blocks[k] == list(range(s0 + k * bs, s0 + k * bs + len(blocks[k])))
    # hand-worked: s0 = 1, tail = 2, n = 13 -> candidates [1, 11) in blocks of 4:
    # [1..4] sum 1.0, [5..8] sum 2.0, [9, 10] sum 1.5; keep = 7 - 1 - 2 = 4 ... then budget 9
    sc = np.array([9.0, .1, .2, .3, .4, .5, .5, .5, .5, 1.0, .5])
    np.testing.assert_array_equal(oracle.select_blocks(sc, 13, 1, 2, 7, 4),
                                  [0, 5, 6, 7, 8, 11, 12])          # block [5..8] whole
    np.testing.assert_array_equal(oracle.select_blocks(sc, 13, 1, 2, 9, 4),
                                  [0, 5, 6, 7, 8, 9, 10, 11, 12])   # then [9, 10] (fits)
    np.testing.assert_array_equal(oracle.select_blocks(sc, 13, 1, 2, 10, 4),
                                  [0, 1, 5, 6, 7, 8, 9, 10, 11, 12])  # then a prefix of [1..4]


def _span_kept_counts(wl):
    t = inputs.make_inputs(wl)
    Q, K, V = (inputs.bf16_bits(t[x]) for x in "QKV")
    starts = inputs.span_positions(wl, 0)
    kept_span, outs = 0, []
    for h in range(wl.Hkv):
        out = oracle.evict_unit(Q[0, 0, h * wl.G:(h + 1) * wl.G], K[0, 0, h], V[0, 0, h],
                                variant=wl.variant, m=wl.m, tail=wl.tail, sinks=wl.sinks,
                                budget=wl.budgets[0], pool_kind=wl.pool, kernel=wl.pool_kernel)
        kept = set(out["idx"].tolist())
        kept_span += sum(len(set(range(p0, p0 + wl.span_len)) & kept) for p0 in starts.tolist())
        np.testing.assert_array_equal(out["Kc"], K[0, 0, h][out["idx"]])
        np.testing.assert_array_equal(out["Vc"], V[0, 0, h][out["idx"]])
        outs.append(out)
    return kept_span, wl.Hkv * len(starts) * wl.span_len, outs


def test_planted_spans_with_known_kept_set(oracle_lib):
    """Spans whose keys have cosine 0.8 with a draft row, no sink: every span is kept.

    Each span key then carries ~e^6.4 of its draft row's weight against ~e^0.5
    for a noise key, so the kept set must contain all span positions (and the
    protected tail), whatever the noise realisation.
    """
    wl = inputs.WORKLOADS["c1_tiny"].with_(span_cos=0.8, sink_scale=1.0)
    kept, total, outs = _span_kept_counts(wl)
    assert kept == total
    for out in outs:
        assert set(range(wl.n - wl.tail, wl.n)) <= set(out["idx"].tolist())


def test_planted_spans_enriched_tiny_workload(oracle_lib):
    """The tiny workload as specified (cos 0.5, 8x sink): spans are strongly enriched.

    There the sink takes most of some draft rows' mass, so not every span
    survives; the kept fraction of span positions must still be well above
    the budget's base rate (B - t)/(n - t).
    """
    wl = inputs.WORKLOADS["c1_tiny"]
    kept, total, outs = _span_kept_counts(wl)
    base = (wl.budgets[0] - wl.tail) / (wl.n - wl.tail)
    assert kept / total >= 3 * base
    for out in outs:
        assert 0 in out["idx"]                              # the 8x sink
        assert out["raw"].sum() < wl.G * wl.m               # tail mass is not scored


def test_cache_byte_arithmetic_matches_paper():
    """App. G's cache sizes and App. E's ~60 MB/layer of prompt queries."""
    for row in _read_golden("cache_bytes.txt"):
        tok, L, H, d, tensors, eb = (int(x) for x in row[:6])
        nbytes = tok * L * H * d * tensors * eb
        if row[6] == "MB":
            assert round(nbytes / 1e6, 1) == float(row[7])
        else:
            assert round(nbytes / 2**30, 2) == float(row[6])
