"""The roofline arithmetic of bench.py against the figures worked out for each configuration
from the cache shapes alone (bf16 rows of d values, K read once, the gather read and written):

- c2: 512 MiB of K + 256 MiB of gather = 805.3 MB a step, 262,144 KV tokens;
- c3: 8 GiB of K + 1.13 GiB of gather (the 2048 -> 256 ramp, 36,879 rows per head) = 9.80 GB,
  4,194,304 KV tokens, 1.442 ms at the measured 6795.5 GB/s copy;
- c4 (H2O): one causal pass over every cache position of the 4 query heads of each group,
  7.04e13 flop;
- c5: R = 528 rows against 131,072 keys, 1.13e13 flop for one pass; the SLM gather floor
  2.68 GB.
A slip in the byte or flop model (a dropped factor of 2, V left out of the gather, the tail
counted twice) would move one of these.
"""
import pytest

import bench
from paper_2609_33334_gb300 import inputs

WL = inputs.WORKLOADS


def test_c2_bytes_and_tokens():
    wl = WL["c2_8b_8k"]
    assert bench.step_bytes(wl) == 805_306_368
    assert bench.kernel_bytes(wl, "score_tc") == 512 * 2**20
    assert bench.tokens_per_step(wl) == 262_144


def test_c3_bytes_tokens_and_roofline_time():
    wl = WL["c3_8b_32k_pyramid"]
    assert sum(wl.budgets) == 36_879
    assert bench.kernel_bytes(wl, "score_tc") == 8 * 2**30
    assert bench.kernel_bytes(wl, "compact") == 4 * 4 * 8 * 36_879 * 128 * 2
    assert bench.step_bytes(wl) == 9_798_385_664
    assert bench.tokens_per_step(wl) == 4_194_304
    assert bench.step_bytes(wl) / 6795.5e9 * 1e3 == pytest.approx(1.442, abs=5e-4)


def test_h2o_flops_are_one_causal_pass():
    wl = WL["c4_h2o_8k"]
    n = wl.n
    assert bench.causal_pairs(wl, "h2o_tc_lse") == n * (n + 1) // 2
    flops = bench.kernel_flops(wl, "h2o_tc_lse")
    assert flops == pytest.approx(7.04e13, rel=2e-3)
    # the column pass covers keys below P only, so it is a little smaller
    assert bench.kernel_flops(wl, "h2o_tc_colsum") < flops


def test_c5_flops_and_slm_floor():
    wl = WL["c5_70b_128k"]
    assert wl.G * wl.m == 528
    assert bench.kernel_flops(wl, "score_tc") == pytest.approx(1.13e13, rel=5e-3)
    slm = WL["c5_slm"]
    assert bench.step_bytes(slm) == pytest.approx(2.68e9, rel=2e-3)
    assert bench.tokens_per_step(slm) == 10_485_760


def test_traffic_digest_follows_the_kernels_own_source(tmp_path, monkeypatch):
    """An ncu traffic figure stays valid while its kernel's own source and the shared headers
    are unchanged, whatever happens to another kernel's file, and is voided by either."""
    csrc = tmp_path / "paper_2609_33334_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (tmp_path / "include").mkdir()
    (tmp_path / "include" / "dge.h").write_text("// api\n")
    (tmp_path / "profiles").mkdir()
    for name, text in (("score_tc.cu", "a"), ("select_compact.cu", "b"), ("h2o_tc.cu", "c"),
                       ("common.cuh", "h")):
        (csrc / name).write_text(text)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    d_tc = bench.source_digest("score_tc")
    (tmp_path / "profiles" / "dram_traffic.txt").write_text(
        f"# header\nscore_tc c3_8b_32k_pyramid 123 {d_tc}\n")
    assert bench.ncu_traffic("score_tc", "c3_8b_32k_pyramid") == 123.0
    assert bench.ncu_traffic("score_tc", "c2_8b_8k") is None           # another workload
    (csrc / "select_compact.cu").write_text("b2")                        # another kernel's file
    assert bench.source_digest("score_tc") == d_tc
    assert bench.ncu_traffic("score_tc", "c3_8b_32k_pyramid") == 123.0
    (csrc / "score_tc.cu").write_text("a2")                              # its own file
    assert bench.ncu_traffic("score_tc", "c3_8b_32k_pyramid") is None
    (csrc / "score_tc.cu").write_text("a")
    assert bench.ncu_traffic("score_tc", "c3_8b_32k_pyramid") == 123.0
    (csrc / "common.cuh").write_text("h2")                               # a shared header
    assert bench.ncu_traffic("score_tc", "c3_8b_32k_pyramid") is None
    # the two H2O launches are one source file: one digest
    assert bench.source_digest("h2o_tc_lse") == bench.source_digest("h2o_tc_colsum")
