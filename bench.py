#!/usr/bin/env python3
"""Throughput of the DGE score -> select -> compact pass on GB300.

One step = one dge_evict call over the whole synthetic workload (every layer,
sequence and KV head: scores, pooling, top-B selection, K/V gather).  The
default workload is the 8B-shaped cache at 32K tokens with the PyramidKV
layer ramp (4 sequences x 32 layers x 32768 positions, w=32 + k=2 observation
rows, avg-pool 7).  Its 8 GiB of K plus 8 GiB of V exceed the 129 MB L2, so
no flush is needed between steps.

Prints one JSON line (rank 0).  ``--impl reference`` times the fp64 CPU oracle
on a bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import csv
import hashlib
import io
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "KV tokens scored+compacted/s at 1 GB300; achieved HBM GB/s vs peak"
UNIT = "KV tokens/s"
DEFAULT_WORKLOAD = "c3_8b_32k_pyramid"
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--layers", type=int, default=0,
                    help="run only the first N layers of the workload (small profiling case)")
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-one-pass", action="store_true",
                    help="skip the extra timing with the row normalisers supplied")
    ap.add_argument("--page-size", type=int, default=0,
                    help="lay K and V out as a paged cache with pages of this many positions")
    ap.add_argument("--page-head-major", action="store_true",
                    help="paged pools as [page][head][slot][d] instead of [page][slot][head][d]")
    ap.add_argument("--page-order", default="random", choices=["random", "sequential", "runs"],
                    help="order in which sequences get their pages")
    ap.add_argument("--lse-supplied", action="store_true",
                    help="time the one-pass scoring with the row normalisers supplied "
                         "(dge_buffers.lse_in), computed once before the timed region")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="target CPU time of the oracle baseline sample")
    return ap.parse_args()


# --- distributed plumbing -------------------------------------------------------------

def dist_setup(backend):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world, device):
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def select_workload(args):
    from paper_2609_33334_gb300 import inputs
    wl = inputs.WORKLOADS[args.workload]
    if args.layers and args.layers < wl.L:
        wl = wl.with_(name=f"{wl.name}[L={args.layers}]", L=args.layers,
                      budgets=wl.budgets[:args.layers])
    if getattr(args, "lse_supplied", False):
        wl = wl.with_(name=f"{wl.name}+lse")
    if getattr(args, "page_size", 0):
        hm = "h" if getattr(args, "page_head_major", False) else ""
        order = getattr(args, "page_order", "random")
        wl = wl.with_(name=f"{wl.name}+pages{args.page_size}{hm}"
                           + ("" if order == "random" else f"-{order}"))
    return wl


# --- workload arithmetic ------------------------------------------------------------------

def tokens_per_step(wl):
    """KV tokens: one cache position of one layer of one sequence (all KV heads)."""
    return wl.b * wl.L * wl.n


def kernel_bytes(wl, name):
    """Algorithmic DRAM bytes of one launch of a library kernel over the workload."""
    U = wl.L * wl.b * wl.Hkv
    P = wl.n - wl.tail
    rows = wl.b * wl.Hkv * sum(wl.budgets)
    row_bytes = wl.d * 2
    if name in ("lse_partial", "score_tc", "score_tc_lse"):
        return U * wl.n * row_bytes              # K read once (score_tc: both phases)
    if name in ("colsum_rows", "colsum_keys"):
        return U * P * row_bytes                 # K[0, P) read once
    if name == "compact":
        return 4 * rows * row_bytes              # K, V rows read + Kc, Vc written
    if name == "select":
        return U * P * 4 + rows * 4              # scores read + idx written
    if name == "pool_select":
        return U * P * 4 + rows * 4              # raw scores read + idx written
    if name == "pool":
        return 2 * U * P * 4
    if name == "combine_lse":
        return 0
    if name in ("h2o_tc_lse", "h2o_tc_colsum"):
        # every query row of the cache (G heads x n positions) plus the keys, read once
        q_bytes = U * wl.G * wl.n * row_bytes
        return q_bytes + U * (wl.n if name == "h2o_tc_lse" else P) * row_bytes
    return 0


def causal_pairs(wl, name):
    """(row, key) products of one H2O pass: rows see keys <= their position; the column pass
    only keys below P."""
    n, P = wl.n, wl.n - wl.tail
    if name in ("h2o_tc_colsum", "colsum_keys"):
        return P * n - P * (P - 1) // 2
    return n * (n + 1) // 2


def kernel_flops(wl, name):
    """Algorithmic tensor flops of one launch: one pass of Q.K^T over the rows the kernel
    scores (the second pass of a two-pass kernel is implementation work)."""
    U = wl.L * wl.b * wl.Hkv
    if wl.variant == 1:    # H2O: every cache position of the group's query heads, causal
        if name in ("h2o_tc_lse", "h2o_tc_colsum", "lse_partial", "colsum_keys"):
            return 2 * wl.d * wl.G * U * causal_pairs(wl, name)
        return 0
    if name in ("score_tc", "score_tc_lse", "lse_partial", "colsum_rows"):
        return 2 * wl.G * wl.m * wl.n * wl.d * U
    return 0


def step_bytes(wl):
    """Algorithmic bytes of one whole step: K once + the gather (reads and writes)."""
    if wl.variant == 2:
        return kernel_bytes(wl, "compact")
    U = wl.L * wl.b * wl.Hkv
    return U * wl.n * wl.d * 2 + kernel_bytes(wl, "compact")


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            pk = json.load(f)
        return (float(pk["hbm_gbs"]), float(pk.get("bf16_tflops_sustained", pk["bf16_tflops"])),
                "measured")
    except Exception:
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS_SUSTAINED, "fallback"


# The source file of each kernel whose DRAM traffic profiles/dram_traffic.txt records.
KERNEL_SOURCE = {"score_tc": "score_tc.cu", "h2o_tc_lse": "h2o_tc.cu",
                 "h2o_tc_colsum": "h2o_tc.cu", "pool_select": "select_compact.cu",
                 "compact": "select_compact.cu", "select": "select_compact.cu"}


def source_digest(kernel=None):
    """sha256 over a kernel's source file and every shared header (csrc/*.cuh, csrc/*.h,
    include/dge.h), or over all kernel sources when `kernel` is None or unknown.  It ties an
    ncu traffic figure to the code it measured: a change to another kernel's file leaves the
    figure valid, a change to this kernel or to a header voids it."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_33334_gb300", "csrc")
    own = KERNEL_SOURCE.get(kernel)
    files = [os.path.join(csrc, fn) for fn in sorted(os.listdir(csrc))
             if fn.endswith((".cuh", ".h")) or (fn.endswith(".cu") and (own is None or fn == own))]
    files.append(os.path.join(ROOT, "include", "dge.h"))
    for path in files:
        with open(path, "rb") as f:
            h.update(os.path.basename(path).encode() + f.read())
    return h.hexdigest()[:16]


def ncu_traffic(kernel, workload):
    """DRAM bytes per launch from profiles/dram_traffic.txt when it matches the current code."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    if not os.path.exists(path):
        return None
    digest = source_digest(kernel)
    with open(path) as f:
        for line in f:
            parts = line.split()
            if len(parts) >= 4 and not line.startswith("#") and parts[0] == kernel and \
                    parts[1] == workload and parts[3] == digest:
                return float(parts[2])
    return None


# --- clocks ---------------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device):
        self.proc = None
        self.out = None
        try:
            uuid = str(torch.cuda.get_device_properties(device).uuid)
            self.ident = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
        except Exception:
            self.ident = None

    def mark(self, which):
        setattr(self, "t_" + which, time.time())

    def start(self):
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
               "-lms", "50"]
        if self.ident:
            cmd.insert(1, f"--id={self.ident}")
        try:
            self.out = io.StringIO()
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
        except Exception:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if not self.proc:
            return None
        time.sleep(0.12)
        self.proc.terminate()
        try:
            text, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            text, _ = self.proc.communicate()
        return self.summarise(text, getattr(self, "t_begin", None), getattr(self, "t_end", None))

    @staticmethod
    def summarise(text, t0=None, t1=None):
        import datetime
        rows = [r for r in csv.reader(io.StringIO(text)) if len(r) >= 10]
        if t0 is not None and t1 is not None:
            kept = []
            for r in rows:
                try:
                    ts = datetime.datetime.strptime(r[0].strip(), "%Y/%m/%d %H:%M:%S.%f")
                    t = ts.timestamp()
                except ValueError:
                    continue
                if t0 - 0.06 <= t <= t1 + 0.06:
                    kept.append(r)
            rows = kept or rows[-1:]
        if not rows:
            return None
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[2]))
                mx = float(r[3])
            except ValueError:
                continue
            for name, val in zip(names, r[6:10]):
                if val.strip().lower() == "active":
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# --- our arm ----------------------------------------------------------------------------------

def run_ours(args):
    rank, world, local = dist_setup("nccl")
    if not torch.cuda.is_available():
        raise SystemExit("bench.py: no CUDA device")
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    from paper_2609_33334_gb300 import _build, api, inputs
    from paper_2609_33334_gb300 import binding as B
    _build.build()
    wl = select_workload(args)
    tens = inputs.make_inputs(wl, device=device)
    paging = None
    if args.page_size:
        # The same cache as page pools behind a block table (pages in a seeded random order).
        hm = args.page_head_major
        K, bt = inputs.paged_layout(tens["K"], args.page_size, seed=1, head_major=hm,
                                    order=args.page_order)
        V, _ = inputs.paged_layout(tens["V"], args.page_size, seed=1, head_major=hm,
                                   order=args.page_order)
        tens = dict(tens, K=K, V=V, bt=bt)
        paging = api.Paging(block_table=bt, page_size=args.page_size, head_major=hm)
    p = api.problem_from_workload(wl)
    Q = tens["Q"] if wl.variant != inputs.STREAMING else None
    ws = api.workspace(p, device)
    if args.lse_supplied:
        # The row normalisers an attention pass over the observation rows would hand over;
        # here the library's own two-pass scoring computes them once, outside the timing.
        tens = dict(tens, lse=api.evict(p, tens["K"], tens["V"], Q, ws=ws, want_lse=True,
                                        paging=paging)["lse"])
    out = api.evict(p, tens["K"], tens["V"], Q, ws=ws, lse_in=tens.get("lse"),
                    paging=paging)  # outputs once
    stream = torch.cuda.current_stream(device)

    def step():
        api.evict(p, tens["K"], tens["V"], Q, ws=ws, out=out, stream=stream,
                  lse_in=tens.get("lse"), paging=paging)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(device)
    status = api.device_status(ws)
    if status != 0:
        raise SystemExit(f"device status {status} after warm-up")

    clocks = ClockSampler(device)
    clocks.start()
    barrier(world)
    torch.cuda.synchronize(device)
    B.dge_profile_begin()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks.mark("begin")
    ev0.record(stream)
    for _ in range(args.steps):
        step()
    ev1.record(stream)
    torch.cuda.synchronize(device)
    clocks.mark("end")
    prof = B.dge_profile_end()
    barrier(world)
    clk = clocks.stop()
    ms_total = ev0.elapsed_time(ev1)
    ms_total = max_over_ranks(ms_total, world, device)
    ms_step = ms_total / args.steps
    tok = tokens_per_step(wl) * world
    value = tok / (ms_step / 1e3)

    hbm, tflops, peak_kind = measured_peaks()
    launches = sum(x[1] for x in prof)
    dom = max(prof, key=lambda x: x[2]) if prof else None
    roofline = None
    kernels = {}
    for name, n_launch, tot in prof:
        kernels[name] = {"launches": n_launch, "ms_per_launch": tot / max(n_launch, 1),
                         "share": tot / max(sum(x[2] for x in prof), 1e-12)}
    if dom:
        name, n_launch, tot = dom
        per = tot / n_launch
        alg = kernel_bytes(wl, name)
        flops = kernel_flops(wl, name)
        # The kernel's bound: whichever of its algorithmic bytes (at the copy peak) and flops
        # (at the sustained bf16 peak: it runs inside a long step) takes longer.
        if flops / (tflops * 1e12) > alg / (hbm * 1e9):
            ach = flops / (per / 1e3) / 1e12
            roofline = {"bound": "tensor", "kernel": name, "achieved": round(ach, 1),
                        "peak": tflops, "unit": "TFLOP/s", "frac": round(ach / tflops, 4),
                        "traffic": ncu_traffic(name, wl.name),
                        "alg_flops_per_launch": flops, "alg_bytes_per_launch": alg,
                        "peak_source": f"{peak_kind} bf16_tflops_sustained"}
        else:
            ach = alg / (per / 1e3) / 1e9
            roofline = {"bound": "hbm", "kernel": name, "achieved": round(ach, 1), "peak": hbm,
                        "unit": "GB/s", "frac": round(ach / hbm, 4),
                        "traffic": ncu_traffic(name, wl.name),
                        "alg_bytes_per_launch": alg, "peak_source": f"{peak_kind} hbm_gbs"}
    step_gbs = step_bytes(wl) / (ms_step / 1e3) / 1e9

    # end to end: pinned host inputs -> device -> dge_evict -> host outputs
    e2e = None
    if not args.no_e2e and args.e2e_steps > 0:
        e2e = run_e2e(args, wl, p, tens, out, ws, device, stream, world, api)

    # The same step with the row normalisers supplied -- as the model's own attention passes over
    # the observation rows return them -- so the scoring reads K once.  Reported beside the
    # configuration's two-pass number; `value` stays the two-pass one.
    one_pass = None
    if not args.lse_supplied and not args.no_one_pass and wl.variant != inputs.STREAMING:
        lse = api.evict(p, tens["K"], tens["V"], Q, ws=ws, want_lse=True, paging=paging)["lse"]

        def step1():
            api.evict(p, tens["K"], tens["V"], Q, ws=ws, out=out, stream=stream, lse_in=lse,
                      paging=paging)

        for _ in range(max(2, args.warmup)):
            step1()
        torch.cuda.synchronize(device)
        barrier(world)
        torch.cuda.synchronize(device)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            step1()
        e1.record(stream)
        torch.cuda.synchronize(device)
        ms1 = max_over_ranks(e0.elapsed_time(e1), world, device) / args.steps
        gbs1 = step_bytes(wl) / (ms1 / 1e3) / 1e9
        one_pass = {"what": "row normalisers supplied (lse_in), one pass over K",
                    "ms_per_step": round(ms1, 4),
                    "value": round(tokens_per_step(wl) * world / (ms1 / 1e3), 1),
                    "step_roofline_frac": round(gbs1 / hbm, 4)}
        del lse

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(wl, args.cpu_seconds)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic",
            "config": {"workload": workload_text(wl), "name": wl.name,
                       "tokens_per_step_per_gpu": tokens_per_step(wl),
                       "l2": "inputs larger than L2 (no flush)",
                       "accumulate": "fp32 (bf16 tensor-core products, fp32 softmax)",
                       "parallelism": f"weak: {world} GPU(s), each the full workload, no "
                                      "collective on the data path"},
            "step_roofline": {"achieved": round(step_gbs, 1), "peak": hbm, "unit": "GB/s",
                              "frac": round(step_gbs / hbm, 4),
                              "alg_bytes_per_step": step_bytes(wl)},
            "roofline": roofline, "kernels": kernels, "gpu_launches": launches,
            "e2e": e2e, "cpu_baseline": cpu, "clocks": clk, "one_pass": one_pass,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


E2E_COPY_STREAMS = 4
E2E_WARMUP = 3


def run_e2e(args, wl, p, tens, out, ws, device, stream, world, api):
    """Same metric through the public call with host buffers: H2D copies of every input,
    the pass, D2H of the kept indices and the compact K/V, all inside the timed region.

    Steps are pipelined as a serving loop would run them: the device inputs are double
    buffered, so step k+1's inputs go over the host link (copy streams) while step k is
    scored and its outputs come back (`stream`).  Every step still copies all of its inputs
    in and its outputs out inside the timed region; the region starts with nothing in
    flight and ends when the last step's outputs are on the host."""
    host_in = {k: torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
               for k, t in tens.items() if t.numel()}
    for k in host_in:
        host_in[k].copy_(tens[k])
    host_out = {k: torch.empty(out[k].shape, dtype=out[k].dtype, pin_memory=True)
                for k in ("idx", "Kc", "Vc")}
    dev_in = [{k: torch.empty_like(tens[k]) for k in host_in} for _ in range(2)]
    h2d = sum(t.numel() * t.element_size() for t in host_in.values())
    d2h = sum(t.numel() * t.element_size() for t in host_out.values())

    def paging_of(buf):
        if "bt" not in buf:
            return None
        hm = args.page_head_major
        return api.Paging(block_table=buf["bt"], page_size=buf["K"].shape[3 if hm else 2],
                          head_major=hm)

    # The inputs go over the host link as E2E_COPY_STREAMS concurrent copies (each tensor cut
    # into that many contiguous pieces); `stream` waits for all of them before the pass.
    copy_streams = [torch.cuda.Stream(device) for _ in range(E2E_COPY_STREAMS)]

    def pieces_of(buf):
        pieces = []
        for k in host_in:
            src, dst = host_in[k].reshape(-1), buf[k].reshape(-1)
            cut = [src.numel() * i // E2E_COPY_STREAMS for i in range(E2E_COPY_STREAMS + 1)]
            pieces.append([(dst[cut[i]:cut[i + 1]], src[cut[i]:cut[i + 1]])
                           for i in range(E2E_COPY_STREAMS)])
        return pieces

    pieces = [pieces_of(b) for b in dev_in]
    freed = [None, None]   # event: the pass that last read buffer b is done

    def step(k):
        b = k & 1
        for i, cs in enumerate(copy_streams):
            if freed[b] is not None:
                cs.wait_event(freed[b])
            with torch.cuda.stream(cs):
                for per_tensor in pieces[b]:
                    dst, src = per_tensor[i]
                    if src.numel():
                        dst.copy_(src, non_blocking=True)
            done = torch.cuda.Event()
            done.record(cs)
            stream.wait_event(done)
        buf = dev_in[b]
        Q = buf.get("Q") if wl.variant != 2 else None
        api.evict(p, buf["K"], buf["V"], Q, ws=ws, out=out, stream=stream,
                  lse_in=buf.get("lse"), paging=paging_of(buf))
        freed[b] = torch.cuda.Event()
        freed[b].record(stream)
        for key in host_out:
            host_out[key].copy_(out[key], non_blocking=True)

    # Warm-up: the first passes over freshly pinned buffers run at about half the link's rate.
    for k in range(E2E_WARMUP):
        step(k)
    torch.cuda.synchronize(device)
    barrier(world)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start = torch.cuda.Event()
    start.record(stream)
    for cs in copy_streams:
        cs.wait_event(start)
    ev0.record(stream)
    for k in range(args.e2e_steps):
        step(E2E_WARMUP + k)
    ev1.record(stream)
    torch.cuda.synchronize(device)
    ms = max_over_ranks(ev0.elapsed_time(ev1), world, device) / args.e2e_steps
    return {"value": round(tokens_per_step(wl) * world / (ms / 1e3), 1), "unit": UNIT,
            "ms_per_step": round(ms, 3), "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "pipelined": "double-buffered device inputs: step k+1's H2D overlaps step k's pass "
                         "and D2H"}


def workload_text(wl):
    kind = {0: "SnapKV/PyramidKV scores", 1: "H2O accumulated scores", 2: "StreamingLLM gather"}
    pool = {0: "no pool", 1: f"max-pool {wl.pool_kernel}", 2: f"avg-pool {wl.pool_kernel}"}
    bud = (f"B={wl.budgets[0]}" if len(set(wl.budgets)) == 1
           else f"B {wl.budgets[0]}->{wl.budgets[-1]} (sum {sum(wl.budgets)})")
    return (f"{wl.name}: L={wl.L} b={wl.b} Hq={wl.Hq} Hkv={wl.Hkv} d={wl.d} n={wl.n} "
            f"w={wl.w}+k={wl.k} {kind[wl.variant]}, {pool[wl.pool]}, {bud}, bf16 K/V/Q N(0,1), "
            f"sink x{wl.sink_scale:g}, {wl.n_spans} planted spans"
            + (", row normalisers supplied (one pass over K)" if "+lse" in wl.name else "")
            + (paged_text(wl.name.split("+pages")[1]) if "+pages" in wl.name else ""))


def paged_text(tag):
    size, _, order = tag.partition("-")
    head = size.endswith("h")
    return (f", paged cache ({size.rstrip('h')}-position pages" + (", head-major" if head else "")
            + f", {order or 'random'} page order, block table)")


# --- CPU oracle (baseline leg and reference arm) ----------------------------------------

def oracle_sample(wl, n_units, seed=0):
    """A deterministic sample of units (all KV heads of a few seeded (layer, sequence)
    slices, so each slice is generated once), as host bf16 bits."""
    from paper_2609_33334_gb300 import inputs
    rng = np.random.default_rng(seed)
    n_slices = min(wl.L * wl.b, -(-n_units // wl.Hkv))
    slices = sorted(rng.choice(wl.L * wl.b, size=n_slices, replace=False).tolist())
    units, data = [], []
    for sl in slices:
        l, b = sl // wl.b, sl % wl.b
        t = inputs.make_inputs(wl, layers=range(l, l + 1), batches=range(b, b + 1))
        for h in range(wl.Hkv):
            if len(units) == n_units:
                break
            G = wl.G
            Qg = inputs.bf16_bits(t["Q"][0, 0, h * G:(h + 1) * G]) if wl.variant != 2 else None
            units.append((l, b, h))
            data.append((l, Qg, inputs.bf16_bits(t["K"][0, 0, h]),
                         inputs.bf16_bits(t["V"][0, 0, h])))
    return units, data


def oracle_pass(wl, data):
    """Run the oracle's whole pass (scores, pool, select, gather) on sampled units."""
    import oracle
    if wl.variant != 2:
        G = wl.G
        Q = np.stack([d[1].reshape(-1, wl.d) for d in data])
        K = np.stack([d[2] for d in data])
        pos = oracle.h2o_positions(wl.n, G) if wl.variant == 1 else \
            oracle.scored_positions(wl.n, wl.m, G)
        raw = oracle.scores(Q, K, pos, wl.n - wl.tail)
    for i, (l, Qg, Kb, Vb) in enumerate(data):
        if wl.variant == 2:
            idx = oracle.streaming_indices(wl.n, wl.sinks, wl.budgets[l])
        else:
            pooled = oracle.pool(raw[i], wl.pool, wl.pool_kernel) if wl.variant == 0 else raw[i]
            idx = oracle.select(pooled, wl.n, wl.sinks, wl.tail, wl.budgets[l])
        oracle.gather(Kb, idx)
        oracle.gather(Vb, idx)


def cores_used():
    try:
        n = len(os.sched_getaffinity(0))
    except AttributeError:
        n = os.cpu_count() or 1
    omp = os.environ.get("OMP_NUM_THREADS")
    return min(n, int(omp)) if omp and omp.isdigit() else n


def calibrate_units(wl, seconds):
    """Units the oracle finishes in about `seconds` on this host's cores (assuming about
    half of ideal scaling over the cores)."""
    import oracle
    oracle.build()
    _, data = oracle_sample(wl, 1, seed=12345)
    t0 = time.perf_counter()
    oracle_pass(wl, data)
    one = time.perf_counter() - t0
    cores = cores_used()
    n = int(seconds * cores * 0.5 / max(one, 1e-3))
    return max(1, min(wl.L * wl.b * wl.Hkv, n)), cores


def cpu_baseline(wl, seconds):
    n_units, cores = calibrate_units(wl, seconds)
    units, data = oracle_sample(wl, n_units)
    t0 = time.perf_counter()
    oracle_pass(wl, data)
    dt = time.perf_counter() - t0
    tok = len(units) * wl.n / wl.Hkv
    return {"value": round(tok / dt, 1), "unit": UNIT, "cores": cores, "kind": "oracle",
            "seconds": round(dt, 2),
            "sample": f"{len(units)} of {wl.L * wl.b * wl.Hkv} (layer, seq, kv-head) units of "
                      f"{wl.name}, fp64 C oracle (scores+pool+select+gather), OpenMP over units"}


def run_reference(args):
    rank, world, local = dist_setup("gloo")
    if rank != 0:
        return
    sys.path.insert(0, ROOT)
    wl = select_workload(args)
    per_step = min(20.0, max(2.0, 60.0 / max(1, args.steps + args.warmup)))
    n_units, cores = calibrate_units(wl, per_step)
    units, data = oracle_sample(wl, n_units)
    for _ in range(args.warmup):
        oracle_pass(wl, data)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_pass(wl, data)
    dt = (time.perf_counter() - t0) / max(args.steps, 1)
    tok = len(units) * wl.n / wl.Hkv
    value = tok / dt
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 1), "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(dt * 1e3, 3), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": workload_text(wl), "name": wl.name,
                       "sample_units_per_step": len(units)},
            "cpu_baseline": {"value": round(value, 1), "unit": UNIT, "cores": cores,
                             "kind": "oracle",
                             "sample": f"{len(units)} of {wl.L * wl.b * wl.Hkv} units per step"},
            "e2e": {"value": round(value, 1), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
