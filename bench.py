#!/usr/bin/env python3
"""Throughput of the SALSA block sweep on GB300.

One step = one full stochastic sweep of the connectome-shaped workload
(139,255 x 139,255, power-law out-degree with mean 20, ~2.8M nonzeros,
r = 64, blocks of 4096; seeded synthetic data): for every block step the
Gram matrix and its inverse, the fused Z-panel tensor-core kernel, the sparse
support correction and the least-squares/momentum update.  Metric: Z entries
per second = 2 m n / sweep time (a sweep touches every entry of Z twice).

Default (``--impl ours``): the CUDA library through its C ABI, inputs resident
in HBM, device time with CUDA events over exactly K sweeps after W warm-up
sweeps.  ``e2e`` repeats the measurement through the public API with host
buffers: per step the factors are copied in from pinned host memory, one
sweep runs, and the factors are copied back.  ``--impl reference`` times the
fp64 CPU oracle on the host cores on a bounded sample of the same workload.

Under torchrun (N > 1 GPUs) every rank runs an independent replica of the
workload (the sweep has no data-path collective); rank 0 prints the
whole-job rate over the slowest rank's time.
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
WORKLOADS = {
    # name: (generator key, r, block, precision default)
    "connectome_r64": ("connectome_r64", 64, 4096),
    "connectome_r256": ("connectome_r256", 256, 8192),
    "planted_medium": ("planted_medium", 32, 2048),
    "identity": ("identity", 3, 512),
    "planted_tiny": ("planted_tiny", 4, 128),
    "connectome_dense_r64": ("connectome_dense_r64", 64, 4096),
    "communities_r64": ("communities_r64", 64, 8192),
    "communities_planted_r64": ("communities_planted_r64", 64, 8192),
}


# DRAM bytes (read + write) of one dense-kernel launch, from an ncu capture of
# the same workload (dram__bytes_read.sum + dram__bytes_write.sum); valid only
# while the kernel's sources hash to the digest recorded with it (else null)
DENSE_TRAFFIC = {
    # (workload, precision, epilogue): (bytes per launch, dense_source_digest() of the code measured)
    ("connectome-139255-r64", "bf16", "z"): (18395392, "5094500fd5d511bc"),
}


def chunks_per_sweep(sol, wl, exact, N):
    """(128-row M tile, Q chunk) pairs of the dense kernel in one sweep."""
    _, bn = sol.range_mask(N.NMD_COL, 0, N.NMD_STOCH)   # the chunk size (the mask itself is not used)

    def cdiv(a, b):
        return -(-a // b)

    m, n, br, bc = wl.m, wl.n, wl.block_rows, wl.block_cols
    if exact:   # b rows against a whole factor, per block
        return (sum(cdiv(min(br, m - i), 128) * cdiv(n, bn) for i in range(0, m, br)) +
                sum(cdiv(min(bc, n - j), 128) * cdiv(m, bn) for j in range(0, n, bc)))
    return (sum(cdiv(m, 128) * cdiv(min(bc, n - j), bn) for j in range(0, n, bc)) +
            sum(cdiv(n, 128) * cdiv(min(br, m - i), bn) for i in range(0, m, br)))


def skip_mode(args, N):
    if args.range_search:
        return N.NMD_SKIP_RANGE
    return N.NMD_SKIP_VOTE if args.skip_zero_chunks else N.NMD_SKIP_NONE


def dense_source_digest():
    """Digest of the dense kernel's code (panel_tc.cu, tc_ptx.cuh) with line
    comments and blank lines removed: a recorded DRAM-traffic figure stays
    valid across comment edits and lapses when the code changes."""
    import hashlib
    h = hashlib.sha256()
    for f in ("panel_tc.cu", "tc_ptx.cuh"):
        with open(os.path.join(ROOT, "paper_2608_21607_gb300", "csrc", f), encoding="utf-8") as fh:
            for line in fh:
                code = line.split("//", 1)[0].rstrip()
                if code:
                    h.update(code.encode() + b"\n")
    return h.hexdigest()[:16]


def support_bytes_per_sweep(wl, elem_bytes):
    """Algorithmic DRAM bytes of the support term over one sweep (each step
    once), and the q-row gathers on top of them.  DRAM: per support entry its
    index and value (8 B); per M-side row with support in the step's panel
    its m row (r elements) and its row of Rs (r fp32 values, written); each
    step's Q-side block once (r elements per row: over a sweep, both factors
    once).  Gathers: per support entry its q row (r elements), which the
    kernels read from L2 or from the block staged in shared memory.  Every
    nonzero is in one column step and one row step; the panel rows are
    counted per step."""
    import numpy as np
    S = wl.S
    rows = np.repeat(np.arange(S.m, dtype=np.int64), np.diff(S.row_ptr))
    cols = np.asarray(S.col_idx, np.int64)
    # column steps: (row, column block) pairs; row steps: (column, row block) pairs
    col_pairs = np.unique(rows * (-(-S.n // wl.block_cols)) + cols // wl.block_cols).size
    row_pairs = np.unique(cols * (-(-S.m // wl.block_rows)) + rows // wl.block_rows).size
    nnz = int(S.row_ptr[-1])
    dram = 2 * nnz * 8 + (col_pairs + row_pairs) * (elem_bytes * wl.r + 4 * wl.r) + (S.m + S.n) * elem_bytes * wl.r
    return dram, 2 * nnz * elem_bytes * wl.r


def measure_support(sol, wl, N):
    """The support-term kernels alone (nmd_support_term, no other work on the
    GPU) over every step of one sweep: device ms of the kernels (CUDA events
    the library records around each step's support-term launches, on the
    stream they run on; the hook's clearing of its output buffer is outside)."""
    import torch
    pr, pc = sol.block_order(0, N.NMD_ROW), sol.block_order(0, N.NMD_COL)
    if wl.schedule == "exact":
        order = [(N.NMD_ROW, b, N.NMD_EXACT) for b in pr] + [(N.NMD_COL, b, N.NMD_EXACT) for b in pc]
    else:   # alternating stochastic sweep
        order = []
        for t in range(max(len(pr), len(pc))):
            if t < len(pc):
                order.append((N.NMD_COL, int(pc[t]), N.NMD_STOCH))
            if t < len(pr):
                order.append((N.NMD_ROW, int(pr[t]), N.NMD_STOCH))
    buf = torch.empty(max(wl.m, wl.n) * sol.r_pad, dtype=torch.float32, device=sol.device)
    for side, block, kind in order[:4]:
        sol.support_term(side, block, kind, buf)
    sol.sync()
    sol.profile(True)
    for side, block, kind in order:
        sol.support_term(side, block, kind, buf)
    ms, _ = sol.profile_read(N.NMD_K_SPARSE)
    sol.profile(False)
    return ms, len(order)


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + q,
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for name, v in zip(["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                                "sw_power_cap"], f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def oracle_sample(wl, budget_s=20.0):
    """Time the fp64 oracle on block steps of the workload until the budget
    (at least one COL/STOCH and one ROW/STOCH step); Z entries per second."""
    import numpy as np
    import oracle as O
    st = O.State(wl.S, wl.W0, wl.H0, O.Options(block_rows=wl.block_rows, block_cols=wl.block_cols,
                                                 schedule=O.EXACT if wl.schedule == "exact" else O.STOCH,
                                                 eta=wl.eta, gamma=wl.gamma))
    steps = st.sweep_steps(0)
    entries, t_used, done = 0, 0.0, []
    for side, block, kind in steps:
        M, _, (m0, m1), _, _, (c0, c1) = st._roles(side, block, kind)
        t0 = time.perf_counter()
        st.block_update(side, block, kind)
        dt = time.perf_counter() - t0
        entries += (m1 - m0) * (c1 - c0)
        t_used += dt
        done.append((side, block))
        if t_used >= budget_s and len(done) >= 2:
            break
    return entries / t_used, len(done), t_used


# The paper's kernel-throughput table (Sec. 4.2): the fused kernel on m =
# 250000 rows against a block of n = 2500, TFLOP/s counted as 4 m n r
# (both products), TF32 operands; H100 PCIe and RTX Pro 6000 figures.
PAPER_KERNEL_TABLE = {16: (215.30, 191.72), 32: (283.73, 203.06), 64: (285.10, 206.11), 128: (279.19, 189.80)}


def embed_bench(args):
    """The cell embedding and held-out 1-NN search of Sec. 5.3 at full size: a
    block-structured graph of 139,255 cells in 64 communities (runs of 128
    cells taken in turn), r = 64, fitted for a few sweeps from its clustered
    start; then per timed step one embedding (nmd_embed) and one all-pairs
    nearest-neighbour search of the 2r = 128-dimensional cells
    (nmd_nearest_neighbors) with the community labels.  The search is a dense
    contraction of N^2 d multiply-adds, each coordinate in three bf16 pieces
    (three tensor-core products per pair)."""
    import torch
    from paper_2608_21607_gb300 import build as B
    from paper_2608_21607_gb300 import nmd as N
    from paper_2608_21607_gb300 import workloads as WLm
    from paper_2608_21607_gb300.replicas import env as replica_env
    _, rank, local = replica_env()
    if rank != 0:
        return 0
    torch.cuda.set_device(local)
    B.build()
    wl = WLm.workload("communities_r64", seed=0)
    labels = torch.from_numpy(WLm.community_of(wl.n, wl.info["clusters"], wl.info["run"]).astype("int32")).cuda()
    sol = N.Solver(wl.S, wl.r, block_rows=wl.block_rows, block_cols=wl.block_cols, eta=wl.eta, gamma=wl.gamma)
    sol.set_factors(wl.W0, wl.H0)
    for _ in range(3):
        sol.sweep()
    n, d = wl.n, 2 * wl.r
    xi = torch.empty((n, d), dtype=torch.float32, device="cuda")
    sig = torch.empty(wl.r, dtype=torch.float32, device="cuda")
    ws = torch.empty(N.nmd_nn_workspace_bytes(n, d), dtype=torch.uint8, device="cuda")
    nn = torch.empty(n, dtype=torch.int32, device="cuda")
    best = torch.empty(n, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()
    clocks = ClockSampler(local)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
           torch.cuda.Event(enable_timing=True)) for _ in range(args.warmup + args.steps)]
    errors = []
    for i, (e0, e1, e2) in enumerate(ev):
        if i == args.warmup:
            clocks.start()
        e0.record(stream)
        N.nmd_embed(sol.h, xi, sig)
        e1.record(stream)
        errors.append(N.nmd_nearest_neighbors(xi, n, d, labels, nn, best, ws, stream.cuda_stream))
        e2.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    t_embed = [e0.elapsed_time(e1) for e0, e1, _ in ev[args.warmup:]]
    t_nn = [e1.elapsed_time(e2) for _, e1, e2 in ev[args.warmup:]]
    ms = statistics.median(a + b for a, b in zip(t_embed, t_nn))
    nn_ms = statistics.median(t_nn)
    pk, pk_kind = peaks()
    flops = 2.0 * n * n * d * 3
    tf = flops / (nn_ms / 1e3) / 1e12
    peak = pk.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    print(json.dumps({
        "metric": "cells embedded and 1-NN searched per second", "value": n / (ms / 1e3), "unit": "cells/s",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "dtype": "bf16x3 (fp32 accumulation)", "data": "synthetic",
        "config": {"workload": wl.name, "cells": n, "r": wl.r, "d": d, "sweeps_before": 3,
                   "labels": "communities (%d)" % wl.info["clusters"]},
        "embed_ms": statistics.median(t_embed), "nn_ms": nn_ms, "one_nn_error_rate": errors[-1] / n,
        "roofline": {"bound": "tensor", "kernel": "panel_tc_kernel nearest-neighbour pass", "achieved": tf,
                     "peak": peak, "unit": "TFLOP/s (three bf16 products per pair)", "frac": tf / peak,
                     "peak_kind": "%s bf16 dense, burst" % pk_kind},
        "clocks": clk}))
    return 0


def kernel_table(args):
    """Each step here is one stochastic column step (all m rows of W against
    a block of 2500 rows of B) run alone, synchronised after every step; the
    dense kernel's own time comes from the library's CUDA-event profile."""
    import numpy as np
    import torch
    from paper_2608_21607_gb300 import build as B
    from paper_2608_21607_gb300 import nmd as N
    from paper_2608_21607_gb300 import workloads as WLm
    from paper_2608_21607_gb300.replicas import env as replica_env
    _, rank, local = replica_env()
    if rank != 0:
        return 0
    torch.cuda.set_device(local)
    B.build()
    m, nb = 250000, 2500
    S = WLm.identity(m)
    for prec_name, prec in (("bf16", N.NMD_BF16), ("fp32", N.NMD_FP32)):
        for r in (16, 32, 64, 128):
            W0, H0 = WLm.init_factors(m, m, r, 0)
            sol = N.Solver(S, r, block_rows=nb, block_cols=nb, precision=prec, eta=0.5, gamma=0.0)
            sol.set_factors(W0, H0)
            for b in range(args.warmup):
                sol.block_update(N.NMD_COL, b, N.NMD_STOCH)
                sol.sync()
            sol.profile(True)
            for b in range(args.steps):
                sol.block_update(N.NMD_COL, args.warmup + b, N.NMD_STOCH)
                sol.sync()
            ms, n = sol.profile_read(N.NMD_K_DENSE)
            sol.profile(False)
            us = 1e3 * ms / n
            tf = 4.0 * m * nb * r / (us * 1e-6) / 1e12
            h100, rtx = PAPER_KERNEL_TABLE[r]
            print(json.dumps({"metric": "dense kernel TFLOP/s at the paper's kernel-table shape (4 m n r per launch)",
                              "value": tf, "unit": "TFLOP/s", "higher_is_better": True, "r": r,
                              "dtype": prec_name, "m": m, "block": nb, "launches": n, "us_per_launch": us,
                              "paper_h100_tf32": h100, "paper_rtx_pro_6000_tf32": rtx,
                              "data": "synthetic (identity S, N(0, 0.01) factors)"}))
            del sol
            torch.cuda.empty_cache()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=sorted(WORKLOADS), default="connectome_r64")
    ap.add_argument("--precision", choices=["bf16", "fp32"], default="bf16")
    ap.add_argument("--epilogue", choices=["z", "delta"], default="z")
    ap.add_argument("--skip-zero-chunks", action="store_true",
                    help="Delta form: skip the second product of chunks whose rectified tile is zero")
    ap.add_argument("--range-search", action="store_true",
                    help="Delta form: skip both dense products of the chunks a range search over the "
                         "normalised factor rows clears (Sec. 4.3)")
    ap.add_argument("--schedule", choices=["workload", "exact", "stoch"], default="workload",
                    help="sweep kind: the workload's own, or exact / stochastic")
    ap.add_argument("--init", choices=["normal", "paper"], default="normal",
                    help="factor start: iid N(0, 0.01), or the sign-structured start W > 0, H < 0")
    ap.add_argument("--no-cpu-baseline", action="store_true", help="skip the oracle timing on the host")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end leg (profiling runs)")
    ap.add_argument("--no-modes", action="store_true", help="skip the fp32-accurate mode's sweep timing")
    ap.add_argument("--support-only", action="store_true",
                    help="only the support term alone over one sweep's steps (profiling; rank 0 only)")
    ap.add_argument("--embed", action="store_true",
                    help="time the cell embedding and 1-NN search (Sec. 5.3) on a block-structured graph")
    ap.add_argument("--kernel-table", action="store_true",
                    help="dense kernel alone at the paper's kernel-table shape (m = 250000 rows against a "
                         "block of 2500), one JSON line per factor rank r and precision (rank 0 only)")
    args = ap.parse_args()
    assert args.warmup >= 3, "at least 3 warm-up steps"
    if args.kernel_table:
        return kernel_table(args)
    if args.embed:
        return embed_bench(args)

    from paper_2608_21607_gb300.replicas import env as replica_env
    ws, rank, local = replica_env()
    metric = "Z entries/s per full ALS sweep (2*m*n / sweep time)"
    from paper_2608_21607_gb300 import workloads as WLm
    gen, r, block = WORKLOADS[args.workload]

    if args.impl == "reference":
        if rank != 0:
            return 0
        wl = WLm.workload(gen, seed=0)
        cores = os.cpu_count()
        vals = []
        for i in range(args.warmup + args.steps):
            v, nsteps, t = oracle_sample(wl, budget_s=max(1.0, 60.0 / (args.warmup + args.steps)))
            if i >= args.warmup:
                vals.append((v, nsteps, t))
        value = statistics.median(v for v, _, _ in vals)
        tsum = sum(t for _, _, t in vals)
        sample = ("%d block steps of the sweep per timed step (the first blocks of "
                  "sweep 0), fp64 oracle, numpy on %d host cores" % (vals[0][1], cores))
        line = {"impl": "reference", "metric": metric, "value": value, "unit": "Z entries/s",
                "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": 1e3 * tsum / len(vals), "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": {"workload": wl.name, "m": wl.m, "n": wl.n, "nnz": wl.S.nnz, "r": r,
                           "block": block, "schedule": wl.schedule, "parallelism": "host cores"},
                "cpu_baseline": {"value": value, "unit": "Z entries/s", "cores": cores, "kind": "oracle",
                                 "sample": sample},
                "e2e": {"value": value, "unit": "Z entries/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return 0

    import numpy as np
    import torch
    from paper_2608_21607_gb300 import build as B
    from paper_2608_21607_gb300 import nmd as N

    from paper_2608_21607_gb300.replicas import Replicas
    torch.cuda.set_device(local)
    rep = Replicas(device=torch.device("cuda", local))
    B.build()
    wl = WLm.workload(gen, seed=0)
    prec = {"bf16": N.NMD_BF16, "fp32": N.NMD_FP32}[args.precision]
    epi = {"z": N.NMD_EPI_Z, "delta": N.NMD_EPI_DELTA}[args.epilogue]
    exact = wl.schedule == "exact" if args.schedule == "workload" else args.schedule == "exact"
    sol = N.Solver(wl.S, wl.r, block_rows=wl.block_rows, block_cols=wl.block_cols,
                   schedule=N.NMD_EXACT if exact else N.NMD_STOCH,
                   eta=wl.eta, gamma=wl.gamma, precision=prec, epilogue=epi, seed=0,
                   skip_zero_chunks=skip_mode(args, N))
    W0, H0 = wl.W0, wl.H0
    if args.init == "paper":
        W0, H0 = WLm.init_factors(wl.m, wl.n, wl.r, 0, signs="paper")
    sol.set_factors(W0, H0)
    stream = sol.stream
    if args.support_only:
        if rank == 0:
            pk, pk_kind = peaks()
            hbm = pk.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"])
            ms, nst = measure_support(sol, wl, N)
            by, gb = support_bytes_per_sweep(wl, 2 if prec == N.NMD_BF16 else 4)
            print(json.dumps({"metric": "support term alone, algorithmic DRAM GB/s", "value": by / (ms / 1e3) / 1e9,
                              "unit": "GB/s", "frac": by / (ms / 1e3) / 1e9 / hbm, "ms_per_sweep": ms,
                              "steps": nst, "bytes_per_sweep": by, "gather_bytes_per_sweep": gb,
                              "with_gathers_gbs": (by + gb) / (ms / 1e3) / 1e9, "workload": wl.name,
                              "precision": args.precision}))
        rep.close()
        return 0

    def barrier():
        torch.cuda.synchronize()
        rep.barrier()
        torch.cuda.synchronize()

    # ---------------- device-resident timing ----------------
    for _ in range(args.warmup):
        sol.sweep()
    sol.sync()
    barrier()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    # Workloads whose whole workspace fits in L2 (129 MB) are timed sweep by
    # sweep with L2 flushed before each (a 512 MB write, outside the timed
    # interval); the others already stream more than L2 per sweep.
    ws_bytes = sol.workspace.numel() * sol.workspace.element_size()
    flush = ws_bytes < 256 * 2**20
    scratch = torch.empty(512 * 2**20, dtype=torch.uint8, device="cuda") if flush else None
    l0 = sol.launches
    sol.skip_count(reset=True)
    ms_total = 0.0
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps if flush else 1)]
    if flush:
        for e0, e1 in ev:
            with torch.cuda.stream(stream):
                scratch.fill_(1)
            e0.record(stream)
            sol.sweep()
            e1.record(stream)
    else:
        ev[0][0].record(stream)
        for _ in range(args.steps):
            sol.sweep()
        ev[0][1].record(stream)
    sol.sync()
    ms_total = sum(e0.elapsed_time(e1) for e0, e1 in ev)
    launches = sol.launches - l0
    skipped = sol.skip_count(reset=True)
    clk = clocks.stop()
    barrier()
    # Per-kernel device times for the roofline come from separate sweeps with
    # an event pair around every launch (the events cost time of their own,
    # so the sweeps timed above run without them).
    def sweeps(s, k, profile):
        """k sweeps of solver s, one at a time (L2 flushed before each where
        the workspace fits in it): their total device time (ms) and, with
        profile, the per-class kernel times read back from the library."""
        s.profile(bool(profile))
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ms = 0.0
        for _ in range(k):
            if flush:
                with torch.cuda.stream(s.stream):
                    scratch.fill_(1)
            t0.record(s.stream)
            s.sweep()
            t1.record(s.stream)
            s.sync()
            ms += t0.elapsed_time(t1)
        classes = {name: s.profile_read(c) for name, c in
                   [("dense", N.NMD_K_DENSE), ("sparse", N.NMD_K_SPARSE), ("gram_inverse", N.NMD_K_GRAM),
                    ("update", N.NMD_K_UPDATE)]} if profile else None
        s.profile(False)
        return ms, classes

    k_prof = min(args.steps, 5)
    ms_prof, other = sweeps(sol, k_prof, True)
    dense_ms, dense_n = other.pop("dense")
    barrier()
    entries = 2.0 * wl.m * wl.n
    value, t_max_s = rep.job_rate(entries * args.steps, ms_total / 1e3)   # replicas: weak scaling
    t_max = 1e3 * t_max_s

    # dense kernel roofline: 4 M K r algorithmic flops per launch (2 M K r for
    # L = M Q^T and 2 M K r for R = P Q), summed over the launches of a sweep
    Kr = -(-wl.m // wl.block_rows)
    Kc = -(-wl.n // wl.block_cols)
    flops_sweep = 4.0 * wl.r * (wl.m * wl.n + wl.n * wl.m)   # COL steps: M=m, sum K = n; ROW steps: M=n, sum K=m
    launches_per_sweep = Kr + Kc
    flops_per_launch = flops_sweep / launches_per_sweep
    pk, pk_kind = peaks()
    peak = pk.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
    burst = pk.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    achieved = flops_sweep * k_prof / (dense_ms / 1e3) / 1e12 if dense_ms > 0 else None
    traffic = None
    rec = DENSE_TRAFFIC.get((wl.name, args.precision, args.epilogue))
    if rec and rec[1] == dense_source_digest():
        traffic = rec[0]
    roofline = {"bound": "tensor", "kernel": "panel_tc_kernel (fused Z-panel, tcgen05)",
                "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": (achieved / peak) if achieved else None,
                "frac_of_burst": (achieved / burst) if achieved else None, "traffic": traffic,
                "traffic_unit": "bytes per launch (ncu dram__bytes_read.sum + dram__bytes_write.sum)",
                "peak_kind": "%s bf16 dense, sustained" % pk_kind,
                "flops_per_launch": flops_per_launch, "launches": dense_n,
                "avg_launch_us": 1e3 * dense_ms / max(dense_n, 1),
                "share_of_step": dense_ms / ms_prof if ms_prof > 0 else None,
                "profiled_sweeps": k_prof, "profiled_ms_per_sweep": ms_prof / k_prof,
                "other_kernels_ms_per_sweep": {k: v[0] / k_prof for k, v in other.items()}}
    if prec == N.NMD_FP32:
        roofline["note"] = "fp32-accurate mode issues 3 bf16 MMAs per product; flops counted once"

    # support term alone (HBM roofline by algorithmic bytes)
    hbm = pk.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"])
    sp_ms, sp_steps = measure_support(sol, wl, N)
    sp_bytes, sp_gather = support_bytes_per_sweep(wl, 2 if prec == N.NMD_BF16 else 4)
    sp_gbs = sp_bytes / (sp_ms / 1e3) / 1e9
    roofline_sparse = {"bound": "hbm", "kernel": "support term (sparse_group_kernel, sparse_long_kernel, "
                                                 "sparse_reduce_kernel; sparse_smem_kernel where the Q-side "
                                                 "block fits in shared memory), alone",
                       "achieved": sp_gbs, "peak": hbm, "unit": "GB/s", "frac": sp_gbs / hbm,
                       "traffic": None, "peak_kind": "%s copy bandwidth" % pk_kind,
                       "bytes_per_sweep": sp_bytes, "ms_per_sweep": sp_ms, "steps": sp_steps,
                       "bytes_rule": "DRAM: per support entry 8 B; per panel row r operand elements + 4 r B "
                                     "(Rs); each step's Q-side block once; operands bf16 in the bf16 mode",
                       "gather_bytes_per_sweep": sp_gather,
                       "with_gathers_gbs": (sp_bytes + sp_gather) / (sp_ms / 1e3) / 1e9,
                       "gather_rule": "per support entry the r operand elements of its q row (from L2 or "
                                      "shared memory)"}

    # the fp32-accurate mode on the same workload and start, same run
    modes = None
    if prec == N.NMD_BF16 and not args.no_modes:
        sol2 = N.Solver(wl.S, wl.r, block_rows=wl.block_rows, block_cols=wl.block_cols,
                        schedule=N.NMD_EXACT if exact else N.NMD_STOCH, eta=wl.eta, gamma=wl.gamma,
                        precision=N.NMD_FP32, epilogue=epi, seed=0)
        sol2.set_factors(W0, H0)
        for _ in range(args.warmup):
            sol2.sweep()
        sol2.sync()
        k2 = min(args.steps, 5)
        clocks2 = ClockSampler(local)
        clocks2.start()
        ms2, _ = sweeps(sol2, k2, False)
        clk2 = clocks2.stop()
        _, c2 = sweeps(sol2, k2, True)
        d2_ms, d2_n = c2["dense"]
        ach2 = flops_sweep * k2 / (d2_ms / 1e3) / 1e12 if d2_ms > 0 else None
        modes = {"fp32": {"ms_per_sweep": ms2 / k2, "value": entries * k2 / (ms2 / 1e3), "unit": "Z entries/s",
                          "sweeps": k2, "dense_tflops_algorithmic": ach2,
                          "dense_frac_of_burst": (ach2 / burst) if ach2 else None,
                          "dense_avg_launch_us": 1e3 * d2_ms / max(d2_n, 1), "clocks": clk2,
                          "note": "fp32-accurate mode (three bf16 pieces per factor; the tensor cores run 3 "
                                  "MMAs per first product and 4 per second); flops counted once"}}
        del sol2
        torch.cuda.empty_cache()

    # ---------------- end to end through the public API, host buffers -------
    Wh = torch.from_numpy(np.ascontiguousarray(W0, np.float32)).pin_memory()
    Hh = torch.from_numpy(np.ascontiguousarray(H0, np.float32)).pin_memory()
    Wo = torch.empty_like(Wh).pin_memory()
    Ho = torch.empty_like(Hh).pin_memory()
    h2d = (Wh.numel() + Hh.numel()) * 4
    d2h = (Wo.numel() + Ho.numel()) * 4

    def e2e_step():
        N.nmd_set_factors(sol.h, Wh, Hh, False)
        N.nmd_sweep(sol.h)
        N.nmd_get_factors(sol.h, Wo, Ho, False)

    e2e = None
    if not args.no_e2e:
        for _ in range(args.warmup):
            e2e_step()
        barrier()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            e2e_step()
        torch.cuda.synchronize()
        e2e_value, e2e_s = rep.job_rate(entries * args.steps, time.perf_counter() - t0)
        e2e = {"value": e2e_value, "unit": "Z entries/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": 1e3 * e2e_s / args.steps}

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        v, nsteps, t = oracle_sample(wl, budget_s=15.0)
        cpu = {"value": v, "unit": "Z entries/s", "cores": os.cpu_count(), "kind": "oracle",
               "sample": "%d block steps (%.1f s) of sweep 0 of the same workload, fp64 oracle (numpy)"
                         % (nsteps, t)}

    if rank == 0:
        line = {"metric": metric, "value": value, "unit": "Z entries/s", "n_gpus": ws, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": t_max / args.steps, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": args.precision if prec == N.NMD_BF16 else "f32",
                "data": "synthetic",
                "config": {"workload": wl.name, "m": wl.m, "n": wl.n, "nnz": wl.S.nnz, "r": wl.r,
                           "block": wl.block_rows,
                           "schedule": "exact (row blocks, then column blocks)" if exact else "stochastic, alternating",
                           "eta": wl.eta,
                           "gamma": wl.gamma, "precision": args.precision,
                           "epilogue": args.epilogue, "init": args.init,
                           "skip_zero_chunks": ["none", "vote", "range"][skip_mode(args, N)],
                           "skipped_chunks_per_sweep": skipped / args.steps,
                           "chunks_per_sweep": chunks_per_sweep(sol, wl, exact, N),
                           "parallelism": "replicas" if ws > 1 else "single GPU",
                           "workspace_mb": round(ws_bytes / 2**20, 1),
                           "l2": ("workspace smaller than L2: L2 flushed (512 MB write) before each timed sweep"
                                  if flush else "workspace larger than L2 (%.0f MB): no flush" % (ws_bytes / 2**20))},
                "e2e": e2e, "roofline": roofline, "roofline_sparse": roofline_sparse, "modes": modes,
                "cpu_baseline": cpu, "clocks": clk,
                "gpu_launches": launches}
        print(json.dumps(line))
    rep.close()
    return 0


if __name__ == "__main__":
    sys.exit(main())
