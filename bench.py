#!/usr/bin/env python
"""Benchmark of the CRVQ code-search hot path on GB300.

A step is the whole hot path (Alg. 1 from prequantization to the refinement loop: Hessian,
prequantize, importance + reorder, base k-means, extended codebooks, least-squares refinement
with beam re-encode, losses) over one workload, through crvq_quantize_layer. The default
workload is the largest one that fits a GPU: the seven matrices of a LLaMA-2-7B decoder block
(q, k, v, o 4096 x 4096 and gate, up 11008 x 4096 sharing one 4096-token X; down 4096 x 11008
with its own SwiGLU-like X; d = 8, K = 256, 2 extended codebooks on 2% channels, B = 8, 10
Lloyd iterations). `--config c1..c4` runs a single matrix instead. The metric is code-search
throughput: scored (hypothesis, codeword) pairs per second over the whole step; the per-step
(block) time is reported beside it.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl crvq|reference] [--config c5]

With N > 1 (torchrun, one rank per GPU) every rank quantizes its own block (independent
problems, no collective on the data path): weak scaling; value = all ranks' scores / the
slowest rank's time. `--impl reference` times the fp64 CPU oracle on bounded row samples of
the same workload on every host core (the paper ships no code; the oracle is the reference
arm).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synthetic as S  # noqa: E402


def schedule_scores(cfg, M, N):
    """(hypothesis, codeword) pairs scored by one matrix through the schedule."""
    d, T = cfg.d, cfg.kmeans_iters
    G = N // d
    Gc = min(G, int(np.ceil(np.float32(cfg.crit_frac) * N / d - 1e-12))) if cfg.crit_frac > 0 else 0
    n_all, n_crit = M * G, M * Gc
    n_base = getattr(cfg, "n_base", 1)

    def beam(stages):                                      # pairs per vector of a beam pass
        total, parents = 0, 1
        for K in stages:
            total += parents * K
            parents = min(cfg.B, parents * K)
        return total

    s = (1 + n_base) * (T + 1) * n_all * cfg.K_base       # prequantize + base k-means
    s += cfg.n_ext * (T + 1) * n_crit * cfg.K_ext          # extended k-means
    s += cfg.refine_rounds * (n_crit * beam([cfg.K_base] * n_base + [cfg.K_ext] * cfg.n_ext) +
                              (n_all - n_crit) * beam([cfg.K_base] * n_base))
    return float(s)


# dram__bytes_read.sum + dram__bytes_write.sum per arg-min launch, averaged over every
# argmin_tc_kernel launch of one step of the workload (one ncu capture of the launch list with
# the two DRAM counters; the summary is kept with the other profiles). None for a workload
# whose counters have not been taken, and whenever the kernel changes until they are taken
# again.
ARGMIN_TRAFFIC = {"c5": 106.24e6}

# The tf32 tensor rate relative to bf16 (nominal dense figures of the part: 1.1 vs 2.25
# PFLOP/s). Only the bf16 rate is measured; the arg-min's MMAs are kind::tf32.
TF32_PER_BF16 = 1.1 / 2.25

# Instructions on the integer ALU pipe per scored pair over the whole arg-min kernel (the
# block minima, selects and merges of the epilogue plus the per-row prologue, certificate and
# statistics): the ncu ALU pipe activity of one launch on the 4096 x 4096 layer (49.1% of
# 41.45 M SM-cycles at two warp instructions per SM-cycle, 32 lanes each) over its 536.9 M
# scored pairs.
ALU_OPS_PER_SCORE = 2.43


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return json.load(f), "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "sm_max_mhz": 2070.0}, "fallback"


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.gpu_id = gpu_id
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(self.gpu_id)], stdout=subprocess.PIPE,
                stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (OSError, FileNotFoundError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.t.join(timeout=2)
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax = float(f[2])
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower() in ("active", "1", "yes"):
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


# Rough fp64-oracle throughput on a few host cores, only to size the CPU samples below.
ORACLE_RATE_EST = 1.5e7


def cpu_oracle_sample(cfg, X=None, budget_s=20.0, max_rows=64):
    """Times the fp64 oracle, as it stands, on a bounded sample of the workload (about
    `budget_s` of CPU work). The whole schedule on the first rows of W (full X) when enough rows
    for K fit the budget; otherwise (a 65536-entry codebook needs 65536 vectors) one encode
    pass, the schedule's dominant step, of the first rows over the first 32 groups against a
    seeded K_base-entry codebook. Returns (scores/s, seconds, cores used, description)."""
    from oracle import crvq_oracle as O
    d = cfg.d
    G = cfg.N // d
    Gc = O.n_crit_groups(cfg.N, d, cfg.crit_frac)
    need = max(cfg.K_base / G, cfg.K_ext / Gc if cfg.n_ext > 0 and Gc > 0 else 0.0)
    per_row = schedule_scores(cfg, 1, cfg.N)
    fit = int(budget_s * ORACLE_RATE_EST / per_row)
    rows = min(cfg.M, max(int(np.ceil(need)), min(fit, max_rows)))
    X = S.gen_X(cfg) if X is None else X
    c0 = time.process_time()
    if rows >= need and per_row * rows <= 3.0 * budget_s * ORACLE_RATE_EST:
        W = S.gen_W(cfg, np.arange(rows))
        t0 = time.perf_counter()
        O.quantize_layer(W, X, cfg)
        wall = time.perf_counter() - t0
        sc = schedule_scores(cfg, rows, cfg.N)
        desc = f"whole schedule on rows 0..{rows - 1} of {cfg.name} (full X)"
    else:
        gs = min(G, 32)
        _, _, Hb, _ = O.hessian(np.ascontiguousarray(X[:, :gs * d]), cfg.damp_rel, d)
        C = np.random.default_rng(0).normal(0.0, 0.02, (cfg.K_base, d)).astype(np.float32)
        W1 = np.ascontiguousarray(S.gen_W(cfg, np.arange(1))[:, :gs * d])
        t0 = time.perf_counter()                       # one row sizes the sample
        O.encode_beam(W1, d, Hb, [O.Codebook(C, None, gs)], 0, 1)
        t1 = time.perf_counter() - t0
        rows = max(1, min(cfg.M, max_rows, int(budget_s / max(t1, 1e-6))))
        W = np.ascontiguousarray(S.gen_W(cfg, np.arange(rows))[:, :gs * d])
        c0 = time.process_time()
        t0 = time.perf_counter()
        O.encode_beam(W, d, Hb, [O.Codebook(C, None, gs)], 0, 1)
        wall = time.perf_counter() - t0
        sc = float(rows) * gs * cfg.K_base
        desc = (f"one encode pass of rows 0..{rows - 1} x groups 0..{gs - 1} of {cfg.name} "
                f"against a seeded {cfg.K_base}-entry codebook")
    cpu = time.process_time() - c0
    return sc / wall, wall, max(1, int(round(cpu / max(wall, 1e-9)))), desc


def _pool_init(cfg, threads_env):
    os.environ.update(threads_env)
    global _POOL_X
    _POOL_X = S.gen_X(cfg)


def _pool_job(cfg, r0, rows):
    """One worker's sample: the whole schedule of the oracle on rows r0 .. r0 + rows - 1."""
    from oracle import crvq_oracle as O
    W = S.gen_W(cfg, np.arange(r0, r0 + rows))
    t0 = time.perf_counter()
    O.quantize_layer(W, _POOL_X, cfg)
    return t0, time.perf_counter()


class OraclePool:
    """The fp64 oracle, as it stands, on every host core: one process per core (started with
    spawn, so that it is safe after CUDA initialisation), each running the whole schedule on its
    own block of rows of the workload's first matrix with the full X. Throughput = all samples'
    scores / the wall time from the first start to the last end."""

    def __init__(self, cfg, workers=None):
        import multiprocessing as mp
        from concurrent.futures import ProcessPoolExecutor
        self.cfg = cfg
        self.workers = workers or len(os.sched_getaffinity(0))
        env = {k: "1" for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
        self.ex = ProcessPoolExecutor(max_workers=self.workers,
                                      mp_context=mp.get_context("spawn"),
                                      initializer=_pool_init, initargs=(cfg, env))
        list(self.ex.map(int, range(self.workers)))   # start the workers, build their X

    def rows_for(self, budget_s):
        cfg = self.cfg
        need = rows_needed(cfg)
        per_row = schedule_scores(cfg, 1, cfg.N)
        rate = ORACLE_RATE_EST / 1.5                  # per process, every core busy
        return min(cfg.M // self.workers, max(need, int(budget_s * rate / per_row)))

    def run(self, budget_s):
        rows = self.rows_for(budget_s)
        futs = [self.ex.submit(_pool_job, self.cfg, w * rows, rows) for w in range(self.workers)]
        spans = [f.result() for f in futs]
        wall = max(b for _, b in spans) - min(a for a, _ in spans)
        sc = self.workers * schedule_scores(self.cfg, rows, self.cfg.N)
        desc = (f"whole schedule on {self.workers} row blocks of {rows} rows of {self.cfg.name} "
                f"(full X), one process per host core")
        return sc / wall, wall, self.workers, desc

    def close(self):
        self.ex.shutdown()


def rows_needed(cfg):
    """Rows a whole-schedule sample needs so that every codebook can draw its K vectors."""
    G = cfg.N // cfg.d
    Gc = min(G, int(np.ceil(np.float32(cfg.crit_frac) * cfg.N / cfg.d - 1e-12)))
    return int(np.ceil(max(cfg.K_base / G, cfg.K_ext / Gc if cfg.n_ext > 0 else 0.0)))


def pool_workers(cfg):
    """Host cores the pool can use: one block of rows each, each block large enough for K
    (0 or 1: run one process; a 65536-entry codebook needs 65536 vectors per sample)."""
    need = rows_needed(cfg)
    if need > 64:
        return 0
    return min(len(os.sched_getaffinity(0)), cfg.M // max(need, 1))


def inference_matvec(P, work, flush, stream, reps=20):
    """The inference product from codes (crvq_lut_matvec; the paper's inference setting) on each
    distinct matrix shape of the workload, with one input (the decode matrix-vector product),
    using the codes and codebooks the timed steps produced. The L2 is flushed before every
    call; the time is the library's CUDA events around its two kernels (slice products and the
    ordered reduction) on the launching stream. Algorithmic bytes: every code (4 B), the input,
    the permutation and the output once. A dense bf16 matrix-vector product of the same shape
    (torch), timed with events around the call, is given as context only."""
    import torch
    from paper_2412_09282_gb300 import Codebook
    rows, seen = [], set()
    for w in work:
        cfg, out = w["cfg"], w["out"]
        key = (cfg.M, cfg.N)
        if key in seen:
            continue
        seen.add(key)
        G = cfg.N // cfg.d
        Gc = out.report["n_crit_groups"]
        cbs = [Codebook(out.C_base, out.codes_base, G)] + \
            [Codebook(out.C_ext[t].contiguous(), out.codes_ext[t], Gc) for t in range(cfg.n_ext)]
        x = torch.randn((1, cfg.N), device=out.C_base.device)
        y = torch.empty((1, cfg.M), device=x.device)
        for _ in range(3):
            P.crvq_lut_matvec(x, out.perm, cbs, cfg.M, Y=y)
        P.crvq_profile_filter("matvec")
        P.crvq_profile_begin()
        for _ in range(reps):
            flush.fill_(1.0)
            P.crvq_lut_matvec(x, out.perm, cbs, cfg.M, Y=y)
        torch.cuda.synchronize()
        st = P.crvq_profile_end()
        P.crvq_profile_filter(None)
        P.crvq_sync()
        ms = sum(k["ms"] for k in st) / reps
        kern = {k["name"]: 1e3 * k["ms"] / reps for k in st}
        Wb = w["W_d"].to(torch.bfloat16)
        xb = x[0].to(torch.bfloat16)
        ts = []
        for _ in range(reps + 3):
            flush.fill_(1.0)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            torch.mv(Wb, xb)
            b.record(stream)
            b.synchronize()
            ts.append(a.elapsed_time(b))
        dense = statistics.median(ts[3:])
        nbytes = 4 * (cfg.M * G + cfg.n_ext * cfg.M * Gc) + 4 * cfg.N * 2 + 4 * cfg.M
        rows.append({"matrix": cfg.name.split("/")[-1], "M": cfg.M, "N": cfg.N, "b": 1,
                     "us": 1e3 * ms, "kernels_us": kern, "bytes": nbytes,
                     "gbs": nbytes / (ms / 1e3) / 1e9, "dense_bf16_mv_us": 1e3 * dense})
        del Wb
    return rows


def coupled_sweep_line(P, work, stream):
    """One Gauss-Seidel sweep of the base codebook under the full loss (crvq_coupled_sweep) on
    the workload's first matrix, from the codes the timed steps produced (on a copy): the dense
    H of its X taken to the layer's channel order, the sweep timed with CUDA events around the
    call (its kernels and their launches), the full loss tr(dW H dW^T) before and after."""
    import torch
    from paper_2412_09282_gb300 import Codebook
    w = work[0]
    cfg, out = w["cfg"], w["out"]
    G, Gc = cfg.N // cfg.d, out.report["n_crit_groups"]
    H, _, _, _ = P.crvq_hessian(w["X_d"], cfg.damp_rel, cfg.d)
    perm = out.perm.long()
    Hs = H[perm][:, perm].contiguous()
    del H
    Ws = w["W_d"][:, perm].contiguous()
    cbs = [Codebook(out.C_base, out.codes_base.clone(), G)] + \
        [Codebook(out.C_ext[t].contiguous(), out.codes_ext[t].clone(), Gc)
         for t in range(cfg.n_ext)]
    l0 = P.crvq_coupled_sweep(Ws, Hs, cbs, 0, sweeps=0)[0]
    torch.cuda.synchronize()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(stream)
    P.crvq_coupled_sweep(Ws, Hs, cbs, 0, sweeps=1, want_loss=False)
    b.record(stream)
    b.synchronize()
    P.crvq_sync()
    ms = a.elapsed_time(b)
    l1 = P.crvq_coupled_sweep(Ws, Hs, cbs, 0, sweeps=0)[0]
    return {"call": "crvq_coupled_sweep (one sweep of the base codebook, cross-group terms)",
            "matrix": cfg.name.split("/")[-1], "M": cfg.M, "N": cfg.N, "groups": G,
            "sweep_ms": ms, "loss_full_before": l0, "loss_full_after": l1,
            "loss_full_reduction": 1.0 - l1 / l0,
            "tensor_work": "2 M N^2 flop per sweep (the lazy block products H[block] D^T)"}


def sweep_grid(name):
    """The synthetic analogs of the paper's ablations on one matrix (no datasets: the block
    losses stand in for perplexity): Table 2's reorder strategies (random, W-only, W-A), the
    critical ratio lambda, the number of extended codebooks m - 1 (Sec. 6.3-6.4) and two base
    codebooks, alone and with three extended ones (Sec. 6.4's m = 2 setting at d = 8)."""
    base = S.C5[0] if name == "c5" else S.CONFIGS[name]
    grid = []
    for mode in (2, 1, 0):                                   # Table 2: random, W-only, W-A
        grid.append(("reorder", base.with_(importance_mode=mode, n_ext=1, crit_frac=0.02)))
    for lam in (0.01, 0.02, 0.05, 0.10):                     # lambda
        grid.append(("lambda", base.with_(crit_frac=lam, n_ext=1)))
    for n_ext in (0, 1, 2, 4):                               # m - 1 extended codebooks
        grid.append(("m", base.with_(n_ext=n_ext, crit_frac=0.02)))
    for n_ext in (0, 3):                                     # two base codebooks
        grid.append(("m_base", base.with_(n_base=2, n_ext=n_ext, crit_frac=0.02)))
    return grid


def avg_bits_of(P, cfg):
    """Bits per weight of a setting (Sec. 3.2 Eq. (bitwidth), App. A.1, the reorder index
    included), with e = log2 K_base for every codebook."""
    e = int(np.log2(cfg.K_base))
    return P.crvq_avg_bits_bases(e, cfg.d, cfg.n_base, cfg.n_ext, float(cfg.crit_frac), cfg.M,
                                 cfg.N, True)


def run_sweep(args):
    """One JSON line per grid point of sweep_grid: losses of the quantized matrix, its time
    (CUDA events around crvq_quantize_layer, inputs resident) and the average bits per weight
    of the setting (Eq. bitwidth with e = log2 K, d = 8, the reorder index included)."""
    import torch
    import paper_2412_09282_gb300 as P
    from paper_2412_09282_gb300 import build as B
    B.build()
    dev = torch.device("cuda", 0)
    stream = torch.cuda.current_stream(dev)
    cache = {}
    for axis, cfg in sweep_grid(args.config):
        key = (cfg.name, cfg.x_tag)
        if key not in cache:
            cache[key] = (torch.from_numpy(S.gen_W(cfg)).to(dev),
                          torch.from_numpy(S.gen_X(cfg)).to(dev))
        W, X = cache[key]
        out = P.crvq_quantize_layer(W, X, cfg)                # captured / warm
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        out = P.crvq_quantize_layer(W, X, cfg, out=out)
        b.record(stream)
        b.synchronize()
        P.crvq_sync()
        rep = out.report
        bits = avg_bits_of(P, cfg)
        print(json.dumps({"sweep": axis, "matrix": cfg.name, "importance_mode": cfg.importance_mode,
                          "crit_frac": cfg.crit_frac, "n_base": cfg.n_base, "n_ext": cfg.n_ext,
                          "n_crit_groups": rep["n_crit_groups"], "avg_bits": bits,
                          "loss_block": rep["loss_block"], "loss_crit": rep["loss_crit"],
                          "loss_full": rep["loss_full"], "loss_pre": rep["loss_pre"],
                          "ms": a.elapsed_time(b)}), flush=True)


def dist_init():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if _cuda_ok() else "gloo")
    return ws, rank, local


def rank_aggregate(tot_ms, scores, ws, device):
    """Whole-job figures of a weak-scaling run: the slowest rank's time and every rank's scores
    (value = all ranks' scores / the slowest rank's time). One process per GPU; the two
    reductions go through torch.distributed (NCCL on GPUs, gloo on CPU)."""
    if ws <= 1:
        return float(tot_ms), float(scores)
    import torch
    import torch.distributed as dist
    t = torch.tensor([tot_ms], dtype=torch.float64, device=device)
    sc = torch.tensor([scores], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(sc, op=dist.ReduceOp.SUM)
    return float(t[0]), float(sc[0])


def _cuda_ok():
    import torch
    return torch.cuda.is_available()


def run_reference(args, layers, ws, rank):
    """Reference arm: the fp64 CPU oracle on bounded samples of the workload's first matrix on
    every host core (one process per core, each its own rows; sized so the whole run stays
    within a few minutes), rank 0 only. Workloads whose codebook needs more rows than a sample
    can hold (K = 65536) time one encode pass in one process instead."""
    if rank != 0:
        return
    cfg = layers[0]
    budget = min(20.0, max(2.0, 150.0 / max(1, args.steps + (args.warmup if args.ref_warmup
                                                              else 0))))
    workers = pool_workers(cfg)
    pool = OraclePool(cfg, workers) if workers > 1 else None
    X = None if pool else S.gen_X(cfg)

    def sample():
        if pool:
            return pool.run(budget)
        return cpu_oracle_sample(cfg, X, budget, args.ref_rows)

    for _ in range(args.warmup if args.ref_warmup else 0):
        sample()
    tot, sc_tot, cores, desc = 0.0, 0.0, 1, ""
    for _ in range(args.steps):
        v, wall, cores, desc = sample()
        tot += wall
        sc_tot += v * wall
    if pool:
        pool.close()
    value = sc_tot / tot
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "scores/s",
        "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * tot / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": DATA,
        "config": workload_dict(args.config, layers, rows_note=desc),
        "cpu_baseline": {"value": value, "unit": "scores/s", "cores": cores, "kind": "oracle",
                         "sample": desc},
        "e2e": {"value": value, "unit": "scores/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


METRIC = "code-search scores/s (whole-layer CRVQ quantize, S1-S7)"
DATA = ("synthetic: seeded SplitMix64/Box-Muller LLaMA-2-shaped weights and calibration "
        "activations (no real weights or Red_Pajama text)")


def assign_lanes(sizes, streams):
    """Matrices (by size) to at most `streams` lanes: largest first, each to the least loaded
    lane. Returns the lanes' matrix indices, in the order each lane runs them."""
    n = max(1, min(streams, len(sizes)))
    lanes = [[] for _ in range(n)]
    load = [0] * n
    for j in sorted(range(len(sizes)), key=lambda j: (-sizes[j], j)):
        q = load.index(min(load))
        lanes[q].append(j)
        load[q] += sizes[j]
    return lanes


def config_dict(cfg, rows_note=None):
    c = {"workload": cfg.name, "M": cfg.M, "N": cfg.N, "n_tok": cfg.n_tok, "d": cfg.d,
         "K_base": cfg.K_base, "n_ext": cfg.n_ext, "K_ext": cfg.K_ext,
         "crit_frac": cfg.crit_frac, "B": cfg.B, "kmeans_iters": cfg.kmeans_iters,
         "refine_rounds": cfg.refine_rounds,
         "l2": "flushed between timed steps (512 MB write)"}
    if rows_note:
        c["sample"] = rows_note
    return c


def workload_dict(name, layers, rows_note=None):
    """config of the JSON line: the layer's settings, or the block's matrices."""
    if len(layers) == 1:
        return config_dict(layers[0], rows_note)
    c = config_dict(layers[0], rows_note)
    c["workload"] = "c5_llama2_7b_decoder_block (7 matrices, one step = the whole block)"
    c["matrices"] = [{"name": L.name.split("/")[-1], "M": L.M, "N": L.N} for L in layers]
    c["shared_X"] = "q,k,v,o,gate,up share one 4096 x 4096 X; down_proj its own 4096 x 11008"
    for k in ("M", "N"):
        c.pop(k)
    return c


def workload_layers(name):
    """The matrices one step quantizes: one layer, or the seven matrices of the decoder block."""
    if name == "c5":
        return list(S.C5)
    return [S.CONFIGS[name]]


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="crvq", choices=["crvq", "reference"])
    ap.add_argument("--config", default="c5", choices=sorted(S.CONFIGS) + ["c5"])
    ap.add_argument("--ref-rows", type=int, default=64,
                    help="most rows a whole-schedule oracle sample takes beyond what K needs")
    ap.add_argument("--ref-warmup", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--streams", type=int, default=3,
                    help="streams (and host threads) the matrices of a step run on")
    ap.add_argument("--no-infer", action="store_true",
                    help="skip the inference-product and coupled-sweep lines after the timed "
                         "steps")
    ap.add_argument("--sweep", action="store_true",
                    help="run the reorder / lambda / m sweep on the workload's first matrix "
                         "instead of the benchmark (one JSON line per setting)")
    args = ap.parse_args()
    if args.sweep:
        run_sweep(args)
        return
    layers = workload_layers(args.config)
    ws, rank, local = dist_init()
    if args.impl == "reference":
        run_reference(args, layers, ws, rank)
        return

    import torch
    import paper_2412_09282_gb300 as P
    from paper_2412_09282_gb300 import build as B
    B.build()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    # each rank quantizes its own matrices; layers of a block that share X share one buffer
    xs = {}
    work = []
    for cfg in layers:
        cfg_r = cfg.with_(seed=cfg.seed + rank)
        tag = cfg_r.x_tag or cfg_r.name
        if tag not in xs:
            Xn = S.gen_X(cfg_r)
            X_h = torch.from_numpy(Xn).pin_memory()
            xs[tag] = (Xn, X_h, X_h.to(dev))
        Xn, X_h, X_d = xs[tag]
        W_h = torch.from_numpy(S.gen_W(cfg_r)).pin_memory()
        work.append({"cfg": cfg_r, "W_h": W_h, "W_d": W_h.to(dev), "X_h": X_h, "X_d": X_d,
                     "Xn": Xn, "out": None, "h_out": None})
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    # The matrices of a step are independent problems. With --streams S > 1 they run on S
    # streams from S host threads (the library replays each matrix's graph on its own stream
    # without holding its cache lock), balanced by size, largest first.
    lanes = assign_lanes([w["cfg"].M * w["cfg"].N for w in work], args.streams)
    nstr = len(lanes)
    streams = [stream] if nstr == 1 else [torch.cuda.Stream(dev) for _ in range(nstr)]
    pool = None
    if nstr > 1:
        from concurrent.futures import ThreadPoolExecutor
        pool = ThreadPoolExecutor(nstr)

    def run_lane(q, host, start):
        s = streams[q]
        sc = 0.0
        with torch.cuda.device(dev):
            if start is not None:
                s.wait_event(start)
            for j in lanes[q]:
                w = work[j]
                if host:
                    w["h_out"] = P.crvq_quantize_layer(w["W_h"], w["X_h"], w["cfg"],
                                                       out=w["h_out"], stream=s, device=dev)
                    sc += w["h_out"].report["scores"]
                else:
                    w["out"] = P.crvq_quantize_layer(w["W_d"], w["X_d"], w["cfg"],
                                                     out=w["out"], stream=s)
                    sc += w["out"].report["scores"]
        return sc

    def run_step(host=False, sequential=False):
        """One step: every matrix of the workload through crvq_quantize_layer. Returns the
        scores of the step."""
        if sequential:  # the matrices one after another on the main stream
            sc = 0.0
            for w in work:
                w["out"] = P.crvq_quantize_layer(w["W_d"], w["X_d"], w["cfg"], out=w["out"],
                                                 stream=stream)
                sc += w["out"].report["scores"]
            return sc
        if pool is None:
            return run_lane(0, host, None)
        start = torch.cuda.Event()
        start.record(stream)
        sc = sum(f.result() for f in [pool.submit(run_lane, q, host, start)
                                      for q in range(nstr)])
        for s in streams:  # every call has synchronized its stream; order the main one after
            stream.wait_stream(s)
        return sc

    for _ in range(args.warmup):
        run_step()
    torch.cuda.synchronize()

    def barrier():
        if ws > 1:
            import torch.distributed as dist
            dist.barrier()
        torch.cuda.synchronize()

    clocks = ClockSampler(local)
    try:
        clocks.gpu_id = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        clocks.gpu_id = local
    # events only around the arg-min launches (the roofline kernel): the other launches of
    # the timed steps run unbracketed. The library replays a captured CUDA graph of each
    # matrix per profiling state; one untimed step captures the ones the timed steps use.
    P.crvq_profile_filter("encode_argmin")
    P.crvq_profile_begin()
    run_step()
    torch.cuda.synchronize()
    P.crvq_profile_end()
    barrier()
    clocks.start()
    launches0 = P.crvq_launch_count()
    P.crvq_profile_begin()
    step_ms = []
    scores = 0.0
    for _ in range(args.steps):
        flush.fill_(1.0)                                     # evict the 129 MB L2
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        scores += run_step()
        b.record(stream)
        b.synchronize()
        step_ms.append(a.elapsed_time(b))
    barrier()
    argmin_stats = [k for k in P.crvq_profile_end()
                    if k["name"] in ("encode_argmin", "encode_argmin_lloyd")]
    launches = P.crvq_launch_count() - launches0
    clk = clocks.stop()
    # With several streams the arg-min launches of the timed steps share the GPU with the other
    # streams' kernels. One more step, untimed, runs the matrices one after another for the
    # kernel's own launch time beside the live one.
    iso_stats = None
    if nstr > 1:
        P.crvq_profile_filter("encode_argmin")
        P.crvq_profile_begin()
        run_step(sequential=True)
        torch.cuda.synchronize()
        iso_stats = [k for k in P.crvq_profile_end()
                     if k["name"] in ("encode_argmin", "encode_argmin_lloyd")]
    # per-kernel breakdown: one more step, untimed, the matrices one after another, every
    # launch bracketed
    P.crvq_profile_filter(None)
    P.crvq_profile_begin()
    run_step(sequential=True)
    torch.cuda.synchronize()
    kstats = P.crvq_profile_end()
    tot_ms_max, scores_all = rank_aggregate(sum(step_ms), scores, ws, dev)
    value = scores_all / (tot_ms_max / 1e3)

    # End to end through the public C ABI with host buffers (pinned): H2D of W and X and D2H
    # of every output inside the timed region, wall clock around synchronizing calls.
    e2e_times = []
    e2e_scores = 0.0
    for i in range(args.e2e_steps + 1 if args.e2e_steps > 0 else 0):
        t0 = time.perf_counter()
        sc = run_step(host=True)
        dt = time.perf_counter() - t0
        if i > 0:
            e2e_times.append(dt)
            e2e_scores = sc
    e2e = None
    if e2e_times:
        h2d = sum(w["W_h"].numel() * 4 + w["X_h"].numel() * 4 for w in work)
        d2h = 0
        for w in work:
            o = w["h_out"]
            d2h += sum(t.numel() * t.element_size() for t in
                       [o.perm, o.C_base, o.codes_base, o.C_ext, o.codes_ext, o.W_hat,
                        o.importance] if t is not None) + 48
        e2e = {"value": ws * e2e_scores / statistics.mean(e2e_times),
               "unit": "scores/s", "h2d_bytes_per_step": int(h2d),
               "d2h_bytes_per_step": int(d2h),
               "ms_per_step": 1e3 * statistics.mean(e2e_times)}

    infer = inference_matvec(P, work, flush, stream) if not args.no_infer else None
    coupled = coupled_sweep_line(P, work, stream) if not args.no_infer else None

    if rank != 0:
        return
    peaks, peak_src = load_peaks()
    props = torch.cuda.get_device_properties(dev)
    nsm = props.multi_processor_count
    ks = sorted(kstats, key=lambda k: -k["ms"])
    total_k = sum(k["ms"] for k in ks) or 1.0
    # The dominant kernel is the tensor-core arg-min (argmin_tc_kernel): tcgen05 computes the
    # certified lower bound of every (vector, codeword) score as a 3xTF32 dot product of length
    # 32 (64 tf32 flop issued per score), and its epilogue keeps the two smallest of each row.
    # The roofline is the score contraction's algorithmic work, 2 d = 16 flop per score, against
    # the tf32 tensor peak (the measured bf16 rate scaled by the nominal tf32 / bf16 ratio; the
    # sustained figure, since the kernel is timed inside a long step). The issued-flop fraction
    # and the integer ALU pipe that binds the epilogue are reported beside it.
    enc_ms = sum(k["ms"] for k in argmin_stats)
    enc_units = sum(k["units"] for k in argmin_stats)
    enc_launches = sum(k["launches"] for k in argmin_stats)
    sec = enc_ms / 1e3 if enc_ms > 0 else float("inf")
    bf16 = peaks.get("bf16_tflops_sustained", peaks.get("bf16_tflops", 1700.0))
    tf32_peak = TF32_PER_BF16 * bf16
    alg_tflops = enc_units * 16.0 / sec / 1e12
    issued_tflops = enc_units * 64.0 / sec / 1e12
    mhz = peaks.get("sm_max_mhz", 2070.0)
    alu_peak = nsm * 64 * mhz * 1e6 / 1e12
    alu_achieved = enc_units * ALU_OPS_PER_SCORE / sec / 1e12
    traffic = ARGMIN_TRAFFIC.get(args.config)
    roof = {"kernel": "argmin_tc_kernel (tensor-core arg-min, all passes of the step)",
            "bound": "tensor", "achieved": alg_tflops, "peak": tf32_peak, "unit": "TFLOP/s",
            "frac": alg_tflops / tf32_peak, "traffic": traffic,
            "work": "2 d = 16 flop per scored (vector, codeword) pair (the score contraction)",
            "peak_source": (f"tf32 = {TF32_PER_BF16:.4f} x bf16 sustained {bf16} TFLOP/s "
                            f"({peak_src}, MEASURED_PEAKS.json) of measured"),
            "avg_launch_ms": enc_ms / max(enc_launches, 1), "launches": enc_launches,
            "scores_per_launch": enc_units / max(enc_launches, 1),
            "issued": {"achieved": issued_tflops, "frac": issued_tflops / tf32_peak,
                       "work": "64 tf32 flop per scored pair issued (K = 32 split operands)"},
            "alu": {"achieved": alu_achieved, "peak": alu_peak, "unit": "TOP/s",
                    "frac": alu_achieved / alu_peak,
                    "work": (f"{ALU_OPS_PER_SCORE} integer ALU ops per scored pair (the "
                             "kernel's ALU pipe instructions, measured by ncu)"),
                    "peak_source": f"{nsm} SMs x 64 ALU lanes x {mhz:.0f} MHz"}}
    if iso_stats:
        roof["streams"] = nstr
        roof["note"] = (f"live: the timed steps, the matrices on {nstr} streams, so arg-min "
                        "launches share the GPU with other streams' kernels; isolated: one "
                        "untimed step with the matrices one after another")
        i_ms = sum(k["ms"] for k in iso_stats)
        i_units = sum(k["units"] for k in iso_stats)
        i_launches = sum(k["launches"] for k in iso_stats)
        i_sec = i_ms / 1e3 if i_ms > 0 else float("inf")
        i_alg = i_units * 16.0 / i_sec / 1e12
        roof["isolated"] = {
            "achieved": i_alg, "frac": i_alg / tf32_peak,
            "avg_launch_ms": i_ms / max(i_launches, 1), "launches": i_launches,
            "issued_frac": i_units * 64.0 / i_sec / 1e12 / tf32_peak,
            "alu_frac": i_units * ALU_OPS_PER_SCORE / i_sec / 1e12 / alu_peak}
    last = work[-1]["out"].report if len(work) == 1 else None
    line = {
        "metric": METRIC, "value": value, "unit": "scores/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": tot_ms_max / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": DATA, "config": dict(workload_dict(args.config, layers), streams=nstr),
        "layer_time_s": tot_ms_max / args.steps / 1e3 / len(work),
        "roofline": roof,
        "e2e": e2e,
        "gpu_launches": int(launches),
        "exact_fallback_decisions_per_step": sum(w["out"].report["flagged"] for w in work),
        "kernels": [{"name": k["name"], "launches": k["launches"], "ms": k["ms"],
                     "share": k["ms"] / total_k} for k in ks[:12]],
        "clocks": clk,
    }
    if infer:
        for r in infer:
            r["hbm_frac"] = r["gbs"] / peaks.get("hbm_gbs", 6800.0)
        line["inference_matvec"] = {
            "call": "crvq_lut_matvec (Y = x W_hat^T from the codes, one input)",
            "peak_gbs": peaks.get("hbm_gbs"), "peak_source": f"hbm_gbs ({peak_src}) burst",
            "shapes": infer}
    if coupled:
        line["coupled_sweep"] = coupled
    if last is not None:
        line["losses"] = {k: last[k] for k in ("loss_pre", "loss_block", "loss_crit",
                                                "loss_full")}
    else:
        line["block_time_s"] = tot_ms_max / args.steps / 1e3
        line["losses"] = {w["cfg"].name: {k: w["out"].report[k] for k in
                                          ("loss_pre", "loss_block", "loss_crit", "loss_full")}
                          for w in work}
    if ws == 1 and not args.no_cpu_baseline:
        w0 = work[0]
        v1, wall1, cores1, desc1 = cpu_oracle_sample(w0["cfg"], w0["Xn"], 20.0, args.ref_rows)
        one = {"value": v1, "unit": "scores/s", "cores": cores1, "kind": "oracle",
               "sample": f"{desc1}, {wall1:.1f} s"}
        workers = pool_workers(w0["cfg"])
        if workers > 1:
            pool = OraclePool(w0["cfg"], workers)
            v, wall, cores, desc = pool.run(15.0)
            pool.close()
            line["cpu_baseline"] = {"value": v, "unit": "scores/s", "cores": cores,
                                    "kind": "oracle", "sample": f"{desc}, {wall:.1f} s",
                                    "one_core": one}
        else:
            line["cpu_baseline"] = one
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
