#!/usr/bin/env python
"""Throughput of the BaKron solve on GB300: weight entries quantized per second.

Workload (default): the 4096 x 4096 attention-projection layer -- W bf16
~N(0, 0.02^2) with 0.1% outlier columns x10, A and B power-law Grams from 8192
samples, 1% damping, 4-bit per-row grid -- drawn by ``workloads`` on the GPU.
A step is one bakron_solve (grid, leaf wavefronts and all band products) on
one resident W with the factors prepared beforehand, replayed from a CUDA
graph captured once (``--no-graph`` launches eagerly); the device prepare is
timed separately and reported in ``prepare_ms``.  L2 is flushed (256 MiB
write) between timed steps, outside the timed events.

Also reported: ``e2e`` (the same solve with W copied from pinned host memory
and codes/scales/zeros copied back inside the timed region), ``roofline`` of
the dominant kernel family (timed live with CUDA events on the launch stream
through the library's profiling hooks), ``cpu_baseline`` (the float64 oracle
on a bounded exact sub-problem: the top-left block, whose codes depend on
nothing else), clocks sampled during the timed region, and ``gpu_launches``.

``--impl reference`` times the oracle itself (the reference arm) on the host
cores, each step a bounded top-left block of the same workload.
Multi-GPU: the solve does not shard (2-D wavefront); ``--gpus N`` under
torchrun runs N independent replicas ("replicas only", weak scaling), with a
barrier and max-over-ranks timing and no data-path collective.
"""
from __future__ import annotations

import argparse
import glob
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "weight entries quantized/sec (4096x4096 BaKron solve, 1 GB300); % of roofline"
UNIT = "entries/s"
PAPER_4096_S = 0.288          # paper's BaKron time for 4096 x 4096 (RTX PRO 6000), context
TILE = 32                     # leaf tile of the library (intra-tile work is the leaf's)
L2_FLUSH_BYTES = 256 << 20


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(x: float, ws_n: int, device="cpu") -> float:
    """The slowest rank's time: all-reduce MAX of x over the process group
    (identity for one process).  `device` is where the collective's tensor
    lives (the GPU for NCCL, "cpu" for gloo)."""
    if ws_n <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: float, ws_n: int, ms: float) -> float:
    """Units all ranks processed (each rank the same, weak scaling) per second
    of the slowest rank's time."""
    return ws_n * units_per_rank / (ms / 1e3)


def _peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return None


def f_alg(m: int, n: int, identity_b: bool = False) -> float:
    """Algorithmic flops of one m x n solve: twice the multiply-adds with a
    structurally nonzero factor operand in Alg. 4's recursion down to single
    entries -- split the longer side (columns when m < n), first part
    floor(size / 2), each bulk update L^B E L^A^T multiplied in its cheaper
    order, triangular diagonal blocks counted at their strictly-lower part
    (their unit diagonal adds, it does not multiply).  With B = I (GPTQ) the
    output-side factor contributes no products at all.  4096 x 4096: 2.403e11
    (1.75 m n (m + n))."""
    memo = {}

    def tri(d):
        return d * (d - 1) // 2

    def macs(mm, nn):
        if mm == 1 and nn == 1:
            return 0
        key = (mm, nn)
        if key in memo:
            return memo[key]
        if mm < nn:
            h = nn // 2
            upd = mm * h * (nn - h) + (0 if identity_b else tri(mm) * min(h, nn - h))
            r = macs(mm, h) + macs(mm, nn - h) + upd
        else:
            h = mm // 2
            upd = 0 if identity_b else (mm - h) * h * nn + tri(nn) * min(h, mm - h)
            r = macs(h, nn) + macs(mm - h, nn) + upd
        memo[key] = r
        return r

    return 2.0 * macs(int(m), int(n))


def fp32_effective_peak(peaks) -> tuple:
    """FP32-effective tensor rate of the 3xTF32 band products, TFLOP/s: the
    measured bf16 burst rate halved (tf32 runs at half the bf16 rate) and
    divided by the three MMAs of the split.  Burst, because a step is a few
    milliseconds and the timed region well under a second."""
    bf16 = float((peaks or {}).get("bf16_tflops", 1892.3))
    return bf16 / 2.0 / 3.0, "of measured: bf16_tflops (burst) / 2 (tf32 rate) / 3 (3xTF32)"


def host_info() -> dict:
    """What the host oracle runs on: logical CPUs, CPU model, BLAS threads."""
    import platform
    info = {"os_cpu_count": os.cpu_count(), "machine": platform.machine()}
    try:
        for line in open("/proc/cpuinfo"):
            low = line.lower()
            if low.startswith("model name") or low.startswith("cpu part"):
                info["cpu_model"] = line.split(":", 1)[1].strip()
                break
    except Exception:
        pass
    try:
        import threadpoolctl
        blas = [p for p in threadpoolctl.threadpool_info() if p.get("user_api") == "blas"]
        if blas:
            info["blas"] = blas[0].get("internal_api")
            info["blas_threads"] = blas[0].get("num_threads")
    except Exception:
        for var in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
            if os.environ.get(var):
                info["blas_threads"] = int(os.environ[var])
                break
        info.setdefault("blas_threads", "library default (all logical CPUs)")
    return info


# The sources that define the solve's kernels and its launch schedule: the
# DRAM figures in profiles/traffic.txt stand while these are unchanged.
SOLVE_SOURCES = ("common.cuh", "profile.cu", "profile.cuh", "solve.cu", "solve.cuh",
                 "tc_gemm.cu", "tc_gemm.cuh", "tune.cu", "tune.cuh")


def _csrc_hash():
    h = hashlib.sha256()
    for name in SOLVE_SOURCES:
        with open(os.path.join(ROOT, "paper_2608_06291_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def _traffic(workload, family, launches):
    """DRAM bytes (read + write) per launch of a kernel family, from the
    committed ncu summary of this workload (`profiles/traffic.txt`: bytes per
    solve by family), or None when there is none or the kernel sources
    changed since it was taken."""
    p = os.path.join(ROOT, "profiles", "traffic.txt")
    try:
        t = json.load(open(p))
    except Exception:
        return None
    if t.get("csrc_hash") != _csrc_hash() or not launches:
        return None
    per_step = t.get("workloads", {}).get(workload, {}).get(family)
    return None if per_step is None else per_step / launches


def _traffic_warm(workload, family, launches):
    """The same per launch from the launch list taken without ncu's L2 flush
    between launches (`<family>_warm_l2`), or None."""
    return _traffic(workload, family + "_warm_l2", launches)


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons (read only)."""
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, bus_id=None):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
               "-lms", "100"]
        if bus_id:
            cmd += ["-i", bus_id]
        try:
            self.p = subprocess.Popen(cmd, stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.p = None

    def stop(self, t0, t1):
        if self.p is None:
            return None
        time.sleep(0.25)
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except Exception:
            self.p.kill()
        self.f.flush()
        rows = [r.split(",") for r in open(self.f.name).read().strip().splitlines() if r.strip()]
        os.unlink(self.f.name)
        samples = []
        for r in rows:
            try:
                ts = time.mktime(time.strptime(r[0].strip().split(".")[0], "%Y/%m/%d %H:%M:%S"))
                samples.append((ts, float(r[1]), float(r[2]), [x.strip() for x in r[5:9]]))
            except Exception:
                continue
        inside = [s for s in samples if t0 - 1.0 <= s[0] <= t1 + 1.0] or samples
        if not inside:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for s in inside for i, v in enumerate(s[3]) if v == "Active"})
        return {"sm_mhz": statistics.median(s[1] for s in inside),
                "sm_max_mhz": max(s[2] for s in inside), "reasons": reasons,
                "samples": len(inside)}


# ----------------------------------------------------------------- oracle legs
def _grid_block(W64, bits, group, k):
    """The full problem's grid restricted to the top-left k x k block: per-row
    (or per-group) min-max over the whole rows, then the block's columns."""
    import oracle as O
    g = O.quant_grid(W64[:k], bits, group)
    if group:
        return O.Grid(g.s[:, :k // group], g.z[:, :k // group], g.qmax, group)
    return g


def _oracle_block(W64, f, bits, group, k):
    """Time the float64 oracle (Alg. 4, Alg. 3 on 64 x 64 blocks) on the
    top-left k x k block of the workload: entry (i, j) depends only on entries
    up-left of it, so with the full problem's factors and grid restricted to
    the block this is an exact part of the full solve."""
    import oracle as O
    Wb = W64[:k, :k]
    g = _grid_block(W64, bits, group, k)
    c0 = os.times()
    t0 = time.perf_counter()
    O.bakron_recursive(Wb, f.LA[:k, :k], f.LB[:k, :k], g, base=64)
    wall = time.perf_counter() - t0
    c1 = os.times()
    cpu = (c1.user - c0.user) + (c1.system - c0.system)
    return wall, max(1, round(cpu / wall)) if wall > 0 else 1


def _block_note(m, n, k):
    """How the per-entry work of the k x k sample compares with the full m x n
    problem (the oracle's time per entry grows with F_alg / (m n))."""
    ratio = (f_alg(k, k) / (k * k)) / (f_alg(m, n) / (m * n))
    return {"sample_entries": k * k, "per_entry_flops_ratio": ratio}


def _timed(fn):
    """Wall time of fn() and the host threads it kept busy on average (CPU
    time / wall time, at least 1): the `cores` of a cpu_baseline; the host's
    logical CPUs and BLAS threads are reported beside it (`host_info`)."""
    c0 = os.times()
    t0 = time.perf_counter()
    fn()
    wall = time.perf_counter() - t0
    c1 = os.times()
    cpu = (c1.user - c0.user) + (c1.system - c0.system)
    return wall, max(1, round(cpu / wall)) if wall > 0 else 1


def extra_cpu_baseline(workload, data):
    """The oracle, as it stands, on a bounded sample of an extra workload's
    input, in the unit of that workload's line.  `data` holds host float64
    arrays (see run_extra):
      gram     X (k_s x d sample rows): oracle Gram, flop/s d (d + 1) k_s / s
      symgrid  W (rows x n sample): oracle symmetric grid, entries/s
      batched / gptq  W, LA, LB (an exact top-left block: entry (i, j) depends
               only on entries up-left of it), bits: oracle Alg. 4, entries/s"""
    import oracle as O
    if workload == "gram":
        X = data["X"]
        k_s, d = X.shape
        wall, cores = _timed(lambda: O.gram(X, alpha=1.0 / k_s))
        return {"value": d * (d + 1) * k_s / wall, "unit": "flop/s", "cores": cores,
                "kind": "oracle",
                "sample": f"first {k_s} of the rows ({k_s} x {d}), float64 Gram, {wall:.2f} s wall",
                "host": host_info()}
    if workload == "symgrid":
        W = data["W"]
        wall, cores = _timed(lambda: O.symmetric_grid(W.astype(np.float32), 3, 0, 50))
        return {"value": W.size / wall, "unit": "entries/s", "cores": cores, "kind": "oracle",
                "sample": f"first {W.shape[0]} rows ({W.shape[0]} x {W.shape[1]}), l = 3, "
                          f"50 shrink steps, {wall:.2f} s wall", "host": host_info()}
    W, LA, LB, bits = data["W"], data["LA"], data["LB"], data["bits"]
    # the per-row grid of the full rows (data["rows"]), which the block's
    # columns share: the block is then an exact part of the full solve
    g = O.quant_grid(data["rows"], bits, 0)
    wall, cores = _timed(lambda: O.bakron_recursive(W, LA, LB, g, base=64))
    return {"value": W.size / wall, "unit": "entries/s", "cores": cores, "kind": "oracle",
            "sample": f"exact top-left {W.shape[0]} x {W.shape[1]} block (grid from the full "
                      f"rows), float64 Alg. 4 with Alg. 3 on 64 x 64 blocks, {wall:.2f} s wall",
            "host": host_info()}


def _oracle_factors(A, B, damp):
    import oracle as O
    return O.prepare(A.double().cpu().numpy(), B.double().cpu().numpy(), damp, via_inverse=False)


def run_reference(args):
    """The reference arm: the oracle, as it stands, on the host cores."""
    import torch
    import workloads as WL
    ws, rank, local = _dist()
    if rank != 0:
        return 0
    cfg = WL.CONFIGS[args.config]
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    W, A, B = WL.make(cfg, device=dev)
    f = _oracle_factors(A, B, cfg.damp)
    W64 = W.double().cpu().numpy()
    k = args.ref_block
    for _ in range(args.warmup):
        _oracle_block(W64, f, cfg.bits, cfg.group, k)
    times, cores = [], 1
    for _ in range(args.steps):
        t, c = _oracle_block(W64, f, cfg.bits, cfg.group, k)
        times.append(t)
        cores = max(cores, c)
    ms = 1e3 * sum(times) / len(times)
    value = k * k / (ms / 1e3)
    sample = (f"top-left {k}x{k} block of the {cfg.m}x{cfg.n} workload per step (exact "
              f"sub-problem: full-problem factors and grid), float64 Alg. 4 oracle with Alg. 3 "
              f"on 64 x 64 blocks")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": _config_dict(cfg),
        "cpu_baseline": dict({"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                              "sample": sample, "host": host_info()},
                             **_block_note(cfg.m, cfg.n, k)),
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))
    return 0


def _config_dict(cfg):
    return {"workload": f"config {cfg.index}: {cfg.name}, W {str(cfg.w_dtype).split('.')[-1]} "
                        f"{cfg.w_dist}, {cfg.bits}-bit "
                        + ("per-row" if cfg.group == 0 else f"g{cfg.group}") + " grid, "
                        f"power-law Grams from {cfg.n_samples} samples, damp {cfg.damp}",
            "m": cfg.m, "n": cfg.n, "bits": cfg.bits, "group": cfg.group,
            "l2": "flushed between timed steps (256 MiB write)", "factors": "precomputed"}


# --------------------------------------------------------------------- main arm
def run_gpu(args):
    import numpy as np
    import torch

    import paper_2608_06291_gb300 as P
    import workloads as WL

    ws_n, rank, local = _dist()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if ws_n > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    P.build()
    P.lib()
    cfg = WL.CONFIGS[args.config]
    m, n = cfg.m, cfg.n
    W, A, B = WL.make(cfg, device=dev)
    work = P.alloc_workspace(m, n, dev)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    fac = P.bakron_prepare(A, B, cfg.damp, workspace=work)
    torch.cuda.synchronize()
    prepare_ms = 1e3 * (time.perf_counter() - t0)
    G = 1 if cfg.group == 0 else n // cfg.group
    codes = torch.empty(m, n, dtype=torch.uint8, device=dev)
    scales = torch.empty(m, G, dtype=torch.float32, device=dev)
    zeros = torch.empty(m, G, dtype=torch.float32, device=dev)
    out = (codes, scales, zeros, None)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def eager_step():
        P.bakron_solve(W, fac, cfg.bits, cfg.group, workspace=work, sync=False, out=out)

    # the library's own schedule autotune for this shape (outside the timed region)
    sched = P.bakron_get_tuning(m, n)
    sched["autotuned"] = False
    if not args.no_autotune:
        best = P.bakron_autotune(W, fac, cfg.bits, cfg.group, workspace=work)
        sched = {"tc_min_band": best["tc_min_band"], "fused_max_band": best["fused_max_band"],
                 "leaf_block": best["leaf_block"], "autotuned": True}
    for _ in range(max(3, args.warmup)):
        flush.fill_(1)
        eager_step()
    torch.cuda.synchronize()
    if P.bakron_read_status(work) != 0:
        raise RuntimeError("device status set during warm-up")
    launches_per_solve = P.bakron_last_launches()
    graph = None
    if not args.no_graph:
        # the solve's launch sequence depends only on shapes and buffers: capture
        # it once and replay it (no host enqueue cost per kernel)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            eager_step()
        graph.replay()
        torch.cuda.synchronize()

    def step():
        if graph is not None:
            graph.replay()
        else:
            eager_step()

    bus = None
    try:
        bus = torch.cuda.get_device_properties(dev).pci_bus_id
    except Exception:
        pass
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(bus) if rank == 0 else None
    time.sleep(0.3)
    if ws_n > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    w0 = time.time()
    launches = 0
    for i in range(args.steps):
        flush.fill_(i & 0xFF)
        starts[i].record(stream)
        step()
        ends[i].record(stream)
        launches += launches_per_solve
    torch.cuda.synchronize()
    if ws_n > 1:
        torch.distributed.barrier()
    w1 = time.time()
    clocks = sampler.stop(w0, w1) if sampler else None
    ms = sum(s.elapsed_time(e) for s, e in zip(starts, ends)) / args.steps
    ms = max_over_ranks(ms, ws_n, dev)
    if P.bakron_read_status(work) != 0:
        raise RuntimeError("device status set during the timed steps")
    value = whole_job_rate(m * n, ws_n, ms)

    # per-family device time of the step as it is timed: the solve captured
    # once more with the library's timeline stamps (no events between the
    # launches, so the programmatic overlap stays) and replayed; each replay's
    # launches partition its device time
    P.bakron_profile_enable(2)
    if graph is not None:
        pgraph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(pgraph):
            eager_step()
        prof_step = pgraph.replay
    else:
        prof_step = eager_step
    prof_steps = max(3, min(args.steps, 10))
    for i in range(prof_steps):
        flush.fill_(i & 0xFF)
        prof_step()
        P.bakron_profile_collect()
    fam = P.bakron_profile_read()
    nrep, span_ms = P.bakron_profile_timeline()
    P.bakron_profile_enable(False)
    if P.bakron_read_status(work) != 0:
        raise RuntimeError("device status set during the profiling replays")
    fam_ms = {k: v[1] / prof_steps for k, v in fam.items()}
    fam_n = {k: v[0] // prof_steps for k, v in fam.items()}
    fam_fl = {k: v[2] / prof_steps for k, v in fam.items()}
    timeline_ms = span_ms / max(1, nrep)

    peaks = _peaks() or {}
    wl_key = f"config {args.config}"
    F_alg = f_alg(m, n)
    sm_max = float(peaks.get("sm_max_mhz", 2070.0))
    p_eff, p_src = fp32_effective_peak(peaks)
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    fp32_simt_peak = 152 * 128 * 2 * sm_max * 1e6 / 1e12     # TFLOP/s, FFMA on CUDA cores
    groups = {
        "tc": (fam_ms["tc1"] + fam_ms["tc2"], fam_fl["tc1"] + fam_fl["tc2"],
               fam_n["tc1"] + fam_n["tc2"]),
        "simt": (fam_ms["band1"] + fam_ms["band2"] + fam_ms["fused"],
                 fam_fl["band1"] + fam_fl["band2"] + fam_fl["fused"],
                 fam_n["band1"] + fam_n["band2"] + fam_n["fused"]),
        "leaf": (fam_ms["leaf"] + fam_ms["subtree"], 17.0 * m * n,
                 fam_n["leaf"] + fam_n["subtree"]),
    }
    # the band products against the FP32-effective tensor rate (tile products
    # in the band, 2 * 32^3 flops each)
    tc_ms, tc_work, tc_n = groups["tc"]
    tc_roof = None
    if tc_ms > 0:
        tc_ach = tc_work / (tc_ms / 1e3) / 1e12
        tc_roof = {"kernel": "k_tc_band: band products on tcgen05, 3xTF32 (stages 1 and 2)",
                   "bound": "tensor", "achieved": tc_ach, "peak": p_eff, "unit": "TFLOP/s",
                   "frac": tc_ach / p_eff, "peak_source": p_src,
                   "algorithmic_per_step": tc_work, "launches_per_step": tc_n,
                   "ms_per_step": tc_ms, "traffic": _traffic(wl_key, "tc", tc_n),
                   "traffic_warm_l2": _traffic_warm(wl_key, "tc", tc_n)}
    # the leaves against their latency floor: the element anti-diagonals
    # (m + n - 1 dependent rounding steps, Sec. 3.3) at the chain's own
    # measured step time, one tile alone on the GPU
    leaf_ms, leaf_bytes, leaf_n = groups["leaf"]
    cyc = P.bakron_diag_leaf_chain()
    mhz = float((clocks or {}).get("sm_mhz") or sm_max)
    step_ns = cyc / mhz * 1e3
    floor_ms = (m + n - 1) * step_ns * 1e-6
    tile_steps = leaf_n * (2 * TILE - 1)
    leaf_roof = {"kernel": "k_leaf: 32 x 32 tiles, one CTA each, wavefront of 63 in-tile steps",
                 "bound": "latency", "achieved": (m + n - 1) / (leaf_ms / 1e3),
                 "peak": 1e9 / step_ns, "unit": "element anti-diagonals/s",
                 "frac": floor_ms / leaf_ms if leaf_ms > 0 else None,
                 "peak_source": f"measured: bakron_diag_leaf_chain {cyc:.1f} cycles per chain "
                                f"step at the sampled {mhz:.0f} MHz",
                 "floor_ms": floor_ms, "ms_per_step": leaf_ms, "launches_per_step": leaf_n,
                 "schedule_chain_steps": tile_steps,
                 "hbm_gbs": leaf_bytes / (leaf_ms / 1e3) / 1e9 if leaf_ms > 0 else None,
                 "traffic": _traffic(wl_key, "leaf", leaf_n),
                 "traffic_warm_l2": _traffic_warm(wl_key, "leaf", leaf_n)}
    dom = max(groups, key=lambda g: groups[g][0])
    if dom == "tc":
        roof = dict(tc_roof)
    elif dom == "simt":
        g_ms, g_work, g_n = groups["simt"]
        achieved = g_work / (g_ms / 1e3) / 1e12
        roof = {"kernel": "k_band1_simt/k_band2_simt/k_band_fused_simt: narrow band products",
                "bound": "alu", "achieved": achieved, "peak": fp32_simt_peak, "unit": "TFLOP/s",
                "frac": achieved / fp32_simt_peak,
                "peak_source": "152 SMs x 128 FP32 lanes x 2 flop x sm_max_mhz (derived)",
                "algorithmic_per_step": g_work, "launches_per_step": g_n,
                "traffic": _traffic(wl_key, "simt", g_n)}
    else:
        roof = dict(leaf_roof)
    roof["timing"] = ("family times partition the graph-replayed step (timeline stamps, "
                      f"{prof_steps} replays)")
    roof["timeline_ms_per_step"] = timeline_ms
    roof["groups_ms_per_step"] = {k: v[0] for k, v in groups.items()}
    roof["family_ms_per_step"] = fam_ms
    roof["family_launches_per_step"] = fam_n
    roof["family_flops_per_step"] = fam_fl
    # whole-solve roofline: F_alg at the FP32-effective tensor rate plus the
    # leaves' bytes at HBM rate
    t_roof = F_alg / (p_eff * 1e12) + 17.0 * m * n / (hbm * 1e9)
    solve_roof = {"tc_roofline": tc_roof, "leaf_roofline": leaf_roof,
                  "fp32_effective_tflops": p_eff, "f_alg_flops": F_alg,
                  "leaf_bytes": 17.0 * m * n, "hbm_gbs": hbm,
                  "roofline_ms": 1e3 * t_roof, "frac": 1e3 * t_roof / ms,
                  "peak_source": p_src,
                  "formula": "(F_alg / P_fp32eff + 17 B/entry / BW_hbm) / t_solve"}
    # context: the library's own measurement of the instruction it issues
    # (tcgen05 kind::tf32, 128 x 128 x 8, operands resident, every SM)
    try:
        mr = P.bakron_diag_mma_rate(2000)
        t_roof_mma = F_alg / (mr["fp32_effective_tflops"] * 1e12) + 17.0 * m * n / (hbm * 1e9)
        solve_roof["measured_tf32_mma"] = {
            "tf32_tflops": mr["tf32_tflops"], "cycles_per_mma": mr["cycles_per_mma"],
            "fp32_effective_tflops": mr["fp32_effective_tflops"],
            "roofline_ms": 1e3 * t_roof_mma, "frac": 1e3 * t_roof_mma / ms}
    except Exception as exc:   # diagnostic only
        solve_roof["measured_tf32_mma"] = {"error": str(exc)}

    # end to end: pinned host W in, codes/scales/zeros out, inside the timed region
    Wh = W.cpu().pin_memory()
    ch = torch.empty(m, n, dtype=torch.uint8).pin_memory()
    sh = torch.empty(m, G, dtype=torch.float32).pin_memory()
    zh = torch.empty(m, G, dtype=torch.float32).pin_memory()
    e2e_steps = max(3, min(args.steps, 10))
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    tot = 0.0
    for i in range(e2e_steps):
        flush.fill_(i & 0xFF)
        e0.record(stream)
        W.copy_(Wh, non_blocking=True)      # the solve's (captured) input buffer
        step()
        ch.copy_(codes, non_blocking=True)
        sh.copy_(scales, non_blocking=True)
        zh.copy_(zeros, non_blocking=True)
        e1.record(stream)
        e1.synchronize()
        tot += e0.elapsed_time(e1)
    e2e_ms = max_over_ranks(tot / e2e_steps, ws_n, dev)
    e2e = {"value": whole_job_rate(m * n, ws_n, e2e_ms), "unit": UNIT,
           "h2d_bytes_per_step": Wh.numel() * Wh.element_size(),
           "d2h_bytes_per_step": ch.numel() + 4 * (sh.numel() + zh.numel()),
           "ms_per_step": e2e_ms}

    cpu_base = None
    if rank == 0 and not args.no_cpu_baseline:
        f = _oracle_factors(A, B, cfg.damp)
        W64 = W.double().cpu().numpy()
        k = min(args.cpu_block, m, n)
        wall, cores = _oracle_block(W64, f, cfg.bits, cfg.group, k)
        cpu_base = dict({"value": k * k / wall, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"top-left {k}x{k} block of the {m}x{n} workload (exact "
                                   f"sub-problem: the full problem's factors and grid), float64 "
                                   f"Alg. 4 oracle with Alg. 3 on 64 x 64 blocks, {wall:.1f} s "
                                   f"wall; the full problem does 1/per_entry_flops_ratio times "
                                   f"the work per entry",
                         "host": host_info()}, **_block_note(m, n, k))

    if rank == 0:
        vs = value / (4096 * 4096 / PAPER_4096_S) if (m, n) == (4096, 4096) else None
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws_n, "steps": args.steps,
            "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": vs, "dtype": "f32", "data": "synthetic",
            "config": dict(_config_dict(cfg), parallelism=f"replicas x{ws_n}",
                           launch="cuda graph replay" if graph is not None else "eager",
                           schedule=sched),
            "prepare_ms": prepare_ms, "roofline": roof, "cpu_baseline": cpu_base, "e2e": e2e,
            "gpu_launches": launches, "clocks": clocks, "solve_roofline": solve_roof,
        }
        print(json.dumps(line))
    if ws_n > 1:
        torch.distributed.destroy_process_group()
    return 0


def run_extra(args):
    """One JSON line for a workload next to the solve (N = 1 only):
      gram     K-FAC input-side factor A = X^T X / k of the 4096-feature layer
               from k = 65536 bf16 activation rows (32 sequences of 2048
               tokens), one bakron_gram call per step;
      symgrid  the symmetric l = 3 grid with 50 shrink steps of the 4096 x 4096
               weights (one bakron_grid_symmetric call per step);
      batched  the 4096 x 4096 weights as 32 heads of 128 rows, each with its
               own 128 x 128 output-side Gram and the layer's input-side one,
               one bakron_solve_batched call over 32 lanes per step (CUDA graph
               replay; the same call on one lane is timed for context);
      gptq     the 4096 x 4096 solve with B = I (GPTQ, the method's special
               case) under the layer's input-side factor, bakron_solve_gptq,
               graph replay."""
    import torch

    import paper_2608_06291_gb300 as P
    import workloads as WL

    ws_n, rank, local = _dist()
    if rank != 0:
        return 0
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    P.build()
    P.lib()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    peaks = _peaks() or {}
    if args.workload == "gram":
        k, d = 65536, 4096
        g = torch.Generator(device=dev).manual_seed(4096)
        X = (torch.randn(k, d, generator=g, device=dev)
             * torch.linspace(0.2, 3.0, d, device=dev)).to(torch.bfloat16)
        G = torch.empty(d, d, dtype=torch.float32, device=dev)
        wsb = torch.empty(P.bakron_gram_workspace_bytes(d, k, False), dtype=torch.uint8,
                          device=dev)

        def step():
            P.bakron_gram(X, alpha=1.0 / k, G=G, workspace=wsb, sync=False)
        nb = d // 128
        units = d * (d + 1) * k                   # 2k flops per unique entry
        mma = nb * (nb + 1) // 2 * 2 * 128 * 128 * k
        unit, metric = "flop/s", "K-FAC Gram X^T X / k flop/s (4096 features, 65536 bf16 rows)"
        per_launch = 2                            # bf16 transpose + tensor-core Gram
        roof_peak = float(peaks.get("bf16_tflops", 1892.3))   # kind::f16 bf16 MMAs
        roof_src = "of measured: bf16_tflops (burst; the Gram runs bf16 x bf16 MMAs)"
        cfg = {"workload": "kfac_gram", "k": k, "d": d, "dtype_in": "bf16",
               "l2": "flushed (256 MiB write) between steps; X 512 MiB > L2"}

        def cpu_data():
            return {"X": X[:4096].double().cpu().numpy()}
    elif args.workload == "gptq":
        # GPTQ as the method's B = I case (Sec. 1): the 4096 x 4096 weights
        # under the layer's input-side factor only
        cfg2 = WL.CONFIGS[2]
        W, A, B = WL.make(cfg2, device=dev)
        m, n = cfg2.m, cfg2.n
        LA, _, rA, _ = P.bakron_get_factors(P.bakron_prepare(A, B, cfg2.damp))
        fac = P.bakron_set_factors(LA, torch.eye(m, device=dev), rA, torch.ones(m, device=dev))
        wsb = P.alloc_workspace(m, n, dev)
        outg = (torch.empty(m, n, dtype=torch.uint8, device=dev),
                torch.empty(m, 1, dtype=torch.float32, device=dev),
                torch.empty(m, 1, dtype=torch.float32, device=dev), None)
        P.bakron_solve_gptq(W, fac, cfg2.bits, 0, workspace=wsb, out=outg)
        launches_per = P.bakron_last_launches()
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr):
            P.bakron_solve_gptq(W, fac, cfg2.bits, 0, workspace=wsb, sync=False, out=outg)

        def step():
            gr.replay()
        units = m * n
        mma = None
        unit, metric = "entries/s", "GPTQ (BaKron with B = I), 4096x4096 bf16 W, 4-bit per row"
        per_launch = launches_per
        p_eff, roof_src = fp32_effective_peak(peaks)
        hbm = float(peaks.get("hbm_gbs", 6800.0))
        F_alg = f_alg(m, n, identity_b=True)
        roof_peak = p_eff
        cfg = {"workload": "gptq_b_identity", "m": m, "n": n, "bits": 4,
               "launch": "cuda graph replay", "paper_gptq_s_rtx_pro_6000": 0.025,
               "l2": "flushed (256 MiB write) between steps"}

        def cpu_data():
            f = _oracle_factors(A, torch.ones(1, 1), cfg2.damp)      # A's factor only
            b = 512
            return {"W": W[:b, :b].double().cpu().numpy(), "LA": f.LA[:b, :b],
                    "LB": np.eye(b), "bits": cfg2.bits, "rows": W[:b].double().cpu().numpy()}
    elif args.workload == "batched":
        cfg2 = WL.CONFIGS[2]
        W, A, _ = WL.make(cfg2, device=dev)
        Hh, mh, n = 32, 128, cfg2.n
        lanes = int(os.environ.get("BAKRON_BENCH_LANES", "32"))   # one per head
        Ws = [W[h * mh:(h + 1) * mh] for h in range(Hh)]
        # the shared input-side factor once; each head's output-side factor
        # from a small prepare of its own Gram; assembled per head
        Bs = [WL.power_law_gram(mh, cfg2.n_samples, cfg2.alpha_b, 9000 + h, 9100 + h, dev)
              for h in range(Hh)]
        LA, _, rA, _ = P.bakron_get_factors(P.bakron_prepare(A, Bs[0], cfg2.damp))
        fs = []
        for h in range(Hh):
            LBh, _, rBh, _ = P.bakron_get_factors(P.bakron_prepare(Bs[h], Bs[h], cfg2.damp))
            fs.append(P.bakron_set_factors(LA, LBh, rA, rBh))
        outs = [(torch.empty(mh, n, dtype=torch.uint8, device=dev),
                 torch.empty(mh, 1, dtype=torch.float32, device=dev),
                 torch.empty(mh, 1, dtype=torch.float32, device=dev)) for _ in range(Hh)]

        def graph_of(S):
            wsb = torch.empty(P.bakron_batched_workspace_bytes(mh, n, S), dtype=torch.uint8,
                              device=dev)
            P.bakron_solve_batched(Ws, fs, cfg2.bits, 0, streams=S, workspace=wsb, out=outs)
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr):
                P.bakron_solve_batched(Ws, fs, cfg2.bits, 0, streams=S, workspace=wsb,
                                       sync=False, out=outs)
            return gr, wsb
        g1, _ = graph_of(1)
        gS, wsS = graph_of(lanes)
        launches_per = P.bakron_last_launches()   # the timed call's (captured last)

        def one_lane():
            g1.replay()

        def step():
            gS.replay()
        for _ in range(3):
            one_lane()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(3):
            one_lane()
        e1.record(stream)
        e1.synchronize()
        one_lane_ms = e0.elapsed_time(e1) / 3
        units = Hh * mh * n
        mma = None
        unit = "entries/s"
        metric = ("per-head BaKron solves: 32 heads of 128x4096 (bf16, 4-bit), "
                  f"{lanes} lanes, entries/s")
        per_launch = launches_per
        F_alg = Hh * f_alg(mh, n)
        p_eff, roof_src = fp32_effective_peak(peaks)
        hbm = float(peaks.get("hbm_gbs", 6800.0))
        roof_peak = p_eff
        def cpu_data():
            f = _oracle_factors(A, Bs[0], cfg2.damp)                 # head 0's factors
            b = 512
            return {"W": W[:mh, :b].double().cpu().numpy(), "LA": f.LA[:b, :b], "LB": f.LB,
                    "bits": cfg2.bits, "rows": W[:mh].double().cpu().numpy()}
        cfg = {"workload": "batched_heads", "heads": Hh, "m_head": mh, "n": n, "bits": 4,
               "lanes": lanes, "launch": "cuda graph replay",
               "one_lane_ms": one_lane_ms, "A": "shared (4096x4096 layer's)",
               "B": "one 128x128 power-law Gram per head",
               "l2": "flushed (256 MiB write) between steps"}
    else:
        cfg2 = WL.CONFIGS[2]
        W, _, _ = WL.make(cfg2, device=dev)
        m, n = cfg2.m, cfg2.n

        def step():
            P.bakron_grid_symmetric(W, 3, 0, 50)
        units = m * n
        mma = None
        unit, metric = "entries/s", "symmetric l=3 grid, 50 shrink steps, 4096x4096 bf16 W"
        per_launch = 1
        # FP32-pipe operations per entry and candidate: mul, rint, max, min, 2 fma
        roof_peak = 152 * 128 * 2.07e9 / 1e12     # lane-ops/s at the maximum SM clock (T)
        roof_src = "152 SMs x 128 FP32 lanes x 2.07 GHz (one op per lane per clock)"
        cfg = {"workload": "grid_symmetric", "m": m, "n": n, "levels": 3, "shrink_steps": 50,
               "l2": "flushed (256 MiB write) between steps"}

        def cpu_data():
            return {"W": W[:512].double().cpu().numpy()}
    for _ in range(max(3, args.warmup)):
        flush.fill_(1)
        step()
    torch.cuda.synchronize()
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    bus = None
    try:
        bus = torch.cuda.get_device_properties(dev).pci_bus_id
    except Exception:
        pass
    sampler = ClockSampler(bus)
    time.sleep(0.3)
    torch.cuda.synchronize()
    w0 = time.time()
    for i in range(args.steps):
        flush.fill_(i & 0xFF)
        starts[i].record(stream)
        step()
        ends[i].record(stream)
    torch.cuda.synchronize()
    w1 = time.time()
    clocks = sampler.stop(w0, w1)
    ms = sum(a.elapsed_time(b) for a, b in zip(starts, ends)) / args.steps
    value = units / (ms / 1e3)
    if args.workload == "gptq":
        if P.bakron_read_status(wsb) != 0:
            raise RuntimeError("device status set during the timed steps")
        t_roof = F_alg / (p_eff * 1e12) + 17.0 * units / (hbm * 1e9)
        roof = {"bound": "tensor", "achieved": F_alg / (ms / 1e3) / 1e12, "peak": p_eff,
                "unit": "TFLOP/s", "frac": 1e3 * t_roof / ms, "traffic": None,
                "peak_source": roof_src, "roofline_ms": 1e3 * t_roof,
                "note": "bakron_solve_gptq (column recursion, row-parallel leaves): F_alg of "
                        "B = I, m n (n - 1) flops, at the FP32-effective tensor rate plus "
                        "17 B/entry at HBM rate"}
        # family times of the replayed step (timeline stamps), as for the solve
        P.bakron_profile_enable(2)
        pg = torch.cuda.CUDAGraph()
        with torch.cuda.graph(pg):
            P.bakron_solve_gptq(W, fac, cfg2.bits, 0, workspace=wsb, sync=False, out=outg)
        for i in range(5):
            flush.fill_(i & 0xFF)
            pg.replay()
            P.bakron_profile_collect()
        fam = P.bakron_profile_read()
        P.bakron_profile_enable(False)
        roof["family_ms_per_step"] = {k: v[1] / 5 for k, v in fam.items() if v[0]}
        roof["family_launches_per_step"] = {k: v[0] // 5 for k, v in fam.items() if v[0]}
        tc_ms = roof["family_ms_per_step"].get("tc2", 0.0)
        if tc_ms > 0:
            tc_fl = fam["tc2"][2] / 5
            roof["tc_frac"] = tc_fl / (tc_ms / 1e3) / 1e12 / p_eff
    elif args.workload == "batched":
        if P.lib().bakron_read_status_batched(wsS.data_ptr(), mh, n, lanes, None) != 0:
            raise RuntimeError("device status set during the timed steps")
        t_roof = F_alg / (p_eff * 1e12) + 17.0 * units / (hbm * 1e9)
        roof = {"bound": "tensor", "achieved": F_alg / (ms / 1e3) / 1e12, "peak": p_eff,
                "unit": "TFLOP/s", "frac": 1e3 * t_roof / ms, "traffic": None,
                "peak_source": roof_src, "roofline_ms": 1e3 * t_roof,
                "note": "whole-call roofline: sum over heads of F_alg at the FP32-effective "
                        "tensor rate plus 17 B/entry at HBM rate"}
    elif args.workload == "gram":
        roof = {"bound": "tensor", "achieved": value / 1e12, "peak": roof_peak,
                "unit": "TFLOP/s", "frac": value / 1e12 / roof_peak, "traffic": None,
                "peak_source": roof_src,
                "note": "algorithmic flops d(d+1)k over the whole call (split kernel included); "
                        f"MMA flops issued {mma:.3e} per step (whole diagonal blocks)"}
    else:
        ops = 6.0 * units * 51
        roof = {"bound": "alu", "achieved": ops / (ms / 1e3) / 1e12, "peak": roof_peak,
                "unit": "Tops/s", "frac": ops / (ms / 1e3) / 1e12 / roof_peak, "traffic": None,
                "peak_source": roof_src}
    cpu_base = None if args.no_cpu_baseline else extra_cpu_baseline(args.workload, cpu_data())
    print(json.dumps({
        "metric": metric, "value": value, "unit": unit, "n_gpus": 1, "steps": args.steps,
        "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": cfg, "roofline": roof, "gpu_launches": per_launch * args.steps,
        "clocks": clocks, "e2e": None, "cpu_baseline": cpu_base}))
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", type=int, default=2)
    ap.add_argument("--cpu-block", type=int, default=2048,
                    help="side of the top-left block the cpu_baseline oracle solves")
    ap.add_argument("--ref-block", type=int, default=1024,
                    help="side of the top-left block each reference-arm step solves")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-autotune", action="store_true",
                    help="use the library's default schedule thresholds")
    ap.add_argument("--no-graph", action="store_true",
                    help="launch each solve's kernels eagerly instead of replaying a CUDA graph")
    ap.add_argument("--workload", default="solve",
                    choices=["solve", "gram", "symgrid", "batched", "gptq"],
                    help="solve (the headline line), or a line for the Gram accumulation, "
                         "the symmetric grid, the batched per-head solve or GPTQ (B = I)")
    args = ap.parse_args()
    if args.workload != "solve" and args.impl == "ours":
        return run_extra(args)
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
