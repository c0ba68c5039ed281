#!/usr/bin/env python
"""Benchmark of the GRKV prefill compression path on GB300.

One step = one grkv_compress call over the whole workload: window scoring,
pooled top-B selection, target Y and the ridge value merge for every
(layer, KV head) unit.  Default workload: the 32-layer Llama-3.1-8B-shaped
prefill cache (256 units, N = 32768, B = 2048, w = 32, GQA 4), bf16.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun each rank compresses its own batch of units (weak scaling, no
collective on the data path); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import multiprocessing as mp
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "compressed KV tokens/sec per GPU (layer-heads x N) and % of GB300 HBM roofline"
UNIT = "layer-head tokens/s"
NOMINAL_HBM_GBS = 8000.0


def args_():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", default="c2_llama_32k_bf16")
    ap.add_argument("--n", type=int, default=0, help="override N (sweep points)")
    ap.add_argument("--budget", type=int, default=0, help="override B (sweep points)")
    ap.add_argument("--units", type=int, default=0,
                    help="take only the first U units of the workload (profiling slices)")
    ap.add_argument("--cpu-seconds", type=float, default=20.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--path", choices=("default", "one_read", "portable"), default="default",
                    help="scoring kernels: default (two tensor-core launches, K read twice), "
                         "one_read (one launch that reads K from HBM once) or portable (CUDA cores)")
    ap.add_argument("--update-k", action="store_true",
                    help="add the key step (GRKV_UPDATE_K, CG to the library's default residual); "
                         "no CPU baseline is timed for it")
    ap.add_argument("--lambda-k", type=float, default=1e-2)
    a = ap.parse_args()
    if a.update_k:
        a.no_cpu_baseline = True
    return a


def workload(a):
    import grkv_inputs as gi
    wl = gi.workload(a.workload)
    if a.n or a.budget:
        n, bud = a.n or wl.n, a.budget or wl.budget
        wl = wl.replace(name=f"{wl.name}_n{n}_b{bud}", n=n, budget=bud,
                        seed=gi.seed_for(wl.seed, n, bud))
    if a.units:
        wl = wl.replace(name=f"{wl.name}_first{a.units}", units=min(a.units, wl.units))
    return wl


def algorithmic_bytes(wl):
    """K and V read once plus the compressed K and V written (bytes / step)."""
    el = 2 if wl.dtype == "bf16" else 4
    read = 2 * wl.units * wl.n * wl.d * el
    write = 2 * wl.units * wl.budget * wl.d * el
    return read, write


# DRAM bytes (read + write) of one grkv_score call (both k_score_tc launches)
# from one ncu capture of the full workload.  A figure holds only
# for the kernel source it was taken on, so it is keyed by that file's digest
# and reported as null once the kernel changes.
SCORE_SRC = os.path.join("paper_2605_31105_gb300", "csrc", "grkv_score_tc.cu")
# DRAM read + write bytes of one grkv_score call (both k_score_tc launches), from
# the ncu capture in profiles/score_tc_c2_llama_32k.md, keyed by the SHA-256 of the
# kernel source it was taken on.
SCORE_TRAFFIC = {
    "c2_llama_32k_bf16": ("0ea59ba48bb5a0be128f6060b1dd07717b01f47bfca8e89e80517f105e7d52bc",
                          6532132864),
}


SCORE_KERNEL = {
    "default": "grkv_score stage (k_score_tc: window scoring + target, two launches)",
    "one_read": "grkv_score stage (k_score_pipe: window scoring + target, one read of K)",
    "portable": "grkv_score stage (CUDA-core kernels: k_stats_chunk, k_stats_reduce, k_prob_chunk, k_y_reduce)",
}


def score_traffic(wl):
    rec = SCORE_TRAFFIC.get(wl.name)
    if rec is None:
        return None
    with open(os.path.join(ROOT, SCORE_SRC), "rb") as f:
        digest = hashlib.sha256(f.read()).hexdigest()
    return rec[1] if digest == rec[0] else None


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# ------------------------------------------------------------ CPU oracle --
def _oracle_worker(conn, wl_dict, unit):
    """One single-threaded process holding one unit's inputs; each message
    runs the fp64 oracle on it once and replies with the seconds it took."""
    import grkv_inputs as gi
    import oracle as O
    wl = gi.Workload(**wl_dict)
    q, k, v = gi.unit_arrays(wl, unit)
    op = O.Params(group=wl.group, n=wl.n, d=wl.d, window=wl.window, budget=wl.budget,
                  pool_kernel=wl.pool_kernel, lambda_v=wl.lambda_v)
    conn.send("ready")
    while conn.recv() == "run":
        t0 = time.perf_counter()
        O.compress_unit(q, k, v, op)
        conn.send(time.perf_counter() - t0)


class OracleGang:
    """`cores` spawn processes (BLAS single-threaded), unit i on process i.
    Created before the first GPU call; inputs are generated at start-up and
    excluded from every timing."""

    def __init__(self, wl, cores):
        for key in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
            os.environ[key] = "1"
        ctx = mp.get_context("spawn")
        self.wl, self.cores, self.conns, self.procs = wl, cores, [], []
        for i in range(cores):
            a, b = ctx.Pipe()
            pr = ctx.Process(target=_oracle_worker, args=(b, wl.__dict__, i % wl.units),
                             daemon=True)
            pr.start()
            self.conns.append(a)
            self.procs.append(pr)

    def wait_ready(self):
        for c in self.conns:
            assert c.recv() == "ready"

    def step(self) -> float:
        """All processes run their unit once; returns the wall seconds."""
        t0 = time.perf_counter()
        for c in self.conns:
            c.send("run")
        for c in self.conns:
            c.recv()
        return time.perf_counter() - t0

    def close(self):
        for c in self.conns:
            c.send("stop")
        for pr in self.procs:
            pr.join(timeout=10)


def cpu_baseline(gang: OracleGang, seconds: float):
    """The oracle as it stands on a bounded sample of the workload's units."""
    wl = gang.wl
    gang.wait_ready()
    first = gang.step()
    rounds = max(1, int(seconds / max(first, 1e-3)))
    wall = sum(gang.step() for _ in range(rounds))
    value = gang.cores * rounds * wl.n / wall
    return {"value": value, "unit": UNIT, "cores": gang.cores, "kind": "oracle",
            "sample": f"units 0..{gang.cores - 1} of the {wl.units} units of {wl.name}, one per "
                      f"single-threaded process, {rounds} round(s), {wall:.1f} s wall; "
                      f"input generation excluded"}


def _cores():
    return max(1, min(os.cpu_count() or 1, 16))


def run_reference(a):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    wl = workload(a)
    gang = OracleGang(wl, _cores())
    try:
        gang.wait_ready()
        for _ in range(a.warmup):
            gang.step()
        wall = sum(gang.step() for _ in range(a.steps))
    finally:
        gang.close()
    value = gang.cores * wl.n * a.steps / wall
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": a.gpus,
        "steps": a.steps, "warmup": a.warmup, "ms_per_step": 1e3 * wall / a.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded; stands in for LongBench / RULER caches)",
        "config": {"workload": wl.name, "units": wl.units, "n": wl.n, "budget": wl.budget,
                   "window": wl.window, "group": wl.group, "d": wl.d},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": gang.cores, "kind": "oracle",
                         "sample": f"each step: units 0..{gang.cores - 1} of the {wl.units}, "
                                   f"one per single-threaded process (fp64 numpy oracle); "
                                   f"input generation excluded"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------- clocks --
class ClockSampler:
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        self.t0 = self.t1 = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", self.gpu_id, f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            time.sleep(0.5)
        except Exception:
            self.proc = None

    def mark(self, begin: bool):
        if begin:
            self.t0 = time.time()
        else:
            self.t1 = time.time()

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.05)
        self.proc.terminate()
        try:
            out = self.proc.communicate(timeout=5)[0]
        except Exception:
            self.proc.kill()
            out = ""
        rows = []
        for line in out.splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                ts = time.mktime(time.strptime(f[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                ts += float("0." + f[0].split(".")[1]) if "." in f[0] else 0.0
                rows.append((ts, float(f[1]), float(f[2]), f[5:9]))
            except Exception:
                continue
        inside = [r for r in rows if self.t0 - 0.02 <= r[0] <= self.t1 + 0.02] or rows
        if not inside:
            return None
        reasons = sorted({self.NAMES[i] for r in inside for i, s in enumerate(r[3])
                          if s.lower().startswith("active")})
        return {"sm_mhz": statistics.median(r[1] for r in inside),
                "sm_max_mhz": max(r[2] for r in inside), "reasons": reasons,
                "samples": len(inside)}


# ------------------------------------------------------------------ ours --
def rank_workload(wl, rank: int, world: int):
    """Weak scaling: every rank compresses its own batch of units, drawn from
    a seed of its own (the units of different ranks are independent)."""
    import grkv_inputs as gi
    return wl if world <= 1 else wl.replace(seed=gi.seed_for(wl.seed, 7919, rank))


def max_over_ranks(values, dist=None, device="cpu"):
    """The element-wise maximum of `values` over the ranks of the process
    group (the slowest rank sets the job's time); identity without one."""
    if dist is None:
        return [float(x) for x in values]
    import torch
    t = torch.tensor([float(x) for x in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t.tolist()]


def job_throughput(units: int, n: int, world: int, ms: float) -> float:
    """Whole-job layer-head tokens/s: every rank processed units x n tokens in
    at most `ms` milliseconds (the max over ranks)."""
    return units * n * world / (ms * 1e-3)


def run_ours(a):
    import numpy as np
    import torch

    import grkv_inputs as gi
    from paper_2605_31105_gb300 import binding as b

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    gang = None
    if rank == 0 and not a.no_cpu_baseline:
        gang = OracleGang(workload(a), _cores())   # before the first GPU call
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    b.load()

    wl = rank_workload(workload(a), rank, world)
    U, n, B, d, m = wl.units, wl.n, wl.budget, wl.d, wl.m
    qdt = np.uint16 if wl.dtype == "bf16" else np.float32
    tdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    hq = torch.empty((U, wl.group, wl.window, d), dtype=tdt).pin_memory()
    hk = torch.empty((U, n, d), dtype=tdt).pin_memory()
    hv = torch.empty((U, n, d), dtype=tdt).pin_memory()
    view = (lambda t: t.view(torch.int16).numpy().view(np.uint16)) if wl.dtype == "bf16" \
        else (lambda t: t.numpy())
    gi.fill_units(wl, view(hq), view(hk), view(hv))
    dq, dk, dv = hq.cuda(), hk.cuda(), hv.cuda()
    p = b.params(U, wl.group, n, wl.window, B, pool_kernel=wl.pool_kernel,
                 lambda_v=wl.lambda_v, lambda_k=a.lambda_k, dtype=wl.dtype,
                 flags={"default": 0, "one_read": b.GRKV_ONE_READ_SCORE,
                        "portable": b.GRKV_FORCE_SIMT}[a.path]
                 | (b.GRKV_UPDATE_K if a.update_k else 0))
    ws = torch.empty(b.grkv_workspace_size(p), dtype=torch.uint8, device="cuda")
    ko = torch.empty((U, B, d), dtype=tdt, device="cuda")
    vo = torch.empty_like(ko)
    idx = torch.empty((U, B), dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream()

    def step():
        b.grkv_compress(p, dq, dk, dv, ko, vo, idx, ws, stream=stream)

    def barrier():
        if dist is not None:
            dist.barrier()

    for _ in range(a.warmup):
        step()
    torch.cuda.synchronize()
    assert b.grkv_status(ws) == b.GRKV_OK

    props = torch.cuda.get_device_properties(local)
    gpu_id = str(getattr(props, "uuid", local))
    if gpu_id and not gpu_id.startswith("GPU-") and len(gpu_id) > 8:
        gpu_id = "GPU-" + gpu_id
    clocks = ClockSampler(gpu_id)
    clocks.start()

    # ---- timed region: inputs resident in HBM (4.3 GB of K/V at the
    # default workload, far above the 129 MB L2, so no flush is needed)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    launches0 = b.grkv_launch_count()
    barrier()
    torch.cuda.synchronize()
    clocks.mark(True)
    e0.record(stream)
    for _ in range(a.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    clocks.mark(False)
    barrier()
    launches = b.grkv_launch_count() - launches0
    ms = e0.elapsed_time(e1) / a.steps
    clk = clocks.stop()
    assert b.grkv_status(ws) == b.GRKV_OK
    ms, = max_over_ranks([ms], dist, "cuda")

    # ---- dominant kernel: the score stage, timed by itself on the same stream
    P = n - wl.window
    scores = torch.empty((U, P), dtype=torch.float32, device="cuda")
    y = torch.empty((U, m, d), dtype=torch.float32, device="cuda")
    rs = torch.empty((U, m, 2), dtype=torch.float32, device="cuda")
    nst = max(3, min(a.steps, 20))
    for _ in range(2):
        b.grkv_score(p, dq, dk, dv, scores, y, rs, ws, stream=stream)
    s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    s0.record(stream)
    for _ in range(nst):
        b.grkv_score(p, dq, dk, dv, scores, y, rs, ws, stream=stream)
    s1.record(stream)
    torch.cuda.synchronize()
    score_ms = s0.elapsed_time(s1) / nst

    # ---- end to end through the public API with host buffers
    hko = torch.empty((U, B, d), dtype=tdt).pin_memory()
    hvo = torch.empty_like(hko).pin_memory()
    hidx = torch.empty((U, B), dtype=torch.int32).pin_memory()

    def e2e_step():
        dq.copy_(hq, non_blocking=True)
        dk.copy_(hk, non_blocking=True)
        dv.copy_(hv, non_blocking=True)
        b.grkv_compress(p, dq, dk, dv, ko, vo, idx, ws, stream=stream)
        hko.copy_(ko, non_blocking=True)
        hvo.copy_(vo, non_blocking=True)
        hidx.copy_(idx, non_blocking=True)

    e2e_step()
    torch.cuda.synchronize()
    barrier()
    x0, x1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    x0.record(stream)
    for _ in range(a.e2e_steps):
        e2e_step()
    x1.record(stream)
    torch.cuda.synchronize()
    barrier()
    e2e_ms = x0.elapsed_time(x1) / a.e2e_steps
    e2e_ms, score_ms = max_over_ranks([e2e_ms, score_ms], dist, "cuda")
    el = hq.element_size()
    h2d = (hq.numel() + hk.numel() + hv.numel()) * el
    d2h = (hko.numel() + hvo.numel()) * el + hidx.numel() * 4

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return
    read, write = algorithmic_bytes(wl)
    peak, peak_kind = measured_peaks()
    score_bytes = read                      # K and V, each read once
    achieved = score_bytes / (score_ms * 1e-3) / 1e9
    path_gbs = (read + write) / (ms * 1e-3) / 1e9
    line = {
        "metric": METRIC, "value": job_throughput(U, n, world, ms), "unit": UNIT, "n_gpus": world,
        "steps": a.steps, "warmup": a.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype,
        "data": "synthetic (seeded; stands in for LongBench / RULER caches)",
        "config": {"workload": wl.name, "units": U, "n": n, "budget": B, "window": wl.window,
                   "group": wl.group, "d": d, "lambda_v": wl.lambda_v,
                   "pool_kernel": wl.pool_kernel, "l2": "inputs (K+V %.1f GB) exceed L2" %
                   (read / 1e9), "parallelism": f"units sharded, {world} rank(s)",
                   "key_step": bool(a.update_k)},
        "path": a.path,
        "roofline": {"bound": "hbm",
                     "kernel": SCORE_KERNEL["portable" if wl.dtype != "bf16" else a.path],
                     "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "peak_kind": peak_kind,
                     "traffic": score_traffic(wl) if a.path == "default" else None,
                     "algorithmic_bytes_per_launch": score_bytes, "launch_ms": score_ms},
        "path_hbm": {"gbs": path_gbs, "frac_of_measured": path_gbs / peak,
                     "frac_of_8tbs": path_gbs / NOMINAL_HBM_GBS,
                     "bytes_per_step": read + write},
        "e2e": {"value": job_throughput(U, n, world, e2e_ms), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms, "steps": a.e2e_steps},
        "gpu_launches": launches,
        "clocks": clk,
    }
    if gang is not None:
        line["cpu_baseline"] = cpu_baseline(gang, a.cpu_seconds)
        gang.close()
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


def main():
    a = args_()
    if a.impl == "reference":
        run_reference(a)
    else:
        run_ours(a)


if __name__ == "__main__":
    main()
