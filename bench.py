#!/usr/bin/env python3
"""Throughput of the batched scheduler simulator on one GB300 (or N, one replica per GPU).

One step = one pass of the whole path over the 1024-instance workload (1024 instances x 1000
requests, all arriving at t=0, M=16384, s~U{1..64}, o~U{1..512}, alpha in {1/5,1/2,4/5,1}):
for each of A_max, A_min and H-SF, load the (device-resident) request arrays through sim_load
(staging: validation + sort of the waiting set) and simulate every instance with sim_run; then
compute the competitive ratios TEL(A_max)/TEL(H-SF) and TEL(A_min)/TEL(H-SF).

The metric is simulated request-steps per second: the sum over instances and policies of
sum_t |batch_t| (tokens generated, wasted A_min tokens included), divided by the device time.

  python bench.py [--gpus N --steps K --warmup W]          # the CUDA path
  python bench.py --impl reference [...]                     # the CPU oracle on a bounded sample
Under torchrun each rank simulates its own 1024 instances (weak scaling; no collective on the
data path: instances are independent); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time
from pathlib import Path

import numpy as np

ROOT = Path(__file__).resolve().parent
sys.path.insert(0, str(ROOT))

METRIC = "simulated request-steps/s (A_min, A_max)"
UNIT = "request-steps/s"
WORKLOAD = "c2"
WORKLOAD_DESC = ("1024 instances x n=1000 requests at t=0, M=16384, s~U{1..64}, o~U{1..512}, "
                 "alpha in {1/5,1/2,4/5,1} (256 seeds each); policies A_max, A_min, H-SF + CR")
POLICY_NAMES = ("A_max", "A_min", "H-SF")
# Algorithmic work model of one request-step (one token of one batch member): tokens += 1,
# compare with the true length, add to the step's memory and to the request-step count.
OPS_PER_REQUEST_STEP = 4
INT32_LANES_PER_SM = 128


def _dram_traffic(kernel: str) -> int | None:
    """DRAM bytes per launch of `kernel` on this workload, from the committed ncu summary, or None
    when the simulation kernel's sources changed since those counters were taken."""
    import hashlib
    p = ROOT / "profiles" / "dram_traffic.json"
    if not p.exists():
        return None
    entry = json.loads(p.read_text()).get(kernel)
    if not entry:
        return None
    h = hashlib.sha256()
    for f in entry["sources"]:
        h.update((ROOT / f).read_bytes())
    return int(entry["bytes_per_launch"]) if h.hexdigest() == entry["sources_sha256"] else None


def _peaks() -> dict:
    p = ROOT / "MEASURED_PEAKS.json"
    if p.exists():
        return json.loads(p.read_text())
    return {"hbm_gbs": 6800.0, "sm_max_mhz": 2070.0, "_fallback": True}


class ClockSampler:
    """nvidia-smi clocks and throttle reasons while the timed region runs."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = Path(f"/tmp/simgb_clocks_{os.getpid()}.csv")

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self) -> dict:
        try:
            rows = [r.split(",") for r in self.path.read_text().strip().splitlines() if r.strip()]
        except Exception:
            rows = []
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(r[1]) for r in rows if len(r) > 2 and r[1].strip().replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if len(r) > 2 and r[2].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in rows:
            for k, nm in enumerate(names):
                if len(r) > 5 + k and r[5 + k].strip().lower() == "active":
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(rows)}


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def make_rank_workload(rank: int):
    from paper_2508_14544_gb300 import workloads as W
    return W.make_workload(WORKLOAD, W.rank_instances(WORKLOAD, rank))


def cpu_baseline(w, max_seconds: float = 20.0) -> dict:
    """The CPU oracle as it stands, on the whole workload once per policy, all host cores.

    One pass of the three policies over every instance is ~1.6 s of wall time on 16 Arm cores
    (about 25 CPU-seconds); later policies are skipped if the budget of max_seconds runs out."""
    from oracle import plain
    cores = os.cpu_count() or 1
    rs = 0
    t0 = time.perf_counter()
    c0 = time.process_time()
    done = 0
    for pol in (0, 1, 2):
        r = plain.run_workload(pol, w, n_threads=cores)
        rs += int(r["request_steps"].sum())
        done += 1
        if time.perf_counter() - t0 > max_seconds:
            break
    dt = time.perf_counter() - t0
    cpu_s = time.process_time() - c0
    return {"value": rs / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"all {w.n_instances} instances x {done} policies (A_max, A_min, H-SF), "
                      f"oracle/plain.c with {cores} threads: {dt:.1f} s wall, {cpu_s:.1f} CPU-s"}


def run_reference(args) -> None:
    rank, world, local = dist_env()
    if rank != 0:
        return
    w = make_rank_workload(0)
    t_all = []
    rs_all = 0
    from oracle import plain
    cores = os.cpu_count() or 1
    sample = w.subset(range(0, w.n_instances, 4))
    for it in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        rs = 0
        for pol in (0, 1, 2):
            r = plain.run_workload(pol, sample, n_threads=cores)
            rs += int(r["request_steps"].sum())
        dt = time.perf_counter() - t0
        if it >= args.warmup:
            t_all.append(dt)
            rs_all += rs
    total = sum(t_all)
    value = rs_all / total
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * total / max(args.steps, 1),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int32",
            "data": "synthetic",
            "config": {"workload": WORKLOAD_DESC, "sample": f"{sample.n_instances} instances (every 4th)"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"{sample.n_instances} of {w.n_instances} instances x 3 policies per step"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_ours(args) -> None:
    import torch
    import torch.distributed as dist

    import __graft_entry__
    __graft_entry__.build()
    from paper_2508_14544_gb300 import SIM_AELL, SIM_AMAX, SIM_AMIN, SIM_AR, SIM_HSF, Simulator

    rank, world, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    stream = torch.cuda.Stream(device=dev)
    sh = stream.cuda_stream

    w = make_rank_workload(rank)
    host = [np.ascontiguousarray(x) for x in (w.arrival, w.prompt, w.lower, w.upper, w.true_o)]
    d_in = [torch.from_numpy(x).to(dev) for x in host]
    pinned = [torch.from_numpy(x).pin_memory() for x in host]
    # residency (one or two simulation warps per scheduler) is tuned on the first warm-up run of
    # each policy: a launch is as long as its slowest instance, and which residency is faster
    # depends on how uneven the instances are
    sims = [Simulator(p, w.M, w.n_instances, tune_residency=1) for p in (SIM_AMAX, SIM_AMIN, SIM_HSF)]
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)  # > 129 MB L2
    torch.cuda.synchronize()

    def step(inputs):
        res = []
        for sim in sims:
            sim.load(w.offsets, *inputs)
            res.append(sim.run(sh))
        cr = [sims[0].competitive_ratio(sims[2], sh), sims[1].competitive_ratio(sims[2], sh)]
        return res, cr

    # warm-up (also checks that every instance finished)
    for _ in range(max(args.warmup, 0)):
        res, _ = step(d_in)
    for r in res:
        assert np.all(r["status"] == 0), r["status"]
    rs_per_step = int(sum(int(r["request_steps"].sum()) for r in res))
    launches0 = sum(s.kernel_launches() for s in sims)

    # timed region: K steps, device time by CUDA events on the simulator's stream
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    load_starts = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    run_starts = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    run_ends = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        time.sleep(0.3)
        for k in range(args.steps):
            with torch.cuda.stream(stream):
                flush.fill_(k & 0xff)
            torch.cuda.synchronize()
            starts[k].record(stream)
            for j, sim in enumerate(sims):
                load_starts[k][j].record(stream)
                sim.load(w.offsets, *d_in)
                run_starts[k][j].record(stream)
                res[j] = sim.run(sh)
                run_ends[k][j].record(stream)
            sims[0].competitive_ratio(sims[2], sh)
            sims[1].competitive_ratio(sims[2], sh)
            ends[k].record(stream)
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    launches = sum(s.kernel_launches() for s in sims) - launches0
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    run_ms = [[run_starts[k][j].elapsed_time(run_ends[k][j]) for j in range(3)] for k in range(args.steps)]
    load_ms = [[load_starts[k][j].elapsed_time(run_starts[k][j]) for j in range(3)] for k in range(args.steps)]
    total_s = sum(step_ms) / 1000.0
    if world > 1:
        t = torch.tensor([total_s], device=dev, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_s = float(t.item())
    value = rs_per_step * args.steps * world / total_s

    # end to end through the public API with host (pinned) buffers: H2D inside sim_load, D2H of
    # the per-instance results inside sim_run and of the ratios
    e2e_steps = max(1, min(args.steps, 5))
    host_in = [p.numpy() for p in pinned]
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        step(host_in)
    torch.cuda.synchronize()
    e2e_s = time.perf_counter() - t0
    if world > 1:
        t = torch.tensor([e2e_s], device=dev, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        e2e_s = float(t.item())
    e2e_val = rs_per_step * e2e_steps * world / e2e_s

    # the paper's two further policies on the same instances (outside the step): A_r (Algorithm
    # random, permutation drawn by the workload generator) and A_ell (Algorithm promote_l);
    # sim_run device time by CUDA events, median of 3 after a warm-up
    further = {}
    for name, pol in (("A_r", SIM_AR), ("A_ell", SIM_AELL)):
        with Simulator(pol, w.M, w.n_instances, tune_residency=1) as sim:
            rk = torch.from_numpy(w.ranks()).to(dev) if pol == SIM_AR else None
            sim.load(w.offsets, *d_in, rank=rk)
            r = sim.run(sh)
            assert np.all(r["status"] == 0), (name, r["status"])
            ms = []
            for _ in range(3):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                torch.cuda.synchronize()
                e0.record(stream)
                sim.run(sh)
                e1.record(stream)
                torch.cuda.synchronize()
                ms.append(e0.elapsed_time(e1))
        rsn = int(r["request_steps"].sum())
        further[name] = {"sim_run_ms": round(statistics.median(ms), 3), "request_steps": rsn,
                         "request_steps_per_s": rsn / (statistics.median(ms) / 1000.0)}

    # the Lemma-thm:Amin evaluator on 2^20 histograms of 64 lengths (512 MB of doubles, read once):
    # 20 FP64 flops per length (6 FMA + 8 other), so GB300's FP64 rate bounds it, not HBM
    from paper_2508_14544_gb300 import cr_amin_lemma
    hx = torch.rand((1 << 20, 64), dtype=torch.float64, device=dev)
    for _ in range(3):
        cr_amin_lemma(hx, 1, 0.0, stream=sh)
    lm = []
    for _ in range(5):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        cr_amin_lemma(hx, 1, 0.0, stream=sh)
        e1.record(stream)
        torch.cuda.synchronize()
        lm.append(e0.elapsed_time(e1))
    lemma_bytes = hx.numel() * 8 + hx.shape[0] * 8
    lemma_gbs = lemma_bytes / (statistics.median(lm) / 1000.0) / 1e9
    lemma_tflops = 20.0 * hx.numel() / (statistics.median(lm) / 1000.0) / 1e12
    del hx
    h2d = 3 * 5 * w.n_total * 4
    d2h = 3 * w.n_instances * 56 + 2 * w.n_instances * 8

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return
    peaks = _peaks()
    clocks = clk.summary()
    # roofline of the dominant kernel (the simulation kernel of the slowest policy): integer issue
    per_pol_ms = [statistics.mean(run_ms[k][j] for k in range(args.steps)) for j in range(3)]
    rs_pol = [int(r["request_steps"].sum()) for r in res]
    dom = int(np.argmax(per_pol_ms))
    achieved_ops = OPS_PER_REQUEST_STEP * rs_pol[dom] / (per_pol_ms[dom] / 1000.0)
    n_sm = torch.cuda.get_device_properties(dev).multi_processor_count
    peak_ops = n_sm * INT32_LANES_PER_SM * float(peaks.get("sm_max_mhz", 2070.0)) * 1e6
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": statistics.mean(step_ms), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int32", "data": "synthetic",
        "config": {"workload": WORKLOAD_DESC, "instances_per_gpu": w.n_instances, "requests_per_instance": 1000,
                   "parallelism": f"instances sharded, {world} replica(s), no collective on the data path",
                   "l2": "256 MB buffer written between timed steps (inputs are 20 MB < L2)",
                   "residency": "SIM_OPT_TUNE_RESIDENCY: one or two warps per scheduler, chosen per policy on the first warm-up run",
                   "request_steps_per_step": rs_per_step,
                   "sim_run_ms": dict(zip(POLICY_NAMES, [round(x, 3) for x in per_pol_ms])),
                   "sim_load_ms": dict(zip(POLICY_NAMES, [round(statistics.mean(load_ms[k][j] for k in range(args.steps)), 3)
                                                          for j in range(3)])),
                   "batches_per_s": {POLICY_NAMES[j]: int(res[j]["steps"].sum()) / (per_pol_ms[j] / 1000.0)
                                     for j in range(3)},
                   "us_per_instance": {POLICY_NAMES[j]: round(1000.0 * per_pol_ms[j] / w.n_instances, 3)
                                       for j in range(3)},
                   "further_policies_not_in_step": further,
                   "lemma_evaluator": {"histograms": 1 << 20, "lengths": 64, "ms": round(statistics.median(lm), 4),
                                       "GB_per_s": round(lemma_gbs, 1),
                                       "frac_of_measured_hbm": round(lemma_gbs / float(_peaks().get("hbm_gbs", 6800.0)), 3),
                                       "fp64_tflops": round(lemma_tflops, 3),
                                       "frac_of_nominal_fp64_1.25": round(lemma_tflops / 1.25, 3)}},
        "roofline": {"bound": "alu", "kernel": f"k_run<{POLICY_NAMES[dom]}>",
                     "achieved": achieved_ops / 1e12, "peak": peak_ops / 1e12,
                     "unit": "Tops/s (int32)", "frac": achieved_ops / peak_ops,
                     "traffic": _dram_traffic(f"k_run<{POLICY_NAMES[dom]}>"),
                     "model": f"{OPS_PER_REQUEST_STEP} int ops per request-step; peak = {n_sm} SMs x "
                              f"{INT32_LANES_PER_SM} int32 lanes x {peaks.get('sm_max_mhz', 2070.0)} MHz"},
        "e2e": {"value": e2e_val, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": launches,
        "clocks": clocks,
    }
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w)
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
