#!/usr/bin/env python3
"""Throughput of the batched scheduler simulator on one GB300 (or N, one replica per GPU).

One step = one pass of the whole path over the alpha-sweep workload (alpha = 1/10 .. 10/10 x 4096
seeds = 40960 instances x 2000 requests, all arriving at t=0, M=32768, s~U{16..256}, bimodal o:
70% U{1..32}, 30% U{512..2048}), the largest of the five configurations: for each of A_max, A_min
and H-SF, load the (device-resident) request arrays through sim_load (staging: validation + sort
of the waiting set) and simulate every instance with sim_run; then compute the competitive ratios
TEL(A_max)/TEL(H-SF) and TEL(A_min)/TEL(H-SF).

The metric is simulated request-steps per second: the sum over instances and policies of
sum_t |batch_t| (tokens generated, wasted A_min tokens included), divided by the device time.
After the timed region the other four configurations are timed per policy (sub-records), the
per-step method's work is counted (SIM_OPT_COUNT_WORK) for the roofline, whose integer-issue and
shared-memory ceilings are measured on the GPU (sim_measure_peaks).

  python bench.py [--gpus N --steps K --warmup W]          # the CUDA path
  python bench.py --impl reference [...]                     # the CPU oracle on a bounded sample
Under torchrun each rank simulates its own copy of the workload's shape (weak scaling; no
collective on the data path: instances are independent); rank 0 prints one JSON line.
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
WORKLOAD = "c4"
WORKLOAD_DESC = ("alpha in {1/10..10/10} x 4096 seeds = 40960 instances x n=2000 requests at t=0, M=32768, "
                 "s~U{16..256}, o: 70% U{1..32}, 30% U{512..2048}; policies A_max, A_min, H-SF + CR")
SUB_WORKLOADS = ("c1", "c2", "c3", "c5")
POLICY_NAMES = ("A_max", "A_min", "H-SF")

# Work of the paper's per-step method (Theorem complexity) per unit, for the roofline:
#   per request-step (one token of one batch member): 4 int ops (tokens + 1, compare with the true
#     length, add to the step's memory and to the request-step count), 8 bytes of shared memory;
#   per S2 add (memory accounting of the active set): 1 int op;
#   per S3 compare-exchange (sorting the active set on an overflow): 3 int ops, 8 bytes;
#   per S5 endpoint evaluation (binary-searched admission): 6 int ops, 16 bytes;
#   per S4 queue operation (one insert and one removal per admission): 1 int op, 16 bytes each;
#   global memory: the 20-byte request once, the 56-byte result, and the bytes the waiting queue
#     moves (counted by the kernel).
OPS = {"request_step": 4, "s2": 1, "s3": 3, "s5": 6, "s4": 1}
SMEM_B = {"request_step": 8, "s3": 8, "s5": 16, "s4": 16}


def _dram_traffic(kernel: str) -> int | None:
    """DRAM bytes per launch of `kernel` on the bench workload, from the committed ncu summary, or
    None when the simulation kernel's sources changed since those counters were taken."""
    import hashlib
    p = ROOT / "profiles" / "dram_traffic.json"
    if not p.exists():
        return None
    entry = json.loads(p.read_text()).get(kernel)
    if not entry or entry.get("workload_key") != WORKLOAD:
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


def make_rank_workload(rank: int, name: str = WORKLOAD):
    from paper_2508_14544_gb300 import workloads as W
    return W.make_workload(name, W.rank_instances(name, rank))


def cpu_baseline(w, budget_s: float = 20.0) -> dict:
    """The CPU oracle as it stands (oracle/plain.c, all host cores, one instance per task) on a
    bounded sample of the workload: every k-th instance, all three policies, k chosen from a
    first timed pass so that the whole sample takes about budget_s of wall time."""
    from oracle import plain
    cores = os.cpu_count() or 1
    first = w.subset(range(0, w.n_instances, 320))  # 128 instances, all alphas
    t0 = time.perf_counter()
    for pol in (0, 1, 2):
        plain.run_workload(pol, first, n_threads=cores)
    per_inst = (time.perf_counter() - t0) / first.n_instances
    stride = max(1, int(w.n_instances / max(1.0, budget_s / max(per_inst, 1e-6))))
    sample = w.subset(range(0, w.n_instances, stride))
    rs = 0
    t0 = time.perf_counter()
    c0 = time.process_time()
    for pol in (0, 1, 2):
        rs += int(plain.run_workload(pol, sample, n_threads=cores)["request_steps"].sum())
    dt = time.perf_counter() - t0
    cpu_s = time.process_time() - c0
    out = {"value": rs / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
           "sample": f"every {stride}th instance ({sample.n_instances} of {w.n_instances}, all alphas) x 3 policies "
                     f"(A_max, A_min, H-SF), oracle/plain.c with {cores} threads: {dt:.1f} s wall, {cpu_s:.1f} CPU-s",
           "cpu": _cpu_model()}
    # the same oracle on one thread (16 instances, all alphas), and the literal Python oracle on
    # the 50-request instance: the other two timing modes of the oracle
    one = w.subset(range(0, w.n_instances, max(1, w.n_instances // 16)))
    t0 = time.perf_counter()
    rs1 = sum(int(plain.run_workload(pol, one, n_threads=1)["request_steps"].sum()) for pol in (0, 1, 2))
    dt1 = time.perf_counter() - t0
    out["single_thread"] = {"value": rs1 / dt1, "unit": UNIT, "sample": f"{one.n_instances} instances x 3 policies, "
                                                                       f"oracle/plain.c on one thread: {dt1:.1f} s"}
    from oracle import literal
    from paper_2508_14544_gb300 import workloads as W
    c1 = W.make_workload("c1").instance(0)
    t0 = time.perf_counter()
    rsl = sum(int(literal.simulate(pol, c1["M"], c1["a"], c1["s"], c1["l"], c1["u"], c1["o"])["request_steps"])
              for pol in (0, 1, 2))
    dtl = time.perf_counter() - t0
    out["literal_c1"] = {"value": rsl / dtl, "unit": UNIT, "sample": f"the 50-request instance x 3 policies, "
                                                                    f"oracle/literal.py: {dtl:.2f} s"}
    return out


def _cpu_model() -> str:
    """The host CPU as /proc/cpuinfo names it (x86 model name, or Arm implementer / part)."""
    import platform
    try:
        info = Path("/proc/cpuinfo").read_text().splitlines()
    except OSError:
        info = []
    for key in ("model name", "CPU part"):
        for line in info:
            if line.startswith(key):
                val = line.split(":", 1)[1].strip()
                if key == "CPU part":
                    impl = next((x.split(":", 1)[1].strip() for x in info if x.startswith("CPU implementer")), "?")
                    return f"{platform.machine()} implementer {impl} part {val}"
                return f"{platform.machine()} {val}"
    return platform.machine()


def run_reference(args) -> None:
    rank, world, local = dist_env()
    if rank != 0:
        return
    from oracle import plain
    from paper_2508_14544_gb300 import workloads as W
    cores = os.cpu_count() or 1
    n_all = W.WORKLOADS[WORKLOAD].n_instances
    sample = W.make_workload(WORKLOAD, range(0, n_all, 320))  # 128 instances per step, all alphas
    t_all, rs_all = [], 0
    for it in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        rs = 0
        for pol in (0, 1, 2):
            rs += int(plain.run_workload(pol, sample, n_threads=cores)["request_steps"].sum())
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
            "config": {"workload": WORKLOAD_DESC, "sample": f"{sample.n_instances} instances (every 320th) per step"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"{sample.n_instances} of {n_all} instances x 3 policies per step"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def _time_runs(sim, stream, load_args, reps: int, with_load: bool = True):
    """(median sim_load ms, median sim_run ms, last results) by CUDA events on the stream."""
    import torch
    lm, rm, res = [], [], None
    for _ in range(reps):
        e0, e1, e2 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
        torch.cuda.synchronize()
        e0.record(stream)
        if with_load:
            sim.load(*load_args)
        e1.record(stream)
        res = sim.run(stream.cuda_stream)
        e2.record(stream)
        torch.cuda.synchronize()
        lm.append(e0.elapsed_time(e1))
        rm.append(e1.elapsed_time(e2))
    return statistics.median(lm), statistics.median(rm), res


def algorithmic_work(res, wc, n_requests: int) -> dict:
    """Per-launch work of the per-step method from the results and the kernel's work counters."""
    rs = int(res["request_steps"].sum())
    ev = int(res["evictions"].sum())
    s2, s3, s5, gq = (int(x) for x in wc.sum(axis=0))
    s4 = 2 * (n_requests + ev)
    ops = OPS["request_step"] * rs + OPS["s2"] * s2 + OPS["s3"] * s3 + OPS["s5"] * s5 + OPS["s4"] * s4
    smem = SMEM_B["request_step"] * rs + SMEM_B["s3"] * s3 + SMEM_B["s5"] * s5 + SMEM_B["s4"] * s4
    hbm = 20 * n_requests + 56 * len(res) + gq
    return {"request_steps": rs, "s2_adds": s2, "s3_compare_exchanges": s3, "s5_endpoint_evals": s5,
            "s4_queue_ops": s4, "queue_global_bytes": gq, "int_ops": ops, "smem_bytes": smem, "hbm_bytes": hbm}


def sub_record(name: str, dev_id, stream, peaks_live: dict) -> dict:
    """One of the other configurations: per policy sim_load and sim_run device time (median of 10
    after two warm-ups), request-steps/s, steps/s, time per instance, the dominant kernel; on the
    10^5-request workload also the global-memory rate of the per-step method's queue traffic."""
    import torch

    from paper_2508_14544_gb300 import SIM_AMAX, SIM_AMIN, SIM_HSF, Simulator
    w = make_rank_workload(0, name)
    d_in = [torch.from_numpy(np.ascontiguousarray(x)).to(dev_id) for x in
            (w.arrival, w.prompt, w.lower, w.upper, w.true_o)]
    rec = {"instances": w.n_instances, "requests": w.n_total}
    per = {}
    for pname, pol in zip(POLICY_NAMES, (SIM_AMAX, SIM_AMIN, SIM_HSF)):
        with Simulator(pol, w.M, w.n_instances, tune_residency=1) as sim:
            sim.set_tie_seeds(w.tie_seeds())
            sim.load(w.offsets, *d_in)
            r = sim.run(stream.cuda_stream)  # warm-up (and residency tuning)
            assert np.all(r["status"] == 0), (name, pname, int(r["status"].min()))
            sim.run(stream.cuda_stream)  # second warm-up
            lms, rms, r = _time_runs(sim, stream, (w.offsets, *d_in), 10)
            rs = int(r["request_steps"].sum())
            p = {"sim_load_ms": round(lms, 3), "sim_run_ms": round(rms, 3), "request_steps": rs,
                 "request_steps_per_s": rs / (rms / 1000.0),
                 "steps_per_s": int(r["steps"].sum()) / (rms / 1000.0),
                 "us_per_instance": round(rms * 1000.0 / w.n_instances, 3)}
            if name == "c5":
                sim.set_option("count_work", 1)
                r2 = sim.run(stream.cuda_stream)
                wk = algorithmic_work(r2, sim.work_counts(), w.n_total)
                p["hbm_bytes_per_launch"] = wk["hbm_bytes"]
                p["hbm_GBps"] = round(wk["hbm_bytes"] / (rms / 1000.0) / 1e9, 2)
            per[pname] = p
    dom = max(per, key=lambda k: per[k]["sim_run_ms"])
    step_ms = sum(v["sim_load_ms"] + v["sim_run_ms"] for v in per.values())
    rec.update({"policies": per, "dominant_kernel": f"k_run<{dom}>",
                "request_steps_per_s": sum(v["request_steps"] for v in per.values()) / (step_ms / 1000.0)})
    if name == "c5":
        gb = per[dom]["hbm_GBps"]
        rec["hbm_of_measured"] = round(gb / float(_peaks().get("hbm_gbs", 6800.0)), 5)
    return rec


def critical_path_c2(dev_id, stream) -> dict:
    """A_min on the 1024-instance workload: the launch time against its slowest instance alone."""
    import torch

    from paper_2508_14544_gb300 import SIM_AMIN, Simulator
    w = make_rank_workload(0, "c2")
    with Simulator(SIM_AMIN, w.M, w.n_instances, tune_residency=1) as sim:
        sim.load_workload(w)
        r = sim.run(stream.cuda_stream)
        _, full_ms, r = _time_runs(sim, stream, None, 3, with_load=False)
    slow = int(np.argmax(r["evictions"]))
    one = w.subset([slow])
    with Simulator(SIM_AMIN, one.M, 1) as sim:
        sim.load_workload(one)
        sim.run(stream.cuda_stream)
        _, alone_ms, _ = _time_runs(sim, stream, None, 3, with_load=False)
    return {"workload": "c2 (1024 x n=1000)", "policy": "A_min", "launch_ms": round(full_ms, 3),
            "slowest_instance": slow, "its_cancellations": int(r["evictions"][slow]),
            "alone_ms": round(alone_ms, 3), "launch_over_alone": round(full_ms / alone_ms, 3)}


def run_ours(args) -> None:
    import torch
    import torch.distributed as dist

    import __graft_entry__
    __graft_entry__.build()
    from paper_2508_14544_gb300 import SIM_AELL, SIM_AMAX, SIM_AMIN, SIM_AR, SIM_HSF, Simulator, cr_amin_lemma
    from paper_2508_14544_gb300 import _lib as L

    rank, world, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    stream = torch.cuda.Stream(device=dev)
    sh = stream.cuda_stream
    peaks_live = L.measure_peaks()

    w = make_rank_workload(rank)
    host = [np.ascontiguousarray(x) for x in (w.arrival, w.prompt, w.lower, w.upper, w.true_o)]
    d_in = [torch.from_numpy(x).to(dev) for x in host]
    pinned = [torch.from_numpy(x).pin_memory() for x in host]
    # residency (one or two simulation warps per scheduler) is tuned on the first warm-up run of
    # each policy: a launch is as long as its slowest instance, and which residency is faster
    # depends on how uneven the instances are
    sims = [Simulator(p, w.M, w.n_instances, tune_residency=1) for p in (SIM_AMAX, SIM_AMIN, SIM_HSF)]
    for s in sims:
        s.set_tie_seeds(w.tie_seeds())
    torch.cuda.synchronize()

    def step(inputs):
        res = []
        for sim in sims:
            sim.load(w.offsets, *inputs)
            res.append(sim.run(sh))
        cr = [sims[0].competitive_ratio(sims[2], sh), sims[1].competitive_ratio(sims[2], sh)]
        return res, cr

    # warm-up (also checks that every instance finished)
    for _ in range(max(args.warmup, 1)):
        res, cr = step(d_in)
    for r in res:
        assert np.all(r["status"] == 0), r["status"]
    rs_per_step = int(sum(int(r["request_steps"].sum()) for r in res))
    launches0 = sum(s.kernel_launches() for s in sims)

    # timed region: K steps, device time by CUDA events on the simulator's stream; the inputs
    # (1.6 GB per policy) are larger than the 129 MB L2, so no flush is needed between steps
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ev = [[[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(3)] for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        time.sleep(0.3)
        for k in range(args.steps):
            starts[k].record(stream)
            for j, sim in enumerate(sims):
                ev[k][j][0].record(stream)
                sim.load(w.offsets, *d_in)
                ev[k][j][1].record(stream)
                res[j] = sim.run(sh)
                ev[k][j][2].record(stream)
            sims[0].competitive_ratio(sims[2], sh)
            sims[1].competitive_ratio(sims[2], sh)
            ends[k].record(stream)
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    launches = sum(s.kernel_launches() for s in sims) - launches0
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    run_ms = [[ev[k][j][1].elapsed_time(ev[k][j][2]) for j in range(3)] for k in range(args.steps)]
    load_ms = [[ev[k][j][0].elapsed_time(ev[k][j][1]) for j in range(3)] for k in range(args.steps)]
    total_s = sum(step_ms) / 1000.0
    if world > 1:
        t = torch.tensor([total_s], device=dev, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_s = float(t.item())
    value = rs_per_step * args.steps * world / total_s

    # end to end through the public API from pinned host buffers: every step copies its inputs
    # (the five request arrays, shared by the three policies) host to device on a copy stream and
    # reads every policy's per-instance results and the ratios back.  A step stages all three
    # policies first, then starts the next step's copy (into the other buffer), then simulates: the
    # copy runs under the simulation, and the small copies inside sim_load do not queue behind it
    # on the copy engine.  Step 0's copy is not hidden.  One untimed pass first (the first
    # transfers from a pinned buffer are slower than the rest).
    e2e_steps = args.steps
    copy_stream = torch.cuda.Stream(device=dev)
    bufs = [[torch.empty_like(t) for t in d_in] for _ in range(2)]
    copied = [torch.cuda.Event() for _ in range(2)]

    def copy_in(k):
        with torch.cuda.stream(copy_stream):
            for dst, src in zip(bufs[k % 2], pinned):
                dst.copy_(src, non_blocking=True)
            copied[k % 2].record(copy_stream)

    def e2e_run(n_steps):
        copy_in(0)
        for k in range(n_steps):
            copied[k % 2].synchronize()
            for sim in sims:
                sim.load(w.offsets, *bufs[k % 2])
            if k + 1 < n_steps:
                copy_in(k + 1)  # the other buffer: its last reader, step k-1's staging, has finished
            for sim in sims:
                sim.run(sh)
            sims[0].competitive_ratio(sims[2], sh)
            sims[1].competitive_ratio(sims[2], sh)
        torch.cuda.synchronize()

    e2e_run(1)
    if world > 1:
        dist.barrier()
    t0 = time.perf_counter()
    e2e_run(e2e_steps)
    e2e_s = time.perf_counter() - t0
    if world > 1:
        t = torch.tensor([e2e_s], device=dev, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        e2e_s = float(t.item())
    e2e_val = rs_per_step * e2e_steps * world / e2e_s
    h2d = 5 * w.n_total * 4
    d2h = 3 * w.n_instances * 56 + 2 * w.n_instances * 8

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    # ---- outside the timed region (rank 0) ----
    # the per-step method's work in each policy's launch (SIM_OPT_COUNT_WORK; same results)
    per_pol_ms = [statistics.mean(run_ms[k][j] for k in range(args.steps)) for j in range(3)]
    work = []
    for j, sim in enumerate(sims):
        sim.set_option("count_work", 1)
        r = sim.run(sh)
        for f in ("total_latency", "request_steps", "evictions", "steps"):
            assert np.array_equal(r[f], res[j][f]), f
        work.append(algorithmic_work(r, sim.work_counts(), w.n_total))
        sim.set_option("count_work", 0)
    dom = int(np.argmax(per_pol_ms))
    wd = work[dom]
    sec = per_pol_ms[dom] / 1000.0
    alu = {"achieved": wd["int_ops"] / sec / 1e12, "peak": peaks_live["int_ops_per_s"] / 1e12, "unit": "Tops/s"}
    alu["frac"] = alu["achieved"] / alu["peak"]
    smem = {"achieved": wd["smem_bytes"] / sec / 1e12, "peak": peaks_live["smem_bytes_per_s"] / 1e12, "unit": "TB/s"}
    smem["frac"] = smem["achieved"] / smem["peak"]
    hbm_peak = float(_peaks().get("hbm_gbs", 6800.0))
    hbm = {"achieved": wd["hbm_bytes"] / sec / 1e9, "peak": hbm_peak, "unit": "GB/s",
           "frac": wd["hbm_bytes"] / sec / 1e9 / hbm_peak}

    # the other configurations, and the latency regime of the 1024-instance workload
    subs = {name: sub_record(name, dev, stream, peaks_live) for name in SUB_WORKLOADS}
    crit = critical_path_c2(dev, stream)

    # the paper's two further policies on the same instances (outside the step): A_r (Algorithm
    # random, permutation drawn by the workload generator) and A_ell (Algorithm promote_l)
    further = {}
    for name, pol in (("A_r", SIM_AR), ("A_ell", SIM_AELL)):
        with Simulator(pol, w.M, w.n_instances, tune_residency=1) as sim:
            rk = torch.from_numpy(w.ranks()).to(dev) if pol == SIM_AR else None
            sim.load(w.offsets, *d_in, rank=rk)
            r = sim.run(sh)
            assert np.all(r["status"] == 0), (name, r["status"])
            _, ms, r = _time_runs(sim, stream, None, 2, with_load=False)
        rsn = int(r["request_steps"].sum())
        further[name] = {"sim_run_ms": round(ms, 3), "request_steps": rsn, "request_steps_per_s": rsn / (ms / 1000.0)}

    # the Lemma-thm:Amin evaluator on 2^20 histograms of 64 lengths (512 MB of doubles, read once):
    # 20 FP64 flops per length (6 FMA + 8 other), so GB300's FP64 rate bounds it, not HBM
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

    clocks = clk.summary()
    rs_pol = [int(r["request_steps"].sum()) for r in res]
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": statistics.mean(step_ms), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int32", "data": "synthetic",
        "config": {"workload": WORKLOAD_DESC, "workload_key": WORKLOAD, "instances_per_gpu": w.n_instances,
                   "requests_per_instance": 2000,
                   "parallelism": f"instances sharded, {world} replica(s), no collective on the data path",
                   "l2": "inputs larger than L2 (1.6 GB per policy against 129 MB); no flush",
                   "residency": "SIM_OPT_TUNE_RESIDENCY: one or two warps per scheduler, chosen per policy on the first warm-up run",
                   "tie_seeds": "A_min cancellation ties: SplitMix64, seed 3000000 + instance id",
                   "request_steps_per_step": rs_per_step,
                   "request_steps": dict(zip(POLICY_NAMES, rs_pol)),
                   "sim_run_ms": dict(zip(POLICY_NAMES, [round(x, 3) for x in per_pol_ms])),
                   "sim_load_ms": dict(zip(POLICY_NAMES, [round(statistics.mean(load_ms[k][j] for k in range(args.steps)), 3)
                                                          for j in range(3)])),
                   "batches_per_s": {POLICY_NAMES[j]: int(res[j]["steps"].sum()) / (per_pol_ms[j] / 1000.0)
                                     for j in range(3)},
                   "us_per_instance": {POLICY_NAMES[j]: round(1000.0 * per_pol_ms[j] / w.n_instances, 4)
                                       for j in range(3)},
                   "mean_cr": {"A_max": float(np.nanmean(cr[0])), "A_min": float(np.nanmean(cr[1]))},
                   "other_configs": subs,
                   "critical_path": crit,
                   "further_policies_not_in_step": further,
                   "lemma_evaluator": {"histograms": 1 << 20, "lengths": 64, "ms": round(statistics.median(lm), 4),
                                       "GB_per_s": round(lemma_gbs, 1),
                                       "frac_of_measured_hbm": round(lemma_gbs / hbm_peak, 3),
                                       "fp64_tflops": round(lemma_tflops, 3),
                                       "frac_of_nominal_fp64_1.25": round(lemma_tflops / 1.25, 3)}},
        "roofline": {"bound": "alu", "kernel": f"k_run<{POLICY_NAMES[dom]}>",
                     "achieved": alu["achieved"], "peak": alu["peak"], "unit": alu["unit"], "frac": alu["frac"],
                     "traffic": _dram_traffic(f"k_run<{POLICY_NAMES[dom]}>"),
                     "smem": smem, "hbm": hbm,
                     "peaks": "measured live by sim_measure_peaks (integer issue: add/xor chains; shared memory: "
                              "conflict-free 16-byte loads); HBM: MEASURED_PEAKS.json copy bandwidth",
                     "work_per_launch": wd,
                     "model": "work of the per-step method (Theorem complexity) counted by SIM_OPT_COUNT_WORK: "
                              "4 ops/8 B per request-step, 1 op per S2 add, 3 ops/8 B per S3 compare-exchange, "
                              "6 ops/16 B per S5 endpoint evaluation, 1 op/16 B per S4 queue operation; "
                              "achieved = that work / the launch's CUDA-event time"},
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
