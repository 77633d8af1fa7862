"""Command-line runner: simulate a named synthetic workload under one policy through the C ABI.

  python -m paper_2508_14544_gb300.run --workload c2 --policy A_min [--instances 0:1024[:step]] [--repeat 1]
                                       [--warps-per-block W] [--warps-per-sm S] [--evict-ties-by-index]
                                       [--dense]

Prints one JSON line per run with the wall time of sim_run, totals of the result fields, the
throughput and a sha256 of the per-instance result records (equal across runs and launch shapes).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import time

import numpy as np

from . import POLICIES, Simulator
from . import workloads as W


def main(argv=None) -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="c2", choices=sorted(W.WORKLOADS))
    ap.add_argument("--policy", default="A_min", choices=sorted(POLICIES))
    ap.add_argument("--instances", default=None, help="a:b or a:b:step range of instance ids (default: all)")
    ap.add_argument("--repeat", type=int, default=1)
    ap.add_argument("--warps-per-block", type=int, default=0)
    ap.add_argument("--warps-per-sm", type=int, default=0, help="residency limit (4: one warp per scheduler)")
    ap.add_argument("--evict-ties-by-index", action="store_true", help="A_min: cancellation ties by index")
    ap.add_argument("--dense", action="store_true", help="12 simulating warps per SM, 384 active-set slots")
    args = ap.parse_args(argv)
    ids = None
    if args.instances:
        ids = range(*(int(x) for x in args.instances.split(":")))
    w = W.make_workload(args.workload, ids)
    import torch
    dev = [torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in (w.arrival, w.prompt, w.lower, w.upper, w.true_o)]
    rank = torch.from_numpy(w.ranks()).cuda() if POLICIES[args.policy] == 3 else None
    opts = {}
    if args.warps_per_block:
        opts["warps_per_block"] = args.warps_per_block
    if args.warps_per_sm:
        opts["warps_per_sm"] = args.warps_per_sm
    if args.evict_ties_by_index:
        opts["evict_ties"] = 1
    if args.dense:
        opts["dense_residency"] = 1
    with Simulator(POLICIES[args.policy], w.M, w.n_instances, **opts) as sim:
        sim.set_tie_seeds(w.tie_seeds())
        for _ in range(args.repeat):
            sim.load(w.offsets, *dev, rank=rank)
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            res = sim.run()
            dt = time.perf_counter() - t0
            rs, st = int(res["request_steps"].sum()), int(res["steps"].sum())
            digest = hashlib.sha256(np.ascontiguousarray(res).tobytes()).hexdigest()
            print(json.dumps({"workload": args.workload, "policy": args.policy, "instances": w.n_instances,
                              "sim_run_s": dt, "request_steps": rs, "steps": st,
                              "request_steps_per_s": rs / dt, "steps_per_s": st / dt,
                              "total_latency": int(res["total_latency"].sum()),
                              "evictions": int(res["evictions"].sum()),
                              "most_evictions": [int(ids[int(np.argmax(res["evictions"]))]) if ids else
                                                 int(np.argmax(res["evictions"])),
                                                 int(res["evictions"].max())],
                              "worst_status": int(res["status"].min()), "results_sha256": digest}), flush=True)


if __name__ == "__main__":
    main()
