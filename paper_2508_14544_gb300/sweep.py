"""The paper's load sweep (Section 6) on the synthetic stand-in for its dataset, through the C ABI.

  python -m paper_2508_14544_gb300.sweep [--experiments rough,buckets,overlap:1/10,...]
                                         [--policies A_max,A_min,H-SF] [--seeds 4] [--M 10000]

For every experiment (interval construction) and policy, all loads n = 200, 400, .., 2000 and all
seeds are simulated in one batch on the GPU; the average end-to-end latency (TEL / n, in batches)
is averaged over the seeds.  Prints one JSON line per (experiment, policy) and a table.
"""
from __future__ import annotations

import argparse
import json
import time

import numpy as np

from . import POLICIES, Simulator
from . import workloads as W


def run_sweep(experiment: str, policies, seeds: int, M: int, loads=tuple(range(200, 2001, 200))) -> dict:
    w = W.make_sweep(experiment, loads=loads, seeds=seeds, M=M)
    n = np.diff(w.offsets)
    out = {}
    for name in policies:
        with Simulator(POLICIES[name], w.M, w.n_instances) as sim:
            sim.load_workload(w)
            t0 = time.perf_counter()
            res = sim.run()
            dt = time.perf_counter() - t0
        if np.any(res["status"] != 0):
            raise RuntimeError(f"{experiment} {name}: instance status {res['status'].min()}")
        avg = res["total_latency"] / n
        per_load = {int(L): float(avg[n == L].mean()) for L in loads}
        out[name] = dict(avg_latency=per_load, sim_run_s=dt, evictions=int(res["evictions"].sum()))
    return out


def main(argv=None) -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--experiments", default="rough,buckets,overlap:1/10,overlap:19/20,overlap:99/100")
    ap.add_argument("--policies", default="A_max,A_min,H-SF")
    ap.add_argument("--seeds", type=int, default=4)
    ap.add_argument("--M", type=int, default=10000)
    args = ap.parse_args(argv)
    pols = args.policies.split(",")
    for exp in args.experiments.split(","):
        res = run_sweep(exp, pols, args.seeds, args.M)
        for name, r in res.items():
            print(json.dumps({"experiment": exp, "policy": name, "M": args.M, "seeds": args.seeds, **r}), flush=True)
        loads = sorted(next(iter(res.values()))["avg_latency"])
        print(f"# {exp}: average latency (batches) by load")
        print("# n     " + "  ".join(f"{p:>9s}" for p in pols))
        for L in loads:
            print(f"# {L:<6d}" + "  ".join(f"{res[p]['avg_latency'][L]:9.1f}" for p in pols))


if __name__ == "__main__":
    main()
