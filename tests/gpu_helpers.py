"""Helpers for the GPU parity tests: run a Workload through the C ABI and through the C oracle."""
from __future__ import annotations

import os

import numpy as np

FIELDS = ("total_latency", "makespan", "peak_memory", "evictions", "steps", "request_steps", "status")


def n_threads() -> int:
    return max(1, min(32, os.cpu_count() or 1))


def gpu_run(policy, w, device_load=True, completions=False, rank=None, **opts):
    """A_r (policy 3) takes ``rank`` or, if None, the workload's own ranks()."""
    import torch

    from paper_2508_14544_gb300 import Simulator
    if policy == 3 and rank is None:
        rank = w.ranks()
    with Simulator(policy, w.M, w.n_instances, record_completions=int(completions), **opts) as sim:
        if device_load:
            sim.set_tie_seeds(w.tie_seeds())
            dev = [torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in
                   (w.arrival, w.prompt, w.lower, w.upper, w.true_o)]
            rk = None if rank is None else torch.from_numpy(np.ascontiguousarray(np.asarray(rank, np.int32))).cuda()
            sim.load(w.offsets, *dev, rank=rk)
        elif rank is not None:
            sim.set_tie_seeds(w.tie_seeds())
            sim.load(w.offsets, w.arrival, w.prompt, w.lower, w.upper, w.true_o, rank=np.asarray(rank, np.int32))
        else:
            sim.load_workload(w)
        res = sim.run()
        comp = sim.completions(w.n_total) if completions else None
    return res, comp


def oracle_run(policy, w, completions=False, step_cap=0, evict_ties="hash"):
    from oracle import plain
    return plain.run_workload(policy, w, step_cap=step_cap, n_threads=n_threads(), completions=completions,
                              evict_ties=evict_ties)


def assert_same(got, ref, rows=None, tag=""):
    rows = np.arange(len(ref)) if rows is None else np.asarray(rows)
    for f in FIELDS:
        g = np.asarray(got[f])[rows] if len(got) != len(ref) else np.asarray(got[f])
        r = np.asarray(ref[f])
        bad = np.nonzero(g != r)[0]
        assert bad.size == 0, f"{tag}: field {f} differs at rows {bad[:10].tolist()}: gpu {g[bad[:5]].tolist()} oracle {r[bad[:5]].tolist()}"
