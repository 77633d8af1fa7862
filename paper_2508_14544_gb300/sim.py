"""A small object wrapper over the C ABI: one ``Simulator`` per (policy, M, n_instances) context."""
from __future__ import annotations

import numpy as np

from . import _lib as L


def _i32_host(x) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(x, dtype=np.int32))


class Simulator:
    """Owns a sim_ctx.  ``load`` accepts numpy arrays (host) or int32 CUDA tensors (device)."""

    def __init__(self, policy: int, M: int, n_instances: int, **options):
        self.policy, self.M, self.n_instances = int(policy), int(M), int(n_instances)
        self.ctx = L.sim_create(policy, M, n_instances)
        self._keep = None
        for k, v in options.items():
            self.set_option(k, v)

    OPTIONS = {"step_cap": L.SIM_OPT_STEP_CAP, "record_completions": L.SIM_OPT_RECORD_COMPLETIONS,
               "warps_per_block": L.SIM_OPT_WARPS_PER_BLOCK, "smem_active_cap": L.SIM_OPT_SMEM_ACTIVE_CAP,
               "warps_per_sm": L.SIM_OPT_WARPS_PER_SM, "debug_checks": L.SIM_OPT_DEBUG_CHECKS,
               "tune_residency": L.SIM_OPT_TUNE_RESIDENCY, "evict_ties": L.SIM_OPT_EVICT_TIES,
               "count_work": L.SIM_OPT_COUNT_WORK, "batch_time": L.SIM_OPT_BATCH_TIME,
               "dense_residency": L.SIM_OPT_DENSE_RESIDENCY}

    def set_option(self, name: str, value: int) -> None:
        rc = L.sim_set_option(self.ctx, self.OPTIONS[name], int(value))
        if rc != L.SIM_OK:
            raise L.SimError(rc, L.sim_last_error(self.ctx))

    def set_tie_seeds(self, seeds) -> None:
        """Seeds of A_min's random cancellation ties, one per instance (None: all 0)."""
        if seeds is not None:
            assert len(seeds) == self.n_instances
        self._check(L.sim_set_tie_seeds(self.ctx, seeds))

    def _check(self, rc: int, allow_instance_status: bool = False) -> int:
        if rc != L.SIM_OK and not (allow_instance_status and rc in (L.SIM_E_INVAL, L.SIM_E_INFEASIBLE,
                                                                     L.SIM_E_STEPCAP)):
            raise L.SimError(rc, L.sim_last_error(self.ctx))
        return rc

    def load(self, offsets, a, s, l, u, o, rank=None) -> None:
        """Load requests (host numpy arrays or CUDA int32 tensors).  ``rank`` is A_r's permutation
        (same layout and memory kind); when given, sim_load_ranked_csr is used."""
        offsets = np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))
        dev = hasattr(a, "is_cuda") and a.is_cuda
        src = (a, s, l, u, o) if rank is None else (a, s, l, u, o, rank)
        if dev:
            arrs = [x.contiguous() for x in src]
            for x in arrs:
                assert str(x.dtype) == "torch.int32"
        else:
            arrs = [_i32_host(x) for x in src]
        if rank is None:
            self._check(L.sim_load_csr(self.ctx, offsets, *arrs, 1 if dev else 0))
        else:
            self._check(L.sim_load_ranked_csr(self.ctx, offsets, *arrs, 1 if dev else 0))

    def load_workload(self, w) -> None:
        """Load a seeded ``Workload`` with its A_min tie seeds; under A_r its ranks() are the
        permutation."""
        rank = w.ranks() if self.policy == L.SIM_AR else None
        self.set_tie_seeds(w.tie_seeds())
        self.load(w.offsets, w.arrival, w.prompt, w.lower, w.upper, w.true_o, rank=rank)

    def run(self, stream: int = 0) -> np.ndarray:
        out = np.zeros(self.n_instances, dtype=L.RESULT_DTYPE)
        self.last_rc = self._check(L.sim_run(self.ctx, out, stream), allow_instance_status=True)
        return out

    def work_counts(self) -> np.ndarray:
        """[n_instances, 4] int64 work counters of the last run (option count_work=1)."""
        out = np.zeros(4 * self.n_instances, dtype=np.int64)
        self._check(L.sim_get_work_counts(self.ctx, out))
        return out.reshape(self.n_instances, 4)

    def batch_time(self, coef, stream: int = 0) -> np.ndarray:
        """[n_instances, 2] (total latency, makespan) in time units under the linear batch-time
        model coef = (c0, c1, c2, c3, c_idle) (option batch_time=1 for the last run)."""
        out = np.zeros(2 * self.n_instances, dtype=np.float64)
        self._check(L.sim_batch_time(self.ctx, coef, out, stream))
        return out.reshape(self.n_instances, 2)

    def batch_time_sums(self) -> np.ndarray:
        """[n_instances, 6] int64: X0..X3, F2, F3 of the last run (option batch_time=1)."""
        out = np.zeros(6 * self.n_instances, dtype=np.int64)
        self._check(L.sim_get_batch_time_sums(self.ctx, out))
        return out.reshape(self.n_instances, 6)

    def completions(self, n_total: int) -> np.ndarray:
        out = np.zeros(max(n_total, 1), dtype=np.int64)
        self._check(L.sim_get_completions(self.ctx, out))
        return out[:n_total]

    def competitive_ratio(self, hsf: "Simulator", stream: int = 0) -> np.ndarray:
        out = np.zeros(self.n_instances, dtype=np.float64)
        self._check(L.sim_competitive_ratio(self.ctx, hsf.ctx, out, stream))
        return out

    def kernel_launches(self) -> int:
        return L.sim_kernel_launches(self.ctx)

    def close(self) -> None:
        if getattr(self, "ctx", None):
            L.sim_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
