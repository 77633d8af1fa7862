"""ctypes wrapper of the plain C oracle (``oracle/plain.c``).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this module.  It shares no code with the CUDA path.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from pathlib import Path

import numpy as np

_HERE = Path(__file__).resolve().parent
_SRC = _HERE / "plain.c"
_SO = _HERE / "_build" / "liboracle.so"

RESULT_DTYPE = np.dtype([
    ("total_latency", "<i8"), ("makespan", "<i8"), ("peak_memory", "<i8"),
    ("evictions", "<i8"), ("steps", "<i8"), ("request_steps", "<i8"),
    ("status", "<i4"), ("pad", "<i4"),
])
FIELDS = ("total_latency", "makespan", "peak_memory", "evictions", "steps", "request_steps", "status")

_lib = None


def build(force: bool = False) -> Path:
    """Compile the C oracle into oracle/_build/liboracle.so (plain gcc, -O2)."""
    _SO.parent.mkdir(parents=True, exist_ok=True)
    if force or not _SO.exists() or _SO.stat().st_mtime < _SRC.stat().st_mtime:
        tmp = _SO.with_suffix(f".so.{os.getpid()}")
        subprocess.run(["gcc", "-O2", "-std=c11", "-D_GNU_SOURCE", "-ffp-contract=off", "-shared", "-fPIC", "-o", str(tmp),
                        str(_SRC), "-lpthread"], check=True)
        os.replace(tmp, _SO)
    return _SO


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(str(_SO))
        i32p = ctypes.POINTER(ctypes.c_int32)
        i64p = ctypes.POINTER(ctypes.c_int64)
        L.oracle_run.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, i32p, i32p, i32p, i32p,
                                 i32p, ctypes.c_int64, ctypes.c_void_p, i64p]
        L.oracle_run.restype = ctypes.c_int
        L.oracle_run_batch.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, i64p, i32p, i32p,
                                       i32p, i32p, i32p, ctypes.c_int64, ctypes.c_void_p, i64p,
                                       ctypes.c_int32]
        L.oracle_run_batch.restype = ctypes.c_int
        L.oracle_run_ex.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, i32p, i32p, i32p, i32p,
                                    i32p, i32p, ctypes.c_int64, ctypes.c_void_p, i64p]
        L.oracle_run_ex.restype = ctypes.c_int
        L.oracle_run_batch_ex.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, i64p, i32p, i32p,
                                          i32p, i32p, i32p, i32p, ctypes.c_int64, ctypes.c_void_p, i64p,
                                          ctypes.c_int32]
        L.oracle_run_batch_ex.restype = ctypes.c_int
        u64p = ctypes.POINTER(ctypes.c_uint64)
        L.oracle_run_seeded.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, i32p, i32p, i32p, i32p,
                                        i32p, i32p, ctypes.c_uint64, ctypes.c_int, ctypes.c_int64,
                                        ctypes.c_void_p, i64p]
        L.oracle_run_seeded.restype = ctypes.c_int
        L.oracle_run_batch_seeded.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, i64p, i32p, i32p,
                                              i32p, i32p, i32p, i32p, u64p, ctypes.c_int, ctypes.c_int64,
                                              ctypes.c_void_p, i64p, ctypes.c_int32]
        L.oracle_run_batch_seeded.restype = ctypes.c_int
        L.oracle_run_full.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, i32p, i32p, i32p, i32p,
                                      i32p, i32p, ctypes.c_uint64, ctypes.c_int, ctypes.c_int64,
                                      ctypes.c_void_p, i64p, i64p]
        L.oracle_run_full.restype = ctypes.c_int
        L.oracle_run_batch_full.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, i64p, i32p, i32p,
                                            i32p, i32p, i32p, i32p, u64p, ctypes.c_int, ctypes.c_int64,
                                            ctypes.c_void_p, i64p, i64p, ctypes.c_int32]
        L.oracle_run_batch_full.restype = ctypes.c_int
        L.oracle_batch_time.argtypes = [i64p, ctypes.c_void_p, ctypes.POINTER(ctypes.c_double),
                                        ctypes.POINTER(ctypes.c_double)]
        L.oracle_batch_time.restype = None
        L.oracle_tie_key.argtypes = [ctypes.c_uint64, ctypes.c_int64, ctypes.c_int32]
        L.oracle_tie_key.restype = ctypes.c_uint32
        L.oracle_default_step_cap.argtypes = [ctypes.c_int32, i32p]
        L.oracle_default_step_cap.restype = ctypes.c_int64
        _lib = L
    return _lib


def _i32(x) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(x, dtype=np.int32))


def _p32(x: np.ndarray | None):
    if x is None:
        return ctypes.POINTER(ctypes.c_int32)()
    return x.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


def _p64(x: np.ndarray | None):
    if x is None:
        return ctypes.POINTER(ctypes.c_int64)()
    return x.ctypes.data_as(ctypes.POINTER(ctypes.c_int64))


def _evict_index(evict_ties: str) -> int:
    if evict_ties not in ("hash", "index"):
        raise ValueError(evict_ties)
    return 1 if evict_ties == "index" else 0


def tie_key(seed: int, t: int, i: int) -> int:
    """A_min's random tie key of request i at step t (the C oracle's own SplitMix64)."""
    return int(lib().oracle_tie_key(int(seed) & ((1 << 64) - 1), int(t), int(i)))


def run(policy: int, M: int, a, s, l, u, o, step_cap: int = 0, completions: bool = False,
        rank=None, tie_seed: int = 0, evict_ties: str = "hash", time_sums: bool = False) -> dict:
    """One instance.  Returns the result fields (and 'completion' if asked).  ``rank`` is A_r's
    permutation (rank[i] = position of request i); ``tie_seed`` seeds A_min's random eviction
    ties (``evict_ties="index"``: by request index instead)."""
    a, s, l, u, o = (_i32(v) for v in (a, s, l, u, o))
    rank = None if rank is None else _i32(rank)
    n = int(o.shape[0])
    res = np.zeros(1, dtype=RESULT_DTYPE)
    comp = np.zeros(max(n, 1), dtype=np.int64) if completions else None
    ts = np.zeros(6, dtype=np.int64) if time_sums else None
    lib().oracle_run_full(int(policy), int(M), n, _p32(a), _p32(s), _p32(l), _p32(u), _p32(o), _p32(rank),
                          int(tie_seed) & ((1 << 64) - 1), _evict_index(evict_ties), int(step_cap),
                          res.ctypes.data, _p64(comp), _p64(ts))
    out = {k: int(res[0][k]) for k in FIELDS}
    if time_sums:
        out["time_sums"] = ts.tolist()
        out["_res"] = res
    if completions:
        out["completion"] = comp[:n].tolist()
    return out


def run_batch(policy: int, M: int, offsets, a, s, l, u, o, step_cap: int = 0, n_threads: int = 1,
              completions: bool = False, rank=None, tie_seeds=None, evict_ties: str = "hash",
              time_sums: bool = False):
    """Many instances in CSR layout.  Returns a structured array (RESULT_DTYPE), then optionally
    the per-request completion steps and the [n_instances, 6] batch-time sums.  ``tie_seeds``: one
    uint64 per instance (default 0 for all)."""
    offsets = np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))
    a, s, l, u, o = (_i32(v) for v in (a, s, l, u, o))
    rank = None if rank is None else _i32(rank)
    n_inst = int(offsets.shape[0] - 1)
    seeds = None
    if tie_seeds is not None:
        seeds = np.ascontiguousarray(np.asarray(tie_seeds, dtype=np.uint64))
        assert seeds.shape == (n_inst,)
    res = np.zeros(n_inst, dtype=RESULT_DTYPE)
    comp = np.zeros(max(int(offsets[-1]), 1), dtype=np.int64) if completions else None
    sp = ctypes.POINTER(ctypes.c_uint64)() if seeds is None else seeds.ctypes.data_as(ctypes.POINTER(ctypes.c_uint64))
    ts = np.zeros((max(n_inst, 1), 6), dtype=np.int64) if time_sums else None
    lib().oracle_run_batch_full(int(policy), int(M), n_inst, _p64(offsets), _p32(a), _p32(s), _p32(l),
                                _p32(u), _p32(o), _p32(rank), sp, _evict_index(evict_ties), int(step_cap),
                                res.ctypes.data, _p64(comp), _p64(ts), int(n_threads))
    out = (res,)
    if completions:
        out += (comp[: int(offsets[-1])],)
    if time_sums:
        out += (ts[:n_inst],)
    return out[0] if len(out) == 1 else out


def run_workload(policy: int, w, step_cap: int = 0, n_threads: int = 1, completions: bool = False,
                 evict_ties: str = "hash", time_sums: bool = False):
    """Convenience: run a ``Workload`` (from the seeded generator) through the C oracle, with the
    workload's own A_min tie seeds."""
    return run_batch(policy, w.M, w.offsets, w.arrival, w.prompt, w.lower, w.upper, w.true_o,
                     step_cap=step_cap, n_threads=n_threads, completions=completions,
                     rank=w.ranks() if policy == 3 else None, tie_seeds=w.tie_seeds(),
                     evict_ties=evict_ties, time_sums=time_sums)


def batch_time(res, time_sums, coef) -> np.ndarray:
    """[n, 2] (total latency, makespan) in time units under coef = (c0, c1, c2, c3, c_idle), by the
    C oracle's own evaluation (res: RESULT_DTYPE rows, time_sums: [n, 6])."""
    res = np.ascontiguousarray(np.atleast_1d(res))
    ts = np.ascontiguousarray(np.asarray(time_sums, dtype=np.int64).reshape(-1, 6))
    cf = np.ascontiguousarray(np.asarray(coef, dtype=np.float64))
    assert cf.shape == (5,) and ts.shape[0] == res.shape[0]
    out = np.zeros((res.shape[0], 2), dtype=np.float64)
    dp = ctypes.POINTER(ctypes.c_double)
    for i in range(res.shape[0]):
        lib().oracle_batch_time(ts[i].ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), res[i:i + 1].ctypes.data,
                                cf.ctypes.data_as(dp), out[i].ctypes.data_as(dp))
    return out


def default_step_cap(o) -> int:
    o = _i32(o)
    return int(lib().oracle_default_step_cap(int(o.shape[0]), _p32(o)))
