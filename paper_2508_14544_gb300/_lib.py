"""ctypes binding of libsim.so (include/sim.h).

Argument marshalling only: every step of the simulation runs in the library's CUDA kernels.
There is no CPU fallback; if the library is missing or fails to load, ``lib()`` raises.
"""
from __future__ import annotations

import ctypes
import os
from pathlib import Path

import numpy as np

from .build import LIB

SIM_AMAX, SIM_AMIN, SIM_HSF, SIM_AR, SIM_AELL = 0, 1, 2, 3, 4
SIM_OK, SIM_E_INVAL, SIM_E_INFEASIBLE, SIM_E_STEPCAP, SIM_E_CUDA, SIM_E_STATE, SIM_E_NOMEM = 0, -1, -2, -3, -4, -5, -6
SIM_OPT_STEP_CAP, SIM_OPT_RECORD_COMPLETIONS, SIM_OPT_WARPS_PER_BLOCK, SIM_OPT_SMEM_ACTIVE_CAP = 1, 2, 3, 4
SIM_OPT_WARPS_PER_SM = 5
SIM_OPT_DEBUG_CHECKS = 6
SIM_OPT_TUNE_RESIDENCY = 7
SIM_OPT_EVICT_TIES = 8
SIM_OPT_COUNT_WORK = 9
SIM_OPT_BATCH_TIME = 10
SIM_OPT_DENSE_RESIDENCY = 11

STATUS_NAMES = {0: "SIM_OK", -1: "SIM_E_INVAL", -2: "SIM_E_INFEASIBLE", -3: "SIM_E_STEPCAP", -4: "SIM_E_CUDA",
                -5: "SIM_E_STATE", -6: "SIM_E_NOMEM"}


class sim_result(ctypes.Structure):
    _fields_ = [("total_latency", ctypes.c_int64), ("makespan", ctypes.c_int64), ("peak_memory", ctypes.c_int64),
                ("evictions", ctypes.c_int64), ("steps", ctypes.c_int64), ("request_steps", ctypes.c_int64),
                ("status", ctypes.c_int32), ("_pad", ctypes.c_int32)]


RESULT_DTYPE = np.dtype([
    ("total_latency", "<i8"), ("makespan", "<i8"), ("peak_memory", "<i8"), ("evictions", "<i8"),
    ("steps", "<i8"), ("request_steps", "<i8"), ("status", "<i4"), ("_pad", "<i4"),
])
assert RESULT_DTYPE.itemsize == ctypes.sizeof(sim_result) == 56

EXPORTS = ("sim_create", "sim_load", "sim_load_csr", "sim_load_ranked_csr", "sim_run", "sim_get_completions", "sim_competitive_ratio",
           "sim_set_option", "sim_set_tie_seeds", "sim_get_work_counts", "sim_batch_time",
           "sim_get_batch_time_sums", "sim_last_error", "sim_destroy", "sim_kernel_launches", "sim_run_noalloc",
           "sim_cr_amin_lemma", "sim_cr_amin_rho", "sim_measure_peaks")

_lib = None


class SimError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(code, code)}: {msg}")
        self.code = code


def lib_path() -> Path:
    p = os.environ.get("SIMGB_LIB")
    return Path(p) if p else LIB


def lib() -> ctypes.CDLL:
    """Load libsim.so (it must have been built, e.g. by __graft_entry__.build())."""
    global _lib
    if _lib is not None:
        return _lib
    path = lib_path()
    if not path.exists():
        raise RuntimeError(f"libsim.so not found at {path}: build it first (python -m paper_2508_14544_gb300.build)")
    L = ctypes.CDLL(str(path))
    vp, i32p, i64p = ctypes.c_void_p, ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int64)
    L.sim_create.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, ctypes.POINTER(vp)]
    L.sim_create.restype = ctypes.c_int
    L.sim_load.argtypes = [vp, ctypes.c_int32, vp, vp, vp, vp, vp, ctypes.c_int]
    L.sim_load.restype = ctypes.c_int
    L.sim_load_csr.argtypes = [vp, vp, vp, vp, vp, vp, vp, ctypes.c_int]
    L.sim_load_csr.restype = ctypes.c_int
    L.sim_load_ranked_csr.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, ctypes.c_int]
    L.sim_load_ranked_csr.restype = ctypes.c_int
    L.sim_run.argtypes = [vp, vp, vp]
    L.sim_run.restype = ctypes.c_int
    L.sim_get_completions.argtypes = [vp, vp]
    L.sim_get_completions.restype = ctypes.c_int
    L.sim_competitive_ratio.argtypes = [vp, vp, vp, vp]
    L.sim_competitive_ratio.restype = ctypes.c_int
    L.sim_set_option.argtypes = [vp, ctypes.c_int, ctypes.c_int64]
    L.sim_set_option.restype = ctypes.c_int
    L.sim_set_tie_seeds.argtypes = [vp, vp]
    L.sim_set_tie_seeds.restype = ctypes.c_int
    L.sim_get_work_counts.argtypes = [vp, vp]
    L.sim_get_work_counts.restype = ctypes.c_int
    L.sim_batch_time.argtypes = [vp, vp, vp, vp]
    L.sim_batch_time.restype = ctypes.c_int
    L.sim_get_batch_time_sums.argtypes = [vp, vp]
    L.sim_get_batch_time_sums.restype = ctypes.c_int
    L.sim_last_error.argtypes = [vp]
    L.sim_last_error.restype = ctypes.c_char_p
    L.sim_destroy.argtypes = [vp]
    L.sim_destroy.restype = None
    L.sim_kernel_launches.argtypes = [vp]
    L.sim_kernel_launches.restype = ctypes.c_int64
    L.sim_run_noalloc.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, vp, vp, vp, vp, vp, vp, vp, vp]
    L.sim_run_noalloc.restype = ctypes.c_int
    L.sim_cr_amin_lemma.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_double, vp, vp,
                                    ctypes.c_int, vp]
    L.sim_cr_amin_lemma.restype = ctypes.c_int
    L.sim_cr_amin_rho.argtypes = [ctypes.c_int32, vp, vp]
    L.sim_cr_amin_rho.restype = ctypes.c_int
    L.sim_measure_peaks.argtypes = [vp]
    L.sim_measure_peaks.restype = ctypes.c_int
    _lib = L
    return L


# ---- thin wrappers with the C names -------------------------------------------------------------

def sim_create(policy: int, M: int, n_instances: int) -> ctypes.c_void_p:
    h = ctypes.c_void_p()
    rc = lib().sim_create(int(policy), int(M), int(n_instances), ctypes.byref(h))
    if rc != SIM_OK:
        raise SimError(rc, sim_last_error(None))
    return h


def sim_last_error(ctx) -> str:
    s = lib().sim_last_error(ctx)
    return s.decode() if s else ""


def sim_set_option(ctx, key: int, value: int) -> int:
    return lib().sim_set_option(ctx, int(key), int(value))


def sim_set_tie_seeds(ctx, seeds) -> int:
    """Seeds of A_min's random cancellation ties: one uint64 per instance (host), or None."""
    if seeds is None:
        return lib().sim_set_tie_seeds(ctx, None)
    arr = np.ascontiguousarray(np.asarray(seeds, dtype=np.uint64))
    return lib().sim_set_tie_seeds(ctx, arr.ctypes.data)


def _ptr(x) -> int:
    """Address of a contiguous int32 host array or device tensor (torch)."""
    if isinstance(x, np.ndarray):
        return x.ctypes.data
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    raise TypeError(type(x))


def sim_load(ctx, n_per_instance: int, a, s, l, u, o, device_ptrs: int) -> int:
    return lib().sim_load(ctx, int(n_per_instance), _ptr(a), _ptr(s), _ptr(l), _ptr(u), _ptr(o), int(device_ptrs))


def sim_load_csr(ctx, offsets: np.ndarray, a, s, l, u, o, device_ptrs: int) -> int:
    assert offsets.dtype == np.int64 and offsets.flags.c_contiguous
    return lib().sim_load_csr(ctx, offsets.ctypes.data, _ptr(a), _ptr(s), _ptr(l), _ptr(u), _ptr(o),
                              int(device_ptrs))


def sim_load_ranked_csr(ctx, offsets: np.ndarray, a, s, l, u, o, rank, device_ptrs: int) -> int:
    assert offsets.dtype == np.int64 and offsets.flags.c_contiguous
    return lib().sim_load_ranked_csr(ctx, offsets.ctypes.data, _ptr(a), _ptr(s), _ptr(l), _ptr(u), _ptr(o),
                                     _ptr(rank) if rank is not None else None, int(device_ptrs))


def sim_run(ctx, out: np.ndarray, stream: int = 0) -> int:
    assert out.dtype == RESULT_DTYPE and out.flags.c_contiguous
    return lib().sim_run(ctx, out.ctypes.data, ctypes.c_void_p(stream or None))


def sim_get_work_counts(ctx, out: np.ndarray) -> int:
    assert out.dtype == np.int64 and out.flags.c_contiguous
    return lib().sim_get_work_counts(ctx, out.ctypes.data)


def sim_batch_time(ctx, coef, out: np.ndarray, stream: int = 0) -> int:
    cf = np.ascontiguousarray(np.asarray(coef, dtype=np.float64))
    assert cf.shape == (5,) and out.dtype == np.float64 and out.flags.c_contiguous
    return lib().sim_batch_time(ctx, cf.ctypes.data, out.ctypes.data, ctypes.c_void_p(stream or None))


def sim_get_batch_time_sums(ctx, out: np.ndarray) -> int:
    assert out.dtype == np.int64 and out.flags.c_contiguous
    return lib().sim_get_batch_time_sums(ctx, out.ctypes.data)


def sim_get_completions(ctx, out: np.ndarray) -> int:
    assert out.dtype == np.int64 and out.flags.c_contiguous
    return lib().sim_get_completions(ctx, out.ctypes.data)


def sim_competitive_ratio(ctx_policy, ctx_hsf, out: np.ndarray, stream: int = 0) -> int:
    assert out.dtype == np.float64 and out.flags.c_contiguous
    return lib().sim_competitive_ratio(ctx_policy, ctx_hsf, out.ctypes.data, ctypes.c_void_p(stream or None))


def sim_kernel_launches(ctx) -> int:
    return int(lib().sim_kernel_launches(ctx))


def sim_run_noalloc(policy: int, M: int, offsets: np.ndarray, a, s, l, u, o, results, stream: int = 0) -> int:
    """Stage and simulate without any device allocation by the library (see include/sim.h).
    a..o and results are device tensors; offsets is a host int64 array."""
    assert offsets.dtype == np.int64 and offsets.flags.c_contiguous
    n_inst = int(offsets.shape[0] - 1)
    return lib().sim_run_noalloc(int(policy), int(M), n_inst, offsets.ctypes.data, _ptr(a), _ptr(s), _ptr(l),
                                 _ptr(u), _ptr(o), _ptr(results), ctypes.c_void_p(stream or None))


def sim_destroy(ctx) -> None:
    lib().sim_destroy(ctx)


def cr_amin_lemma(x, l: int, s: float, stream: int = 0):
    """Lemma thm:Amin for each row of ``x`` (host float64 array [n_hist, len] or a CUDA float64
    tensor; a tensor gives a tensor, computed asynchronously on ``stream``)."""
    if hasattr(x, "is_cuda") and x.is_cuda:
        import torch
        x = x.contiguous()
        assert x.dtype == torch.float64 and x.dim() == 2
        out = torch.empty(x.shape[0], dtype=torch.float64, device=x.device)
        rc = lib().sim_cr_amin_lemma(int(x.shape[0]), int(x.shape[1]), int(l), float(s), x.data_ptr(),
                                     out.data_ptr(), 1, ctypes.c_void_p(stream or None))
    else:
        x = np.ascontiguousarray(np.asarray(x, dtype=np.float64))
        if x.ndim == 1:
            x = x[None, :]
        out = np.zeros(x.shape[0], dtype=np.float64)
        rc = lib().sim_cr_amin_lemma(int(x.shape[0]), int(x.shape[1]), int(l), float(s), x.ctypes.data,
                                     out.ctypes.data, 0, ctypes.c_void_p(stream or None))
    if rc != SIM_OK:
        raise SimError(rc, sim_last_error(None))
    return out


def cr_amin_rho(u_values) -> np.ndarray:
    """Spectral radius of B_u^{-1} A_u for each u (Corollary A/B)."""
    us = np.ascontiguousarray(np.asarray(u_values, dtype=np.int32).ravel())
    out = np.zeros(us.shape[0], dtype=np.float64)
    rc = lib().sim_cr_amin_rho(int(us.shape[0]), us.ctypes.data, out.ctypes.data)
    if rc != SIM_OK:
        raise SimError(rc, sim_last_error(None))
    return out


def measure_peaks() -> dict:
    """Measured integer-issue and shared-memory-read ceilings of the current device
    (include/sim_peaks.h)."""
    out = np.zeros(4, dtype=np.float64)
    rc = lib().sim_measure_peaks(out.ctypes.data)
    if rc != 0:
        raise SimError(rc, "sim_measure_peaks failed")
    return {"int_ops_per_s": float(out[0]), "smem_bytes_per_s": float(out[1]), "int_ms": float(out[2]),
            "smem_ms": float(out[3])}
