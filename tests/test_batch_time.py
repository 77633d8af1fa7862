"""Latency in time units under a linear batch-time model (Section 6: each batch is timed by a linear
regression predictor; the paper prints no coefficients, so they are inputs), pinned on the CPU
oracles (no GPU).

A processed step t takes f(B_t) = c0 + c1 |B_t| + c2 mem(t) + c3 prefill(t); an idle step c_idle.
Both oracles keep the integer sums X0..X3 (over requests, of the features of the steps
a_i .. C_i - 1) and F2, F3 (feature totals): the literal one per request and per step, the plain
one by prefix sums.
"""
from fractions import Fraction

import numpy as np
import pytest

from oracle import literal, plain
from tests import pins

COEF = (0.7, 0.013, 1.1e-4, 3.3e-3, 0.25)


def _tri(W):
    return W * (W + 1) // 2


def test_wave_closed_forms():
    """Identical jobs with exact intervals run in W waves of k, each o steps long (the wave pins):
    every step of a wave has k jobs, memory k (s + g) at its g-th step, and its first step starts
    k prompts.  A job of wave w spans waves 0..w, so X0 = k o W(W+1)/2 = TEL,
    X1 = k^2 o W(W+1)/2, X2 = k^2 (s o + o(o+1)/2) W(W+1)/2, X3 = k^2 s W(W+1)/2,
    F2 = W k (s o + o(o+1)/2), F3 = n s."""
    for (k, W, s, o, r), M, a, ss, l, u, oo, exp in pins.wave_cases():
        want = [k * o * _tri(W), k * k * o * _tri(W), k * k * (s * o + o * (o + 1) // 2) * _tri(W),
                k * k * s * _tri(W), W * k * (s * o + o * (o + 1) // 2), k * W * s]
        for p in (0, 1, 2):
            r1 = literal.simulate(p, M, a, ss, l, u, oo)
            r2 = plain.run(p, M, a, ss, l, u, oo, time_sums=True)
            assert r1["time_sums"] == want, ((k, W, s, o), p)
            assert r2["time_sums"] == want, ((k, W, s, o), p)
            assert r1["time_sums"][0] == r1["total_latency"]


def test_idle_steps_count_only_in_the_makespan():
    """One request arriving at step 5 with s = 3, o = 2 (M = 10): steps 0..4 are idle, steps 5 and
    6 run it with memory 4 and 5; it starts (prefill 3) at 5 and completes at 7.  Latency in time
    units = f(step 5) + f(step 6); makespan = 5 c_idle + the same."""
    c0, c1, c2, c3, ci = COEF
    for p in (0, 1, 2):
        r1 = literal.simulate(p, 10, [5], [3], [2], [2], [2])
        r2 = plain.run(p, 10, [5], [3], [2], [2], [2], time_sums=True)
        assert r1["time_sums"] == r2["time_sums"] == [2, 2, 9, 3, 9, 3]
        tel, span = literal.batch_time(r1, COEF)
        assert tel == c0 * 2 + c1 * 2 + c2 * 9 + c3 * 3
        assert span == c0 * 2 + c1 * 2 + c2 * 9 + c3 * 3 + ci * 5
        assert tuple(plain.batch_time(r2["_res"], [r2["time_sums"]], COEF)[0]) == (tel, span)


def test_arrival_after_processed_steps():
    """H-SF, M = 10: request 0 (a 0, s 1, o 3) runs steps 0..2; request 1 (a 2, s 1, o 2) arrives at
    step 2, fits beside it, and runs steps 2..3.  Steps 0..3 have batch sizes 1, 1, 2, 1, memories
    2, 3, 6, 3 and prefill 1, 0, 1, 0.  Request 0 spans steps 0..2, request 1 steps 2..3:
    X = (3 + 2, 4 + 3, 11 + 9, 2 + 1) = (5, 7, 20, 3), F2 = 14, F3 = 2."""
    for p in (0, 1, 2):
        r1 = literal.simulate(p, 10, [0, 2], [1, 1], [3, 2], [3, 2], [3, 2])
        r2 = plain.run(p, 10, [0, 2], [1, 1], [3, 2], [3, 2], [3, 2], time_sums=True)
        assert r1["completion"] == [3, 4]
        assert r1["time_sums"] == r2["time_sums"] == [5, 7, 20, 3, 14, 2]


def test_unit_model_gives_steps():
    """c0 = c_idle = 1, the rest 0: every step takes one unit, so the latency in time units is the
    total latency in steps and the makespan the makespan."""
    rng = np.random.default_rng(17)
    for trial in range(60):
        n = int(rng.integers(1, 9))
        o = rng.integers(1, 9, n)
        l = np.array([rng.integers(1, x + 1) for x in o])
        u = o + rng.integers(0, 5, n)
        s = rng.integers(1, 5, n)
        a = rng.integers(0, 8, n)
        M = int(max(s + u) + rng.integers(0, 10))
        for p in (0, 1, 2, 4):
            r = literal.simulate(p, M, a, s, l, u, o, tie_seed=trial)
            assert literal.batch_time(r, (1, 0, 0, 0, 1)) == (float(r["total_latency"]), float(r["makespan"]))


def test_sums_equal_the_per_step_definition_in_exact_arithmetic():
    """With rational coefficients, c0 X0 + c1 X1 + c2 X2 + c3 X3 equals the sum over requests of the
    time of the steps in [a_i, C_i), each step's time computed from the literal trace."""
    rng = np.random.default_rng(23)
    cf = [Fraction(7, 10), Fraction(13, 1000), Fraction(11, 100000), Fraction(33, 10000)]
    for trial in range(40):
        n = int(rng.integers(1, 8))
        o = rng.integers(1, 8, n)
        l = np.array([rng.integers(1, x + 1) for x in o])
        u = o + rng.integers(0, 4, n)
        s = rng.integers(1, 4, n)
        a = rng.integers(0, 6, n)
        M = int(max(s + u) + rng.integers(0, 8))
        for p in (0, 1, 2):
            tr = []
            r = literal.simulate(p, M, a, s, l, u, o, tie_seed=trial, trace=tr)
            dur = {rec["t"]: cf[0] + cf[1] * len(rec["batch"]) + cf[2] * rec["mem"]
                   + cf[3] * sum(int(s[i]) for i in rec["admitted"]) for rec in tr}
            direct = sum(d for i in range(n) for t, d in dur.items() if a[i] <= t < r["completion"][i])
            x = r["time_sums"]
            assert direct == cf[0] * x[0] + cf[1] * x[1] + cf[2] * x[2] + cf[3] * x[3]


@pytest.mark.parametrize("p", [0, 1, 2, 3, 4])
def test_literal_equals_plain_sums_and_times(p):
    rng = np.random.default_rng(100 + p)
    for trial in range(150):
        n = int(rng.integers(1, 9))
        o = rng.integers(1, 9, n)
        l = np.array([rng.integers(1, x + 1) for x in o])
        u = o + rng.integers(0, 6, n)
        s = rng.integers(1, 5, n)
        a = rng.integers(0, 6, n)
        M = int(max(s + u) + rng.integers(0, 14))
        rank = list(rng.permutation(n)) if p == 3 else None
        r1 = literal.simulate(p, M, a, s, l, u, o, rank=rank, tie_seed=trial)
        r2 = plain.run(p, M, a, s, l, u, o, rank=rank, tie_seed=trial, time_sums=True)
        assert r1["time_sums"] == r2["time_sums"]
        coef = rng.uniform(0, 2, 5)
        assert tuple(plain.batch_time(r2["_res"], [r2["time_sums"]], coef)[0]) == literal.batch_time(r1, coef)


def test_unfinished_instance_has_no_time():
    r = plain.run(1, 10, [0, 0], [1, 1], [1, 1], [5, 5], [5, 5], step_cap=3, time_sums=True)
    assert r["status"] == -3 and r["time_sums"] == [0] * 6
    assert np.all(np.isnan(plain.batch_time(r["_res"], [r["time_sums"]], COEF)))


# ---- planted mistakes in the batch-time code of both oracles (on the CPU) ----------------------

def _time_pins_fail(run) -> bool:
    """True if `run(p, M, a, s, l, u, o) -> time_sums` misses a closed form or the idle pin."""
    for (k, W, s, o, r), M, a, ss, l, u, oo, exp in pins.wave_cases():
        want = [k * o * _tri(W), k * k * o * _tri(W), k * k * (s * o + o * (o + 1) // 2) * _tri(W),
                k * k * s * _tri(W), W * k * (s * o + o * (o + 1) // 2), k * W * s]
        if run(0, M, a, ss, l, u, oo) != want:
            return True
    return (run(2, 10, [5], [3], [2], [2], [2]) != [2, 2, 9, 3, 9, 3] or
            run(2, 10, [0, 2], [1, 1], [3, 2], [3, 2], [3, 2]) != [5, 7, 20, 3, 14, 2])


LIT_TIME_MUTATIONS = {
    "interval_includes_completion_step": ("if a[i] <= tt < completion[i]:", "if a[i] <= tt <= completion[i]:"),
    "interval_from_zero": ("if a[i] <= tt < completion[i]:", "if 0 <= tt < completion[i]:"),
    "prefill_of_whole_batch": ("step_log.append((t, len(batch), mem, sum(s[i] for i in admitted)))",
                               "step_log.append((t, len(batch), mem, sum(s[i] for i in batch)))"),
}

PLAIN_TIME_MUTATIONS = {
    "completion_adds_step_memory": ("xs[2] += ncomp * memsum;", "xs[2] += ncomp * mem;"),
    "arrival_keeps_prefill": ("            xs[3] -= pfsum;\n", "\n"),
    "memory_prefix_before_the_step": (
        "        memsum += mem;\n        xs[0] += ncomp * steps; /* prefixes up to C = t + 1 */\n"
        "        xs[1] += ncomp * rsteps;\n        xs[2] += ncomp * memsum;\n",
        "        xs[0] += ncomp * steps;\n        xs[1] += ncomp * rsteps;\n        xs[2] += ncomp * memsum;\n"
        "        memsum += mem;\n"),
}


@pytest.mark.parametrize("name", sorted(LIT_TIME_MUTATIONS))
def test_literal_time_mutation_is_caught(name):
    import types
    src = (pins.GOLDEN.parent.parent / "oracle" / "literal.py").read_text()
    old, new = LIT_TIME_MUTATIONS[name]
    assert src.count(old) == 1
    mod = types.ModuleType("literal_time_mutant")
    exec(compile(src.replace(old, new), "literal_time_mutant.py", "exec"), mod.__dict__)
    assert _time_pins_fail(lambda p, M, a, s, l, u, o: mod.simulate(p, M, a, s, l, u, o)["time_sums"])


@pytest.mark.parametrize("name", sorted(PLAIN_TIME_MUTATIONS))
def test_plain_time_mutation_is_caught(name, tmp_path):
    import ctypes
    import subprocess
    src = (pins.GOLDEN.parent.parent / "oracle" / "plain.c").read_text()
    old, new = PLAIN_TIME_MUTATIONS[name]
    assert src.count(old) == 1
    c, so = tmp_path / "mut.c", tmp_path / "libmut.so"
    c.write_text(src.replace(old, new))
    subprocess.run(["gcc", "-O1", "-std=c11", "-D_GNU_SOURCE", "-shared", "-fPIC", "-o", str(so), str(c),
                    "-lpthread", "-lm"], check=True)
    L = ctypes.CDLL(str(so))
    i32p, i64p = ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int64)
    L.oracle_run_full.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, i32p, i32p, i32p, i32p, i32p, i32p,
                                  ctypes.c_uint64, ctypes.c_int, ctypes.c_int64, ctypes.c_void_p, i64p, i64p]

    def run(p, M, a, s, l, u, o):
        arrs = [np.ascontiguousarray(np.asarray(v, np.int32)) for v in (a, s, l, u, o)]
        res = np.zeros(1, plain.RESULT_DTYPE)
        ts = np.zeros(6, np.int64)
        L.oracle_run_full(p, M, len(o), *[x.ctypes.data_as(i32p) for x in arrs], i32p(), 0, 0, 0, res.ctypes.data,
                          i64p(), ts.ctypes.data_as(i64p))
        return ts.tolist()

    assert _time_pins_fail(run)
