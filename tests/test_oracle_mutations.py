"""Plant plausible mistakes in copies of the oracles (on the CPU) and check the pins catch each.

Every mutation below is a one-token slip of the kind the pins are meant to catch: a dropped +1 in
the memory of a step, an endpoint off by one, a reversed sort, the literal 'bound <- tokens'
refinement, the wrong length estimate, a completion one step early.  The mutated oracle must
fail at least one pin (paper example, hand trace, closed form) or trip an internal invariant.
"""
import ctypes
import importlib.util
import subprocess
import sys
import types
from pathlib import Path

import numpy as np
import pytest

from tests import pins

ROOT = Path(__file__).resolve().parent.parent
LIT = (ROOT / "oracle" / "literal.py").read_text()
PLAIN = (ROOT / "oracle" / "plain.c").read_text()

LIT_MUTATIONS = {
    "memory_without_plus_one": ("total += sj + (tp - p) + 1", "total += sj + (tp - p)"),
    "endpoint_one_late": ("e = start[j] + est_len(j) - 1", "e = start[j] + est_len(j)"),
    "new_endpoint_one_early": ("jobs.append((t, t + est_len(j) - 1, s[j]))", "jobs.append((t, t + est_len(j) - 2, s[j]))"),
    "evict_descending": ("order = sorted(active, key=lambda i: (otil[i], tie_key(tie_seed, t, i), i))",
                         "order = sorted(active, key=lambda i: (-otil[i], tie_key(tie_seed, t, i), i))"),
    "evict_ties_by_index": ('tie_seed: int = 0, evict_ties: str = "hash",', 'tie_seed: int = 0, evict_ties: str = "index",'),
    "evict_ties_descending": ("order = sorted(active, key=lambda i: (otil[i], tie_key(tie_seed, t, i), i))",
                              "order = sorted(active, key=lambda i: (otil[i], -tie_key(tie_seed, t, i), i))"),
    "tie_key_fixed_per_request": ("return splitmix64(seed & _MASK64, ((t << 32) | i) + 1) >> 32",
                                  "return splitmix64(seed & _MASK64, i + 1) >> 32"),
    "tie_key_low_half": ("return splitmix64(seed & _MASK64, ((t << 32) | i) + 1) >> 32",
                         "return splitmix64(seed & _MASK64, ((t << 32) | i) + 1) & 0xFFFFFFFF"),
    "splitmix_wrong_shift": ("z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK64",
                             "z = ((z ^ (z >> 28)) * 0x94D049BB133111EB) & _MASK64"),
    "refine_to_tokens": ("new_bound = max(otil[i], gen[i]) if refine == \"max\" else gen[i]",
                         "new_bound = gen[i]"),
    "admit_longest_first": ("            waiting.sort(key=lambda i: (key(i), i))", "            waiting.sort(key=lambda i: (-key(i), i))"),
    "amax_uses_lower": ("        if policy == AMAX:\n            return u[i]", "        if policy == AMAX:\n            return l[i]"),
    "hsf_uses_upper": ("        if policy in (HSF, AR):\n            return o[i]", "        if policy == AR:\n            return o[i]\n        if policy == HSF:\n            return u[i]"),
    "evict_trigger_without_plus_one": ("need = sum(s[i] + gen[i] + 1 for i in active)",
                                       "need = sum(s[i] + gen[i] for i in active)"),
    "completion_one_early": ("completion[i] = t + 1\n", "completion[i] = t\n"),
    "latency_from_start_zero": ("tel += t + 1 - a[i]", "tel += t - a[i]"),
    "evictee_waits": ("same_step: bool = True", "same_step: bool = False"),
    "peak_before_step": ("        mem = sum(s[i] + gen[i] for i in batch)", "        mem = sum(s[i] + gen[i] - 1 for i in batch)"),
    "aell_promotion_ahead_of_arrivals": ("qkey[i] = 2 * t + 1", "qkey[i] = 2 * t - 1"),
    "aell_keeps_lower_estimate": ("                    otil[i] = u[i]\n", "                    otil[i] = o[i] + 1\n"),
    "aell_promotes_one_step_late": ("                if gen[i] == otil[i]:", "                if gen[i] == otil[i] + 1:"),
    "ar_projects_upper": ("        if policy in (HSF, AR):\n            return o[i]", "        if policy == HSF:\n            return o[i]\n        if policy == AR:\n            return u[i]"),
    "ar_ignores_rank": ("        if policy == AR:\n            return rank[i]", "        if policy == AR:\n            return o[i]"),
}


def _load_literal(src: str) -> types.ModuleType:
    mod = types.ModuleType("literal_mutant")
    exec(compile(src, "literal_mutant.py", "exec"), mod.__dict__)
    return mod


def _literal_pins(mod) -> list:
    return pins.check_all(lambda p, M, a, s, l, u, o, rank=None, tie_seed=0:
                          mod.simulate(p, M, a, s, l, u, o, rank=rank, tie_seed=tie_seed), tie_key=mod.tie_key)


@pytest.mark.parametrize("name", sorted(LIT_MUTATIONS))
def test_literal_mutation_is_caught(name):
    old, new = LIT_MUTATIONS[name]
    assert LIT.count(old) == 1, f"mutation anchor not found once: {name}"
    mod = _load_literal(LIT.replace(old, new))
    assert _literal_pins(mod), f"mutation {name} passed every pin"


def test_unmutated_literal_passes():
    assert _literal_pins(_load_literal(LIT)) == []


PLAIN_MUTATIONS = {
    "sweep_ascending": ("return (a->e < b->e) - (a->e > b->e);", "return (a->e > b->e) - (a->e < b->e);"),
    "new_job_c_off_by_one": ("ep[base + nadm].c = s[i] - t + 1;", "ep[base + nadm].c = s[i] - t;"),
    "evict_need_no_plus_one": ("need += s[act[k]] + (t - start[act[k]]) + 1;", "need += s[act[k]] + (t - start[act[k]]);"),
    "no_clamp_for_amin": ("if (policy == O_AMIN && e < t) e = t;", "(void)0;"),
    "refine_to_tokens": ("if (g > otil[i]) otil[i] = (int32_t)g;", "otil[i] = (int32_t)g;"),
    "aell_promotion_key_even": ("qkey[i] = 2 * t + 1;", "qkey[i] = 2 * t;"),
    "aell_estimate_not_raised": ("                    otil[i] = u[i];\n", "                    otil[i] = o[i] + 1;\n"),
    "ar_key_is_length": ("#define QKEY(i) (policy == O_AR ? (uint32_t)rank[i]", "#define QKEY(i) (policy == O_AR ? (uint32_t)o[i]"),
    "evict_ties_by_index": ("ev[k].tie = evict_index ? 0u : oracle_tie_key(tie_seed, t, i);", "ev[k].tie = 0u;"),
    "tie_counter_without_plus_one": ("const uint64_t k = (((uint64_t)t << 32) | (uint32_t)i) + 1u;",
                                     "const uint64_t k = (((uint64_t)t << 32) | (uint32_t)i);"),
    "tie_compare_reversed": ("if (a->tie != b->tie) return (a->tie > b->tie) - (a->tie < b->tie);",
                             "if (a->tie != b->tie) return (a->tie < b->tie) - (a->tie > b->tie);"),
}


def _build_plain(src: str, tmp_path: Path):
    c = tmp_path / "mut.c"
    so = tmp_path / "libmut.so"
    c.write_text(src)
    subprocess.run(["gcc", "-O1", "-std=c11", "-D_GNU_SOURCE", "-shared", "-fPIC", "-o", str(so), str(c),
                    "-lpthread"], check=True)
    L = ctypes.CDLL(str(so))
    i32p = ctypes.POINTER(ctypes.c_int32)
    i64p = ctypes.POINTER(ctypes.c_int64)
    L.oracle_run_seeded.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int32, i32p, i32p, i32p, i32p, i32p,
                                    i32p, ctypes.c_uint64, ctypes.c_int, ctypes.c_int64, ctypes.c_void_p, i64p]
    L.oracle_tie_key.argtypes = [ctypes.c_uint64, ctypes.c_int64, ctypes.c_int32]
    L.oracle_tie_key.restype = ctypes.c_uint32
    from oracle.plain import RESULT_DTYPE, FIELDS

    def sim(p, M, a, s, l, u, o, rank=None, tie_seed=0):
        arrs = [np.ascontiguousarray(np.asarray(v, np.int32)) for v in (a, s, l, u, o)]
        rk = None if rank is None else np.ascontiguousarray(np.asarray(rank, np.int32))
        n = len(o)
        res = np.zeros(1, RESULT_DTYPE)
        comp = np.zeros(max(n, 1), np.int64)
        L.oracle_run_seeded(p, M, n, *[x.ctypes.data_as(i32p) for x in arrs],
                            rk.ctypes.data_as(i32p) if rk is not None else i32p(), tie_seed, 0, 0, res.ctypes.data,
                            comp.ctypes.data_as(i64p))
        out = {k: int(res[0][k]) for k in FIELDS}
        out["completion"] = comp[:n].tolist()
        return out

    sim.tie_key = lambda seed, t, i: int(L.oracle_tie_key(seed, t, i))
    return sim


@pytest.mark.parametrize("name", sorted(PLAIN_MUTATIONS))
def test_plain_mutation_is_caught(name, tmp_path):
    old, new = PLAIN_MUTATIONS[name]
    assert PLAIN.count(old) == 1, name
    sim = _build_plain(PLAIN.replace(old, new), tmp_path)
    assert pins.check_all(sim, tie_key=sim.tie_key), f"mutation {name} passed every pin"


def test_unmutated_plain_passes(tmp_path):
    sim = _build_plain(PLAIN, tmp_path)
    assert pins.check_all(sim, tie_key=sim.tie_key) == []
