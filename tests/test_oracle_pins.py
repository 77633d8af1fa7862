"""Pins of both CPU oracles to values the paper prints or the model fixes (no GPU)."""
import pytest

from oracle import bruteforce as bf
from oracle import literal, plain
from tests import pins

SIMS = {
    "literal": lambda p, M, a, s, l, u, o, rank=None, tie_seed=0: literal.simulate(p, M, a, s, l, u, o, rank=rank,
                                                                                  tie_seed=tie_seed),
    "plain": lambda p, M, a, s, l, u, o, rank=None, tie_seed=0: plain.run(p, M, a, s, l, u, o, completions=True,
                                                                          rank=rank, tie_seed=tie_seed),
}
TIE_KEYS = {"literal": literal.tie_key, "plain": plain.tie_key}


@pytest.mark.parametrize("which", sorted(SIMS))
def test_all_pins(which):
    fails = pins.check_all(SIMS[which], tie_key=TIE_KEYS[which])
    assert not fails, fails


def test_def1_schedules_feasibility():
    """Example after Definition 1: I_1, I_2, I_3 are valid schedules under M=7; starting all four
    jobs together is not (otherwise I_3 could not be optimal)."""
    d = pins.load("paper_examples.json")["def1_example"]
    for name, sch in d["schedules"].items():
        assert literal.is_feasible_schedule(d["M"], d["s"], d["o"], sch["starts"]) == sch["feasible"], name


def test_def1_optimum_is_I3():
    d = pins.load("paper_examples.json")["def1_example"]
    i3 = d["schedules"]["I3"]["starts"]
    assert literal.schedule_tel(d["a"], d["o"], i3) == d["expect"]["OPT"]["total_latency"]
    assert bf.opt_exact(d["M"], d["a"], d["s"], d["o"]) == d["expect"]["OPT"]["total_latency"]
    # I_1 and I_2 are feasible but worse
    for name in ("I1", "I2"):
        assert literal.schedule_tel(d["a"], d["o"], d["schedules"][name]["starts"]) > 12


def test_def1_hsf_starts():
    d = pins.load("paper_examples.json")["def1_example"]
    tr = []
    r = literal.simulate(literal.HSF, d["M"], d["a"], d["s"], d["o"], d["o"], d["o"], trace=tr)
    starts = [None] * 4
    for rec in tr:
        for i in rec["admitted"]:
            starts[i] = rec["t"]
    assert starts == d["expect"]["HSF"]["starts"]
    assert r["completion"] == d["expect"]["HSF"]["completion"]


def test_example1_opt_and_amax_ratio():
    """Example 1: H-SF is optimal there (TEL 5) and A_max pays 9."""
    e = pins.load("paper_examples.json")["example1"]
    assert bf.opt_exact(e["M"], e["a"], e["s"], e["o"]) == 5


def test_validation_statuses():
    # l > o, o > u, s < 1, a < 0 -> INVAL; s + o > M -> INFEASIBLE; s + u > M only for A_max
    base = dict(M=10, a=[0], s=[1], l=[1], u=[2], o=[1])
    for key, val, st in [("l", [2], -1), ("u", [0], -1), ("s", [0], -1), ("a", [-1], -1),
                         ("o", [10], -2)]:
        c = dict(base)
        c[key] = val
        if key == "o":
            c["u"] = [10]
        for p in (0, 1, 2):
            assert literal.simulate(p, c["M"], c["a"], c["s"], c["l"], c["u"], c["o"])["status"] == st
            assert plain.run(p, c["M"], c["a"], c["s"], c["l"], c["u"], c["o"])["status"] == st
    # s + u > M: A_max infeasible, the others fine
    c = dict(base, u=[10])
    assert plain.run(0, c["M"], c["a"], c["s"], c["l"], c["u"], c["o"])["status"] == -2
    assert plain.run(1, c["M"], c["a"], c["s"], c["l"], c["u"], c["o"])["status"] == 0
    assert plain.run(2, c["M"], c["a"], c["s"], c["l"], c["u"], c["o"])["status"] == 0


def test_step_cap():
    """A cap of 3 processed batches on an instance that needs more stops with STEPCAP after 3."""
    M, a, s, l, u, o = 4, [0, 0], [1, 1], [3, 3], [3, 3], [3, 3]
    for p in (0, 1, 2):
        r1 = literal.simulate(p, M, a, s, l, u, o, step_cap=3)
        r2 = plain.run(p, M, a, s, l, u, o, step_cap=3)
        assert r1["status"] == r2["status"] == -3
        assert r1["steps"] == r2["steps"] == 3
        for k in pins.FIELDS:
            assert r1[k] == r2[k]


def test_empty_instance():
    for p in (0, 1, 2):
        r = plain.run(p, 10, [], [], [], [], [])
        assert r["status"] == 0 and r["steps"] == 0 and r["total_latency"] == 0
