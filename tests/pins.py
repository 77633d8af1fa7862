"""Checks of an oracle implementation against values the paper and the mathematics fix.

``check_all(sim)`` runs every pin against ``sim(policy, M, a, s, l, u, o, rank=None) -> dict`` (a
dict with the result fields and 'completion'; ``rank`` is A_r's permutation) and returns the list of
failures.  The pin tests call it on
both oracles; the mutation tests call it on deliberately broken copies of the literal oracle and
expect failures.
"""
from __future__ import annotations

import json
from pathlib import Path

GOLDEN = Path(__file__).resolve().parent / "golden"
AMAX, AMIN, HSF, AR, AELL = 0, 1, 2, 3, 4
POL = {"AMAX": AMAX, "AMIN": AMIN, "HSF": HSF, "AR": AR, "AELL": AELL}
FIELDS = ("total_latency", "makespan", "peak_memory", "evictions", "steps", "request_steps")


def load(name: str) -> dict:
    return json.loads((GOLDEN / name).read_text())


def wave_cases():
    """Identical jobs with exact intervals (l = u = o), n = k*W, M in [k(s+o), k(s+o)+s]:
    nothing can start while a wave runs (a job started d steps into a wave would need
    s + o - d more tokens of room at the wave's last step, and the slack is at most s < s+o-d),
    so the jobs run in W waves of k, each lasting o steps.  Closed form from the model of
    Section 2: TEL = k*o*W(W+1)/2, makespan W*o, peak k(s+o), steps W*o, request steps n*o."""
    out = []
    for (k, W, s, o, r) in [(1, 3, 1, 1, 0), (2, 3, 1, 4, 1), (3, 4, 2, 5, 2), (5, 2, 3, 2, 0),
                            (4, 5, 1, 3, 1), (2, 6, 4, 1, 3), (7, 3, 2, 6, 2)]:
        n = k * W
        M = k * (s + o) + r
        exp = dict(total_latency=k * o * W * (W + 1) // 2, makespan=W * o, peak_memory=k * (s + o),
                   evictions=0, steps=W * o, request_steps=n * o)
        out.append(((k, W, s, o, r), M, [0] * n, [s] * n, [o] * n, [o] * n, [o] * n, exp))
    return out


def amax_wave_cases():
    """A_max on identical jobs whose true length o is below the upper bound u, M = k(s+u):
    A_max projects every job to u, so it starts k jobs at a time and nothing else fits until
    the wave completes (after o steps) -- Example 1 generalised.  TEL = sum over waves w of
    |wave_w| * (w+1) * o, with waves of k and a last partial wave."""
    out = []
    for (k, n, s, o, u) in [(2, 5, 1, 1, 4), (3, 7, 2, 2, 5), (1, 4, 3, 3, 3), (4, 9, 1, 2, 9)]:
        M = k * (s + u)
        tel, w, left = 0, 0, n
        while left > 0:
            m = min(k, left)
            tel += m * (w + 1) * o
            left -= m
            w += 1
        exp = dict(total_latency=tel, makespan=w * o, evictions=0, steps=w * o, request_steps=n * o,
                   peak_memory=min(k, n) * (s + o))
        out.append(((k, n, s, o, u), M, [0] * n, [s] * n, [o] * n, [u] * n, [o] * n, exp))
    return out


def aell_wave_cases():
    """A_ell on the two-point family (Algorithm promote_l): n = k*W requests with equal s, each of
    length l or u (estimate l first), M = k(s+l) and M - k_u(s+u) <= s with k_u = floor(M/(s+u)).
    First pass: FIFO waves of k, wave w runs steps w*l .. (w+1)*l - 1 and fills M exactly at its
    last step, so nothing else starts meanwhile; its short requests complete at (w+1)*l, its long
    ones have used up l unfinished and are promoted at step (w+1)*l behind all first-pass
    requests.  Second pass, from W*l: the N_u long requests (estimate u = o) in promotion order,
    waves of k_u lasting u steps (the slack below s+1 again lets nothing start inside a wave).
    TEL = sum_short (w+1)*l + sum over long waves j of |wave_j| * (W*l + (j+1)*u); evictions =
    N_u; request steps = n*l + N_u*u; steps = makespan = W*l + ceil(N_u/k_u)*u; peak = M."""
    out = []
    for (k, W, s, l, u, pattern) in [(4, 2, 1, 2, 5, "SLLSSLSL"), (2, 3, 3, 3, 9, "LSSLLS"),
                                     (3, 3, 2, 4, 7, "SSLLSLSLL"), (4, 3, 1, 2, 5, "LLLLSSSSLSLS"),
                                     (2, 2, 1, 3, 3, "SSSS")]:
        n = k * W
        assert len(pattern) == n
        M = k * (s + l)
        ku = M // (s + u)
        assert ku >= 1 and M - ku * (s + u) <= s
        o = [l if c == "S" else u for c in pattern]
        tel, longs = 0, []
        for w in range(W):
            for i in range(w * k, (w + 1) * k):
                if o[i] == l:
                    tel += (w + 1) * l
                else:
                    longs.append(i)
        nu = len(longs)
        nw = -(-nu // ku)
        for j in range(nw):
            tel += min(ku, nu - j * ku) * (W * l + (j + 1) * u)
        span = W * l + nw * u
        exp = dict(total_latency=tel, makespan=span, peak_memory=M, evictions=nu, steps=span,
                   request_steps=n * l + nu * u)
        out.append(((k, W, s, l, u, pattern), M, [0] * n, [s] * n, [l] * n, [u] * n, o, exp))
    return out


def tie_vectors():
    """(seed, k, expected high 32 bits of SplitMix64 output k) from the published vectors."""
    out = []
    for v in load("splitmix64.json")["vectors"]:
        outs = [int(x, 16) for x in v["outputs_hex"]] if "outputs_hex" in v else [int(x) for x in v["outputs"]]
        for k, z in enumerate(outs, start=1):
            out.append((int(v["seed"]), k, z >> 32))
    return out


def check_all(sim, tie_key=None) -> list:
    """Run every pin against ``sim``; ``tie_key(seed, t, i)`` (optional) is checked against the
    published SplitMix64 vectors and the tie keys listed in the hand traces."""
    fails = []

    def chk(tag, got, exp):
        for key, val in exp.items():
            if key == "completion_sorted":
                if sorted(got["completion"]) != val:
                    fails.append((tag, key, sorted(got["completion"]), val))
            elif key == "starts":
                continue
            elif got.get(key) != val:
                fails.append((tag, key, got.get(key), val))

    def run(tag, *args, rank=None, tie_seed=None):
        kw = {}
        if rank is not None:
            kw["rank"] = rank
        if tie_seed is not None:
            kw["tie_seed"] = tie_seed
        try:
            return sim(*args, **kw)
        except AssertionError as e:  # an internal invariant tripped
            fails.append((tag, "assertion", str(e), None))
            return None

    if tie_key is not None:
        for seed, k, hi in tie_vectors():
            got = tie_key(seed, 0, k - 1)
            if got != hi:
                fails.append((f"splitmix64/{seed}/{k}", "tie_key", got, hi))

    pe = load("paper_examples.json")
    ex = pe["example1"]
    for pname, exp in ex["expect"].items():
        r = run("example1/" + pname, POL[pname], ex["M"], ex["a"], ex["s"], ex["l"], ex["u"], ex["o"])
        if r is not None:
            chk("example1/" + pname, r, exp)
    d1 = pe["def1_example"]
    r = run("def1/HSF", HSF, d1["M"], d1["a"], d1["s"], d1["o"], d1["o"], d1["o"])
    if r is not None:
        chk("def1/HSF", r, d1["expect"]["HSF"])

    ht = load("hand_traces.json")
    for name, case in ht.items():
        if name.startswith("_"):
            continue
        r = run(name, POL[case["policy"]], case["M"], case["a"], case["s"], case["l"], case["u"], case["o"],
                rank=case.get("rank"), tie_seed=case.get("tie_seed"))
        if r is not None:
            chk(name, r, case["expect"])
        if tie_key is not None and "tie_keys" in case:
            for t, keys in case["tie_keys"].items():
                for i, want in enumerate(keys):
                    got = tie_key(case["tie_seed"], int(t), i)
                    if got != want:
                        fails.append((name, f"tie_key({t},{i})", got, want))

    for tag, M, a, s, l, u, o, exp in wave_cases():
        for p in (AMAX, AMIN, HSF):
            r = run(f"waves{tag}/{p}", p, M, a, s, l, u, o)
            if r is not None:
                chk(f"waves{tag}/{p}", r, exp)
    for tag, M, a, s, l, u, o, exp in amax_wave_cases():
        r = run(f"amaxwaves{tag}", AMAX, M, a, s, l, u, o)
        if r is not None:
            chk(f"amaxwaves{tag}", r, exp)
    for tag, M, a, s, l, u, o, exp in aell_wave_cases():
        r = run(f"aellwaves{tag}", AELL, M, a, s, l, u, o)
        if r is not None:
            chk(f"aellwaves{tag}", r, exp)
    # exact waves with l = u = o: A_r in index order and A_ell (no long request) are plain FIFO
    for tag, M, a, s, l, u, o, exp in wave_cases():
        r = run(f"waves{tag}/AR", AR, M, a, s, l, u, o, rank=list(range(len(o))))
        if r is not None:
            chk(f"waves{tag}/AR", r, exp)
        r = run(f"waves{tag}/AELL", AELL, M, a, s, l, u, o)
        if r is not None:
            chk(f"waves{tag}/AELL", r, exp)
    return fails
