"""Literal CPU oracle of the batched schedulers (A_max, A_min, H-SF, A_r, A_ell).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this module.  The CUDA path shares no code with it.

This is the slowest, most literal reading of the paper: it keeps the waiting set R_t and the active
set S_t as explicit Python lists, and checks the future-memory constraint at *every* step t' from t
to the last projected step (no endpoint shortcut).  Pure Python loops: small instances only.

Model (Section 2, "Batch Processing, Memory Constraint, and Cancellation of Requests"):
one worker with a KV cache of M tokens; a batch takes one unit of time; every member of the batch
generates one output token; a job's memory is its prompt size plus the tokens generated so far
(eq. constraintM); cancelling a job discards its tokens and returns it to the waiting set, its true
output length o_i unchanged.  TEL = sum over jobs of (completion step - arrival step) (eq. latency;
with all arrivals at 0 this is the paper's L_i = t + o_i of a job whose final start is t).

Readings of the text that this oracle fixes (each is also listed in the design notes):

* Memory timing ("W reading").  Step t processes batch B_t; each member's token count g goes up by
  one; the memory of step t is  sum_{i in B_t} (s_i + g_i)  with g taken after the step, and must
  be <= M.  A job started at step p with length L occupies steps p..p+L-1 (memory s+1 .. s+L) and
  completes at C = p + L.  Completed jobs free their memory before the next step.  This is eq.
  constraintM evaluated at the end of each batch.  It accepts both schedules I_1 and I_2 of the
  example after Definition 1 and makes I_3 optimal there (TEL 12), and reproduces Example 1.
* Future feasibility (eq. Constraint).  A candidate set U started at t is feasible with the active
  set S' iff for every step t' >= t:
      sum_{j in S' u U, t' <= e_j} (s_j + (t' - p_j) + 1) <= M,
  where p_j is the job's (last) start (t for members of U) and e_j = p_j + Lhat_j - 1 its last
  projected step.  Lhat is the policy's length estimate: o (H-SF, Section 3.1), u (A_max,
  Algorithm malb) or the running lower bound õ (A_min, Algorithm milb).  For an active A_min job
  that has already passed its estimate, e_j = max(p_j + õ_j - 1, t): it is known to be unfinished,
  so it is projected for at least the current step.  The check covers every t' >= t (as stated
  for A_max and H-SF), so if S' alone fails at some future step nothing is admitted.
* Admission order.  The eligible waiting set (arrived, not active, not done) is sorted by
  (key, request index) with key = u (A_max), õ (A_min) or o (H-SF); the policy admits the largest
  feasible *prefix* ("in order", Algorithm milb).  The paper's "break ties uniformly at random"
  becomes "smaller request index first": the workload generator draws the requests i.i.d., so
  the index order of requests that have not yet run is a uniformly random order that the policy
  has observed nothing about, and a fixed random order of such requests admits the same
  subsets, in law, as a fresh draw every step.
* A_min eviction (Algorithm milb / milbrevise).  If sum_{i in S_t} (s_i + g_i + 1) > M, sort S_t by
  õ_i ascending, ties "uniformly at random", and remove jobs one at a time until the rest fits.
  The random tie order is drawn afresh at every step: job i's tie key at step t is
  ``tie_key(seed, t, i)``, a counter-based draw (SplitMix64, below), and S_t is sorted by
  (õ_i, tie key, index).  The seed is an input (one per instance), so runs are reproducible.
  A fixed order such as the request index would not be a fair draw here: admission also takes
  ties in index order, so among active jobs of equal õ the lowest index started first and has
  generated the most tokens, and an index rule would always cancel the most advanced of them.
  Each removed job: eviction count + 1, õ_i <- max(õ_i, g_i) (the refinement never lowers a
  certified lower bound), g_i <- 0, back to the waiting set, and eligible in the same step's
  admission ("unprocessed or restartable requests", Section 4).  The max, the same-step
  eligibility and the tie rule are switchable for sensitivity studies (``refine``, ``same_step``,
  ``evict_ties="index"`` for the index order).
* A_r (Algorithm random, Appendix B).  The true lengths o, and a fixed random permutation given as
  ``rank`` (rank[i] = position of request i; the draw is an input, not made here).  Admission is
  the largest feasible prefix of the waiting set in (rank, index) order, as for the other
  policies.
* A_ell (Algorithm promote_l, Section 5 and Appendix).  The waiting set is a FIFO queue: a request
  enters it at its arrival step, and a promoted request re-enters it at the end at the step of its
  promotion (key 2 a_i for an arrival, 2 t + 1 for a promotion at step t, so promotions follow the
  arrivals of the same step; simultaneous promotions in index order).  The length estimate starts
  at l_i.  At the start of a step, an active request that has generated its estimate of tokens
  without finishing (it then has more than l_i tokens to go) is removed, its tokens discarded,
  its estimate set to u_i, and it is appended to the queue, eligible in the same step.  The text
  says "more than l tokens"; running a request past its estimate would use memory the feasibility
  check did not reserve, so the removal happens as soon as the estimate is used up ("as soon as
  the currently served request generates l tokens", Section 5).  Promotions count as evictions.
  The paper states A_ell for the two-point family o in {l, u}; with per-request intervals it uses
  each request's own l_i and u_i.  Like A_max it needs s_i + u_i <= M.
* Arrivals (an extension: the paper has all a_i = 0).  Request i is eligible from step a_i on;
  when nothing is active or eligible, time jumps to the next arrival.  Makespan = max C_i.
* Step cap.  A run that has processed ``step_cap`` batches without finishing stops with status
  STEPCAP.  Default cap: 64 * (n + sum_i o_i).
* Batch time (Section 6: the experiments time each batch with a linear regression predictor).
  The paper prints no coefficients, so the model is an input: a processed step t takes
  f(B_t) = c0 + c1 |B_t| + c2 mem(t) + c3 prefill(t), where mem(t) is the step's memory (its KV
  tokens) and prefill(t) the prompt tokens of the requests started at t; a step with nothing to
  run takes c_idle.  A request's latency in time units is the time of the steps a_i .. C_i - 1.
  Summed over the requests that latency is c0 X0 + c1 X1 + c2 X2 + c3 X3 with the integer sums
  X_k = sum_i sum_{t in [a_i, C_i), processed} feature_k(t) (no step inside a request's interval
  is idle), and the makespan in time units is c0 F0 + c1 F1 + c2 F2 + c3 F3 + c_idle F4 with the
  feature totals F of steps 0 .. makespan - 1 (F4 the idle steps).  ``batch_time`` evaluates both
  from the sums in that order, in IEEE double.
"""
from __future__ import annotations

from typing import Sequence

AMAX, AMIN, HSF, AR, AELL = 0, 1, 2, 3, 4
POLICY_NAMES = {AMAX: "A_max", AMIN: "A_min", HSF: "H-SF", AR: "A_r", AELL: "A_ell"}

OK, E_INVAL, E_INFEASIBLE, E_STEPCAP = 0, -1, -2, -3

_WAITING, _ACTIVE, _DONE = 0, 1, 2


_MASK64 = (1 << 64) - 1


def splitmix64(seed: int, k: int) -> int:
    """Output number k (k >= 1) of the SplitMix64 generator seeded with ``seed`` (Steele, Lea and
    Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014, with the finalizer of
    Vigna's public-domain splitmix64.c): the state after k steps is seed + k * 0x9E3779B97F4A7C15
    (mod 2^64), and the output is that state passed through two xor-shift-multiply rounds and a
    final xor-shift."""
    z = (seed + k * 0x9E3779B97F4A7C15) & _MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK64
    return z ^ (z >> 31)


def tie_key(seed: int, t: int, i: int) -> int:
    """Random tie key of request i at step t for A_min's eviction order: the high 32 bits of
    SplitMix64 output number (t * 2^32 + i) + 1.  One counter per (step, request), so every step
    draws a fresh, independent order of the tied jobs."""
    return splitmix64(seed & _MASK64, ((t << 32) | i) + 1) >> 32


def default_step_cap(o: Sequence[int]) -> int:
    return 64 * (len(o) + sum(int(x) for x in o))


def validate(policy: int, M: int, a, s, l, u, o, rank=None) -> int:
    """Per-instance input check: 1 <= l <= o <= u, s >= 1, a >= 0, rank >= 0 (A_r), s + o <= M
    (s + u <= M for A_max and A_ell)."""
    if policy not in POLICY_NAMES or (policy == AR and rank is None):
        return E_INVAL
    for i in range(len(o)):
        if s[i] < 1 or a[i] < 0 or l[i] < 1 or l[i] > o[i] or o[i] > u[i]:
            return E_INVAL
        if policy == AR and rank[i] < 0:
            return E_INVAL
    for i in range(len(o)):
        if s[i] + o[i] > M:
            return E_INFEASIBLE
        if policy in (AMAX, AELL) and s[i] + u[i] > M:
            return E_INFEASIBLE
    return OK


def _empty_result(status: int, n: int) -> dict:
    return dict(total_latency=0, makespan=0, peak_memory=0, evictions=0, steps=0,
                request_steps=0, status=status, completion=[0] * n, time_sums=[0] * 6)


def batch_time(res: dict, coef: Sequence[float]) -> tuple[float, float]:
    """(total latency, makespan) in time units under the linear batch-time model
    coef = (c0, c1, c2, c3, c_idle), from a result's ``time_sums`` = [X0, X1, X2, X3, F2, F3]
    (F0 = steps, F1 = request steps, F4 = makespan - steps), each a sum of products evaluated left
    to right in IEEE double; NaN for an instance that did not finish."""
    if res["status"] != OK:
        return float("nan"), float("nan")
    c0, c1, c2, c3, ci = (float(c) for c in coef)
    x0, x1, x2, x3, f2, f3 = (float(v) for v in res["time_sums"])
    tel = c0 * x0 + c1 * x1 + c2 * x2 + c3 * x3
    span = (c0 * float(res["steps"]) + c1 * float(res["request_steps"]) + c2 * f2 + c3 * f3
            + ci * float(res["makespan"] - res["steps"]))
    return tel, span


def simulate(policy: int, M: int, a, s, l, u, o, step_cap: int | None = None,
             refine: str = "max", same_step: bool = True, trace: list | None = None,
             rank: Sequence[int] | None = None, tie_seed: int = 0, evict_ties: str = "hash",
             admit_ties: str = "index") -> dict:
    """Run one instance; return the result record plus per-request completion steps.

    ``trace`` (optional list) receives one dict per processed step: t, the batch, the admitted
    and the evicted (A_min) or promoted (A_ell) request indices, and the step's memory.
    ``rank`` is A_r's permutation (rank[i] = position of request i), required for A_r only.
    ``tie_seed`` seeds A_min's random eviction ties (``evict_ties="hash"``, the paper's rule);
    ``evict_ties="index"`` breaks them by request index instead (sensitivity studies only).
    ``admit_ties="hash"`` (sensitivity studies only) orders the waiting set by (key, fresh random
    draw, index) at every step, the draw being ``tie_key(~tie_seed, t, i)``, instead of by
    (key, index).
    """
    if evict_ties not in ("hash", "index") or admit_ties not in ("hash", "index"):
        raise ValueError((evict_ties, admit_ties))
    n = len(o)
    a = [int(x) for x in a]
    s = [int(x) for x in s]
    l = [int(x) for x in l]
    u = [int(x) for x in u]
    o = [int(x) for x in o]
    rank = None if rank is None else [int(x) for x in rank]
    st = validate(policy, M, a, s, l, u, o, rank)
    if st != OK:
        return _empty_result(st, n)
    if n == 0:
        return _empty_result(OK, 0)
    cap = default_step_cap(o) if step_cap is None else int(step_cap)

    state = [_WAITING] * n
    start = [None] * n  # last start p_i
    gen = [0] * n  # tokens generated since the last start, g_i
    otil = list(l)  # õ_i: the running lower bound (A_min), the current estimate l_i or u_i (A_ell)
    qkey = [2 * x for x in a]  # A_ell queue position: 2 a_i on arrival, 2 t + 1 after a promotion
    completion = [0] * n

    tel = makespan = peak = evictions = steps = request_steps = 0
    status = OK
    step_log = []  # (t, |B_t|, mem(t), prefill(t)) of every processed step
    t = min(a)
    n_done = 0

    def est_len(i: int) -> int:
        if policy in (HSF, AR):
            return o[i]
        if policy == AMAX:
            return u[i]
        return otil[i]

    def key(i: int) -> int:
        if policy == AR:
            return rank[i]
        if policy == AELL:
            return qkey[i]
        return est_len(i)  # A_max, A_min, H-SF: the sort key is the length estimate

    def feasible(active: list, new: list) -> bool:
        """eq. Constraint at every step t' from t to the last projected step (literal)."""
        jobs = []  # (start, last projected step, prompt)
        for j in active:
            e = start[j] + est_len(j) - 1
            if policy == AMIN:
                e = max(e, t)
            jobs.append((start[j], e, s[j]))
        for j in new:
            jobs.append((t, t + est_len(j) - 1, s[j]))
        if not jobs:
            return True
        horizon = max(e for _, e, _ in jobs)
        for tp in range(t, horizon + 1):
            total = 0
            for p, e, sj in jobs:
                if tp <= e:
                    total += sj + (tp - p) + 1
            if total > M:
                return False
        return True

    while n_done < n:
        if steps >= cap:
            status = E_STEPCAP
            break
        waiting = [i for i in range(n) if state[i] == _WAITING and a[i] <= t]
        active = [i for i in range(n) if state[i] == _ACTIVE]
        if not waiting and not active:
            t = min(a[i] for i in range(n) if state[i] == _WAITING)
            continue

        evicted = []
        if policy == AMIN:
            need = sum(s[i] + gen[i] + 1 for i in active)
            if need > M:
                if evict_ties == "hash":
                    order = sorted(active, key=lambda i: (otil[i], tie_key(tie_seed, t, i), i))
                else:
                    order = sorted(active, key=lambda i: (otil[i], i))
                for i in order:
                    if need <= M:
                        break
                    need -= s[i] + gen[i] + 1
                    new_bound = max(otil[i], gen[i]) if refine == "max" else gen[i]
                    assert new_bound >= otil[i] or refine != "max"
                    otil[i] = new_bound
                    gen[i] = 0
                    start[i] = None
                    state[i] = _WAITING
                    evictions += 1
                    evicted.append(i)
                active = [i for i in active if state[i] == _ACTIVE]
                if same_step:
                    waiting = waiting + evicted
                    waiting = [i for i in range(n) if i in set(waiting)]

        if policy == AELL:
            # promote-l: a request that has used up its estimate without finishing leaves the
            # batch, loses its tokens, takes u_i as its estimate and goes to the end of the queue
            for i in active:
                if gen[i] == otil[i]:
                    otil[i] = u[i]
                    gen[i] = 0
                    start[i] = None
                    state[i] = _WAITING
                    qkey[i] = 2 * t + 1
                    evictions += 1
                    evicted.append(i)
            if evicted:
                active = [i for i in active if state[i] == _ACTIVE]
                waiting = waiting + evicted

        if admit_ties == "hash":
            waiting.sort(key=lambda i: (key(i), tie_key(~tie_seed & _MASK64, t, i), i))
        else:
            waiting.sort(key=lambda i: (key(i), i))
        admitted = []
        for i in waiting:
            if feasible(active, admitted + [i]):
                admitted.append(i)
            else:
                break
        for i in admitted:
            state[i] = _ACTIVE
            start[i] = t
            gen[i] = 0

        batch = active + admitted
        for i in batch:
            gen[i] += 1
        mem = sum(s[i] + gen[i] for i in batch)
        assert mem <= M, (t, mem, M)
        step_log.append((t, len(batch), mem, sum(s[i] for i in admitted)))
        peak = max(peak, mem)
        request_steps += len(batch)
        steps += 1
        finished = []
        for i in batch:
            if gen[i] == o[i]:
                state[i] = _DONE
                completion[i] = t + 1
                tel += t + 1 - a[i]
                makespan = max(makespan, t + 1)
                n_done += 1
                finished.append(i)
                assert completion[i] - start[i] == o[i]
        if policy == AMIN:
            for i in batch:
                assert otil[i] <= o[i]
        if policy == AELL:
            for i in batch:
                assert gen[i] <= otil[i]
        if trace is not None:
            trace.append(dict(t=t, batch=sorted(batch), admitted=list(admitted),
                              evicted=list(evicted), finished=sorted(finished), mem=mem))
        t += 1

    time_sums = [0] * 6
    if status == OK:
        for i in range(n):
            for (tt, nb, mm, pf) in step_log:
                if a[i] <= tt < completion[i]:
                    time_sums[0] += 1
                    time_sums[1] += nb
                    time_sums[2] += mm
                    time_sums[3] += pf
        time_sums[4] = sum(mm for (_, _, mm, _) in step_log)
        time_sums[5] = sum(pf for (_, _, _, pf) in step_log)
    return dict(total_latency=tel, makespan=makespan, peak_memory=peak, evictions=evictions,
                steps=steps, request_steps=request_steps, status=status, completion=completion,
                time_sums=time_sums)


def is_feasible_schedule(M: int, s: Sequence[int], o: Sequence[int], starts: Sequence[int]) -> bool:
    """Check a non-preemptive schedule (job i runs steps starts[i] .. starts[i]+o[i]-1) against
    eq. constraintM under the W reading: at every step the batch's memory sum (s_i + g_i), with g_i
    counted after the step, is at most M."""
    if not starts:
        return True
    end = max(p + oi for p, oi in zip(starts, o))
    for tp in range(min(starts), end):
        total = 0
        for p, si, oi in zip(starts, s, o):
            if p <= tp <= p + oi - 1:
                total += si + (tp - p) + 1
        if total > M:
            return False
    return True


def schedule_tel(a: Sequence[int], o: Sequence[int], starts: Sequence[int]) -> int:
    """TEL of a schedule given final starts (eq. latency): sum (p_i + o_i - a_i)."""
    return sum(p + oi - ai for p, oi, ai in zip(starts, o, a))
