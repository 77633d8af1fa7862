"""CPU oracles of the paper's schedulers (A_max, A_min, H-SF).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import, call, link or execute anything in this package.  The CUDA path
(``paper_2508_14544_gb300``) shares no code with it and never falls back to it.

* ``literal``    - pure-Python transcription; checks eq. Constraint at every future step.
* ``plain``      - plain C (``plain.c``) with endpoint evaluation; also the timed CPU baseline.
* ``bruteforce`` - exact optimum over all non-preemptive schedules and over all orders of the
                   auxiliary random-permutation policy, for tiny instances.
"""
AMAX, AMIN, HSF = 0, 1, 2
