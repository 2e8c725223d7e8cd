"""The oracle, as it stands, run in one process per logical CPU at once: the
all-cores figure of the benchmark's CPU-baseline leg (test infrastructure; no
arithmetic of the method lives here).

Processes are spawned, not forked: the calling process may already hold a GPU
context, and a forked child of one can hang.
"""
from __future__ import annotations

import multiprocessing as mp
import os
import time

_SAMPLE = None


def _init(sample):
    global _SAMPLE
    _SAMPLE = sample


def _work(job):
    """One process: the oracle over the whole sample (base rows in top-k mode,
    lookahead rows statistics only), repeated for budget_s; (rows/s, rows)."""
    from . import default
    k_max, budget_s = job
    o = default()
    rb, rr = _SAMPLE
    done, t0, elapsed = 0, time.perf_counter(), 0.0
    while elapsed < budget_s:
        o.row_stats(rb, k_max)
        o.row_stats(rr, 0)
        done += len(rb) + len(rr)
        elapsed = time.perf_counter() - t0
    return done / elapsed, done


def rows_per_second_all_cores(sample, k_max: int, budget_s: float, procs: int | None = None):
    """(sum of the processes' rows/s, rows scored in all, processes)."""
    procs = procs or os.cpu_count() or 1
    with mp.get_context("spawn").Pool(procs, initializer=_init, initargs=(sample,)) as pool:
        res = pool.map(_work, [(k_max, budget_s)] * procs)
    return sum(r[0] for r in res), sum(r[1] for r in res), procs
