"""The fp64 oracle's paged attention over a whole batch, spread over the
host cores.

Each thread runs the oracle on its own subset of the sequences (the
oracle's ``seq_ids`` option: longest first, dealt round-robin so the
threads get similar work); ctypes releases the interpreter lock during the
C call, so the threads run at once.  The subsets' rows are merged into one
array; every row comes from exactly one oracle call, so the result is the
single call's result bit for bit (pinned on the CPU by
``tests/test_bench_ranks_cpu.py``).  Test infrastructure only.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np

import oracle


def host_threads(cap: int = 32) -> int:
    try:
        n = len(os.sched_getaffinity(0))
    except (AttributeError, OSError):
        n = os.cpu_count() or 1
    return max(1, min(cap, n))


def paged_attention(pool, n_pages, page_elems, bs, Hkv, d, q, table, lens, scale, seq_ids=None,
                    threads: int | None = None) -> np.ndarray:
    """fp64 [S, Hq, d]; rows outside ``seq_ids`` (when given) are NaN."""
    lens = np.ascontiguousarray(lens, dtype=np.int32)
    ids = np.arange(lens.size, dtype=np.int32) if seq_ids is None else np.asarray(seq_ids, np.int32)
    T = min(threads or host_threads(), max(1, ids.size))
    order = ids[np.argsort(-lens[ids].astype(np.int64), kind="stable")]
    subsets = [order[i::T] for i in range(T)]
    q = np.ascontiguousarray(q)
    table = np.ascontiguousarray(table, dtype=np.int32)

    def run(sub):
        return sub, oracle.paged_attention(pool, n_pages, page_elems, bs, Hkv, d, q, table, lens, scale,
                                           seq_ids=sub)

    out = np.full((q.shape[0], q.shape[1], d), np.nan, dtype=np.float64)
    with ThreadPoolExecutor(T) as ex:
        for sub, part in ex.map(run, subsets):
            out[sub] = part[sub]
    return out
