"""Row-parallel driver for the float64 oracle (test infrastructure).

Runs ``grpo_objective.token_logprobs`` over row ranges of a large logits array on a
``spawn`` process pool; the array is shared with the workers through
``multiprocessing.shared_memory``. Rows are independent, so splitting them changes
no arithmetic. Only tests and bench.py's CPU legs use this module.
"""

from __future__ import annotations

import multiprocessing as mp
import os
from multiprocessing import shared_memory

import numpy as np

_STATE = {}


def _init(name, shape, dtype_str, np_dtype, ids):
    shm = shared_memory.SharedMemory(name=name)
    _STATE.update(shm=shm, raw=np.ndarray(shape, dtype=np_dtype, buffer=shm.buf), dtype=dtype_str, ids=ids)


def _rows(span):
    from oracle import grpo_objective as O

    lo, hi = span
    return lo, O.token_logprobs(_STATE["raw"][lo:hi], _STATE["dtype"], _STATE["ids"][lo:hi])


def token_logprobs_parallel(raw: np.ndarray, dtype: str, ids: np.ndarray, workers: int | None = None,
                            rows_per_job: int = 256):
    """(logp, H, lse) float64 for every row of ``raw`` (uint16 bf16 bits or float32)."""
    workers = workers or len(os.sched_getaffinity(0))
    n = raw.shape[0]
    shm = shared_memory.SharedMemory(create=True, size=max(1, raw.nbytes))
    try:
        np.ndarray(raw.shape, dtype=raw.dtype, buffer=shm.buf)[:] = raw
        spans = [(i, min(n, i + rows_per_job)) for i in range(0, n, rows_per_job)]
        logp = np.empty(n)
        H = np.empty(n)
        lse = np.empty(n)
        ctx = mp.get_context("spawn")
        with ctx.Pool(workers, initializer=_init,
                      initargs=(shm.name, raw.shape, dtype, raw.dtype, np.ascontiguousarray(ids))) as pool:
            for lo, (lp, h, ls) in pool.imap_unordered(_rows, spans):
                logp[lo:lo + len(lp)] = lp
                H[lo:lo + len(lp)] = h
                lse[lo:lo + len(lp)] = ls
    finally:
        shm.close()
        shm.unlink()
    return logp, H, lse
