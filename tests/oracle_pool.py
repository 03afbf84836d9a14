"""A pool of oracle worker processes for the sampled-row parity tests.

The oracle is serial NumPy; on the long workloads (a 1080p chunk sees up to
244 800 keys) one head's 256 sampled rows take about a third of a second, so
every chunk and every head of the 1080p and windowed 1080p streams would take
minutes in one process.  The rows of different heads are independent, so the
tests hand each (chunk, batch, head) to a worker process.  Workers run the
unchanged oracle (`oracle.attention.softmax_attention`) on the exact bf16
input values, passed as their 16-bit patterns and widened to float64 here
(bf16 is the upper half of a float32, so the widening is exact).

The pool is started with `spawn` (a fresh interpreter per worker, nothing
inherited from a process that has touched the GPU) and with one BLAS thread
per worker.  Only the tests use this module.
"""
from __future__ import annotations

import atexit
import collections
import multiprocessing as mp
import os
from typing import Callable, Optional

import numpy as np

_POOL = None
_WORKERS = 0


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact float64 values of bfloat16 numbers given as 16-bit patterns."""
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def head_rows(task):
    """One head's sampled rows: (q_bits [R, d], k_bits [Lk, d], v_bits
    [Lk, d], scale) -> (o [R, d], lse [R]) from the oracle in float64."""
    from oracle import attention as OA
    q, k, v, scale = task
    return OA.softmax_attention(bf16_bits_to_f64(q), bf16_bits_to_f64(k),
                                bf16_bits_to_f64(v), scale)


def pool(workers: Optional[int] = None):
    """The shared pool (created on first use, closed at exit)."""
    global _POOL, _WORKERS
    if _POOL is None:
        n = workers or max(1, min(16, len(os.sched_getaffinity(0))))
        keys = ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS")
        saved = {k: os.environ.get(k) for k in keys}
        for k in keys:
            os.environ[k] = "1"
        try:
            _POOL = mp.get_context("spawn").Pool(n)
        finally:
            for k, v in saved.items():
                if v is None:
                    os.environ.pop(k, None)
                else:
                    os.environ[k] = v
        _WORKERS = n
        atexit.register(_close)
    return _POOL


def _close():
    global _POOL
    if _POOL is not None:
        _POOL.terminate()
        _POOL.join()
        _POOL = None


class Pending:
    """Submits head tasks and runs `done(key, (o, lse))` on each result in
    submission order, keeping at most 2 tasks per worker in flight so that
    the queued inputs stay bounded."""

    def __init__(self, done: Callable):
        self.p = pool()
        self.done = done
        self.q = collections.deque()

    def submit(self, key, task) -> None:
        self.q.append((key, self.p.apply_async(head_rows, (task,))))
        while len(self.q) > 2 * _WORKERS:
            self._pop()

    def _pop(self) -> None:
        key, res = self.q.popleft()
        self.done(key, res.get())

    def finish(self) -> None:
        while self.q:
            self._pop()
