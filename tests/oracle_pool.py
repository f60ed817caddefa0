"""Whole oracle steps in a pool of worker processes (test infrastructure).

The full-size parity tests need the fp64 oracle on every projected row of many steps.  One
oracle step spends most of its time in single-threaded numpy (softmax and entropy over the
full vocabulary), so independent steps run in separate processes.  Each worker draws the LM
head itself from its seed (``workloads.make_head``, deterministic), so only a step's hidden
states and mask cross the process boundary, and the result (``oracle.rpd_oracle.StepResult``:
per-position arrays) comes back.  The pool uses the ``spawn`` start method, which is safe
after the parent has initialised CUDA.
"""
from __future__ import annotations

import multiprocessing as mp
import os

import numpy as np

_HEAD = {}


def _bits(t):
    return t.contiguous().view(__import__("torch").int16).numpy().view(np.uint16)


def _init(V: int, d: int, seed: int, w_std: float, blas_threads: int):
    os.environ.setdefault("OPENBLAS_NUM_THREADS", str(blas_threads))
    import workloads as WL
    W, g = WL.make_head(V, d, seed, w_std=w_std)
    _HEAD["W"], _HEAD["g"] = _bits(W), _bits(g)


def _run(task):
    from oracle import rpd_oracle as O
    hidden_bits, mask, eps, tau, budget, rule = task
    return O.rpd_step(hidden_bits, mask, _HEAD["g"], _HEAD["W"], eps, tau, budget, rule)


def oracle_steps(V: int, d: int, seed: int, tasks, workers: int = 0, w_std: float = 0.02):
    """``tasks``: list of (hidden bits [K][N][d] uint16, mask [N] uint8, eps, tau, budget, rule)
    for a head drawn by ``make_head(V, d, seed, w_std)``; returns the oracle's StepResult of
    each, in order."""
    cores = os.cpu_count() or 1
    workers = workers or max(1, min(len(tasks), cores // 4, 6))
    ctx = mp.get_context("spawn")
    with ctx.Pool(workers, initializer=_init,
                  initargs=(V, d, seed, w_std, max(1, cores // workers))) as pool:
        return pool.map(_run, tasks, chunksize=1)
