"""Runs the oracle's selection over many rows in spawned worker processes (test helper).

The workers receive the pooled inputs and W_o once, at start-up, and select disjoint chunks
of rows; the result is the same {(h, i): RowSelection} that a single ress_select call over
all the rows returns (every row is independent).  The pool is spawned, never forked, so it
is safe to start after the test process has used the GPU; each worker runs one BLAS thread.
This module imports no torch, so workers start quickly.
"""
from __future__ import annotations

import os

import oracle as O

_STATE = {}


def _init(pooled, W_o, c_h, rounds, rho, variant):
    _STATE.update(pooled=pooled, W_o=W_o, c_h=c_h, rounds=rounds, rho=rho, variant=variant)


def _select(rows):
    s = _STATE
    return O.ress_select(s["pooled"], s["W_o"], s["c_h"], s["rounds"], s["rho"], rows=rows,
                         variant=s["variant"])


def select_rows(pooled, W_o, c_h, rounds, rho, rows, variant=O.RESS, workers=None, chunk=48):
    """Oracle selection of `rows` on `workers` spawned processes (default: every core)."""
    import multiprocessing as mp
    workers = workers or os.cpu_count() or 1
    saved = {k: os.environ.get(k) for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS",
                                            "MKL_NUM_THREADS")}
    for k in saved:
        os.environ[k] = "1"
    try:
        ctx = mp.get_context("spawn")
        with ctx.Pool(workers, initializer=_init,
                      initargs=(pooled, W_o, list(c_h), rounds, rho, variant)) as pool:
            chunks = [rows[k:k + chunk] for k in range(0, len(rows), chunk)]
            out = {}
            for part in pool.imap_unordered(_select, chunks):
                out.update(part)
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    return out
