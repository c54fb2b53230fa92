"""Process pool for the fp64 oracle in the full-size GPU tests.

The oracle's layers are independent (the method runs per layer, its state is
per layer), so a step's layers are scored in parallel.  Workers are started
with ``spawn`` (never forked from a process that holds a CUDA context) and
import only the oracle and numpy, one BLAS thread each.  Inputs travel as the
raw bf16 bits (uint16) and are widened exactly in the worker.
"""
from __future__ import annotations

import os

# one BLAS thread per worker process (set before numpy is imported there)
for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, "1")

import concurrent.futures as cf  # noqa: E402
import multiprocessing as mp  # noqa: E402

import numpy as np  # noqa: E402


def bf16_bits(t) -> np.ndarray:
    """The bits of a bf16 torch tensor as a uint16 array (no rounding)."""
    import torch
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def _widen(bits: np.ndarray) -> np.ndarray:
    """bf16 bits -> float64 (exact)."""
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def _layer_job(job):
    """One layer through the oracle: group score map (or the given one), then
    the selection; returns the output and the advanced layer state."""
    from oracle import starkv_oracle as O
    q, k, window, meta, cur_frame, budget, R, C, st, p, per_head, S = job
    if S is None:
        S = O.score_layer(_widen(q), _widen(k), window, p)
    sel = O.select_layer_per_head if per_head else O.select_layer
    out = sel(S, *meta, cur_frame, budget, R, C, st, p)
    out["S"] = S
    out["lp"] = S.shape[1]
    return out, st


def _init_worker(root):
    import sys
    if root not in sys.path:
        sys.path.insert(0, root)


class OraclePool:
    """``map(jobs)`` runs ``_layer_job`` over the jobs on spawned workers."""

    def __init__(self, workers: int | None = None):
        n = workers or min(16, os.cpu_count() or 1)
        root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
        self.ex = cf.ProcessPoolExecutor(max_workers=n, mp_context=mp.get_context("spawn"),
                                         initializer=_init_worker, initargs=(root,))

    def map(self, jobs):
        return list(self.ex.map(_layer_job, jobs))

    def close(self):
        self.ex.shutdown()


def layer_job(si, layer, wl, st, p, per_head=False, S=None):
    """The arguments of one layer's oracle run for sequence input ``si``."""
    import harness as H
    lay = si.layout[layer]
    meta = tuple(H.layer_meta(lay, f) for f in ("is_visual", "frame", "row", "col"))
    q = None if S is not None else bf16_bits(si.q[layer])
    k = None if S is not None else bf16_bits(si.k[layer])
    return (q, k, wl.window, meta, si.cur_frame, si.budget, wl.grid_rows, wl.grid_cols, st, p, per_head, S)
