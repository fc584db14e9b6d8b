"""Run the oracle's token-range functions in parallel worker processes.

The direction term C (Eq. gij_cij) is a sum over tokens, so a full-size
oracle loss splits into token ranges whose partial C matrices are added in a
fixed order.  Workers are started with the 'spawn' method (never forked from
a process that has touched the GPU) and read the inputs from .npy files
through memory maps.
"""
import multiprocessing as mp
import os
import tempfile

import numpy as np


def _direction_part(args):
    zpath, fpath, gate, t0, t1 = args
    import oracle

    z = np.load(zpath, mmap_mode="r")
    f = np.load(fpath, mmap_mode="r")
    return oracle.direction(np.ascontiguousarray(z[t0:t1]), np.ascontiguousarray(f[t0:t1]), gate)


def direction_parallel(z: np.ndarray, f: np.ndarray, gate: int, workers: int | None = None):
    T = z.shape[0]
    workers = workers or max(1, min(32, os.cpu_count() or 1))
    chunks = max(workers * 2, 1)
    step = (T + chunks - 1) // chunks
    with tempfile.TemporaryDirectory(dir="/tmp") as d:
        zp, fp = os.path.join(d, "z.npy"), os.path.join(d, "f.npy")
        np.save(zp, z)
        np.save(fp, f)
        jobs = [(zp, fp, gate, t0, min(T, t0 + step)) for t0 in range(0, T, step)]
        ctx = mp.get_context("spawn")
        with ctx.Pool(workers) as pool:
            parts = pool.map(_direction_part, jobs)
    C = np.zeros_like(parts[0])
    for p in parts:
        C += p
    return C
