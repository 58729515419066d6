"""Comparison of the CUDA path's outputs with the oracle's.

Tolerances (applied by every GPU parity test):
  p            relative 1e-6 (p = 0 exactly where g = 0)
  kept sets    identical, except coordinates whose draw u_i lies within 1e-6
               of p_i (counted and reported; expected to be ~0)
  values       relative 1e-5 on the common kept coordinates
  idx order    strictly ascending on both sides, compared exactly
  sparse sum   |gpu - oracle| <= 1e-5 * sum_m |Q_m[i]| (relative to the
               magnitude of the terms, since terms of both signs may cancel)
"""
import concurrent.futures as cf
import os

import numpy as np

import oracle

P_RTOL = 1e-6
V_RTOL = 1e-5
FLIP_BAND = 1e-6


def compare_probabilities(p_gpu, g_row, kappa, iters):
    p_ref, info = oracle.probabilities(g_row, kappa, iters)
    p_gpu = np.asarray(p_gpu, dtype=np.float64)
    zero = p_ref == 0
    assert np.all(p_gpu[zero] == 0), "p must be 0 exactly where g is 0"
    rel = np.abs(p_gpu[~zero] - p_ref[~zero]) / p_ref[~zero]
    worst = float(rel.max()) if rel.size else 0.0
    assert worst <= P_RTOL, f"p relative error {worst:.3g} > {P_RTOL}"
    return info, worst


def compare_sparse(idx, val, g_row, kappa, iters, seed, step, worker, i0=0, ref=None):
    """Check one worker's (idx, val) against the oracle; returns the number of
    boundary flips (coordinates kept on one side only, all within the band)."""
    idx = np.asarray(idx, dtype=np.int64)
    val = np.asarray(val, dtype=np.float32)
    if idx.size > 1:
        assert np.all(np.diff(idx) > 0), "indices must be strictly ascending"
    if ref is None:
        ri, rv, info = oracle.sparsify(g_row, kappa, iters, seed, step, worker, i0)
    else:
        ri, rv, info = ref
    ri = ri.astype(np.int64)
    if idx.size == ri.size and np.array_equal(idx, ri):
        # the usual case: identical kept sets (no sort needed)
        common, ia, ib = idx, np.arange(idx.size), np.arange(idx.size)
        only = np.empty(0, dtype=np.int64)
    else:
        common, ia, ib = np.intersect1d(idx, ri, assume_unique=True, return_indices=True)
        only = np.setdiff1d(np.union1d(idx, ri), common)
    lam = info["lambda"]
    for i in only:
        a = abs(float(g_row[i - i0]))
        p = min(lam * a, 1.0)
        u = float(oracle.uniforms(seed, step, worker, int(i), 1)[0])
        assert abs(u - p) < FLIP_BAND, f"coordinate {i}: kept on one side only, u={u!r} p={p!r}"
    if common.size:
        a, b = val[ia].astype(np.float64), rv[ib].astype(np.float64)
        rel = np.abs(a - b) / np.maximum(np.abs(b), 1e-300)
        worst = float(rel.max())
        assert worst <= V_RTOL, f"value relative error {worst:.3g} > {V_RTOL}"
    return int(only.size)


def compare_sum(out_gpu, idx_list, val_list, d):
    ref = oracle.aggregate(idx_list, val_list, d)
    mag = np.zeros(d, dtype=np.float64)
    for i, v in zip(idx_list, val_list):
        i = np.asarray(i, dtype=np.int64)
        assert i.size < 2 or np.all(np.diff(i) > 0), "oracle lists are strictly ascending"
        mag[i] += np.abs(np.asarray(v, dtype=np.float64))   # distinct indices within one list
    err = np.abs(np.asarray(out_gpu, dtype=np.float64) - ref.astype(np.float64))
    bad = err > V_RTOL * mag
    assert not bad.any(), f"sparse sum differs at {int(bad.sum())} coordinates"
    return ref


def oracle_rows(fn, rows, *args, threads=None, workers=None, **kw):
    """fn(rows[j], *args, worker=workers[j], **kw) for every row (workers
    defaults to 0, 1, ...), run on host threads (the oracle is plain C called
    through ctypes, which releases the interpreter lock, and keeps no state
    between calls).  Returns the results in row order."""
    n = len(rows)
    workers = list(range(n)) if workers is None else list(workers)
    threads = threads or min(n, os.cpu_count() or 1)
    with cf.ThreadPoolExecutor(max_workers=max(1, threads)) as ex:
        futs = [ex.submit(fn, rows[j], *args, worker=workers[j], **kw) for j in range(n)]
        return [f.result() for f in futs]
