"""ctypes wrapper of the CPU oracle (oracle/gs_oracle.c).

TEST INFRASTRUCTURE ONLY: imported by tests/, by __graft_entry__.smoke() and by
bench.py's cpu_baseline / reference leg, never by the product package.  The
functions follow the paper's definitions in fp64 (see gs_oracle.c for the
section / algorithm each one restates).
"""
import ctypes
import os

import numpy as np

from . import build as _build

_LIB = None


class Info(ctypes.Structure):
    _fields_ = [("lambda_", ctypes.c_double), ("capped", ctypes.c_int64), ("iters_run", ctypes.c_int32),
                ("pad", ctypes.c_int32), ("sum_p", ctypes.c_double), ("l1", ctypes.c_double)]

    def as_dict(self):
        return {"lambda": self.lambda_, "capped": self.capped, "iters_run": self.iters_run,
                "sum_p": self.sum_p, "l1": self.l1}


class OracleError(RuntimeError):
    def __init__(self, code):
        super().__init__(f"oracle returned status {code}")
        self.code = code


def lib():
    global _LIB
    if _LIB is None:
        path = _build.build()
        L = ctypes.CDLL(path)
        P = ctypes.POINTER
        L.gso_philox4x32_10.argtypes = [P(ctypes.c_uint32), P(ctypes.c_uint32), P(ctypes.c_uint32)]
        L.gso_word.argtypes = [ctypes.c_uint64, ctypes.c_uint32, ctypes.c_uint32, ctypes.c_int64]
        L.gso_word.restype = ctypes.c_uint32
        L.gso_uniform.argtypes = [ctypes.c_uint64, ctypes.c_uint32, ctypes.c_uint32, ctypes.c_int64]
        L.gso_uniform.restype = ctypes.c_double
        L.gso_uniforms.argtypes = [ctypes.c_uint64, ctypes.c_uint32, ctypes.c_uint32, ctypes.c_int64,
                                   ctypes.c_int64, ctypes.c_void_p]
        L.gso_greedy_lambda.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_double, ctypes.c_int, P(Info)]
        L.gso_greedy_pvector.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_double, ctypes.c_int,
                                         ctypes.c_void_p, P(ctypes.c_int32)]
        L.gso_probabilities.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_double, ctypes.c_int,
                                        ctypes.c_void_p, P(Info)]
        L.gso_sparsify.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_double, ctypes.c_int, ctypes.c_uint64,
                                   ctypes.c_uint32, ctypes.c_uint32, ctypes.c_int64, ctypes.c_void_p,
                                   ctypes.c_void_p, P(ctypes.c_int64), P(Info)]
        L.gso_segmented_sparsify.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int, ctypes.c_double,
                                             ctypes.c_int, ctypes.c_uint64, ctypes.c_uint32, ctypes.c_uint32,
                                             ctypes.c_void_p, ctypes.c_void_p, P(ctypes.c_int64), ctypes.c_void_p]
        L.gso_aggregate.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int, ctypes.c_int64,
                                    ctypes.c_void_p]
        for f in ("gso_greedy_lambda", "gso_greedy_pvector", "gso_probabilities", "gso_sparsify",
                  "gso_segmented_sparsify", "gso_aggregate"):
            getattr(L, f).restype = ctypes.c_int
        _LIB = L
    return _LIB


def _f32(g):
    g = np.ascontiguousarray(g, dtype=np.float32)
    return g, g.ctypes.data


def _check(rc):
    if rc != 0:
        raise OracleError(rc)


def philox4x32_10(ctr, key):
    c = (ctypes.c_uint32 * 4)(*[int(x) & 0xFFFFFFFF for x in ctr])
    k = (ctypes.c_uint32 * 2)(*[int(x) & 0xFFFFFFFF for x in key])
    o = (ctypes.c_uint32 * 4)()
    lib().gso_philox4x32_10(c, k, o)
    return [o[i] for i in range(4)]


def word(seed, step, worker, i):
    return lib().gso_word(seed, step, worker, i)


def uniforms(seed, step, worker, i0, n):
    u = np.empty(n, dtype=np.float64)
    lib().gso_uniforms(seed, step, worker, i0, n, u.ctypes.data)
    return u


def greedy_lambda(g, kappa, iters):
    g, ptr = _f32(g)
    info = Info()
    _check(lib().gso_greedy_lambda(ptr, g.size, kappa, iters, ctypes.byref(info)))
    return info.as_dict()


def greedy_pvector(g, kappa, iters):
    g, ptr = _f32(g)
    p = np.empty(g.size, dtype=np.float64)
    it = ctypes.c_int32()
    _check(lib().gso_greedy_pvector(ptr, g.size, kappa, iters, p.ctypes.data, ctypes.byref(it)))
    return p, it.value


def probabilities(g, kappa, iters):
    g, ptr = _f32(g)
    p = np.empty(g.size, dtype=np.float64)
    info = Info()
    _check(lib().gso_probabilities(ptr, g.size, kappa, iters, p.ctypes.data, ctypes.byref(info)))
    return p, info.as_dict()


def sparsify(g, kappa, iters, seed, step, worker, i0=0):
    g, ptr = _f32(g)
    idx = np.empty(g.size, dtype=np.int32)
    val = np.empty(g.size, dtype=np.float32)
    n = ctypes.c_int64()
    info = Info()
    _check(lib().gso_sparsify(ptr, g.size, kappa, iters, seed, step, worker, i0, idx.ctypes.data, val.ctypes.data,
                              ctypes.byref(n), ctypes.byref(info)))
    return idx[:n.value].copy(), val[:n.value].copy(), info.as_dict()


def segmented_sparsify(g, offsets, kappa, iters, seed, step, worker):
    g, ptr = _f32(g)
    off = np.ascontiguousarray(offsets, dtype=np.int64)
    L = off.size - 1
    idx = np.empty(g.size, dtype=np.int32)
    val = np.empty(g.size, dtype=np.float32)
    lam = np.empty(L, dtype=np.float64)
    n = ctypes.c_int64()
    _check(lib().gso_segmented_sparsify(ptr, off.ctypes.data, L, kappa, iters, seed, step, worker, idx.ctypes.data,
                                        val.ctypes.data, ctypes.byref(n), lam.ctypes.data))
    return idx[:n.value].copy(), val[:n.value].copy(), lam


def aggregate(idx_list, val_list, d):
    M = len(idx_list)
    idxs = [np.ascontiguousarray(x, dtype=np.int32) for x in idx_list]
    vals = [np.ascontiguousarray(x, dtype=np.float32) for x in val_list]
    ip = (ctypes.c_void_p * M)(*[x.ctypes.data for x in idxs])
    vp = (ctypes.c_void_p * M)(*[x.ctypes.data for x in vals])
    nn = np.array([x.size for x in idxs], dtype=np.int64)
    out = np.empty(d, dtype=np.float32)
    _check(lib().gso_aggregate(ip, vp, nn.ctypes.data, M, d, out.ctypes.data))
    return out
