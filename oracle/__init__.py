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


class DenseModel(ctypes.Structure):
    """Quantized model of the dense code (frequencies over 2^15)."""
    _fields_ = [("len_f", ctypes.c_uint32 * 31), ("len_c", ctypes.c_uint32 * 32), ("bit_f1", ctypes.c_uint32 * 30),
                ("val_f", ctypes.c_uint32 * 3), ("val_c", ctypes.c_uint32 * 4)]


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
        L.gso_average.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int, ctypes.c_int64,
                                  ctypes.c_void_p]
        L.gso_hybrid_encode.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_double, ctypes.c_void_p,
                                        ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p,
                                        P(ctypes.c_int64), ctypes.c_void_p, P(ctypes.c_int64), P(ctypes.c_double)]
        L.gso_hybrid_decode.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p,
                                        ctypes.c_int64, ctypes.c_double, ctypes.c_void_p, ctypes.c_void_p,
                                        P(ctypes.c_int64)]
        L.gso_ternary_bits.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64]
        L.gso_ternary_bits.restype = ctypes.c_double
        L.gso_comm_bits.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_double, ctypes.c_int]
        L.gso_comm_bits.restype = ctypes.c_double
        L.gso_closed_form_lambda.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_double, P(Info)]
        L.gso_probabilities_eps.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_double, ctypes.c_void_p,
                                            P(Info)]
        L.gso_sparsify_eps.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_double, ctypes.c_uint64,
                                       ctypes.c_uint32, ctypes.c_uint32, ctypes.c_int64, ctypes.c_void_p,
                                       ctypes.c_void_p, P(ctypes.c_int64), P(Info)]
        L.gso_dense_model_build.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                            ctypes.POINTER(DenseModel)]
        L.gso_dense_encode.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_void_p,
                                       ctypes.c_int64, P(ctypes.c_int64)]
        L.gso_dense_decode.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p]
        for f in ("gso_dense_model_build", "gso_dense_encode", "gso_dense_decode"):
            getattr(L, f).restype = ctypes.c_int
        for f in ("gso_closed_form_lambda", "gso_probabilities_eps", "gso_sparsify_eps", "gso_greedy_lambda", "gso_greedy_pvector", "gso_probabilities", "gso_sparsify",
                  "gso_segmented_sparsify", "gso_aggregate", "gso_average", "gso_hybrid_encode", "gso_hybrid_decode"):
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


def average(idx_list, val_list, d):
    """Algorithm 1 step 6: v = (1/M) sum_m Q(g^m) (fp32 sum in worker order,
    then one fp32 division by M)."""
    M = len(idx_list)
    idxs = [np.ascontiguousarray(x, dtype=np.int32) for x in idx_list]
    vals = [np.ascontiguousarray(x, dtype=np.float32) for x in val_list]
    ip = (ctypes.c_void_p * M)(*[x.ctypes.data for x in idxs])
    vp = (ctypes.c_void_p * M)(*[x.ctypes.data for x in vals])
    nn = np.array([x.size for x in idxs], dtype=np.int64)
    out = np.empty(d, dtype=np.float32)
    _check(lib().gso_average(ip, vp, nn.ctypes.data, M, d, out.ctypes.data))
    return out


def closed_form_lambda(g, eps):
    """Algorithm 2 (section 3.2): lambda of (7) for the smallest k of (6);
    `capped` is that k."""
    g, ptr = _f32(g)
    info = Info()
    _check(lib().gso_closed_form_lambda(ptr, g.size, float(eps), ctypes.byref(info)))
    return info.as_dict()


def probabilities_eps(g, eps):
    """p of Algorithm 2: 1 on the k largest magnitudes, lambda |g_i| elsewhere."""
    g, ptr = _f32(g)
    p = np.empty(g.size, dtype=np.float64)
    info = Info()
    _check(lib().gso_probabilities_eps(ptr, g.size, float(eps), p.ctypes.data, ctypes.byref(info)))
    return p, info.as_dict()


def sparsify_eps(g, eps, seed, step, worker, i0=0):
    """Q(g) with the p of Algorithm 2 and the same Philox draw as sparsify()."""
    g, ptr = _f32(g)
    idx = np.empty(g.size, dtype=np.int32)
    val = np.empty(g.size, dtype=np.float32)
    n = ctypes.c_int64()
    info = Info()
    _check(lib().gso_sparsify_eps(ptr, g.size, float(eps), seed, step, worker, i0, idx.ctypes.data,
                                  val.ctypes.data, ctypes.byref(n), ctypes.byref(info)))
    return idx[:n.value].copy(), val[:n.value].copy(), info.as_dict()


def hybrid_encode(g, lam, idx, val):
    """Section 3.3, eqs. (9)-(10): split the plain coding (idx, val) of Q(g)
    into Q_A (capped: index, value) and Q_B (codes 2 * index + [g_i < 0]);
    returns (qa_idx, qa_val, qb_code, 1 / lambda)."""
    g, gp = _f32(g)
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    val = np.ascontiguousarray(val, dtype=np.float32)
    n = idx.size
    qa_i = np.empty(max(n, 1), np.int32)
    qa_v = np.empty(max(n, 1), np.float32)
    qb = np.empty(max(n, 1), np.uint32)
    na, nb, inv = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_double()
    _check(lib().gso_hybrid_encode(gp, g.size, float(lam), idx.ctypes.data, val.ctypes.data, n,
                                   qa_i.ctypes.data, qa_v.ctypes.data, ctypes.byref(na), qb.ctypes.data,
                                   ctypes.byref(nb), ctypes.byref(inv)))
    return qa_i[:na.value].copy(), qa_v[:na.value].copy(), qb[:nb.value].copy(), inv.value


def hybrid_decode(qa_idx, qa_val, qb_code, inv_lambda):
    """Merge Q_A and Q_B back into the ascending (idx, val) lists."""
    qa_idx = np.ascontiguousarray(qa_idx, dtype=np.int32)
    qa_val = np.ascontiguousarray(qa_val, dtype=np.float32)
    qb_code = np.ascontiguousarray(qb_code, dtype=np.uint32)
    n = qa_idx.size + qb_code.size
    idx = np.empty(max(n, 1), np.int32)
    val = np.empty(max(n, 1), np.float32)
    nn = ctypes.c_int64()
    _check(lib().gso_hybrid_decode(qa_idx.ctypes.data, qa_val.ctypes.data, qa_idx.size, qb_code.ctypes.data,
                                   qb_code.size, float(inv_lambda), idx.ctypes.data, val.ctypes.data,
                                   ctypes.byref(nn)))
    return idx[:nn.value].copy(), val[:nn.value].copy()


def ternary_bits(d, n_neg, n_pos, n_cap):
    """Entropy-coding length of the dense code in {0, -1, +1, 2}^d (section 3.3)."""
    return lib().gso_ternary_bits(int(d), int(n_neg), int(n_pos), int(n_cap))


def comm_bits(d, n_capped, sum_p_uncapped, b=32):
    """One worker's summand of H(T, M) for one step (section 5)."""
    return lib().gso_comm_bits(int(d), int(n_capped), float(sum_p_uncapped), int(b))


def dense_model(d, n_pos, n_neg, n_cap):
    """Frequencies (over 2^15) of the dense code's models: bit lengths of the
    zero runs, each bit below the leading one, and the non-zero values."""
    m = DenseModel()
    _check(lib().gso_dense_model_build(int(d), int(n_pos), int(n_neg), int(n_cap), ctypes.byref(m)))
    return {"len_f": np.array(m.len_f, np.int64), "len_c": np.array(m.len_c, np.int64),
            "bit_f1": np.array(m.bit_f1, np.int64), "val_f": np.array(m.val_f, np.int64),
            "val_c": np.array(m.val_c, np.int64)}


def dense_encode(qt, log2_k=9):
    """Section 3.3: entropy code of q~ in {0, +1, -1, 2}^d (int8 values) as
    16-bit words (header, chunk directory, one rANS stream per chunk of
    2^log2_k non-zero symbols)."""
    qt = np.ascontiguousarray(qt, dtype=np.int8)
    n = ctypes.c_int64()
    _check(lib().gso_dense_encode(qt.ctypes.data, qt.size, int(log2_k), None, 0, ctypes.byref(n)))
    out = np.empty(n.value, dtype=np.uint16)
    _check(lib().gso_dense_encode(qt.ctypes.data, qt.size, int(log2_k), out.ctypes.data, out.size,
                                  ctypes.byref(n)))
    return out


def dense_decode(words, d):
    """Inverse of dense_encode: q~ as int8 values."""
    words = np.ascontiguousarray(words, dtype=np.uint16)
    qt = np.empty(int(d), dtype=np.int8)
    _check(lib().gso_dense_decode(words.ctypes.data, words.size, int(d), qt.ctypes.data))
    return qt
