"""Python binding of libgs.so, the GB300 gradient-sparsification library.

The functions carry the C-ABI names of include/gs.h and only marshal
arguments: tensors become device pointers, shapes become sizes, the current
torch stream becomes the cudaStream_t.  Every step of the computation runs in
the library's CUDA kernels; there is no CPU fallback.  If libgs.so has not
been built the first call raises.

Build it with ``python -c "import __graft_entry__ as g; g.build()"`` (or
``python paper_1710_09854_gb300/build.py``).
"""
import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libgs.so")

(GS_OK, GS_ERR_INVALID_ARG, GS_ERR_CUDA, GS_ERR_CAPACITY, GS_ERR_NONFINITE, GS_ERR_TIMEOUT, GS_ERR_INTERNAL,
 GS_ERR_ABORTED) = range(8)
GS_DTYPE_F32, GS_DTYPE_BF16 = 0, 1
GS_OPT_FORCE_EXACT_SOLVE, GS_OPT_SAMPLE_SIZE, GS_OPT_KERNEL_TIMING, GS_OPT_STREAM_PATH, GS_OPT_SMALL_PATH = 1, 2, 3, 4, 5

# Symbols include/gs.h declares (checked by the tests).
EXPORTS = ("gs_status_string", "gs_last_error", "gs_version", "gs_sync_status", "gs_probabilities", "gs_probabilities_ex",
           "gs_sparsify", "gs_batched_sparsify", "gs_batched_sparsify_hybrid", "gs_probabilities_eps", "gs_batched_sparsify_eps", "gs_segmented_sparsify", "gs_segmented_sparsify_aggregate", "gs_sparse_aggregate",
           "gs_sparsify_aggregate", "gs_sparsify_average_sparsify", "gs_sparsify_noalloc", "gs_pipeline_host", "gs_logreg_grad", "gs_logreg_margins", "gs_row_sq_norms", "gs_sum_rows", "gs_sgd_step",
           "gs_dense_encode", "gs_dense_decode", "gs_random_words", "gs_selftest_timeout", "gs_set_option", "gs_kernel_count", "gs_kernel_name",
           "gs_kernel_times")


class GSError(RuntimeError):
    def __init__(self, code, where):
        self.code = code
        super().__init__(f"{where}: {status_string(code)}")


class Info(ctypes.Structure):
    """Mirror of gs_info (32 bytes)."""
    _fields_ = [("lambda_", ctypes.c_double), ("sum_p", ctypes.c_double), ("capped", ctypes.c_int64),
                ("iters_run", ctypes.c_int32), ("flags", ctypes.c_int32)]


INFO_BYTES = ctypes.sizeof(Info)
_LIB = None


def lib():
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"CUDA library not built: {LIB_PATH} is missing "
                               "(run `python -c \"import __graft_entry__ as g; g.build()\"`)")
        L = ctypes.CDLL(LIB_PATH)
        vp, i64, u64, u32, i32, dbl = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64, ctypes.c_uint32,
                                       ctypes.c_int, ctypes.c_double)
        sig = {
            "gs_status_string": ([i32], ctypes.c_char_p),
            "gs_version": ([], i32),
            "gs_last_error": ([], ctypes.c_char_p),
            "gs_sync_status": ([vp], i32),
            "gs_probabilities": ([vp, i64, dbl, i32, vp, vp], i32),
            "gs_probabilities_ex": ([vp, i64, dbl, i32, vp, vp, vp], i32),
            "gs_sparsify": ([vp, i64, dbl, i32, u64, u32, u32, vp, vp, vp, vp], i32),
            "gs_batched_sparsify": ([vp, i32, i32, i64, dbl, i32, u64, u32, u32, vp, vp, vp, i64, vp, vp], i32),
            "gs_dense_encode": ([vp, vp, vp, vp, i32, i64, i64, i32, vp, i64, vp, vp], i32),
            "gs_dense_decode": ([vp, vp, i32, i64, i64, vp, vp], i32),
            "gs_batched_sparsify_hybrid": ([vp, i32, i32, i64, dbl, i32, u64, u32, u32, vp, vp, vp, vp, vp, vp, i64,
                                            vp, vp], i32),
            "gs_probabilities_eps": ([vp, i64, dbl, vp, vp, vp], i32),
            "gs_batched_sparsify_eps": ([vp, i32, i32, i64, dbl, u64, u32, u32, vp, vp, vp, i64, vp, vp], i32),
            "gs_segmented_sparsify": ([vp, i32, i32, i64, vp, i32, dbl, i32, u64, u32, u32, vp, vp, vp, i64, vp, vp],
                                      i32),
            "gs_segmented_sparsify_aggregate": ([vp, i32, i32, i64, vp, i32, dbl, i32, u64, u32, u32, vp, vp, vp, i64,
                                                 vp, vp, vp], i32),
            "gs_sparse_aggregate": ([vp, vp, vp, i32, i64, vp, vp], i32),
            "gs_sparsify_aggregate": ([vp, i32, i32, i64, dbl, i32, u64, u32, u32, vp, vp, vp, i64, vp, vp, vp], i32),
            "gs_sparsify_average_sparsify": ([vp, i32, i32, i64, dbl, i32, u64, u32, u32, vp, vp, vp, i64, vp, dbl,
                                              i32, u32, vp, vp, vp, vp, vp], i32),
            "gs_sparsify_noalloc": ([vp, i64, dbl, i32, u64, u32, u32, vp, vp, vp, vp, vp, vp], i32),
            "gs_pipeline_host": ([vp, i32, i32, i64, dbl, i32, u64, u32, u32, vp, vp, vp, vp, i64, vp, vp, vp, vp],
                                 i32),
            "gs_random_words": ([u64, u32, u32, i64, i64, vp, vp], i32),
            "gs_selftest_timeout": ([i32, vp], i32),
            "gs_logreg_grad": ([vp, vp, i32, i32, vp, vp, i32, i32, ctypes.c_float, vp, vp, vp], i32),
            "gs_logreg_margins": ([vp, vp, i32, i32, vp, vp, vp], i32),
            "gs_row_sq_norms": ([vp, vp, i32, i64, vp, vp], i32),
            "gs_sum_rows": ([vp, i32, i64, vp, vp], i32),
            "gs_sgd_step": ([vp, vp, i64, ctypes.c_float, ctypes.c_float, ctypes.c_float, i32, vp, vp, i32, vp, vp],
                            i32),
            "gs_set_option": ([i32, i64], i32),
            "gs_kernel_count": ([], i32),
            "gs_kernel_name": ([i32], ctypes.c_char_p),
            "gs_kernel_times": ([vp, vp, i32], i32),
        }
        for name, (args, res) in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _LIB = L
    return _LIB


def status_string(code):
    return lib().gs_status_string(int(code)).decode()


def _check(rc, where):
    if rc != GS_OK:
        if rc == GS_ERR_CUDA:
            where = f"{where} [{lib().gs_last_error().decode()}]"
        raise GSError(rc, where)


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _ptr(t, name, dtypes=None):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    import torch
    cur = torch.cuda.current_device()
    if t.device.index is not None and t.device.index != cur:
        # The library launches on the current device: memory of another
        # device would be read through a pointer that is not valid there.
        raise ValueError(f"{name} is on {t.device} but the current CUDA device is cuda:{cur}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtypes is not None and t.dtype not in dtypes:
        raise ValueError(f"{name} has dtype {t.dtype}, expected one of {dtypes}")
    return t.data_ptr()


def _g_dtype(g):
    import torch
    if g.dtype == torch.float32:
        return GS_DTYPE_F32
    if g.dtype == torch.bfloat16:
        return GS_DTYPE_BF16
    raise ValueError(f"g must be float32 or bfloat16, got {g.dtype}")


def info_tensor(n, device="cuda"):
    """Device buffer for n gs_info records."""
    import torch
    return torch.zeros(n * INFO_BYTES, dtype=torch.uint8, device=device)


def decode_info(t):
    """gs_info records of a (device or host) buffer as a list of dicts."""
    raw = t.cpu().numpy().tobytes() if hasattr(t, "cpu") else bytes(t)
    n = len(raw) // INFO_BYTES
    out = []
    for k in range(n):
        r = Info.from_buffer_copy(raw[k * INFO_BYTES:(k + 1) * INFO_BYTES])
        out.append({"lambda": r.lambda_, "sum_p": r.sum_p, "capped": r.capped, "iters_run": r.iters_run,
                    "flags": r.flags})
    return out


def gs_version():
    return lib().gs_version()


def gs_sync_status(stream=None):
    return lib().gs_sync_status(_stream(stream))


def gs_set_option(option, value):
    _check(lib().gs_set_option(int(option), int(value)), "gs_set_option")


def gs_kernel_count():
    return lib().gs_kernel_count()


def gs_kernel_name(k):
    return lib().gs_kernel_name(int(k)).decode()


def gs_kernel_times():
    """{kernel name: (accumulated ms, launches)} since the previous read; resets."""
    n = gs_kernel_count()
    ms = (ctypes.c_double * n)()
    nl = (ctypes.c_int64 * n)()
    _check(lib().gs_kernel_times(ms, nl, n), "gs_kernel_times")
    return {gs_kernel_name(k): (ms[k], nl[k]) for k in range(n)}


def gs_logreg_grad(X, y, w, batch, lam2, G, gsq, stream=None):
    """Minibatch gradients of eq. (14) for M workers: X (N, d), y (N,), w (d,),
    batch (M, B) int32 row indices; G (M, d) and gsq (M,) are written."""
    import torch
    N, d = X.shape
    M, B = batch.shape
    if y.numel() != N or w.numel() != d or tuple(G.shape) != (M, d) or gsq.numel() != M:
        raise ValueError("shapes: X (N, d), y (N,), w (d,), batch (M, B), G (M, d), gsq (M,)")
    f32 = (torch.float32,)
    _check(lib().gs_logreg_grad(_ptr(X, "X", f32), _ptr(y, "y", f32), N, d, _ptr(w, "w", f32),
                                _ptr(batch, "batch", (torch.int32,)), M, B, float(lam2), _ptr(G, "G", f32),
                                _ptr(gsq, "gsq", f32), _stream(stream)), "gs_logreg_grad")


def gs_logreg_margins(X, y, w, margins, stream=None):
    import torch
    N, d = X.shape
    f32 = (torch.float32,)
    _check(lib().gs_logreg_margins(_ptr(X, "X", f32), _ptr(y, "y", f32), N, d, _ptr(w, "w", f32),
                                   _ptr(margins, "margins", f32), _stream(stream)), "gs_logreg_margins")


def gs_row_sq_norms(val, nnz, out, stream=None):
    """val (M, cap) fp32, nnz (M,) int32 -> out (M,) = sum of the first nnz[m] values squared."""
    import torch
    M, cap = val.shape
    _check(lib().gs_row_sq_norms(_ptr(val, "val", (torch.float32,)), _ptr(nnz, "nnz", (torch.int32,)), M, cap,
                                 _ptr(out, "out", (torch.float32,)), _stream(stream)), "gs_row_sq_norms")


def gs_sum_rows(G, v, stream=None):
    import torch
    M, d = G.shape
    _check(lib().gs_sum_rows(_ptr(G, "G", (torch.float32,)), M, d, _ptr(v, "v", (torch.float32,)),
                             _stream(stream)), "gs_sum_rows")


def gs_sgd_step(w, v, scale, eta0, T0, t, qsq, gsq, log=None, stream=None):
    import torch
    f32 = (torch.float32,)
    _check(lib().gs_sgd_step(_ptr(w, "w", f32), _ptr(v, "v", f32), w.numel(), float(scale), float(eta0), float(T0),
                             int(t), _ptr(qsq, "qsq", f32), _ptr(gsq, "gsq", f32), gsq.numel(),
                             _ptr(log, "log", f32), _stream(stream)), "gs_sgd_step")


def gs_selftest_timeout(kind, stream=None):
    """Launch the bounded-wait self-test (kind 0: mbarrier, 1: flag); the next
    gs_sync_status() returns GS_ERR_TIMEOUT."""
    _check(lib().gs_selftest_timeout(int(kind), _stream(stream)), "gs_selftest_timeout")


def gs_random_words(seed, step, worker, i0, out, stream=None):
    """out: int32 CUDA tensor receiving the words (bit patterns) of coordinates i0 .. i0 + out.numel() - 1."""
    import torch
    _check(lib().gs_random_words(int(seed), int(step), int(worker), int(i0), out.numel(),
                                 _ptr(out, "out", (torch.int32,)), _stream(stream)), "gs_random_words")


def gs_probabilities(g, kappa, iters, p, stream=None):
    import torch
    _check(lib().gs_probabilities(_ptr(g, "g", (torch.float32,)), g.numel(), float(kappa), int(iters),
                                  _ptr(p, "p", (torch.float32,)), _stream(stream)), "gs_probabilities")


def gs_probabilities_ex(g, kappa, iters, p, info=None, stream=None):
    import torch
    _check(lib().gs_probabilities_ex(_ptr(g, "g", (torch.float32,)), g.numel(), float(kappa), int(iters),
                                     _ptr(p, "p", (torch.float32,)), _ptr(info, "info"), _stream(stream)),
           "gs_probabilities_ex")


def gs_sparsify(g, kappa, iters, seed, step, worker, idx, val, nnz, stream=None):
    import torch
    if idx.numel() < g.numel() or val.numel() < g.numel():
        raise ValueError("idx / val need capacity d")
    _check(lib().gs_sparsify(_ptr(g, "g", (torch.float32,)), g.numel(), float(kappa), int(iters), int(seed),
                             int(step), int(worker), _ptr(idx, "idx", (torch.int32,)),
                             _ptr(val, "val", (torch.float32,)), _ptr(nnz, "nnz", (torch.int32,)), _stream(stream)),
           "gs_sparsify")


def gs_sparsify_noalloc(g, kappa, iters, seed, step, worker, idx, val, nnz, status, info=None, stream=None):
    """gs_sparsify on the library's static scratch (d <= 2^22): the call
    itself allocates no device memory.  `status` (one int32 on the device,
    required) receives the call's device-side status code: the only place
    such errors are reported for this call."""
    import torch
    if idx.numel() < g.numel() or val.numel() < g.numel():
        raise ValueError("idx / val need capacity d")
    L = lib()
    rc = L.gs_sparsify_noalloc(_ptr(g, "g", (torch.float32,)), g.numel(), float(kappa), int(iters), int(seed),
                               int(step), int(worker), _ptr(idx, "idx", (torch.int32,)),
                               _ptr(val, "val", (torch.float32,)), _ptr(nnz, "nnz", (torch.int32,)),
                               _ptr(info, "info"), _ptr(status, "status", (torch.int32,)), _stream(stream))
    if rc == GS_ERR_INVALID_ARG and L.gs_last_error():
        raise GSError(rc, f"gs_sparsify_noalloc [{L.gs_last_error().decode()}]")
    _check(rc, "gs_sparsify_noalloc")


def gs_batched_sparsify(g, kappa, iters, seed, step, worker0, idx, val, nnz, info=None, stream=None):
    """g: (M, d) fp32/bf16; idx/val: (M, cap); nnz: (M,)."""
    import torch
    M, d = g.shape
    cap = idx.shape[1]
    if idx.shape[0] != M or tuple(val.shape) != tuple(idx.shape) or nnz.numel() != M:
        raise ValueError("idx / val must be (M, cap) and nnz (M,)")
    _check(lib().gs_batched_sparsify(_ptr(g, "g"), _g_dtype(g), M, d, float(kappa), int(iters), int(seed),
                                     int(step), int(worker0), _ptr(idx, "idx", (torch.int32,)),
                                     _ptr(val, "val", (torch.float32,)), _ptr(nnz, "nnz", (torch.int32,)), cap,
                                     _ptr(info, "info"), _stream(stream)), "gs_batched_sparsify")


def gs_batched_sparsify_hybrid(g, kappa, iters, seed, step, worker0, qa_idx, qa_val, qb_code, n_a, n_b, inv_lam,
                               info=None, stream=None):
    """g: (M, d) fp32/bf16; qa_idx/qa_val/qb_code: (M, cap) int32/fp32/uint32
    (or int32 viewed as codes); n_a/n_b: (M,) int32; inv_lam: (M,) fp32."""
    import torch
    M, d = g.shape
    cap = qa_idx.shape[1]
    if tuple(qa_val.shape) != tuple(qa_idx.shape) or tuple(qb_code.shape) != tuple(qa_idx.shape):
        raise ValueError("qa_idx, qa_val and qb_code must be (M, cap)")
    if qa_idx.shape[0] != M or n_a.numel() != M or n_b.numel() != M or inv_lam.numel() != M:
        raise ValueError("one row / count / 1-over-lambda per worker")
    codes = (torch.int32, torch.uint32) if hasattr(torch, "uint32") else (torch.int32,)
    _check(lib().gs_batched_sparsify_hybrid(_ptr(g, "g"), _g_dtype(g), M, d, float(kappa), int(iters), int(seed),
                                            int(step), int(worker0), _ptr(qa_idx, "qa_idx", (torch.int32,)),
                                            _ptr(qa_val, "qa_val", (torch.float32,)), _ptr(qb_code, "qb_code", codes),
                                            _ptr(n_a, "n_a", (torch.int32,)), _ptr(n_b, "n_b", (torch.int32,)),
                                            _ptr(inv_lam, "inv_lam", (torch.float32,)), cap, _ptr(info, "info"),
                                            _stream(stream)), "gs_batched_sparsify_hybrid")


def gs_dense_encode(qa_idx, qb_code, n_a, n_b, d, log2_k, words, n_words, stream=None):
    """The dense code of section 3.3 from the hybrid lists (M, cap) of
    gs_batched_sparsify_hybrid: words (M, word_cap) int16 (16-bit words) and
    n_words (M,) int64 receive each worker's code and its length."""
    import torch
    M, cap = qa_idx.shape
    if tuple(qb_code.shape) != (M, cap) or n_a.numel() != M or n_b.numel() != M or words.shape[0] != M:
        raise ValueError("qa_idx, qb_code (M, cap); n_a, n_b (M,); words (M, word_cap)")
    codes = (torch.int32, torch.uint32) if hasattr(torch, "uint32") else (torch.int32,)
    w16 = (torch.int16, torch.uint16) if hasattr(torch, "uint16") else (torch.int16,)
    _check(lib().gs_dense_encode(_ptr(qa_idx, "qa_idx", (torch.int32,)), _ptr(qb_code, "qb_code", codes),
                                 _ptr(n_a, "n_a", (torch.int32,)), _ptr(n_b, "n_b", (torch.int32,)), M, int(d), cap,
                                 int(log2_k), _ptr(words, "words", w16), words.shape[1],
                                 _ptr(n_words, "n_words", (torch.int64,)), _stream(stream)), "gs_dense_encode")


def gs_dense_decode(words, n_words, d, qt, stream=None):
    """Decode codes written by gs_dense_encode into qt (M, d) int8 (q~ rows)."""
    import torch
    M, word_cap = words.shape
    if n_words.numel() != M or tuple(qt.shape) != (M, int(d)):
        raise ValueError("words (M, word_cap), n_words (M,), qt (M, d)")
    w16 = (torch.int16, torch.uint16) if hasattr(torch, "uint16") else (torch.int16,)
    _check(lib().gs_dense_decode(_ptr(words, "words", w16), _ptr(n_words, "n_words", (torch.int64,)), M, int(d),
                                 word_cap, _ptr(qt, "qt", (torch.int8,)), _stream(stream)), "gs_dense_decode")


def gs_probabilities_eps(g, eps, p, info=None, stream=None):
    """p of Algorithm 2 (variance budget eps) for one fp32 gradient."""
    import torch
    _check(lib().gs_probabilities_eps(_ptr(g, "g", (torch.float32,)), g.numel(), float(eps),
                                      _ptr(p, "p", (torch.float32,)), _ptr(info, "info"), _stream(stream)),
           "gs_probabilities_eps")


def gs_batched_sparsify_eps(g, eps, seed, step, worker0, idx, val, nnz, info=None, stream=None):
    """gs_batched_sparsify with lambda from Algorithm 2 (variance budget eps)."""
    import torch
    M, d = g.shape
    cap = idx.shape[1]
    if idx.shape[0] != M or tuple(val.shape) != tuple(idx.shape) or nnz.numel() != M:
        raise ValueError("idx / val must be (M, cap) and nnz (M,)")
    _check(lib().gs_batched_sparsify_eps(_ptr(g, "g"), _g_dtype(g), M, d, float(eps), int(seed), int(step),
                                         int(worker0), _ptr(idx, "idx", (torch.int32,)),
                                         _ptr(val, "val", (torch.float32,)), _ptr(nnz, "nnz", (torch.int32,)), cap,
                                         _ptr(info, "info"), _stream(stream)), "gs_batched_sparsify_eps")


def gs_segmented_sparsify(g, seg_offsets, kappa, iters, seed, step, worker0, idx, val, nnz, info=None, stream=None):
    """g: (M, d); seg_offsets: host sequence of L+1 offsets (0 .. d)."""
    import torch
    M, d = g.shape
    cap = idx.shape[1]
    off = np.ascontiguousarray(seg_offsets, dtype=np.int64)
    if idx.shape[0] != M or tuple(val.shape) != tuple(idx.shape) or nnz.numel() != M:
        raise ValueError("idx / val must be (M, cap) and nnz (M,)")
    _check(lib().gs_segmented_sparsify(_ptr(g, "g"), _g_dtype(g), M, d, off.ctypes.data, off.size - 1,
                                       float(kappa), int(iters), int(seed), int(step), int(worker0),
                                       _ptr(idx, "idx", (torch.int32,)), _ptr(val, "val", (torch.float32,)),
                                       _ptr(nnz, "nnz", (torch.int32,)), cap, _ptr(info, "info"), _stream(stream)),
           "gs_segmented_sparsify")


def gs_segmented_sparsify_aggregate(g, seg_offsets, kappa, iters, seed, step, worker0, idx, val, nnz, out,
                                    info=None, stream=None):
    """gs_segmented_sparsify of g (M, d) plus the dense sum of the M rows into out (d,)."""
    import torch
    M, d = g.shape
    cap = idx.shape[1]
    off = np.ascontiguousarray(seg_offsets, dtype=np.int64)
    if idx.shape[0] != M or tuple(val.shape) != tuple(idx.shape) or nnz.numel() != M or out.numel() != d:
        raise ValueError("idx / val must be (M, cap), nnz (M,), out (d,)")
    _check(lib().gs_segmented_sparsify_aggregate(_ptr(g, "g"), _g_dtype(g), M, d, off.ctypes.data, off.size - 1,
                                                 float(kappa), int(iters), int(seed), int(step), int(worker0),
                                                 _ptr(idx, "idx", (torch.int32,)), _ptr(val, "val", (torch.float32,)),
                                                 _ptr(nnz, "nnz", (torch.int32,)), cap, _ptr(info, "info"),
                                                 _ptr(out, "out", (torch.float32,)), _stream(stream)),
           "gs_segmented_sparsify_aggregate")


def gs_sparse_aggregate(idx_list, val_list, nnz, d, out, stream=None):
    """idx_list / val_list: M device tensors (or rows of (M, cap) tensors)."""
    import torch
    M = len(idx_list)
    ip = (ctypes.c_void_p * M)(*[_ptr(x, "idx", (torch.int32,)) for x in idx_list])
    vp = (ctypes.c_void_p * M)(*[_ptr(x, "val", (torch.float32,)) for x in val_list])
    _check(lib().gs_sparse_aggregate(ip, vp, _ptr(nnz, "nnz", (torch.int32,)), M, int(d),
                                     _ptr(out, "out", (torch.float32,)), _stream(stream)), "gs_sparse_aggregate")


def gs_sparsify_aggregate(g, kappa, iters, seed, step, worker0, idx, val, nnz, out, info=None, stream=None):
    """gs_batched_sparsify of g (M, d) into idx / val / nnz plus the dense sum into out (d,)."""
    import torch
    M, d = g.shape
    cap = idx.shape[1]
    if idx.shape[0] != M or tuple(val.shape) != tuple(idx.shape) or nnz.numel() != M or out.numel() != d:
        raise ValueError("idx / val must be (M, cap), nnz (M,), out (d,)")
    _check(lib().gs_sparsify_aggregate(_ptr(g, "g"), _g_dtype(g), M, d, float(kappa), int(iters), int(seed),
                                       int(step), int(worker0), _ptr(idx, "idx", (torch.int32,)),
                                       _ptr(val, "val", (torch.float32,)), _ptr(nnz, "nnz", (torch.int32,)), cap,
                                       _ptr(info, "info"), _ptr(out, "out", (torch.float32,)), _stream(stream)),
           "gs_sparsify_aggregate")


def gs_sparsify_average_sparsify(g, kappa, iters, seed, step, worker0, idx, val, nnz, v, kappa_v, iters_v,
                                 worker_v, idx_v, val_v, nnz_v, info=None, stream=None):
    """Algorithm 1 steps 4-7: Q(g^m) of g (M, d) into idx / val / nnz, their
    average into v (d,), and Q(v) (density kappa_v, iters_v rescalings, worker
    id worker_v) into idx_v / val_v (d,) and nnz_v (1,)."""
    import torch
    M, d = g.shape
    cap = idx.shape[1]
    if idx.shape[0] != M or tuple(val.shape) != tuple(idx.shape) or nnz.numel() != M or v.numel() != d:
        raise ValueError("idx / val must be (M, cap), nnz (M,), v (d,)")
    if idx_v.numel() < d or val_v.numel() < d or nnz_v.numel() != 1:
        raise ValueError("idx_v / val_v need capacity d and nnz_v one entry")
    _check(lib().gs_sparsify_average_sparsify(_ptr(g, "g"), _g_dtype(g), M, d, float(kappa), int(iters), int(seed),
                                              int(step), int(worker0), _ptr(idx, "idx", (torch.int32,)),
                                              _ptr(val, "val", (torch.float32,)), _ptr(nnz, "nnz", (torch.int32,)),
                                              cap, _ptr(v, "v", (torch.float32,)), float(kappa_v), int(iters_v),
                                              int(worker_v), _ptr(idx_v, "idx_v", (torch.int32,)),
                                              _ptr(val_v, "val_v", (torch.float32,)),
                                              _ptr(nnz_v, "nnz_v", (torch.int32,)), _ptr(info, "info"),
                                              _stream(stream)), "gs_sparsify_average_sparsify")


def gs_pipeline_host(g_host, kappa, iters, seed, step, worker0, g_dev, idx, val, nnz, out, out_host, nnz_host,
                     stream=None):
    """g_host: (M, d) pinned CPU tensor; out_host (d,) / nnz_host (M,) pinned CPU tensors."""
    import torch
    M, d = g_host.shape
    cap = idx.shape[1]
    for t, n in ((g_host, "g_host"), (out_host, "out_host"), (nnz_host, "nnz_host")):
        if t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{n} must be a contiguous host tensor")
    _check(lib().gs_pipeline_host(g_host.data_ptr(), _g_dtype(g_host), M, d, float(kappa), int(iters), int(seed),
                                  int(step), int(worker0), _ptr(g_dev, "g_dev"), _ptr(idx, "idx", (torch.int32,)),
                                  _ptr(val, "val", (torch.float32,)), _ptr(nnz, "nnz", (torch.int32,)), cap,
                                  _ptr(out, "out", (torch.float32,)), out_host.data_ptr(), nnz_host.data_ptr(),
                                  _stream(stream)), "gs_pipeline_host")
