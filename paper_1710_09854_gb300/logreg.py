"""The convex experiment of section 5.1 on the GPU: l2-regularised logistic
regression (eq. 14) trained by synchronous SGD over M simulated workers
(Algorithm 1).  Each step, every worker's minibatch gradient is either
sparsified by the library (Algorithm 3, `iters` rescalings, density budget
kappa) or sent dense (the baseline), the workers' vectors are summed, and the
step size is divided by the variance factor var = ||Q(g)||^2 / ||g||^2, as
section 5.1 prescribes for the sparsified SGD.

Every step runs in libgs.so's kernels (gs_logreg_grad, gs_sparsify_aggregate
or gs_sum_rows, gs_row_sq_norms, gs_sgd_step); the host only enqueues the
calls and, every `log_every` steps, evaluates the objective in fp64 from the
margins the device computes.  Minibatch indices are inputs, drawn by the
caller.
"""
import math

import numpy as np

from . import (gs_logreg_grad, gs_logreg_margins, gs_row_sq_norms, gs_sgd_step, gs_sparsify_aggregate, gs_sum_rows,
               gs_sync_status, status_string, GS_OK)

LN2 = math.log(2.0)


def objective_from_margins(margins, w, lam2):
    """Eq. (14) in fp64: mean_n log2(1 + exp(-margin_n)) + lam2 ||w||^2."""
    m = np.asarray(margins, dtype=np.float64)
    w = np.asarray(w, dtype=np.float64)
    return float(np.mean(np.logaddexp(0.0, -m)) / LN2 + lam2 * np.dot(w, w))


def optimum(X, y, lam2, tol=1e-13, max_iter=100):
    """min_w f(w) of eq. (14) by Newton's method with backtracking, in fp64 on
    the host (the reference point of the suboptimality curves)."""
    A = np.asarray(X, dtype=np.float64) * np.asarray(y, dtype=np.float64)[:, None]
    N, d = A.shape
    w = np.zeros(d)

    def f(w):
        return float(np.mean(np.logaddexp(0.0, -(A @ w))) / LN2 + lam2 * np.dot(w, w))

    fw = f(w)
    for _ in range(max_iter):
        z = A @ w
        s = 0.5 * (1.0 - np.tanh(0.5 * z))           # sigma(-z)
        g = -(A.T @ s) / (N * LN2) + 2.0 * lam2 * w
        h = s * (1.0 - s) / (N * LN2)
        H = (A.T * h) @ A + 2.0 * lam2 * np.eye(d)
        step = np.linalg.solve(H, g)
        dec = float(g @ step)
        if dec / 2.0 <= tol:
            break
        t = 1.0
        while True:
            wn = w - t * step
            fn = f(wn)
            if fn <= fw - 0.25 * t * dec or t < 1e-12:
                break
            t *= 0.5
        w, fw = wn, fn
    return fw, w


def smoothness(X, lam2):
    """max_n ||a_n||^2 / (4 ln 2) + 2 lam2: a bound on every sample loss's
    gradient Lipschitz constant (eq. (14) with log2)."""
    X = np.asarray(X, dtype=np.float64)
    return float(np.max(np.sum(X * X, axis=1)) / (4.0 * LN2) + 2.0 * lam2)


def train(X, y, batches, lam2, eta0, T0, kappa=None, iters=2, seed=0, log_every=None, stream=None):
    """Run len(batches) SGD steps from w = 0.

    X (N, d), y (N,): fp32 CUDA tensors; batches: (T, M, B) int32 CUDA tensor
    of row indices.  kappa None trains the dense baseline.  Returns a dict with
    the objective every `log_every` steps (and at the end), the run's var
    (section 5.1: the summed ||Q(g^m)||^2 over the summed ||g^m||^2), each
    step's (eta_t, var_t), the kept entries sent, and the final w (host)."""
    import torch
    N, d = X.shape
    T, M, B = batches.shape
    dev = X.device
    w = torch.zeros(d, dtype=torch.float32, device=dev)
    G = torch.empty((M, d), dtype=torch.float32, device=dev)
    v = torch.empty(d, dtype=torch.float32, device=dev)
    gsq = torch.empty((T, M), dtype=torch.float32, device=dev)
    qsq = torch.empty((T, M), dtype=torch.float32, device=dev)
    logs = torch.empty((T, 2), dtype=torch.float32, device=dev)
    kept = torch.zeros(T, dtype=torch.int64, device=dev)
    margins = torch.empty(N, dtype=torch.float32, device=dev)
    if kappa is not None:
        idx = torch.empty((M, d), dtype=torch.int32, device=dev)
        val = torch.empty((M, d), dtype=torch.float32, device=dev)
        nnz = torch.empty(M, dtype=torch.int32, device=dev)
    curve = []

    def log_point(t):
        gs_logreg_margins(X, y, w, margins, stream=stream)
        curve.append((t, objective_from_margins(margins.cpu().numpy(), w.cpu().numpy(), lam2)))

    log_point(0)
    for t in range(T):
        gs_logreg_grad(X, y, w, batches[t], lam2, G, gsq[t], stream=stream)
        if kappa is None:
            gs_sum_rows(G, v, stream=stream)
            q = gsq[t]
        else:
            gs_sparsify_aggregate(G, kappa, iters, seed, t, 0, idx, val, nnz, v, stream=stream)
            gs_row_sq_norms(val, nnz, qsq[t], stream=stream)
            kept[t] = nnz.sum()
            q = qsq[t]
        gs_sgd_step(w, v, 1.0 / M, eta0, T0, t, q, gsq[t], log=logs[t], stream=stream)
        if log_every and (t + 1) % log_every == 0 and t + 1 < T:
            log_point(t + 1)
    log_point(T)
    rc = gs_sync_status(stream)
    if rc != GS_OK:
        raise RuntimeError(f"device status after training: {status_string(rc)}")
    g2 = float(gsq.double().sum().item())
    q2 = float((gsq if kappa is None else qsq).double().sum().item())
    return {"curve": curve, "var": q2 / g2 if g2 > 0 else 1.0, "steps": T,
            "eta_var": logs.cpu().numpy(), "kept_total": int(kept.sum().item()) if kappa is not None else T * M * d,
            "w": w.cpu().numpy()}
