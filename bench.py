"""Benchmark of the GB300 gradient-sparsification path.

One step = gs_batched_sparsify over M worker gradients + gs_sparse_aggregate
of the M sparse vectors (steps (1)-(6) of the path), on inputs resident in
HBM.  Default workload: M = 16 workers, d = 2^24 fp32, Student-t(3)
gradients with 1% zeros, kappa = 0.01, 3 greedy iterations.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gs|reference]
                  [--workload c1..c5] [--kappa K] [--dtype f32|bf16]

Under torchrun (N > 1) every rank runs its own replica of the workload on
its own GPU (weak scaling; the path has no cross-replica exchange) and rank 0
prints one JSON line with the whole-job throughput.  `--impl reference`
times the CPU oracle (the single-threaded C restatement of the paper) on a
bounded sample of the same workload, on the host cores.
"""
import argparse
import json
import os
import statistics
import subprocess
import tempfile
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads  # noqa: E402

METRIC = "sparsified coords/s and achieved HBM GB/s vs peak (d=2^24, M=16 workers)"
UNIT = "coords/s"
L2_BYTES = 129 * 1024 * 1024


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


# ---------------------------------------------------------------------------
# Distributed plumbing (one process per GPU; replicas only)
# ---------------------------------------------------------------------------
def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def init_dist(backend):
    import torch.distributed as dist
    ws, rank, _ = dist_env()
    if ws > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend, rank=rank, world_size=ws)
    return ws, rank


def barrier():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        dist.barrier()


def max_over_ranks(x, device=None):
    """Largest value of x over all ranks (x itself without a process group)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x, device=None):
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def job_throughput(units_per_rank, ms_max, n_ranks):
    """Whole-job units/s: all ranks' units over the slowest rank's time."""
    return units_per_rank * n_ranks / (ms_max / 1e3)


# ---------------------------------------------------------------------------
# Workload construction
# ---------------------------------------------------------------------------
def make_workload(name, kappa=None, dtype=None, rank=0, workers=None, dim=None):
    import dataclasses
    import torch
    w = {"c1": workloads.C1, "c2": workloads.C2, "c3": workloads.C3, "c4": workloads.C4, "c5": workloads.C5}[name]
    if workers or dim:
        if name == "c4":
            raise SystemExit("--workers / --dim do not apply to the layer-wise workload")
        w = dataclasses.replace(w, M=workers or w.M, d=dim or w.d,
                                name=f"{w.name}_reduced_M{workers or w.M}_d{dim or w.d}")
    kappa = w.kappa if kappa is None else kappa
    dtype = dtype or w.dtype
    off = None
    if name == "c1":
        g = workloads.device_c1(w.d, seed=w.data_seed + 1000 * rank)
    elif name == "c2":
        g = workloads.device_logreg(w.M, w.d, seed0=w.data_seed + 1000 * rank)
    elif name == "c3":
        g = workloads.device_student_t(w.M, w.d, seed0=w.data_seed + 1000 * rank)
    elif name == "c4":
        g, off = workloads.device_layerwise(w.M, seed0=w.data_seed + 1000 * rank)
    else:
        g = workloads.device_lognormal(w.M, w.d, seed0=w.data_seed + 1000 * rank)
    if dtype == "bf16":
        g = g.to(torch.bfloat16)
    torch.cuda.synchronize()
    return w, g, off, kappa, dtype


TIME_EVERY = 10   # the streaming pass of one step in ten carries CUDA events in the timed region


def algorithmic_bytes(M, d, esz, nnz_total):
    """Bytes the path must move at least (one read of g, the (idx, val) codes
    written and read back, the dense sum written)."""
    sparsify = M * d * esz + nnz_total * 8
    aggregate = nnz_total * 8 + d * 4
    return sparsify, aggregate


# ---------------------------------------------------------------------------
# Clock sampling during the timed region
# ---------------------------------------------------------------------------
class Clocks:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        # The raw samples go to $GS_CLOCKS_DIR (kept for inspection) or a
        # temporary directory; the summary goes into the JSON line.
        try:
            out_dir = os.environ.get("GS_CLOCKS_DIR") or tempfile.mkdtemp(prefix="gs_clocks_")
            os.makedirs(out_dir, exist_ok=True)
            self.path = os.path.join(out_dir, f"clocks_rank{self.gpu}.csv")
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.15)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.fh.close()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# ---------------------------------------------------------------------------
# The GPU arm
# ---------------------------------------------------------------------------
def run_gpu(args):
    import torch
    ws, rank = init_dist("nccl")
    _, _, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    import paper_1710_09854_gb300 as gs
    gs.lib()

    w, g, off, kappa, dtype = make_workload(args.workload, args.kappa, args.dtype, rank, args.workers, args.dim)
    M, d = g.shape
    esz = g.element_size()
    cap = d
    idx = torch.empty((M, cap), dtype=torch.int32, device=dev)
    val = torch.empty((M, cap), dtype=torch.float32, device=dev)
    nnz = torch.empty(M, dtype=torch.int32, device=dev)
    out = torch.empty(d, dtype=torch.float32, device=dev)
    idx_rows = [idx[m] for m in range(M)]
    val_rows = [val[m] for m in range(M)]
    stream = torch.cuda.current_stream(dev)

    def step(t):
        if off is None and not args.separate:
            gs.gs_sparsify_aggregate(g, kappa, w.iters, w.seed, t, 0, idx, val, nnz, out, stream=stream)
            return
        if off is None:
            gs.gs_batched_sparsify(g, kappa, w.iters, w.seed, t, 0, idx, val, nnz, stream=stream)
        elif not args.separate:
            gs.gs_segmented_sparsify_aggregate(g, off, kappa, w.iters, w.seed, t, 0, idx, val, nnz, out,
                                               stream=stream)
            return
        else:
            gs.gs_segmented_sparsify(g, off, kappa, w.iters, w.seed, t, 0, idx, val, nnz, stream=stream)
        gs.gs_sparse_aggregate(idx_rows, val_rows, nnz, d, out, stream=stream)

    for t in range(args.warmup):
        step(t)
    torch.cuda.synchronize()
    rc = gs.gs_sync_status(stream)
    if rc != gs.GS_OK:
        raise RuntimeError(f"device status after warm-up: {gs.status_string(rc)}")
    nnz_total = int(nnz.sum().item())

    # ---- timed region: exactly K steps, barrier + synchronize on both sides.
    # The streaming pass of every TIME_EVERY-th step is bracketed by events
    # (mode 2): events around a launch keep it from overlapping its
    # neighbours' programmatic launches, so timing every step would slow it.
    gs.gs_kernel_times()  # reset counters
    clocks = Clocks(local)
    clocks.start()
    barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for t in range(args.steps):
        gs.gs_set_option(gs.GS_OPT_KERNEL_TIMING, 2 if t % TIME_EVERY == 0 else 0)
        step(args.warmup + t)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop()
    ktimes = gs.gs_kernel_times()
    gs.gs_set_option(gs.GS_OPT_KERNEL_TIMING, 0)
    ms_local = e0.elapsed_time(e1) / args.steps
    ms = max_over_ranks(ms_local, dev)
    rc = gs.gs_sync_status(stream)
    if rc != gs.GS_OK:
        raise RuntimeError(f"device status after timing: {gs.status_string(rc)}")

    coords = M * d
    value = job_throughput(coords, ms, ws)
    b_sp, b_ag = algorithmic_bytes(M, d, esz, nnz_total)
    hbm, peak_kind = peaks()
    launches = int(sum(n for _, n in ktimes.values()))
    dom = max(ktimes.items(), key=lambda kv: kv[1][0])
    dom_name, (dom_ms, dom_n) = dom
    n_timed = (args.steps + TIME_EVERY - 1) // TIME_EVERY   # launches of the streaming pass with events
    per_launch_ms = dom_ms / max(n_timed, 1)
    # Algorithmic bytes of the dominant kernel per launch.
    kernel_bytes = {
        "k_stream": M * d * esz,                 # one read of g
        "k_stream_tma": M * d * esz,             # one read of g
        # the cluster path: one read of g, the codes written (and, for one
        # worker, the dense sum it writes itself)
        "k_small": M * d * esz + nnz_total * 8 + (d * 4 if M == 1 else 0),
        "k_small_sum": M * d // 8 + nnz_total * esz + d * 4,   # decision bits, kept g, dense sum
        "k_emit": nnz_total * 8,                 # the (idx, val) codes written
        "k_emit_sum": 2 * nnz_total * 8 + d * 4,  # codes written, codes read, dense sum written
        "k_tiles": nnz_total * 8 + d * 4,        # codes read, dense sum written
    }
    kb = kernel_bytes.get(dom_name, 0)
    achieved = kb / (per_launch_ms / 1e3) / 1e9 if kb else 0.0
    traffic = load_traffic(dom_name, w.name, dtype, kappa)
    roofline = {"kernel": dom_name, "bound": "hbm", "achieved": round(achieved, 1), "peak": hbm,
                "peak_kind": peak_kind, "unit": "GB/s", "frac": round(achieved / hbm, 4),
                "traffic": traffic, "algorithmic_bytes_per_launch": kb,
                "ms_per_launch": round(per_launch_ms, 4), "launches_timed": n_timed}
    pipe_gbs = (b_sp + b_ag) / (ms / 1e3) / 1e9
    # Per-kernel breakdown from a short run after the timed region with every
    # launch timed (those events keep each kernel from overlapping the next
    # one's launch, so these times add up to a little more than ms_per_step).
    n_bd = min(args.steps, 100)
    gs.gs_set_option(gs.GS_OPT_KERNEL_TIMING, 1)
    gs.gs_kernel_times()
    for t in range(n_bd):
        step(args.warmup + args.steps + t)
    torch.cuda.synchronize()
    bd = gs.gs_kernel_times()
    gs.gs_set_option(gs.GS_OPT_KERNEL_TIMING, 0)
    kernels = {k: {"ms_per_step": round(v[0] / n_bd, 4), "launches": v[1]} for k, v in bd.items() if v[1]}
    step_stats = per_step_stats(lambda t: step(args.warmup + args.steps + n_bd + t), n_bd, stream)

    # Sparsify alone (steps 1-5, no sum) against B_sparsify, on the same inputs.
    sp_only = None
    if off is None:
        for t in range(3):
            gs.gs_batched_sparsify(g, kappa, w.iters, w.seed, t, 0, idx, val, nnz, stream=stream)
        torch.cuda.synchronize()
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s0.record(stream)
        for t in range(n_bd):
            gs.gs_batched_sparsify(g, kappa, w.iters, w.seed, args.warmup + t, 0, idx, val, nnz, stream=stream)
        s1.record(stream)
        torch.cuda.synchronize()
        sp_ms = max_over_ranks(s0.elapsed_time(s1) / n_bd, dev)
        sp_gbs = b_sp / (sp_ms / 1e3) / 1e9
        sp_only = {"api": "gs_batched_sparsify", "steps": n_bd, "ms_per_step": round(sp_ms, 4),
                   "algorithmic_bytes": b_sp, "achieved": round(sp_gbs, 1), "peak": hbm,
                   "frac": round(sp_gbs / hbm, 4), "unit": "GB/s"}
        rc = gs.gs_sync_status(stream)
        if rc != gs.GS_OK:
            raise RuntimeError(f"device status after the sparsify-only run: {gs.status_string(rc)}")
    alg3 = run_alg3_state(gs, g, off, kappa, w, idx, val, nnz, stream)
    hybrid = run_hybrid(gs, g, kappa, w, args, dev, stream, n_bd, hbm) if off is None else None
    vbudget = run_variance_budget(gs, g, w, args, dev, stream, n_bd, hbm) if off is None else None
    resp = run_resparsify(gs, g, kappa, w, args, dev, stream, n_bd, hbm, ms) if off is None else None
    lr = run_lr_sgd(dev, stream) if (off is None and not args.no_lr) else None

    # ---- end to end through the host-buffer entry point
    e2e = None
    if not args.no_e2e and off is None:
        e2e = run_e2e(gs, g, kappa, w, args, dev, stream, ws)

    # ---- every configuration (GPU only), after the headline's own buffers are freed
    configs = None
    if not args.no_configs and args.workers is None and args.dim is None:
        del idx, val, idx_rows, val_rows, out
        torch.cuda.empty_cache()
        configs = run_configs(gs, args, dev, stream, hbm, rank)

    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": dtype, "data": "synthetic",
        "config": {"workload": w.name, "M": M, "d": d, "kappa": kappa, "iters": w.iters, "dtype": dtype,
                   "api": (("gs_segmented_sparsify + gs_sparse_aggregate" if args.separate else
                            "gs_segmented_sparsify_aggregate") if off is not None else
                           "gs_batched_sparsify + gs_sparse_aggregate" if args.separate else "gs_sparsify_aggregate"),
                   "parallelism": f"replicas{ws}", "l2": "inputs exceed L2 (%.2f GB of g per step)" % (M * d * esz / 1e9)},
        "hbm_gbs_pipeline": round(pipe_gbs, 1),
        "pipeline_roofline": {"bound": "hbm", "algorithmic_bytes": b_sp + b_ag, "achieved": round(pipe_gbs, 1),
                              "peak": hbm, "frac": round(pipe_gbs / hbm, 4), "unit": "GB/s"},
        "roofline": roofline,
        "sparsify_roofline": sp_only,
        "algorithm3": alg3,
        "hybrid_code": hybrid,
        "variance_budget": vbudget,
        "average_resparsify": resp,
        "lr_sgd": lr,
        "kernels": kernels, "kernels_steps": n_bd, "step_ms_stats": step_stats,
        "nnz_per_step": nnz_total,
        "gpu_launches": launches,
        "clocks": clk,
        "e2e": e2e,
        "configs": configs,
    }
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline_sample(g, off, kappa, w, budget_s=args.cpu_seconds)
    return result, rank


# Every configuration of the path, each timed with the call bench.py times
# for it: c1-c3 and c5 through gs_sparsify_aggregate, c4 through
# gs_segmented_sparsify_aggregate.
CONFIG_SWEEP = (("c1", None, None), ("c2", None, None), ("c3", None, None), ("c4", None, None),
                ("c5", 0.001, "f32"), ("c5", 0.01, "f32"), ("c5", 0.1, "f32"),
                ("c5", 0.001, "bf16"), ("c5", 0.01, "bf16"), ("c5", 0.1, "bf16"))


def per_step_stats(step, n, stream):
    """Median, p10 and p90 of n steps timed one by one (a pair of CUDA events
    around each step, which keeps a step's first launch from overlapping the
    previous step's last, so the median sits a little above ms_per_step)."""
    import torch
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    for t, (a, b) in enumerate(evs):
        a.record(stream)
        step(t)
        b.record(stream)
    torch.cuda.synchronize()
    xs = sorted(a.elapsed_time(b) for a, b in evs)
    q = lambda f: xs[min(len(xs) - 1, int(f * len(xs)))]
    return {"steps": n, "median_ms": round(q(0.5), 5), "p10_ms": round(q(0.1), 5), "p90_ms": round(q(0.9), 5)}


def run_configs(gs, args, dev, stream, hbm, rank):
    """One row per configuration: time per step of the fused call (steps
    1-6), coordinates/s, the whole step against its algorithmic bytes (one
    read of g, the kept pairs written and read back, the dense sum written)
    and the streaming kernel against its one read of g, both as fractions of
    the measured copy peak.  The step time comes from a loop with no events
    between launches; the streaming kernel's time from a second loop in which
    only that kernel carries events."""
    import torch
    rows = []
    for name, kappa_o, dtype_o in CONFIG_SWEEP:
        try:
            w, g, off, kappa, dtype = make_workload(name, kappa_o, dtype_o, rank)
            M, d = g.shape
            esz = g.element_size()
            idx = torch.empty((M, d), dtype=torch.int32, device=dev)
            val = torch.empty((M, d), dtype=torch.float32, device=dev)
            nnz = torch.empty(M, dtype=torch.int32, device=dev)
            out = torch.empty(d, dtype=torch.float32, device=dev)

            def step(t):
                if off is None:
                    gs.gs_sparsify_aggregate(g, kappa, w.iters, w.seed, t, 0, idx, val, nnz, out, stream=stream)
                else:
                    gs.gs_segmented_sparsify_aggregate(g, off, kappa, w.iters, w.seed, t, 0, idx, val, nnz, out,
                                                       stream=stream)
            n = 30 if name == "c5" else 200
            for t in range(5):
                step(t)
            torch.cuda.synchronize()
            if gs.gs_sync_status(stream) != gs.GS_OK:
                raise RuntimeError("device status after warm-up")
            kept = int(nnz.sum().item())
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for t in range(n):
                step(5 + t)
            e1.record(stream)
            torch.cuda.synchronize()
            ms = max_over_ranks(e0.elapsed_time(e1) / n, dev)
            gs.gs_set_option(gs.GS_OPT_KERNEL_TIMING, 2)
            gs.gs_kernel_times()
            for t in range(n):
                step(5 + n + t)
            torch.cuda.synchronize()
            kt = gs.gs_kernel_times()
            gs.gs_set_option(gs.GS_OPT_KERNEL_TIMING, 0)
            if gs.gs_sync_status(stream) != gs.GS_OK:
                raise RuntimeError("device status after timing")
            # The streaming pass, or the cluster-resident kernel on short rows.
            stats = per_step_stats(lambda t: step(5 + 2 * n + t), min(n, 50), stream)
            sk = next((k for k in ("k_stream_tma", "k_stream", "k_small") if kt.get(k, (0, 0))[1]), "k_stream")
            s_ms = kt[sk][0] / max(kt[sk][1], 1)
            b_sp, b_ag = algorithmic_bytes(M, d, esz, kept)
            step_gbs = (b_sp + b_ag) / (ms / 1e3) / 1e9
            s_bytes = M * d * esz + (kept * 8 + (d * 4 if M == 1 else 0) if sk == "k_small" else 0)
            s_gbs = s_bytes / (s_ms / 1e3) / 1e9
            rows.append({"workload": w.name, "M": M, "d": d, "kappa": kappa, "dtype": dtype, "iters": w.iters,
                         "api": "gs_segmented_sparsify_aggregate" if off is not None else "gs_sparsify_aggregate",
                         "steps": n, "ms_per_step": round(ms, 5), "coords_per_s": M * d / (ms / 1e3),
                         "nnz_per_step": kept, "algorithmic_bytes": b_sp + b_ag,
                         "step_gbs": round(step_gbs, 1), "step_frac": round(step_gbs / hbm, 4),
                         "stream_kernel": sk, "stream_ms": round(s_ms, 5), "stream_gbs": round(s_gbs, 1),
                         "stream_frac": round(s_gbs / hbm, 4), "peak": hbm, "step_ms_stats": stats,
                         "l2": ("fits in L2" if M * d * esz < L2_BYTES else "exceeds L2")})
            del g, idx, val, nnz, out
        except Exception as e:  # one failed row never costs the bench line
            rows.append({"workload": name, "kappa": kappa_o, "dtype": dtype_o,
                         "error": f"{type(e).__name__}: {e}"[:300]})
        torch.cuda.empty_cache()
    return rows


def host_cpu():
    """The host's logical CPU count and CPU model (lscpu's model name, else
    the platform's machine name)."""
    import platform
    model = None
    try:
        outp = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in outp.splitlines():
            if line.split(":")[0].strip() in ("Model name", "Model"):
                model = line.split(":", 1)[1].strip()
                if line.startswith("Model name"):
                    break
    except (OSError, subprocess.SubprocessError):
        pass
    return {"nproc": os.cpu_count(), "model": model or platform.machine()}


def run_e2e(gs, g, kappa, w, args, dev, stream, ws):
    import torch
    M, d = g.shape
    gh = g.cpu().pin_memory()
    g_dev = torch.empty_like(g)
    idx = torch.empty((M, d), dtype=torch.int32, device=dev)
    val = torch.empty((M, d), dtype=torch.float32, device=dev)
    nnz = torch.empty(M, dtype=torch.int32, device=dev)
    out = torch.empty(d, dtype=torch.float32, device=dev)
    out_h = torch.empty(d, dtype=torch.float32).pin_memory()
    nnz_h = torch.empty(M, dtype=torch.int32).pin_memory()
    n = max(3, min(args.steps, args.e2e_steps))
    for t in range(2):
        gs.gs_pipeline_host(gh, kappa, w.iters, w.seed, t, 0, g_dev, idx, val, nnz, out, out_h, nnz_h, stream=stream)
    torch.cuda.synchronize()
    barrier()
    h2d = M * d * g.element_size()
    # The same host-to-device copies alone (worker groups alternating between
    # two streams, as the pipelined call issues them): the floor the
    # pipelined step is measured against.
    cs = (torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev))
    G = min(M, 8)

    def copies():
        ev = torch.cuda.Event()
        ev.record(stream)
        m0 = 0
        for k in range(G):
            m1 = M * (k + 1) // G
            c = cs[k & 1]
            c.wait_event(ev)
            with torch.cuda.stream(c):
                g_dev[m0:m1].copy_(gh[m0:m1], non_blocking=True)
            m0 = m1
        stream.wait_stream(cs[0])
        stream.wait_stream(cs[1])

    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(fn):
        e0.record(stream)
        for t in range(n):
            fn(t)
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / n

    # The host link is shared with other work on the host, and its rate moves
    # between runs: both measurements are taken in E2E_ROUNDS interleaved
    # rounds and reported by their medians (and spread).
    copies()
    torch.cuda.synchronize()
    pipe, copy = [], []
    for r in range(E2E_ROUNDS):
        pipe.append(timed(lambda t: gs.gs_pipeline_host(gh, kappa, w.iters, w.seed, 1000 * r + t, 0, g_dev, idx, val,
                                                          nnz, out, out_h, nnz_h, stream=stream)))
        copy.append(timed(lambda t: copies()))
    rc = gs.gs_sync_status(stream)
    if rc != gs.GS_OK:
        raise RuntimeError(f"device status after e2e: {gs.status_string(rc)}")
    med = lambda xs: sorted(xs)[len(xs) // 2]
    ms = max_over_ranks(med(pipe), dev)
    copy_ms = max_over_ranks(med(copy), dev)
    return {"value": job_throughput(M * d, ms, ws), "unit": UNIT, "ms_per_step": ms,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d * 4 + M * 4,
            "h2d_gbs_over_step": round(h2d / (ms / 1e3) / 1e9, 1),
            "copy_only_ms": round(copy_ms, 4), "copy_only_h2d_gbs": round(h2d / (copy_ms / 1e3) / 1e9, 1),
            "step_over_copy": round(ms / copy_ms, 3), "rounds": E2E_ROUNDS, "steps_per_round": n,
            "ms_per_step_rounds": [round(x, 3) for x in pipe], "copy_only_ms_rounds": [round(x, 3) for x in copy],
            "api": "gs_pipeline_host (worker groups copied on two streams while earlier groups compute)",
            "host_memory": "pinned"}


E2E_ROUNDS = 7
KERNEL_SOURCES = {"k_stream_tma": ("gs_stream_tma.cu", "gs_device.cuh")}


def source_digest(kernel):
    """sha256 over the source files that define `kernel`."""
    import hashlib
    src = os.path.join(ROOT, "paper_1710_09854_gb300", "csrc")
    h = hashlib.sha256()
    for fn in KERNEL_SOURCES.get(kernel, ("gs_kernels.cu", "gs_device.cuh")):
        with open(os.path.join(src, fn), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def alg3_summary(recs, kappa, seg_lens):
    """Algorithm 3's state after one call, from its gs_info records (one per
    worker and segment, `seg_lens` their lengths): lambda's range, how close
    sum p came to the budget kappa * d_l (1 at the fixed point), the
    rescalings taken (section 5 runs two) and the segments that needed the
    exact fallback."""
    fill = [r["sum_p"] / (kappa * n) for r, n in zip(recs, seg_lens)]
    lam = [r["lambda"] for r in recs]
    its = [r["iters_run"] for r in recs]
    return {"records": len(recs), "lambda_min": min(lam), "lambda_max": max(lam),
            "sum_p_over_budget_min": round(min(fill), 9), "sum_p_over_budget_max": round(max(fill), 9),
            "iters_run": {str(k): its.count(k) for k in sorted(set(its))},
            "capped_total": sum(r["capped"] for r in recs),
            "exact_fallbacks": sum(1 for r in recs if r["flags"] & 1)}


def run_alg3_state(gs, g, off, kappa, w, idx, val, nnz, stream):
    """One more call, outside every timed region, that returns the gs_info
    records, summarised by alg3_summary."""
    import torch
    M, d = g.shape
    try:
        if off is None:
            info = gs.info_tensor(M)
            gs.gs_batched_sparsify(g, kappa, w.iters, w.seed, 0, 0, idx, val, nnz, info=info, stream=stream)
            lens = [d] * M
        else:
            L = len(off) - 1
            info = gs.info_tensor(M * L)
            gs.gs_segmented_sparsify(g, off, kappa, w.iters, w.seed, 0, 0, idx, val, nnz, info=info, stream=stream)
            lens = [int(off[l + 1]) - int(off[l]) for _ in range(M) for l in range(L)]
        torch.cuda.synchronize()
        rc = gs.gs_sync_status(stream)
        if rc != gs.GS_OK:
            return {"error": gs.status_string(rc)}
        return alg3_summary(gs.decode_info(info), kappa, lens)
    except Exception as e:  # a report of its own: it never costs the bench line
        return {"error": f"{type(e).__name__}: {e}"[:300]}


def run_hybrid(gs, g, kappa, w, args, dev, stream, n_steps, hbm):
    """The hybrid code of section 3.3 (gs_batched_sparsify_hybrid) on the same
    inputs: its time and bytes, and the coding lengths of one step -- plain
    (index, value) pairs, this format (Q_A 64 bits, Q_B 32 bits, 32 bits of
    1/lambda per worker), the paper's hybrid (b + log2 d and log2 d + 1 bits),
    the entropy-coded dense {0, -1, +1, 2} code, and the section 5 summand of
    H(T, M) (b = 32)."""
    import math
    import numpy as np
    import torch
    M, d = g.shape
    qa_i = torch.empty((M, d), dtype=torch.int32, device=dev)
    qa_v = torch.empty((M, d), dtype=torch.float32, device=dev)
    qb = torch.empty((M, d), dtype=torch.int32, device=dev)
    na = torch.empty(M, dtype=torch.int32, device=dev)
    nb = torch.empty(M, dtype=torch.int32, device=dev)
    il = torch.empty(M, dtype=torch.float32, device=dev)
    info = torch.zeros(M * gs.INFO_BYTES, dtype=torch.uint8, device=dev)
    for t in range(3):
        gs.gs_batched_sparsify_hybrid(g, kappa, w.iters, w.seed, t, 0, qa_i, qa_v, qb, na, nb, il, info=info,
                                      stream=stream)
    torch.cuda.synchronize()
    h0, h1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    h0.record(stream)
    for t in range(n_steps):
        gs.gs_batched_sparsify_hybrid(g, kappa, w.iters, w.seed, args.warmup + t, 0, qa_i, qa_v, qb, na, nb, il,
                                      stream=stream)
    h1.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(h0.elapsed_time(h1) / n_steps, dev)
    # coding lengths of one step (step 0's outputs)
    gs.gs_batched_sparsify_hybrid(g, kappa, w.iters, w.seed, 0, 0, qa_i, qa_v, qb, na, nb, il, info=info,
                                  stream=stream)
    torch.cuda.synchronize()
    rc = gs.gs_sync_status(stream)
    if rc != gs.GS_OK:
        raise RuntimeError(f"device status after the hybrid-code run: {gs.status_string(rc)}")
    rec = gs.decode_info(info)
    a, b_ = na.cpu().numpy().astype(np.int64), nb.cpu().numpy().astype(np.int64)
    ld = math.log2(d)
    bits = {"plain": 0.0, "this_format": 0.0, "paper_hybrid": 0.0, "dense_entropy": 0.0, "H_summand": 0.0}
    for m in range(M):
        codes = qb[m, :int(b_[m])].cpu().numpy().view(np.uint32)
        n_neg = int((codes & 1).sum())
        bits["plain"] += 64.0 * (a[m] + b_[m])
        bits["this_format"] += 64.0 * a[m] + 32.0 * b_[m] + 32.0
        bits["paper_hybrid"] += a[m] * (32 + math.ceil(ld)) + b_[m] * (math.ceil(ld) + 1) + 32
        counts = [d - a[m] - b_[m], n_neg, b_[m] - n_neg, a[m]]
        bits["dense_entropy"] += sum(c * math.log2(d / c) for c in counts if c > 0)
        sum_p_uncapped = rec[m]["sum_p"] - rec[m]["capped"]
        bits["H_summand"] += rec[m]["capped"] * (32 + ld) + min(2 * d, ld * sum_p_uncapped) + 32
    esz = g.element_size()
    algo = M * d * esz + 8 * int(a.sum()) + 4 * int(b_.sum()) + 4 * M
    gbs = algo / (ms / 1e3) / 1e9
    dense = run_dense_code(gs, qa_i, qb, na, nb, d, bits["dense_entropy"], dev, stream, n_steps, hbm)
    # The chunk size trades bits (each chunk adds a directory entry and a
    # flushed state) for parallelism (chunks are coded independently).
    if "error" not in dense:
        dense["by_chunk_size"] = []
        for lk in DENSE_LOG2_K_SWEEP:
            r = run_dense_code(gs, qa_i, qb, na, nb, d, bits["dense_entropy"], dev, stream, n_steps, hbm, log2_k=lk)
            dense["by_chunk_size"].append({k: r.get(k) for k in ("log2_k", "bits_per_coordinate", "over_entropy",
                                                                 "encode_ms", "decode_ms", "error") if k in r})
    return {"api": "gs_batched_sparsify_hybrid", "dense_coded": dense, "steps": n_steps, "ms_per_step": round(ms, 4),
            "algorithmic_bytes": algo, "achieved": round(gbs, 1), "peak": hbm, "frac": round(gbs / hbm, 4),
            "unit": "GB/s", "n_a": int(a.sum()), "n_b": int(b_.sum()),
            "bits_per_step": {k: round(v) for k, v in bits.items()},
            "bits_per_coordinate": {k: round(v / (M * d), 4) for k, v in bits.items()}}


DENSE_LOG2_K = 9   # log2 of the non-zero symbols per chunk of the dense code
DENSE_LOG2_K_SWEEP = (5, 6, 7, 8, 10)   # the other chunk sizes the bench line reports


def run_dense_code(gs, qa_i, qb, na, nb, d, entropy_bits, dev, stream, n_steps, hbm, log2_k=None):
    """The dense code of section 3.3 (gs_dense_encode / gs_dense_decode) of one
    step's hybrid lists: its length in bits per coordinate against the model's
    entropy length sum_s d_s log2(d / d_s), and the time of each direction.
    Algorithmic bytes: the lists read (4 bytes per entry) and the code written
    (encoder); the code read and the dense int8 rows written (decoder)."""
    import torch
    log2_k = DENSE_LOG2_K if log2_k is None else log2_k
    M = qa_i.shape[0]
    word_cap = d // 4 + 4096
    words = torch.empty((M, word_cap), dtype=torch.int16, device=dev)
    n_words = torch.zeros(M, dtype=torch.int64, device=dev)
    qt = torch.empty((M, d), dtype=torch.int8, device=dev)

    def timed(fn):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(n_steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / n_steps

    enc = timed(lambda: gs.gs_dense_encode(qa_i, qb, na, nb, d, log2_k, words, n_words, stream=stream))
    dec = timed(lambda: gs.gs_dense_decode(words, n_words, d, qt, stream=stream))
    rc = gs.gs_sync_status(stream)
    if rc != gs.GS_OK:
        return {"error": gs.status_string(rc)}
    total_words = int(n_words.sum().item())
    entries = int(na.sum().item()) + int(nb.sum().item())
    b_enc = 4 * entries + 2 * total_words
    b_dec = 2 * total_words + M * d
    return {"api": "gs_dense_encode / gs_dense_decode", "log2_k": log2_k, "words": total_words,
            "bits_per_coordinate": round(16.0 * total_words / (M * d), 5),
            "entropy_bits_per_coordinate": round(entropy_bits / (M * d), 5),
            "over_entropy": round(16.0 * total_words / entropy_bits, 4) if entropy_bits else None,
            "encode_ms": round(enc, 4), "encode_gbs": round(b_enc / (enc / 1e3) / 1e9, 1),
            "decode_ms": round(dec, 4), "decode_gbs": round(b_dec / (dec / 1e3) / 1e9, 1),
            "coords_per_s_encode": M * d / (enc / 1e3), "peak": hbm}


def run_resparsify(gs, g, kappa, w, args, dev, stream, n_steps, hbm, ms_fused):
    """Algorithm 1 steps 4-7 (gs_sparsify_average_sparsify): the fused
    sparsify + average, then step 7's Q(v) of the average (kappa_v = kappa,
    the same iterations, a worker id of its own).  Step 7's own cost is the
    difference to the fused call's time per step; its algorithmic bytes are one
    read of v (4d) and the kept pairs of Q(v) written."""
    import torch
    M, d = g.shape
    idx = torch.empty((M, d), dtype=torch.int32, device=dev)
    val = torch.empty((M, d), dtype=torch.float32, device=dev)
    nnz = torch.empty(M, dtype=torch.int32, device=dev)
    v = torch.empty(d, dtype=torch.float32, device=dev)
    idx_v = torch.empty(d, dtype=torch.int32, device=dev)
    val_v = torch.empty(d, dtype=torch.float32, device=dev)
    nnz_v = torch.empty(1, dtype=torch.int32, device=dev)
    wv = 2 ** 32 - 1

    def call(t):
        gs.gs_sparsify_average_sparsify(g, kappa, w.iters, w.seed, t, 0, idx, val, nnz, v, kappa, w.iters, wv,
                                        idx_v, val_v, nnz_v, stream=stream)
    for t in range(3):
        call(t)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for t in range(n_steps):
        call(args.warmup + t)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(e0.elapsed_time(e1) / n_steps, dev)
    rc = gs.gs_sync_status(stream)
    if rc != gs.GS_OK:
        raise RuntimeError(f"device status after the step-7 run: {gs.status_string(rc)}")
    kv = int(nnz_v.item())
    nz = int((v != 0).sum().item())
    # Step 7's cost is the difference of two separately timed loops; if noise
    # leaves no positive difference, no step-7 rate is reported.
    step7_ms = ms - ms_fused
    algo = 4 * d + 8 * kv
    gbs = algo / (step7_ms / 1e3) / 1e9 if step7_ms > 0 else None
    return {"api": "gs_sparsify_average_sparsify", "steps": n_steps, "ms_per_step": round(ms, 4),
            "step7_ms": round(step7_ms, 4) if step7_ms > 0 else None, "kappa_v": kappa, "nnz_average": nz,
            "nnz_resparsified": kv, "step7_algorithmic_bytes": algo,
            "step7_achieved": round(gbs, 1) if gbs else None, "peak": hbm,
            "step7_frac": round(gbs / hbm, 4) if gbs else None, "unit": "GB/s"}


def run_lr_sgd(dev, stream, passes=30, kappas=(0.1, 0.02)):
    """The convex experiment of section 5.1 as a training workload around the
    sparsifier (a reported check): l2-regularised logistic regression on the
    section's synthetic data (N = 1024, d = 2048, C1 = 0.6, C2 = 4^-2,
    lam2 = 1/(10 N)), M = 4 workers with minibatches of 8, step size
    eta0 / ((1 + t/T0) var) with eta0 = M B / L (L: the largest sample loss's
    smoothness) and T0 = five data passes.  The dense
    baseline against the sparsified SGD at each density kappa (Algorithm 3,
    two iterations): suboptimality f(w) - f* after 5, 10, 20 and all passes,
    the run's var, the share of coordinates sent and the time per step."""
    import time
    import torch
    import workloads
    from paper_1710_09854_gb300 import logreg
    N, d, M, B = 1024, 2048, 4, 8
    lam2 = 1.0 / (10 * N)
    Xh, yh = workloads.gen_sec51(N, d, 0.6, 1.0 / 16.0, seed=0)
    f_star, _ = logreg.optimum(Xh, yh, lam2)
    per_pass = N // (M * B)
    steps = passes * per_pass
    bh = workloads.minibatches(steps, M, B, N, seed=0)
    X, y, batches = (torch.from_numpy(a).to(dev) for a in (Xh, yh, bh))
    eta0, T0 = M * B / logreg.smoothness(Xh, lam2), 5.0 * per_pass
    runs = {}
    for kappa in (None,) + tuple(kappas):
        name = "dense" if kappa is None else f"kappa_{kappa}"
        res = logreg.train(X, y, batches, lam2, eta0, T0, kappa=kappa, iters=2, seed=1, log_every=per_pass,
                           stream=stream)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        logreg.train(X, y, batches, lam2, eta0, T0, kappa=kappa, iters=2, seed=1, log_every=None, stream=stream)
        torch.cuda.synchronize()
        ms = (time.perf_counter() - t0) * 1e3 / steps
        curve = dict(res["curve"])
        runs[name] = {"kappa": kappa, "var": round(res["var"], 4),
                      "sent_fraction": round(res["kept_total"] / (steps * M * d), 5),
                      "subopt": {str(p): curve[p * per_pass] - f_star for p in (5, 10, 20, passes)},
                      "ms_per_step": round(ms, 4)}
    return {"data": "section 5.1 synthetic, N=1024, d=2048, C1=0.6, C2=1/16, lam2=1/(10N)", "M": M, "B": B,
            "passes": passes, "f_star": f_star, "f_0": float(dict(res["curve"])[0]), "runs": runs}


VARIANCE_BUDGETS = (30.0, 1.0)   # about 1.2% and 21% density on the Student-t gradients


def run_variance_budget(gs, g, w, args, dev, stream, n_steps, hbm):
    """Algorithm 2 (gs_batched_sparsify_eps) on the same gradients for a few
    variance budgets eps: time per step, density, Newton steps, the bytes of
    the call (two reads of g, the kept (idx, val) pairs written) and the
    histogram pass against its one read of g."""
    import torch
    M, d = g.shape
    esz = g.element_size()
    idx = torch.empty((M, d), dtype=torch.int32, device=dev)
    val = torch.empty((M, d), dtype=torch.float32, device=dev)
    nnz = torch.empty(M, dtype=torch.int32, device=dev)
    info = torch.zeros(M * gs.INFO_BYTES, dtype=torch.uint8, device=dev)
    out = []
    for eps in VARIANCE_BUDGETS:
        for t in range(3):
            gs.gs_batched_sparsify_eps(g, eps, w.seed, t, 0, idx, val, nnz, info=info, stream=stream)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for t in range(n_steps):
            gs.gs_batched_sparsify_eps(g, eps, w.seed, args.warmup + t, 0, idx, val, nnz, stream=stream)
        e1.record(stream)
        torch.cuda.synchronize()
        ms = max_over_ranks(e0.elapsed_time(e1) / n_steps, dev)
        # per-kernel times with every launch bracketed (a few steps)
        nb = min(n_steps, 20)
        gs.gs_set_option(gs.GS_OPT_KERNEL_TIMING, 1)
        gs.gs_kernel_times()
        for t in range(nb):
            gs.gs_batched_sparsify_eps(g, eps, w.seed, t, 0, idx, val, nnz, info=info, stream=stream)
        torch.cuda.synchronize()
        bd = gs.gs_kernel_times()
        gs.gs_set_option(gs.GS_OPT_KERNEL_TIMING, 0)
        rc = gs.gs_sync_status(stream)
        if rc != gs.GS_OK:
            raise RuntimeError(f"device status after the variance-budget run: {gs.status_string(rc)}")
        rec = gs.decode_info(info)
        kept = int(nnz.sum().item())
        algo = 2 * M * d * esz + 8 * kept
        gbs = algo / (ms / 1e3) / 1e9
        hist_ms = bd.get("k_eps_hist", (0.0, 0))[0] / nb
        hist_gbs = M * d * esz / (hist_ms / 1e3) / 1e9 if hist_ms > 0 else 0.0
        out.append({"api": "gs_batched_sparsify_eps", "eps": eps, "steps": n_steps, "ms_per_step": round(ms, 4),
                    "coords_per_s": M * d / (ms / 1e3), "density": round(kept / (M * d), 6),
                    "newton_steps_max": max(r["iters_run"] for r in rec),
                    "algorithmic_bytes": algo, "achieved": round(gbs, 1), "peak": hbm, "frac": round(gbs / hbm, 4),
                    "unit": "GB/s",
                    "hist_roofline": {"kernel": "k_eps_hist", "bound": "hbm", "algorithmic_bytes": M * d * esz,
                                      "ms_per_launch": round(hist_ms, 4), "achieved": round(hist_gbs, 1),
                                      "peak": hbm, "frac": round(hist_gbs / hbm, 4)},
                    "kernels": {k: round(v[0] / nb, 4) for k, v in bd.items() if v[1]}})
    return out


def load_traffic(kernel, workload, dtype, kappa):
    """DRAM bytes per launch of `kernel` (ncu dram__bytes_read.sum +
    dram__bytes_write.sum) from profiles/traffic.txt, if that figure was taken
    on the kernel's current source (its sha256 matches); else None.
    Line format: kernel workload dtype kappa bytes_per_launch sha256."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    try:
        lines = open(path).read().splitlines()
        digest = source_digest(kernel)
    except OSError:
        return None
    for line in lines:
        f = line.split()
        if len(f) != 6 or line.startswith("#"):
            continue
        if f[0] == kernel and f[1] == workload and f[2] == dtype and float(f[3]) == float(kappa):
            return int(f[4]) if f[5] == digest else None
    return None


# ---------------------------------------------------------------------------
# CPU oracle timing (reported baseline and the reference arm)
# ---------------------------------------------------------------------------
def oracle_step(g_rows, off, kappa, iters, seed, step):
    import oracle
    il, vl = [], []
    for m, row in enumerate(g_rows):
        if off is None:
            i, v, _ = oracle.sparsify(row, kappa, iters, seed, step, m)
        else:
            i, v, _ = oracle.segmented_sparsify(row, off, kappa, iters, seed, step, m)
        il.append(i)
        vl.append(v)
    oracle.aggregate(il, vl, g_rows[0].size)


def cpu_baseline_sample(g, off, kappa, w, budget_s=15.0):
    """The oracle as it stands, single-threaded: whole workers of the same
    workload sparsified until about `budget_s` seconds of CPU work have run,
    then the sparse sum of their lists, each timed on its own (the rows'
    copies to the host are outside the timed work)."""
    import oracle
    oracle.lib()
    M, d = g.shape
    il, vl = [], []
    t_sp = 0.0
    for m in range(M):
        row = g[m].float().cpu().numpy()
        t = time.perf_counter()
        if off is None:
            i, v, _ = oracle.sparsify(row, kappa, w.iters, w.seed, 0, m)
        else:
            i, v, _ = oracle.segmented_sparsify(row, off, kappa, w.iters, w.seed, 0, m)
        t_sp += time.perf_counter() - t
        il.append(i)
        vl.append(v)
        if t_sp > budget_s:
            break
    t = time.perf_counter()
    oracle.aggregate(il, vl, d)
    t_ag = time.perf_counter() - t
    done = len(il) * d
    return {"value": done / (t_sp + t_ag), "unit": UNIT, "cores": 1, "kind": "oracle", "host": host_cpu(),
            "sparsify_coords_per_s": done / t_sp, "sparsify_s": round(t_sp, 2), "aggregate_s": round(t_ag, 3),
            "sample": f"{len(il)} of {M} workers at full d={d}: sparsify {t_sp:.1f} s, then the sparse sum of "
                      f"their lists {t_ag:.2f} s"}


def run_reference(args):
    """Reference arm: the CPU oracle, timed on the host cores, each step a
    bounded slice of the workload sized so the whole run takes minutes."""
    ws, rank, _ = dist_env()
    if ws > 1:
        import torch.distributed as dist
        init_dist("gloo")
        if rank != 0:
            dist.barrier()
            return None, rank
    import oracle
    oracle.lib()
    w = {"c1": workloads.C1, "c2": workloads.C2, "c3": workloads.C3, "c4": workloads.C4, "c5": workloads.C5}[
        args.workload]
    kappa = w.kappa if args.kappa is None else args.kappa
    # Host copy of the same distribution (numpy generator), one worker at a time.
    if args.workload in ("c3",):
        full = workloads.gen_student_t(1, min(w.d, 1 << 22), seed0=w.data_seed)[0]
    elif args.workload == "c5":
        full = workloads.gen_c5(1, min(w.d, 1 << 22))[0]
    else:
        full = workloads.gen_c1(min(w.d, 1 << 20))
    # Calibrate: coordinates per step so that (K + W) steps take ~150 s.
    probe = full[: 1 << 16]
    t = time.perf_counter()
    oracle_step([probe], None, kappa, w.iters, w.seed, 0)
    rate = probe.size / (time.perf_counter() - t)
    per_step_s = min(10.0, 150.0 / max(1, args.steps + args.warmup))
    n = int(min(full.size, max(1024, rate * per_step_s)))
    sl = full[:n]
    for t in range(args.warmup):
        oracle_step([sl], None, kappa, w.iters, w.seed, t)
    t0 = time.perf_counter()
    for t in range(args.steps):
        oracle_step([sl], None, kappa, w.iters, w.seed, args.warmup + t)
    el = time.perf_counter() - t0
    ms = el / args.steps * 1e3
    value = n / (ms / 1e3)
    sample = f"one worker slice of {n} coordinates per step (sparsify + sparse sum), single thread"
    res = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": w.name, "M": w.M, "d": w.d, "kappa": kappa, "iters": w.iters, "dtype": w.dtype,
                      "api": "oracle (C, fp64)", "parallelism": f"replicas{ws}"},
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample,
                            "host": host_cpu()},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()
    return res, rank


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="gs", choices=["gs", "reference"])
    ap.add_argument("--workload", default="c3", choices=["c1", "c2", "c3", "c4", "c5"])
    ap.add_argument("--kappa", type=float, default=None)
    ap.add_argument("--dtype", default=None, choices=[None, "f32", "bf16"])
    ap.add_argument("--workers", type=int, default=None, help="override M (reduced case for profiling)")
    ap.add_argument("--dim", type=int, default=None, help="override d (reduced case for profiling)")
    ap.add_argument("--separate", action="store_true",
                    help="time gs_batched_sparsify + gs_sparse_aggregate as two calls instead of gs_sparsify_aggregate")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-lr", action="store_true", help="skip the section 5.1 training-loop report")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-configs", action="store_true", help="skip the sweep over every configuration")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        res, rank = run_reference(args)
    else:
        res, rank = run_gpu(args)
    if rank == 0 and res is not None:
        print(json.dumps(res), flush=True)
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
