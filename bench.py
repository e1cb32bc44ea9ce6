#!/usr/bin/env python
"""Benchmark of the cached Picard solver step on GB300.

Workload (default): SD-v1.5-shaped cached Picard DDIM -- T=100, window 100,
batch 1, 4x64x64 fp32 latents, 16-component mixture denoiser, tol 1e-3,
tau_cache 0.05 (synthetic seeded inputs). One bench step = one complete
generation (every Picard iteration until t = T), replayed as one CUDA graph
with one pair of CUDA events around it on the launch stream; L2 (129 MB) is
flushed before every generation by writing a 256 MiB buffer, outside the
events. ``value`` is Picard iterations per second of device time, denoiser
included, whole job (the iterations all ranks ran over the slowest rank's time).

Also reported:
  solver_step   the cache + Picard solver step alone: a graph of the solver's
                kernels with the eps rows recorded from the same generation and
                an empty stand-in kernel where the denoiser ran, no event nodes
                inside; microseconds per iteration and its algorithmic bytes
                per microsecond against the measured HBM copy bandwidth (and
                the nominal 8 TB/s), with L2 flushed per generation, L2 warm,
                and L2 flushed before every iteration;
  roofline      the solver step (update and planning kernels, or the fused
                step where it runs) from the solver-only graph, with the stored
                ncu DRAM bytes of those kernels as ``traffic``;
  denoiser      the denoiser alone: a graph of the same generation's calls on
                the recorded batches;
  uncached      the same generation with tau_cache = 0 (no hits): NFE,
                iterations and time;
  hit_heavy     the same generation with tau_cache = 0.1 (the hit path
                exercised: about a third of the window points hit at the SD
                shape): NFE, hits, iterations and time;
  e2e           the public API with host buffers (copies inside the timing);
  cpu_baseline  the fp64 oracle on the host cores, one thread and all cores,
                whole iterations and the solver step with the denoiser's time
                taken out.

``--impl reference`` times the fp64 CPU oracle (the only reference this
method has: the paper ships no code) on the same workload.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import workload as W  # noqa: E402

METRIC = "Picard+cache solver steps/s and HBM GB/s vs peak at T=100, 4x64x64; NFE"
UNIT = "solver steps/s"
FLUSH_BYTES = 256 << 20
E2E_CHUNK = 4      # Picard iterations issued between two pa_poll calls in the end-to-end run
GMM_FORMS = {2: "one kernel: clusters of 16 CTAs per 8 rows, CUDA-core dot products summed through "
                "distributed shared memory",
             1: "tensor-core dot products (tcgen05 kind::tf32, split operands), then for 16 < K <= 64 the "
                "responsibilities and the output contraction on the tensor cores too, else an output kernel",
             0: "CUDA-core dot products (fp32 FMA) + output kernel"}
PEAKS_PATH = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0
# ncu DRAM bytes (read + write) per launch of the solver step's kernel(s),
# averaged over one generation's launches, keyed by the sha256 of the solver
# kernels' source files at capture time and the workload. These are stored
# figures from an earlier ncu capture of this bench command (profiles/ has it),
# not a measurement of the current run; reported as null once the kernel
# source has changed since.
NCU_TRAFFIC = {
    # per iteration: k_update_lean + k_plan_gather read + write bytes, averaged
    # over the first generation's launches
    ("97d9b1620ebf45c1", "sd15"): 8263616,       # 6,253,184 + 2,010,432 (no DRAM writes)
    ("97d9b1620ebf45c1", "batched"): 30270037,   # 24,571,861 + 5,698,176
    ("97d9b1620ebf45c1", "large"): 79946021,     # 71,099,246 + 8,846,775
}
# ncu average duration per launch (cold cache, serialised) of the solver-step
# and denoiser kernels over the launches of a launch list (`--metrics
# gpu__time_duration.sum`, the launch lists kept under profiles/), the same key.
NCU_LAUNCH_US = {
    ("97d9b1620ebf45c1", "sd15"): {"k_update_lean": 8.77, "k_plan_gather": 7.54, "k_gmm_cluster": 10.01,
                                   "k_init": 4.58},
    ("97d9b1620ebf45c1", "batched"): {"k_update_lean": 18.30, "k_plan_gather": 10.35, "k_gmm_cluster": 20.53,
                                      "k_init": 6.06},
    ("97d9b1620ebf45c1", "large"): {"k_update_lean": 34.57, "k_plan_gather": 10.92, "k_gmm_dots_tc": 40.10,
                                    "k_gmm_resp": 4.36, "k_gmm_out_tc": 25.50, "k_init": 8.95},
}


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=sorted(W.ALL), default="sd15",
                    help="sd15 is the headline; *_taa run the triangular Anderson (ParaTAA-style) update")
    ap.add_argument("--no-flush", action="store_true", help="do not flush L2 between iterations")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--update-kernel", type=int, default=None)
    ap.add_argument("--gmm-form", type=int, default=None,
                    help="denoiser: 2 one cluster kernel, 1 tensor-core dots + output kernel, 0 CUDA-core dots + output kernel")
    ap.add_argument("--cache-thresh", type=float, default=None,
                    help="override the workload's tau_cache (the threshold sweep)")
    ap.add_argument("--cache-bits", type=int, default=32, choices=[16, 32],
                    help="storage of the cache entries: 32 fp32, 16 bfloat16")
    ap.add_argument("--oracle-sample", type=float, default=None, help=argparse.SUPPRESS)
    return ap.parse_args(argv)


# ---------------------------------------------------------------- ranks ----

def rank_info():
    env = os.environ
    return (int(env.get("RANK", 0)), int(env.get("WORLD_SIZE", 1)), int(env.get("LOCAL_RANK", 0)))


def rank_workload(w: W.Workload, rank: int) -> W.Workload:
    """Weak scaling: rank r runs its own trajectories, seeds offset by r * batch."""
    return w.with_(seed=w.seed + rank * w.batch)


def aggregate(units_local, seconds_local, group=None):
    """(sum of units over ranks, max seconds over ranks) -- host-side timing only."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return float(units_local), float(seconds_local)
    dev = "cuda" if dist.get_backend(group) == "nccl" else "cpu"
    u = torch.tensor([float(units_local)], dtype=torch.float64, device=dev)
    s = torch.tensor([float(seconds_local)], dtype=torch.float64, device=dev)
    dist.all_reduce(u, op=dist.ReduceOp.SUM, group=group)
    dist.all_reduce(s, op=dist.ReduceOp.MAX, group=group)
    return float(u.item()), float(s.item())


def barrier():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        dist.barrier()


# -------------------------------------------------------------- helpers ----

def measured_hbm_gbs():
    try:
        with open(PEAKS_PATH) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


UPDATE_KERNEL_SOURCES = ("k_update_bulk.cu", "k_update_lean.cu", "k_solver.cu", "pa_decide.cuh", "pa_bulk.cuh",
                         "pa_internal.h")


def kernel_source_sha():
    """sha256-16 of the update kernel's sources with comments and whitespace
    removed: it changes when the code changes, not when a comment does."""
    import hashlib
    import re
    h = hashlib.sha256()
    for name in UPDATE_KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_2609_36522_gb300", "csrc", name)) as f:
            src = f.read()
        src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
        src = re.sub(r"//[^\n]*", " ", src)
        h.update("".join(src.split()).encode())
    return h.hexdigest()[:16]


def iteration_bytes(log, w: W.Workload, entry_bytes=4, fused=False):
    """Algorithmic bytes per Picard iteration, from the solver's iteration log.

    Per trajectory with window start t, p points, m misses, frontier e and h1
    hits at positions >= 1 (rows of D fp32 values; cache-entry rows of D
    values of entry_bytes each):
      update : x_t, the p - lazy materialised old states, m batch eps rows and
               p - m ehat rows, m ehat and m xhat writes, h1 xhat reads (next
               distances), p new states, and p draws z_i for stochastic steps
      gather : the next iteration's m' batch rows: read and written by the
               planning kernel, written only by the fused step (the new states
               are still in its registers)
      denoiser: m reads + m writes (+ K means)
    Returns (update, gather, denoiser) arrays over the iterations.
    """
    row = w.D * 4
    ent = w.D * entry_bytes
    n = log.shape[0]
    upd, gat, den = np.zeros(n), np.zeros(n), np.zeros(n)
    for k in range(n):
        for b in range(log.shape[1]):
            t, p, m, stride, e, h1 = (int(v) for v in log[k, b, :6])
            if p == 0:
                continue
            lazy = max(0, t + p - e)
            zr = p if w.eta != 0.0 else 0
            if w.sampler == "taa":
                # mixing update: x_t, old states, eps rows, the previous R of
                # states with a history (nh); entries of the misses, G and R
                # written. mix kernel: G, G' of mixed positions, old states,
                # next-hit entries read; the new states written
                nh = max(0, min(p, e - t))
                upd[k] += ((1 + (p - lazy) + m + nh + zr + 2 * p) + (p + max(0, nh - 1) + (p - lazy) + h1 + p)) \
                    * row + ((p - m) + 2 * m) * ent
            else:
                upd[k] += (1 + (p - lazy) + m + p + zr) * row + ((p - m) + 2 * m + h1) * ent
            den[k] += 2 * m * row
            if k + 1 < n:
                gat[k] += (1 if fused else 2) * int(log[k + 1, b, 2]) * row
        den[k] += w.K * row
    return upd, gat, den


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 100 ms."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# --------------------------------------------------------- oracle timing ----

def oracle_sample(workload_name, budget_s, cache_thresh=None):
    """Time the fp64 oracle on whole generations of the workload for about
    budget_s seconds (at least one generation), and within that the time its
    denoiser calls took (the solver step = the rest). Runs in a fresh process."""
    from oracle import run_picard, run_srds
    from oracle.gmm import make_eps_fn
    from oracle.picard import CacheAdaptation
    from oracle.taa import run_taa
    w = W.ALL[workload_name]
    if cache_thresh is not None:
        w = w.with_(cache_thresh=cache_thresh)
    adapt = CacheAdaptation(*w.extra["adapt"]) if w.extra.get("adapt") else None
    a, x0, mu = W.inputs(w)
    f = make_eps_fn(a, mu, w.gmm_std)
    t_eps = [0.0]

    def f_timed(rows, idx):
        t0 = time.perf_counter()
        r = f(rows, idx)
        t_eps[0] += time.perf_counter() - t0
        return r

    iters = gens = 0
    t0 = time.perf_counter()
    while True:
        if w.sampler == "srds":   # a solver step is one evaluation stage
            r = run_srds(a, x0, f_timed, w.tol, w.cache_thresh)
            iters += len(r.batches)
        elif w.sampler == "taa":
            r = run_taa(a, x0, f_timed, w.window, w.tol, w.cache_thresh, depth=1, record=False,
                        eta=w.eta, noise=W.noise(w), adapt=adapt)
            iters += r.iters
        else:
            r = run_picard(a, x0, f_timed, w.window, w.tol, w.cache_thresh, record=False,
                           eta=w.eta, noise=W.noise(w), adapt=adapt)
            iters += r.iters
        gens += 1
        if time.perf_counter() - t0 >= budget_s:
            break
    dt = time.perf_counter() - t0
    return {"iters": iters, "generations": gens, "seconds": dt, "denoiser_seconds": t_eps[0],
            "nfe_per_gen": r.nfe, "iters_per_gen": r.iters}


def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else platform)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.split(":")[0].strip() == "Model name":
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.processor() or platform.machine()


def time_oracle_subprocess(workload_name, budget_s, threads=1, cache_thresh=None):
    env = dict(os.environ)
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[k] = str(threads)
    env["CUDA_VISIBLE_DEVICES"] = ""
    extra = [] if cache_thresh is None else ["--cache-thresh", repr(float(cache_thresh))]
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--workload", workload_name,
                        "--oracle-sample", str(budget_s), *extra], capture_output=True, text=True, env=env)
    if r.returncode != 0:
        raise RuntimeError(f"oracle sample failed: {r.stderr[-2000:]}")
    return json.loads(r.stdout.strip().splitlines()[-1])


def cpu_baseline(workload_name, budget_s=10.0, cache_thresh=None):
    """The oracle on one host thread (the line's value) and on all of them
    (BLAS/OpenMP threads = os.cpu_count(); NumPy's element-wise work stays on
    one thread), with the solver step's share (the denoiser's time taken out)."""
    ncpu = os.cpu_count() or 1
    legs = {}
    for name, thr in (("one_thread", 1), ("all_cores", ncpu)):
        s = time_oracle_subprocess(workload_name, budget_s, threads=thr, cache_thresh=cache_thresh)
        solver_s = max(s["seconds"] - s["denoiser_seconds"], 1e-12)
        legs[name] = {"value": s["iters"] / s["seconds"], "threads": thr,
                      "solver_step_us_per_iteration": 1e6 * solver_s / s["iters"],
                      "solver_steps_per_s_denoiser_excluded": s["iters"] / solver_s,
                      "sample": f"{s['generations']} full generation(s), {s['iters']} solver steps, "
                                f"{s['seconds']:.1f} s ({s['denoiser_seconds']:.1f} s in the denoiser)"}
    one = legs["one_thread"]
    return {"value": one["value"], "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"fp64 NumPy oracle, single-threaded (BLAS/OpenMP threads = 1): {one['sample']}",
            "cpu_model": cpu_model(), "host_cores": ncpu,
            "solver_step_us_per_iteration": one["solver_step_us_per_iteration"],
            "all_cores": legs["all_cores"]}


# ------------------------------------------------------------ reference ----

def workload_config(w: W.Workload, world, steps_per_gen):
    """The ``config`` of a bench line: the workload only, the same for both arms."""
    extra = {"cache_adaptation": dict(zip(("rate", "target", "tau_min", "tau_max"), w.extra["adapt"]))} \
        if w.extra.get("adapt") else {}
    return {**extra, "workload": w.name,
            "step": ("one full cached Parareal generation (solver step = evaluation stage)"
                     if w.sampler == "srds" else "one full cached-Picard generation"),
            "solver_steps_per_step": int(steps_per_gen), "global_batch": w.batch * world, "seq_len": w.T,
            "window": w.window, "latent": "x".join(map(str, w.latent_shape)), "mixture_components": w.K,
            "tol": w.tol, "cache_thresh": w.cache_thresh, "eta": w.eta}


def run_reference(args):
    rank, world, _ = rank_info()
    if rank != 0:
        return 0
    w = W.ALL[args.workload]
    if args.cache_thresh is not None:
        w = w.with_(cache_thresh=args.cache_thresh)
    # each step: one whole generation by the oracle, in its own process
    for _ in range(args.warmup):
        time_oracle_subprocess(args.workload, 0.0, cache_thresh=args.cache_thresh)
    iters = 0
    secs = 0.0
    per_gen = 0
    for _ in range(args.steps):
        s = time_oracle_subprocess(args.workload, 0.0, cache_thresh=args.cache_thresh)
        iters += s["iters"]
        secs += s["seconds"]
        per_gen = s["iters_per_gen"] if w.sampler != "srds" else s["iters"] // max(1, s["generations"])
    value = iters / secs
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1000.0 * secs / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(w, 1, per_gen),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": f"{args.steps} full generation(s), fp64 NumPy oracle, "
                                   f"single-threaded", "cpu_model": cpu_model(),
                         "host_cores": os.cpu_count()},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# ------------------------------------------------------------------ ours ----

def run_ours(args):
    import torch
    import torch.distributed as dist
    from paper_2609_36522_gb300 import abi
    from paper_2609_36522_gb300 import build as pa_build
    from paper_2609_36522_gb300.solver import Solver, GmmDenoiser

    rank, world, local = rank_info()
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    if local == 0 or world == 1:
        pa_build.build()
    barrier()
    w = rank_workload(W.ALL[args.workload], rank)
    if args.cache_thresh is not None:
        w = w.with_(cache_thresh=args.cache_thresh)
    if w.sampler == "srds":
        return run_srds_bench(args, w)
    a, x0, mu = W.inputs(w)
    dev = torch.device("cuda", local)
    stream = torch.cuda.Stream(device=dev)
    torch.cuda.set_stream(stream)
    noise_dev = torch.from_numpy(W.noise(w)).to(dev) if w.eta != 0.0 else None

    def make_solver(cache_thresh):
        sv = Solver(w.T, w.window, w.latent_shape, a, w.tol, cache_thresh, batch=w.batch, stream=stream)
        if args.update_kernel is not None:
            sv.set_update_kernel(args.update_kernel)
        if args.cache_bits == 16:
            sv.set_cache_precision(16)
        if noise_dev is not None:  # stochastic steps: the draws stay resident on the device
            sv.set_noise(w.eta, noise_dev)
        if w.sampler == "taa":     # triangular Anderson mixing of depth 1
            sv.set_anderson(1)
        if w.extra.get("adapt") and cache_thresh > 0.0:   # tau_cache adapted online
            sv.set_cache_adaptation(*w.extra["adapt"])
        return sv

    s = make_solver(w.cache_thresh)
    max_rows = w.batch * s.window
    g = GmmDenoiser(torch.from_numpy(mu).to(dev), w.gmm_std, a, max_rows, stream=stream)
    if args.gmm_form is not None:
        g.set_form(args.gmm_form)
    eps = torch.empty(max_rows, w.D, dtype=torch.float32, device=dev)
    x_dev = torch.from_numpy(x0).to(dev)
    flush = None if args.no_flush else torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream.synchronize()

    def one_iteration(sv=None):
        sv = s if sv is None else sv
        bx, mb, nm = sv.step_async()
        g.eps(bx, mb, nm, eps)
        sv.submit_eps(eps)

    def run_sync(sv, record=None, record_in=None):
        """One generation through the synchronous API; -> iterations. With a
        list in `record`, the denoiser's eps rows of every iteration are kept;
        with a list in `record_in`, its inputs (batch rows, miss list, count)."""
        sv.init(x_dev)
        n = 0
        while True:
            out = sv.step()
            if out is None:
                return n
            if record_in is not None:
                m = max(out.n_miss, 1)
                full = torch.zeros(max_rows, w.D, dtype=torch.float32, device=dev)  # the denoiser may read every row
                full[:out.n_miss].copy_(out.batch_x)
                record_in.append((full,
                                  out.miss_bt[:out.n_miss].clone() if out.n_miss else torch.zeros(1, 2, dtype=torch.int32, device=dev),
                                  torch.tensor([out.n_miss], dtype=torch.int32, device=dev), m))
            g.eps(out.batch_x_ptr, out.miss_bt_ptr, sv.n_miss_dev(), eps)
            if record is not None:
                record.append(eps[: max(out.n_miss, 1)].clone())
            sv.submit_eps(eps)
            n += 1

    # learn the iteration count with the synchronous API (also a warm-up),
    # keeping the eps rows for the solver-only graph
    eps_rec, den_in = [], []
    n_iters = run_sync(s, eps_rec, den_in)
    st0 = s.stats()
    log = s.iter_log()
    nfe, hits = st0["nfe"], st0["hits"]
    fused = st0["update_kernel"] == 3
    upd_bytes, gat_bytes, den_bytes = iteration_bytes(log, w, 2 if args.cache_bits == 16 else 4, fused)
    step_bytes = upd_bytes + gat_bytes          # the solver step of each iteration

    # One generation (pa_init, then n_iters Picard iterations: the denoiser's
    # two kernels and the solver step -- the fused step kernel, or the update
    # and planning kernels) as a CUDA graph. The timed graph also records CUDA
    # events around every denoiser call and every solver-step launch; the
    # plain graph has no event nodes and gives the iteration rate.
    s.init(x_dev)
    one_iteration()                       # eager warm-up of every launch path
    stream.synchronize()

    den_events = []   # (before, after) the denoiser call of every iteration, timed graph only
    den_ms = [0.0]    # their total over the timed replays
    init_launches = 1                     # pa_init: one kernel (first plan, its batch, cleared sums)

    def capture(timed):
        """-> (graph, kernels launched per iteration inside it)"""
        abi.pa_set_kernel_timing(s.h, timed)
        abi.pa_kernel_timing(s.h, reset=True)
        stream.synchronize()
        l0 = s.stats()["launches"] + g.launches()
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=stream):
            s.init(x_dev)                 # x_init copy, then the first plan, its batch and the cleared sums
            for _ in range(n_iters):
                if not timed:
                    one_iteration()
                    continue
                bx, mb, nm = s.step_async()
                # recorded inside the capture: external events keep their timestamps
                ev = (torch.cuda.Event(enable_timing=True, external=True),
                      torch.cuda.Event(enable_timing=True, external=True))
                ev[0].record(stream)
                g.eps(bx, mb, nm, eps)
                ev[1].record(stream)
                den_events.append(ev)
                s.submit_eps(eps)
        abi.pa_set_kernel_timing(s.h, False)
        l1 = s.stats()["launches"] + g.launches()
        return gr, (l1 - l0 - init_launches) // n_iters

    graph_plain, kernels_per_iter = capture(False)
    graph_timed, _ = capture(True)

    def generation(gr, timed):
        """L2 flushed, then one generation (pa_init included) timed with one event pair."""
        if flush is not None:
            flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        gr.replay()
        e1.record(stream)
        e1.synchronize()
        ms = e0.elapsed_time(e1)
        upd = abi.pa_kernel_timing(s.h, reset=False)[0] if timed else 0.0
        if timed:
            den_ms[0] += sum(a.elapsed_time(b) for a, b in den_events)
        return ms, upd

    for _ in range(args.warmup):
        generation(graph_plain, False)
        generation(graph_timed, True)
    stream.synchronize()
    assert s.poll() == 0, "solver did not finish within the learned iteration count"

    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    barrier()
    stream.synchronize()
    wall0 = time.perf_counter()
    dev_ms = upd_ms = 0.0
    den_ms[0] = 0.0
    for _ in range(args.steps):
        a_ms, _ = generation(graph_plain, False)
        dev_ms += a_ms
        assert s.poll() == 0
        _, u_ms = generation(graph_timed, True)     # same work, solver-step launches bracketed by events
        upd_ms += u_ms
        assert s.poll() == 0
    stream.synchronize()
    barrier()
    wall = time.perf_counter() - wall0
    st1 = s.stats()
    assert st1["iters"] == n_iters and st1["nfe"] == nfe, (st1, n_iters, nfe)
    time.sleep(0.2)
    clk = clocks.stop()
    launches = 2 * args.steps * (n_iters * kernels_per_iter + init_launches)   # both graphs, pa_init each
    graph_plain.replay()
    stream.synchronize()
    assert s.poll() == 0
    x_cached = s.result().cpu().numpy()

    # ---- the solver step alone ------------------------------------------
    # The same generation with the recorded eps rows fed to pa_submit_eps and
    # pa_debug_gap (an empty kernel with the same dependent-launch attribute)
    # where the denoiser ran, so every solver kernel sees the dependency
    # structure it has in a generation. pa_init is its own graph, replayed
    # before the timed one; events around the iterations only.
    g_init = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_init, stream=stream):
        s.init(x_dev)
    g_iter = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_iter, stream=stream):
        for k in range(n_iters):
            s.step_async()
            s.submit_eps(eps_rec[k])
            abi.pa_debug_gap(s.stream_ptr)
    # one graph per iteration, for the L2-cold-before-every-iteration figure
    # (captured from a fresh pa_init so that iteration k uses plan copy k mod 2,
    # as after g_init)
    s.init(x_dev)
    stream.synchronize()
    g_each = []
    for k in range(n_iters):
        gk = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gk, stream=stream):
            s.step_async()
            s.submit_eps(eps_rec[k])
            abi.pa_debug_gap(s.stream_ptr)
        g_each.append(gk)

    def solver_only(do_flush, reps):
        tot = 0.0
        for _ in range(reps):
            if do_flush and flush is not None:
                flush.zero_()
            g_init.replay()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            g_iter.replay()
            e1.record(stream)
            e1.synchronize()
            tot += e0.elapsed_time(e1)
        return 1000.0 * tot / (reps * n_iters)    # us per iteration

    def solver_cold(reps):
        """L2 flushed before every iteration, events around each iteration's graph."""
        per = np.zeros(n_iters)
        for _ in range(reps):
            g_init.replay()
            for k in range(n_iters):
                if flush is not None:
                    flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                g_each[k].replay()
                e1.record(stream)
                e1.synchronize()
                per[k] += e0.elapsed_time(e1)
        return 1000.0 * per / reps                 # us per iteration, per iteration index

    solver_only(True, 3)                           # warm-up
    so_reps = max(10, min(args.steps * 5, 200))
    so_us = solver_only(True, so_reps)
    so_warm_us = solver_only(False, so_reps)
    cold_per = solver_cold(max(3, min(args.steps, 20)))
    assert s.poll() == 0
    so_log_ok = bool(np.array_equal(s.iter_log(), log))
    so_x_ok = bool(np.array_equal(s.result().cpu().numpy(), x_cached))
    assert so_log_ok and so_x_ok, "the solver-only replay diverged from the generation it was recorded from"
    peak, peak_kind = measured_hbm_gbs()
    alg_it = float(step_bytes.mean())
    so_gbps = alg_it / (so_us * 1e-6) / 1e9
    so_warm_gbps = alg_it / (so_warm_us * 1e-6) / 1e9
    cold_gbps = float(step_bytes.sum()) / (float(cold_per.sum()) * 1e-6) / 1e9
    sha = kernel_source_sha()
    tkey = args.workload + ("-bf16" if args.cache_bits == 16 else "") + \
        ("" if args.cache_thresh is None else f"-c{args.cache_thresh:g}") + \
        ("" if args.update_kernel is None else f"-k{args.update_kernel}")
    traffic = NCU_TRAFFIC.get((sha, tkey))
    step_kernel = {4: "Anderson-mixing update + mix kernel + planning kernel",
                   3: "fused step (update, grid barrier, decision, next batch from registers)",
                   2: "lean register update + planning kernel",
                   1: "register-resident or staged update + planning kernel"}.get(st1["update_kernel"],
                                                                                 "plain-load update + planning kernel")
    solver_step = {
        "kernels": step_kernel,
        "us_per_iteration": so_us,
        "alg_bytes_per_iteration": alg_it,
        "gbps": so_gbps, "frac_of_measured_hbm": so_gbps / peak, "frac_of_nominal_8tbs": so_gbps / NOMINAL_HBM_GBS,
        "us_per_iteration_warm_l2": so_warm_us, "gbps_warm_l2": so_warm_gbps,
        "frac_warm_l2_of_measured_hbm": so_warm_gbps / peak,
        "cold_l2_us_per_iteration": float(cold_per.mean()), "cold_l2_gbps": cold_gbps,
        "cold_l2_frac_of_measured_hbm": cold_gbps / peak,
        "cold_l2_us_by_iteration": [round(float(v), 2) for v in cold_per],
        "steps_per_s": 1e6 / so_us,
        "event_timed_launch_us": 1000.0 * upd_ms / max(1, args.steps * n_iters),
        "ncu_kernel_avg_us": NCU_LAUNCH_US.get((sha, tkey)),
        "ncu_kernel_avg_note": ("ncu gpu__time_duration per launch, cold cache and serialised, averaged over "
                                "the launches of an earlier ncu launch list of this workload's bench command "
                                "(several generations); a stored figure keyed by the kernel sources' hash (null: "
                                "not captured for these sources)"),
        "timing": ("a CUDA graph of the generation's solver-step launches fed the eps rows recorded "
                   "from the same generation, with pa_debug_gap (an empty kernel with the same "
                   "dependent-launch attribute) where the denoiser ran; pa_init replayed before it, "
                   "one event pair around the iterations, L2 flushed before each replay (warm_l2: "
                   "not flushed). cold_l2: L2 flushed before every iteration, one graph and one event "
                   "pair per iteration. event_timed_launch_us: events around each solver-step launch "
                   "inside the full generation graph (the events cut the dependent-launch overlap)"),
        "checks": "iteration log and x_T bitwise equal to the generation with the denoiser",
    }
    if traffic is not None:  # DRAM bytes (stored ncu figure) over the same time
        solver_step["dram_bytes_per_iteration"] = traffic
        solver_step["dram_gbps"] = traffic / (so_us * 1e-6) / 1e9
        solver_step["dram_frac_of_measured_hbm"] = solver_step["dram_gbps"] / peak
    roofline = {"bound": "hbm", "achieved": so_gbps, "peak": peak, "unit": "GB/s",
                "frac": so_gbps / peak, "traffic": traffic,
                "kernel": "solver step: " + step_kernel,
                "peak_kind": f"{peak_kind} HBM copy bandwidth (of {peak_kind})",
                "alg_bytes_per_launch": alg_it,
                "avg_launch_us": so_us,
                "avg_launch_note": ("per iteration of the solver-only graph (one solver step and one empty "
                                    "stand-in kernel per iteration, events around the whole graph): an upper "
                                    "bound of the step's own launch time"),
                "traffic_note": ("ncu dram read+write bytes per solver step, averaged over one generation; a "
                                 "stored figure from an earlier capture of this command, keyed by the kernel "
                                 "sources' hash (null: not captured for these sources)")}

    # ---- the denoiser alone -----------------------------------------------
    # Its calls of the same generation on the recorded batches (rows, miss
    # list, count), each followed by pa_debug_gap as the solver step's stand-in,
    # as one graph; events around it, L2 flushed before each replay.
    g_den = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_den, stream=stream):
        for bx_k, mb_k, nm_k, _ in den_in:
            g.eps(bx_k.data_ptr(), mb_k.data_ptr(), nm_k.data_ptr(), eps)
            abi.pa_debug_gap(s.stream_ptr)
    den_only = 0.0
    den_reps = max(10, min(args.steps * 5, 200))
    for r in range(den_reps + 3):
        if flush is not None:
            flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        g_den.replay()
        e1.record(stream)
        e1.synchronize()
        if r >= 3:
            den_only += e0.elapsed_time(e1)
    den_only_us = 1000.0 * den_only / (den_reps * n_iters)
    del g_den

    # ---- side runs of the same sample: uncached (tau_cache = 0, every window
    # point evaluated) and hit-heavy (tau_cache = 0.1: the hit path exercised)
    def side_run(thresh):
        su = make_solver(thresh)
        it = run_sync(su)
        st_ = su.stats()
        su.init(x_dev)
        one_iteration(su)
        stream.synchronize()
        gu = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gu, stream=stream):
            su.init(x_dev)
            for _ in range(it):
                one_iteration(su)
        ms = 0.0
        reps = max(5, min(args.steps, 50))
        for r in range(reps + 2):
            if flush is not None:
                flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            gu.replay()
            e1.record(stream)
            e1.synchronize()
            if r >= 2:
                ms += e0.elapsed_time(e1)
        assert su.poll() == 0
        xs = su.result().cpu().numpy()
        del gu
        su.close()
        ms /= reps
        return {"nfe_per_step": st_["nfe"], "hits_per_step": st_["hits"],
                "hit_rate": st_["hits"] / max(1, st_["hits"] + st_["nfe"]), "iters_per_step": it,
                "ms_per_step": ms, "us_per_iteration": 1000.0 * ms / it, "value": it / (ms / 1000.0)}, xs

    uncached, x_uncached = side_run(0.0)
    for k in ("hits_per_step", "hit_rate"):
        uncached.pop(k)
    uncached["cached_speedup_per_generation"] = uncached["ms_per_step"] / (dev_ms / args.steps)
    uncached["nfe_reduction"] = 1.0 - nfe / max(1, uncached["nfe_per_step"])
    hit_heavy, x_hit_heavy = side_run(0.1)
    hit_heavy["cache_thresh"] = 0.1

    # Quality check of the paper's kind with latents in place of CLIP scores:
    # the cached result against serial DDIM, which is the same library with a
    # window of one point and no cache (every step evaluated in order).
    ser = Solver(w.T, 1, w.latent_shape, a, 0.0, 0.0, batch=w.batch, stream=stream)
    if noise_dev is not None:
        ser.set_noise(w.eta, noise_dev)
    run_sync(ser)
    x_serial = ser.result().cpu().numpy()
    ser.close()

    def dev_from_serial(x):
        return float((np.abs(x - x_serial).max(axis=1) / np.abs(x_serial).max(axis=1)).max())

    deviation = dev_from_serial(x_cached)
    uncached["deviation_from_serial_ddim"] = dev_from_serial(x_uncached)
    hit_heavy["deviation_from_serial_ddim"] = dev_from_serial(x_hit_heavy)

    units, secs = aggregate(args.steps * n_iters, dev_ms / 1000.0)
    value = units / secs

    # End to end through the public API with host buffers (no flush): every
    # step copies x_init in from pinned host memory (pa_init), runs the
    # generation and copies x_T out to pinned host memory (pa_result), with
    # host time and device events around the whole loop. Headline: one
    # Solver.generate call per step through the device-driven loop
    # (pa_loop_launch: x_init copied in, pa_init's kernel, one graph launch; pa_poll_begin:
    # no host round trip inside a generation),
    # without waiting, so that each generation is queued behind the previous
    # one's poll (at most two in flight, each checked); finish() at the end.
    # Beside it: the same calls waiting for every generation, and the
    # through eager calls: pa_step_async + pa_gmm_eps + pa_submit_eps issued
    # from Python in chunks of E2E_CHUNK, pa_poll per chunk.
    e2e = None
    if not args.no_e2e:
        x_host = torch.from_numpy(x0).pin_memory()
        out_host = torch.empty(w.batch, w.D, dtype=torch.float32).pin_memory()
        reps = max(3, min(args.steps, 50))

        def denoise(bx, mb, nm):
            g.eps(bx, mb, nm, eps)
            return eps

        def timed(run):
            stream.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            t0 = time.perf_counter()
            polls = run()
            e1.record(stream)
            stream.synchronize()
            return max(e0.elapsed_time(e1) / 1000.0, time.perf_counter() - t0), polls

        def run_generate(wait=False):
            for _ in range(reps):
                s.generate(x_host, denoise, out=out_host, wait=wait)
            s.finish()
            return reps * (1 if s.generate_path() == "device loop" else -(-n_iters // s.last_chunk))

        def run_eager():
            polls = 0
            for _ in range(reps):
                s.init(x_host)
                while True:
                    for _ in range(E2E_CHUNK):
                        bx, mb, nm = s.step_async()
                        g.eps(bx, mb, nm, eps)
                        s.submit_eps(eps)
                    polls += 1
                    if s.poll() == 0:
                        break
                s.result(out_host)
            return polls

        s.generate(x_host, denoise, out=out_host)   # body length learned and loop captured outside the timing
        assert np.array_equal(out_host.numpy(), x_cached), "generate() differs from the graph-replayed generation"
        e2e_s, polls = timed(run_generate)
        assert np.array_equal(out_host.numpy(), x_cached), "pipelined generate() differs"
        wait_s, _ = timed(lambda: run_generate(wait=True))
        eager_s, eager_polls = timed(run_eager)
        units_e, secs_e = aggregate(reps * n_iters, e2e_s)
        units_w, secs_w = aggregate(reps * n_iters, wait_s)
        units_g, secs_g = aggregate(reps * n_iters, eager_s)
        e2e = {"value": units_e / secs_e, "unit": UNIT,
               "h2d_bytes_per_step": int(w.batch * w.D * 4),
               "d2h_bytes_per_step": int((polls // reps) * (w.batch * w.D * 4 + 40)),  # x_T and the 40-byte counters
               "steps": reps,
               "api": (f"Solver.generate(wait=False) per step: pa_loop_launch (host x_init copied in, "
                       f"pa_init's kernel, one launch of a CUDA graph whose conditional WHILE node repeats "
                       f"{s.last_chunk} captured iterations (the iteration count of one host-driven "
                       f"generation at capture, rounded up to even) -- pa_step_async, pa_gmm_eps, "
                       f"pa_submit_eps -- until "
                       f"every trajectory has reached T), pa_poll_begin "
                       "(host x_T and the counters); each generation's poll read and checked once the next "
                       "generation is queued, Solver.finish() after the last"
                       if s.generate_path() == "device loop" else
                       f"Solver.generate: {s.last_chunk} iterations captured as a CUDA graph, replayed with "
                       f"pa_poll_result per replay (the driver refused the conditional graph node: "
                       f"{s.__dict__.get('loop_error')})"),
               "generate_path": s.generate_path(),
               "loop_body_iterations": s.last_chunk,
               "waiting_value": units_w / secs_w,
               "waiting_api": "the same with generate(wait=True): the host waits for each generation's poll",
               "eager_value": units_g / secs_g,
               "eager_api": f"the same calls issued from Python in chunks of {E2E_CHUNK}, pa_poll per chunk"}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args.workload, cache_thresh=args.cache_thresh)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": dev_ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": workload_config(w, world, n_iters),
            "method": {"cache_entries": "bf16" if args.cache_bits == 16 else "fp32",
                       "solver_step_kernels": step_kernel,
                       "kernels_per_iteration": kernels_per_iter,
                       "denoiser": GMM_FORMS.get(g.form(), "?"),
                       "parallelism": f"replicas x{world} (independent trajectories)"},
            "timing": {"l2": ("not flushed" if args.no_flush else
                              "256 MiB write before every generation (between timed steps), outside the "
                              "timed events"),
                       "value": "CUDA events around each generation: one CUDA-graph replay of pa_init and its "
                                "Picard iterations (denoiser and solver-step kernels each) on the launch "
                                "stream"},
            "nfe_per_step": nfe, "hits_per_step": hits,
            "hit_rate": hits / max(1, hits + nfe),
            "deviation_from_serial_ddim": deviation,
            "solver_step": solver_step,
            "uncached": uncached,
            "hit_heavy": hit_heavy,
            "denoiser_us_per_iteration": den_only_us,
            "denoiser_note": ("the denoiser alone: a graph of its calls on the generation's recorded batches, "
                              "each followed by pa_debug_gap, events around the graph, L2 flushed per replay"),
            "denoiser_event_timed_us": 1000.0 * den_ms[0] / max(1, args.steps * n_iters),
            "denoiser_alg_bytes_per_iteration": float(den_bytes.mean()),
            "roofline": roofline,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": int(launches),
            "clocks": clk,
            "wall_s_timed_region": wall,
        }
        print(json.dumps(line))
    del g_iter, g_init, g_each, graph_plain, graph_timed
    s.close()
    g.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


def run_srds_bench(args, w):
    """The Parareal (SRDS-style) sampler: a solver step is one evaluation stage
    (a fine step of every block, or one coarse block, with its cache test,
    compaction, denoiser call and update). One generation = every stage until
    all trajectories converged, captured as one CUDA graph; L2 flushed between
    generations; CUDA events around each replay."""
    import torch
    import torch.distributed as dist
    from paper_2609_36522_gb300.solver import SrdsSolver, GmmDenoiser
    rank, world, local = rank_info()
    a, x0, mu = W.inputs(w)
    dev = torch.device("cuda", local)
    stream = torch.cuda.Stream(device=dev)
    torch.cuda.set_stream(stream)
    s = SrdsSolver(w.T, w.latent_shape, a, w.tol, w.cache_thresh, batch=w.batch, stream=stream)
    g = GmmDenoiser(torch.from_numpy(mu).to(dev), w.gmm_std, a, s.max_rows, stream=stream)
    if args.gmm_form is not None:
        g.set_form(args.gmm_form)
    eps = torch.empty(s.max_rows, w.D, dtype=torch.float32, device=dev)
    x_dev = torch.from_numpy(x0).to(dev)
    flush = None if args.no_flush else torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)

    def one_stage():
        g.eps(*s.step_async(), eps)
        s.submit_eps(eps)

    s.init(x_dev)
    n_stages = 0
    while True:                         # the stage count, through the synchronous API
        out = s.step()
        if out is None:
            break
        g.eps(out.batch_x_ptr, out.miss_bt_ptr, s.n_miss_dev(), eps)
        s.submit_eps(eps)
        n_stages += 1
    st0 = s.stats()
    nfe, hits, iters = st0["nfe"], st0["hits"], st0["iters"]
    stream.synchronize()
    l0 = s.stats()["launches"] + g.launches()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        s.init(x_dev)                     # x_init widened to fp64, cache and sums cleared
        for _ in range(n_stages):
            one_stage()
    launches_per_gen = s.stats()["launches"] + g.launches() - l0

    def generation():
        if flush is not None:
            flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        graph.replay()
        e1.record(stream)
        e1.synchronize()
        return e0.elapsed_time(e1)

    for _ in range(args.warmup):
        generation()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    barrier()
    wall0 = time.perf_counter()
    dev_ms = 0.0
    for _ in range(args.steps):
        dev_ms += generation()
    stream.synchronize()
    barrier()
    wall = time.perf_counter() - wall0
    st1 = s.stats()
    assert st1["nfe"] == nfe and st1["n_active"] == 0, (st1, nfe)
    time.sleep(0.2)
    clk = clocks.stop()
    units, secs = aggregate(args.steps * n_stages, dev_ms / 1000.0)
    value = units / secs
    # lower bound of the bytes every stage must move (fp64 states, fp32 eps):
    # per evaluated row the distance (x, xhat: 16 B) and the update (x in and
    # out, eps: 20 B); per miss the gather (12 B) and the cache entry (12 B)
    row = w.D
    alg = ((nfe + hits) * 36 + nfe * 24) * row
    peak, peak_kind = measured_hbm_gbs()
    achieved = alg * args.steps / (dev_ms / 1000.0) / 1e9
    e2e = None
    if not args.no_e2e:
        x_host = torch.from_numpy(x0).pin_memory()
        out_host = torch.empty(w.batch, w.D, dtype=torch.float32).pin_memory()
        reps = max(3, min(args.steps, 20))

        def denoise(bx, mb, nm):
            g.eps(bx, mb, nm, eps)
            return eps

        def timed(run):
            stream.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            t0 = time.perf_counter()
            polls = run()
            e1.record(stream)
            stream.synchronize()
            return max(e0.elapsed_time(e1) / 1000.0, time.perf_counter() - t0), polls

        def run_generate():
            for _ in range(reps):
                s.generate(x_host, denoise, out=out_host)
            return 0 if s.generate_path() == "device graph" else reps * -(-n_stages // E2E_CHUNK)

        def run_eager():
            polls = 0
            for _ in range(reps):
                s.init(x_host)
                done = False
                while not done:
                    for _ in range(E2E_CHUNK):
                        out = s.step_async()
                        if out is None:
                            done = True
                            break
                        g.eps(*out, eps)
                        s.submit_eps(eps)
                    polls += 1
                    if not done and s.poll() == 0:
                        done = True
                s.result(out_host)
            return polls

        s.generate(x_host, denoise, out=out_host)   # the capture, outside the timing
        e2e_s, polls = timed(run_generate)
        eager_s, _ = timed(run_eager)
        units_e, secs_e = aggregate(reps * n_stages, e2e_s)
        units_g, secs_g = aggregate(reps * n_stages, eager_s)
        e2e = {"value": units_e / secs_e, "unit": UNIT, "h2d_bytes_per_step": int(w.batch * w.D * 4),
               "d2h_bytes_per_step": int(w.batch * w.D * 4 + (polls // reps) * 24), "steps": reps,
               "api": ("SrdsSolver.generate per step: pa_srds_init (host x_init), pa_srds_loop_launch (every "
                       "stage of every Parareal iteration captured once as a CUDA graph of IF nodes, one per "
                       "iteration, the iterations after convergence skipped on the device), pa_srds_result "
                       "(host x_T, one synchronisation)"
                       if s.generate_path() == "device graph" else
                       f"SrdsSolver.generate, stages issued from Python, pa_srds_poll every {E2E_CHUNK} (the "
                       f"driver refused the conditional graph nodes: {s.__dict__.get('loop_error')})"),
               "generate_path": s.generate_path(),
               "eager_value": units_g / secs_g,
               "eager_api": f"pa_srds_init (host x_init), pa_srds_step_async + pa_gmm_eps + pa_srds_submit_eps "
                            f"in chunks of {E2E_CHUNK} stages, pa_srds_poll per chunk, pa_srds_result (host x_T)"}
    # the sampled latents against serial DDIM (the Picard solver with a window
    # of one point and no cache, same inputs and denoiser)
    graph.replay()
    stream.synchronize()
    assert s.poll() == 0
    x_srds = s.result().cpu().numpy()
    from paper_2609_36522_gb300.solver import Solver
    ser = Solver(w.T, 1, w.latent_shape, a, 0.0, 0.0, batch=w.batch, stream=stream)
    ser.init(x_dev)
    while True:
        out = ser.step()
        if out is None:
            break
        g.eps(out.batch_x_ptr, out.miss_bt_ptr, ser.n_miss_dev(), eps)
        ser.submit_eps(eps)
    x_serial = ser.result().cpu().numpy()
    ser.close()
    deviation = float((np.abs(x_srds - x_serial).max(axis=1) / np.abs(x_serial).max(axis=1)).max())
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args.workload)
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": dev_ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64 states, f32 eps", "data": "synthetic",
            "config": {"workload": w.name, "step": "one full cached Parareal generation",
                       "solver_step_unit": "evaluation stage", "stages_per_step": n_stages,
                       "parareal_iterations": iters, "blocks": s.blocks, "block_steps": s.block_steps,
                       "global_batch": w.batch * world, "seq_len": w.T,
                       "latent": "x".join(map(str, w.latent_shape)), "mixture_components": w.K,
                       "tol": w.tol, "cache_thresh": w.cache_thresh,
                       "denoiser": GMM_FORMS.get(g.form(), "?"),
                       "parallelism": f"replicas x{world} (independent trajectories)",
                       "l2": ("not flushed" if args.no_flush else
                              "256 MiB write before every generation (between timed steps), outside the "
                              "timed events"),
                       "timing": "CUDA events around each generation: one CUDA-graph replay of "
                                 "pa_srds_init and its stages"},
            "nfe_per_step": nfe, "hits_per_step": hits, "hit_rate": hits / max(1, hits + nfe),
            "deviation_from_serial_ddim": deviation,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": None,
                         "kernel": "whole evaluation stages (solver kernels and denoiser, one graph)",
                         "traffic_note": "achieved = a lower bound of the stage bytes over the whole "
                                         "generation time (latency-bound stages of B x N rows)",
                         "peak_kind": f"{peak_kind} HBM copy bandwidth (of {peak_kind})"},
            "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": int(args.steps * launches_per_gen),
            "clocks": clk, "wall_s_timed_region": wall,
        }
        print(json.dumps(line))
    s.close()
    g.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


def main(argv=None):
    args = parse_args(argv)
    if args.oracle_sample is not None:
        print(json.dumps(oracle_sample(args.workload, args.oracle_sample, args.cache_thresh)))
        return 0
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
