#!/usr/bin/env python
"""Benchmark of the 1.5-SPSA parameter-space step on GB300.

One step = the whole hot path over one batch of synthetic inputs:
K x (perturb +eps, perturb -2 eps, perturb +eps) over every weight tensor,
the probe-space preconditioner on K seeded loss triples, and the fused
K-probe update (lr = eps). Default workload: the OPT-30B-shaped fp16
parameter set (772 tensors, 29.97e9 weights, 60 GB), K = 256.

Metric: Gparam*probe/s = d * K / step time, whole job over all ranks.
Prints one JSON line (rank 0). Multi-GPU runs (torchrun) are independent
replicas by default: every rank trains its own copy; nothing is exchanged.
--probe-parallel runs the paper's probe-parallel step instead (Algorithm 1,
Sec. 4.3): probe k on rank k mod R (its out-of-place pair pass and its two
forwards), the K x 3 loss table all-gathered, the same preconditioner and
fused update on every rank; K probes per step over the whole job.

--impl reference times the CPU oracle instead (rank 0 only), on a bounded
prefix sample of the same workload.

--config tiny times the small workload's full step instead (d = 2^20 fp32,
quadratic loss, K = 8): the clean loss, per probe the loss at theta + eps z
and at theta - eps z, the preconditioner and the fused update, the losses
computed on the device; its oracle baseline runs the same steps in full.
"""
import argparse
import dataclasses
import hashlib
import re
import json
import os
import platform
import statistics
import subprocess
import tempfile
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from paper_2609_38095_gb300 import workloads as W  # noqa: E402

METRIC = "Gparam·probe/s and HBM GB/s vs peak, fused K-probe update, OPT-30B shape"
UNIT = "Gparam·probe/s"
NOMINAL_HBM_GBS = 7900.0
FALLBACK_HBM_GBS = 6800.0
LANES_PER_SM = 128


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed steps (default 2; 10 for --config tiny, the small workload's ten full steps)")
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["zo", "reference"], default="zo")
    ap.add_argument("--config", default="opt-30b", choices=sorted(W.BY_KEY))
    ap.add_argument("--K", type=int, default=None, help="override the probes per step of --config")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="target CPU time of the oracle sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--single-thread-seconds", type=float, default=4.0,
                    help="target CPU time of the single-threaded oracle sample")
    ap.add_argument("--cpu-workers", type=int, default=None,
                    help="oracle worker processes for the CPU baseline (default: one per host core)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--clocks-csv", default=None,
                    help="keep the nvidia-smi clock samples of the timed region in this file")
    ap.add_argument("--packing", type=int, default=1, choices=[1, 8],
                    help="generated bits per (weight, probe): 1 (the paper's bit packing) or 8")
    ap.add_argument("--schedule", default=None, choices=["fused", "alg1", "pair", "onepass"],
                    help="fused (default): each restore is folded into the next probe's +eps pass and the last "
                         "one into the update (2K+1 passes); alg1: Algorithm 1's +eps, -2eps, +eps per probe "
                         "(3K+1); pair: theta +- eps z_k written out of place by one pass per probe into two extra "
                         "copies of the weights (K+1 passes, 3 copies in device memory); onepass (--config tiny "
                         "only, its default): the fused schedule with each pass and the loss after it in one "
                         "launch")
    ap.add_argument("--probe-parallel", action="store_true",
                    help="the probe-parallel step over the ranks (probe k on rank k mod R, the loss table "
                         "all-gathered, every rank updates); implies the pair schedule")
    ap.add_argument("--no-pair", action="store_true",
                    help="skip the extra measurement of the out-of-place pair schedule")
    ap.add_argument("--no-other-sets", action="store_true",
                    help="skip the short timings of the other parameter sets (and of the aligned-chunk kernels)")
    ap.add_argument("--no-sequential", action="store_true",
                    help="skip timing Algorithm 1's K sequential update passes against the fused update")
    ap.add_argument("--view-offset", type=int, default=0,
                    help="every parameter a view this many elements into its own allocation (e.g. 1: off the "
                         "32-byte grid, the perturbation passes run the aligned-chunk kernel)")
    args = ap.parse_args()
    if args.steps is None:
        args.steps = W.TINY_STEPS if args.config == "tiny" else 2
    if args.schedule is None:
        args.schedule = "onepass" if args.config == "tiny" else "fused"
    if args.schedule == "onepass" and args.config != "tiny":
        ap.error("--schedule onepass needs --config tiny (the loss it fuses is the small workload's)")
    if args.schedule == "pair" and args.config == "tiny":
        ap.error("--config tiny runs the onepass, fused or alg1 schedule")
    return args


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return json.load(f), "measured"
    return {"hbm_gbs": FALLBACK_HBM_GBS, "sm_max_mhz": 2070.0}, "fallback"


# The sources each kernel is compiled from: a traffic figure stays valid
# while they are unchanged.
KERNEL_SOURCES = {
    "perturb_kernel": ("zo_device.cuh", "zo_stream_kernels.cu"),
    "perturb2_kernel": ("zo_device.cuh", "zo_stream_kernels.cu"),
    "perturb_pair_kernel": ("zo_device.cuh", "zo_stream_kernels.cu"),
    "update_lut8_kernel": ("zo_device.cuh", "zo_update_lut8.cu"),
}


def kernel_source_hash(kernel):
    """sha256[:16] of the kernel's sources with comments and blank lines taken
    out: an edited comment leaves the committed traffic figures valid."""
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2609_38095_gb300", "csrc", f), encoding="utf-8") as fh:
            text = re.sub(r"/\*.*?\*/", "", fh.read(), flags=re.S)
        code = [ln.split("//", 1)[0].rstrip() for ln in text.splitlines()]
        h.update("\n".join(ln for ln in code if ln.strip()).encode())
    return h.hexdigest()[:16]


def committed_traffic(kernel, config_key):
    """(DRAM bytes per launch, how they were obtained) from the committed ncu
    summary, or (None, reason) when the summary is missing or was taken on a
    different kernel source."""
    p = os.path.join(ROOT, "profiles", "ncu_traffic.txt")
    if not os.path.exists(p):
        return None, "no ncu summary committed"
    want = kernel_source_hash(kernel)
    for line in open(p):
        parts = line.split()
        if len(parts) >= 4 and parts[0] == kernel and parts[1] == config_key and parts[2] == want:
            how = parts[4] if len(parts) > 4 else "measured"
            if how.startswith("scaled-from-"):
                how = ("one ncu capture of the same kernel on a smaller parameter set, scaled to this launch by "
                       "the ratio of weights streamed: " + how)
            return float(parts[3]), how
    return None, "kernel source changed since the committed ncu capture"


# ----------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_id, path=None):
        self.proc = None
        self.keep = path is not None
        self.path = path or os.path.join(tempfile.gettempdir(), f"zo_bench_clocks_{os.getpid()}.csv")
        self.device_id = device_id

    def start(self):
        try:
            os.makedirs(os.path.dirname(os.path.abspath(self.path)), exist_ok=True)
            self.fh = open(self.path, "w")
            cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200"]
            if self.device_id:
                cmd += ["-i", self.device_id]
            self.proc = subprocess.Popen(cmd, stdout=self.fh, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.fh.close()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not self.keep:
            try:
                os.remove(self.path)
            except OSError:
                pass
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------- ranks (replicas)
def dist_barrier(world, device):
    """Barrier over the ranks, then a device synchronise."""
    import torch
    import torch.distributed as dist
    if world > 1:
        dist.barrier()
    if device.type == "cuda":
        torch.cuda.synchronize(device)


def max_over_ranks(x, world, device):
    """Largest value of x over all ranks (the slowest replica sets the time)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world, d, K, seconds):
    """Gparam*probe/s of the whole job: every replica processes d weights x K
    probes per step."""
    return world * d * K / seconds / 1e9


# ------------------------------------------------------------- oracle arm
def _widen(bits, dtype):
    """Storage bits -> float32 values (exact)."""
    if dtype == W.DT_F32:
        return bits
    if dtype == W.DT_F16:
        return bits.view(np.float16).astype(np.float32)
    return (bits.astype(np.uint32) << 16).view(np.float32)


def _narrow(out_bits, dtype):
    return out_bits.view(np.float32) if dtype == W.DT_F32 else out_bits.astype(np.uint16)


def oracle_block_step(task):
    """One step of the workload on the weights with virtual indices
    [first, first + n) of the first tensor, computed by the CPU oracle's
    element-list routines: K x (+eps, -2 eps, +eps), the preconditioner on the
    step's loss triples and the fused update. Returns the seconds it took
    (input generation excluded). Runs in a worker process."""
    dtype, first, n, K, eps, step, packing = task
    import oracle
    oracle.set_packing(packing)
    bits = W.random_storage(np.random.default_rng([1, first]), n, dtype)
    g = np.arange(first, first + n, dtype=np.uint64)
    seed = W.step_seed(step)
    t0 = time.perf_counter()
    for k in range(K):
        for s in (eps, -2 * eps, eps):
            bits = _narrow(oracle.perturb_elements(dtype, g, _widen(bits, dtype), seed, k, s), dtype)
    rc, c, _, _ = oracle.precondition(W.synthetic_losses(K, step), eps)
    assert rc == 0
    bits = _narrow(oracle.update_elements(dtype, g, _widen(bits, dtype), seed, c, eps), dtype)
    return time.perf_counter() - t0


def cpu_model():
    """The host CPU's model name (from /proc/cpuinfo; Arm hosts give the
    implementer and part codes)."""
    try:
        info = open("/proc/cpuinfo").read().splitlines()
    except OSError:
        return platform.processor() or platform.machine()
    fields = {}
    for line in info:
        if ":" in line:
            k, v = line.split(":", 1)
            fields.setdefault(k.strip(), v.strip())
    if "model name" in fields:
        return fields["model name"]
    arm = [f"{k} {fields[k]}" for k in ("CPU implementer", "CPU part", "CPU variant") if k in fields]
    return (platform.machine() + " " + " ".join(arm)).strip() if arm else platform.machine()


def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def time_oracle(ps, target_s, steps=1, warmup=0, packing=1, workers=None):
    """The oracle on a bounded sample of the workload, one process per host
    core (spawned, so no CUDA state is inherited), each on its own range of
    the first tensor's weights. Returns (value, seconds per step, weights,
    cores, sample description)."""
    import multiprocessing

    import oracle
    oracle.lib()                                    # build once before the workers load it
    P = max(1, workers or host_cores())
    t_cal = oracle_block_step((ps.dtype, 0, 2048, ps.K, ps.eps, 0, packing))
    per = int(2048 * target_s / max(t_cal, 1e-6)) // 16 * 16
    per = max(16, min(per, ps.numels[0] // P // 16 * 16))
    M = per * P
    ctx = multiprocessing.get_context("spawn")
    with ctx.Pool(P) as pool:
        pool.map(oracle_block_step, [(ps.dtype, j * per, 16, 8, ps.eps, 0, packing) for j in range(P)])
        walls = []
        for s in range(warmup + steps):
            tasks = [(ps.dtype, j * per, per, ps.K, ps.eps, s, packing) for j in range(P)]
            t0 = time.perf_counter()
            pool.map(oracle_block_step, tasks, chunksize=1)
            if s >= warmup:
                walls.append(time.perf_counter() - t0)
    dt = sum(walls) / len(walls)
    value = M * ps.K / dt / 1e9
    sample = (f"first {M} weights of the first tensor ({ps.shapes[0][0]}) of the {ps.name} set, K={ps.K}, "
              f"split over {P} worker processes ({per} weights each, one per host core): "
              f"{3 * ps.K} perturb passes + preconditioner + fused update per step, by the oracle's "
              f"element-list routines; wall time of the slowest worker; value = sample weights x K / time "
              f"(extrapolated to the whole set at the same rate)")
    return value, dt, M, P, sample


def time_oracle_single(ps, target_s, packing=1):
    """The oracle's full step on one core: a prefix of the first tensor sized
    for about target_s seconds. Returns (value, weights)."""
    import oracle
    oracle.set_packing(packing)
    t_cal = oracle_block_step((ps.dtype, 0, 2048, ps.K, ps.eps, 0, packing))
    n = max(16, min(int(2048 * target_s / max(t_cal, 1e-6)) // 16 * 16, ps.numels[0] // 16 * 16))
    dt = oracle_block_step((ps.dtype, 0, n, ps.K, ps.eps, 1, packing))
    return n * ps.K / dt / 1e9, n


def cpu_baseline_line(ps, args, v, M, cores, sample):
    """The cpu_baseline object: all host cores, plus one core, the CPU model
    and how the value was obtained."""
    st_v, st_n = time_oracle_single(ps, args.single_thread_seconds, packing=args.packing)
    return {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample,
            "extrapolated": True, "sample_weights": M, "cpu_model": cpu_model(),
            "single_thread": {"value": st_v, "unit": UNIT, "cores": 1, "sample_weights": st_n,
                              "sample": f"first {st_n} weights of {ps.shapes[0][0]}, one full step, one process"}}


def param_set(args):
    ps = W.BY_KEY[args.config]
    if args.K is not None:
        ps = dataclasses.replace(ps, K=args.K)
    return ps


def stream_config(ps, args, world):
    """The `config` of a parameter-set workload: the same dict on both arms
    (how each arm does the work is in its own top-level keys)."""
    pp = bool(getattr(args, "probe_parallel", False))
    return {"workload": ps.name, "K": ps.K, "d": ps.d, "tensors": len(ps.numels), "packing": args.packing,
            "storage": {W.DT_F16: "fp16", W.DT_BF16: "bf16"}.get(ps.dtype, "fp32"),
            "eps": ps.eps, "lr": ps.eps, "parallelism": f"probe-parallel{world}" if pp else f"replicas{world}",
            **({"view_offset": args.view_offset} if args.view_offset else {}),
            "l2": "inputs larger than L2 (every pass streams the whole parameter set)"}


def tiny_config(ps, args, world):
    """The `config` of the small workload, the same dict on both arms."""
    return {"workload": ps.name, "K": ps.K, "d": ps.d, "eps": ps.eps, "lr": W.TINY_LR,
            "loss": "quadratic 1/2 sum a_i theta_i^2, a_i log-uniform in [1e-2, 1e2]",
            "parallelism": f"replicas{world}",
            "l2": f"flushed before every timed step ({L2_FLUSH_BYTES >> 20} MB write outside the events)"}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    ps = param_set(args)
    value, dt, M, cores, sample = time_oracle(ps, args.cpu_seconds / 2, steps=args.steps, warmup=args.warmup,
                                              packing=args.packing, workers=args.cpu_workers)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": stream_config(ps, args, args.gpus),
        "schedule": f"Algorithm 1 order ({3 * ps.K} perturb passes, the preconditioner, the fused update) on a sample",
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample,
                         "extrapolated": True, "sample_weights": M, "cpu_model": cpu_model()},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------- the small workload
# d = 2^20 fp32 weights, quadratic loss f = 1/2 sum a_i theta_i^2, K = 8,
# eps = 1e-3, lr = 1e-2: the full step, losses included, timed as a whole.
L2_FLUSH_BYTES = 256 << 20        # larger than the 129 MB L2


def _tiny_oracle_phase(task):
    """Worker: the probe phase (kind "probes": K x (+eps, loss, -2 eps, loss,
    +eps) with the partial losses of this slice) or the update phase of one
    step on weights [lo, hi) held in shared memory."""
    kind, shm_th, shm_a, n_all, lo, hi, step, K, eps, lr, c = task
    from multiprocessing import shared_memory

    import oracle
    th_m = shared_memory.SharedMemory(name=shm_th)
    a_m = shared_memory.SharedMemory(name=shm_a)
    try:
        th = np.ndarray((n_all,), dtype=np.float32, buffer=th_m.buf)[lo:hi]
        a = np.ndarray((n_all,), dtype=np.float32, buffer=a_m.buf)[lo:hi]
        g = np.arange(lo, hi, dtype=np.uint64)
        seed = W.step_seed(step)
        if kind == "probes":
            rows = np.zeros((K, 2))
            l0 = oracle.quadratic_loss(th, a)
            for k in range(K):
                for j, sc in enumerate((eps, -2 * eps)):
                    th[:] = oracle.perturb_elements(W.DT_F32, g, th, seed, k, sc).view(np.float32)
                    rows[k, j] = oracle.quadratic_loss(th, a)
                th[:] = oracle.perturb_elements(W.DT_F32, g, th, seed, k, eps).view(np.float32)
            return l0, rows
        th[:] = oracle.update_elements(W.DT_F32, g, th, seed, c, lr).view(np.float32)
        return None
    finally:
        del th, a
        th_m.close()
        a_m.close()


def time_tiny_oracle(steps, workers, K, eps, lr):
    """The oracle on the whole small workload, `steps` full steps, split by
    element range over `workers` processes (1 = the plain single-threaded
    oracle on the whole vector). Returns seconds per step."""
    import multiprocessing
    from multiprocessing import shared_memory

    import oracle
    oracle.lib()
    th0, a0 = W.tiny_theta(), W.tiny_curvatures()
    n = th0.size
    if workers <= 1:
        host = [th0.copy()]
        t0 = time.perf_counter()
        for s in range(steps):
            seed = W.step_seed(s)
            l0 = oracle.quadratic_loss(host[0], a0)
            rows = []
            for k in range(K):
                oracle.perturb(host, [W.DT_F32], seed, k, eps)
                lp = oracle.quadratic_loss(host[0], a0)
                oracle.perturb(host, [W.DT_F32], seed, k, -2 * eps)
                lm = oracle.quadratic_loss(host[0], a0)
                oracle.perturb(host, [W.DT_F32], seed, k, eps)
                rows.append([lp, lm, l0])
            rc, c, _, _ = oracle.precondition(np.array(rows), eps)
            assert rc == oracle.OK
            oracle.update(host, [W.DT_F32], seed, c, lr)
        return (time.perf_counter() - t0) / steps
    shm_th = shared_memory.SharedMemory(create=True, size=n * 4)
    shm_a = shared_memory.SharedMemory(create=True, size=n * 4)
    try:
        np.ndarray((n,), dtype=np.float32, buffer=shm_th.buf)[:] = th0
        np.ndarray((n,), dtype=np.float32, buffer=shm_a.buf)[:] = a0
        bounds = np.linspace(0, n // 16, workers + 1).astype(np.int64) * 16
        bounds[-1] = n
        ctx = multiprocessing.get_context("spawn")
        with ctx.Pool(workers) as pool:
            pool.map(_tiny_oracle_phase, [("update", shm_th.name, shm_a.name, n, 0, 0, 0, K, eps, lr,
                                           np.zeros(K))] * workers)          # start the workers
            t0 = time.perf_counter()
            for s in range(steps):
                parts = pool.map(_tiny_oracle_phase, [("probes", shm_th.name, shm_a.name, n, int(lo), int(hi), s,
                                                       K, eps, lr, None) for lo, hi in zip(bounds[:-1], bounds[1:])])
                l0 = sum(p[0] for p in parts)
                rows = np.zeros((K, 3))
                rows[:, :2] = sum(p[1] for p in parts)
                rows[:, 2] = l0
                rc, c, _, _ = oracle.precondition(rows, eps)
                assert rc == oracle.OK
                pool.map(_tiny_oracle_phase, [("update", shm_th.name, shm_a.name, n, int(lo), int(hi), s, K, eps,
                                               lr, c) for lo, hi in zip(bounds[:-1], bounds[1:])])
            return (time.perf_counter() - t0) / steps
    finally:
        shm_th.close()
        shm_th.unlink()
        shm_a.close()
        shm_a.unlink()


def tiny_cpu_baseline(args, K, eps, lr, steps):
    d = 1 << 20
    cores = max(1, args.cpu_workers or host_cores())
    st_s = time_tiny_oracle(steps, 1, K, eps, lr)
    mt_s = time_tiny_oracle(steps, cores, K, eps, lr) if cores > 1 else st_s
    return {"value": d * K / mt_s / 1e9, "unit": UNIT, "cores": cores, "kind": "oracle", "extrapolated": False,
            "sample": f"the whole workload, {steps} full steps (every weight), weights split by range over {cores} "
                      f"worker processes; losses summed from their partial sums", "cpu_model": cpu_model(),
            "ms_per_step": mt_s * 1e3,
            "single_thread": {"value": d * K / st_s / 1e9, "unit": UNIT, "cores": 1, "ms_per_step": st_s * 1e3,
                              "sample": f"the whole workload, {steps} full steps, one process"}}


def run_tiny(args):
    import torch
    import torch.distributed as dist

    import paper_2609_38095_gb300 as zo
    from paper_2609_38095_gb300.quadratic import QuadraticStep

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        if rank != 0:
            return
        ps = param_set(args)
        st_s = time_tiny_oracle(args.steps, max(1, args.cpu_workers or host_cores()), ps.K, ps.eps, W.TINY_LR)
        value = ps.d * ps.K / st_s / 1e9
        cores = max(1, args.cpu_workers or host_cores())
        print(json.dumps({
            "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": 0, "ms_per_step": st_s * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": tiny_config(ps, args, args.gpus),
            "schedule": "Algorithm 1 order, the oracle's full steps",
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"the whole workload, {args.steps} full steps", "cpu_model": cpu_model()},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}), flush=True)
        return
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    zo.set_packing(args.packing)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    ps = param_set(args)
    K, eps, lr, d = ps.K, ps.eps, W.TINY_LR, ps.d
    schedule = args.schedule
    theta = torch.from_numpy(W.tiny_theta()).to(dev)
    a = torch.from_numpy(W.tiny_curvatures()).to(dev)
    q = QuadraticStep(theta, a, K, eps, lr, schedule=schedule)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    for s in range(args.warmup):
        q.step(W.step_seed(s))
    # timed steps, L2 flushed before each (the workload's 8 MB would stay in L2)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    host_s = []
    clocks = ClockSampler(None, args.clocks_csv)
    clocks.start()
    dist_barrier(world, dev)
    for i in range(args.steps):
        flush.zero_()
        ev[i][0].record(stream)
        t0 = time.perf_counter()
        q.step(W.step_seed(args.warmup + i))
        host_s.append(time.perf_counter() - t0)
        ev[i][1].record(stream)
    dist_barrier(world, dev)
    clk = clocks.stop()
    ms_per_step = max_over_ranks(sum(a_.elapsed_time(b_) for a_, b_ in ev) / args.steps, world, dev)
    launches = q.library_launches_per_step()
    if schedule == "onepass":
        calls = 2 * K + 1 + 2                                                # C-ABI calls per step
    else:
        calls = 2 * K + 1 + (2 * K if schedule == "fused" else 3 * K) + 2
    host_us_per_call = 1e6 * statistics.median(host_s) / calls
    # the same step replayed from a CUDA graph (no host cost per call)
    graph_ms = None
    try:
        side = torch.cuda.Stream(dev)
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            q.step(W.step_seed(0))                                            # warm on the capture stream
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=side):
                q.step(W.step_seed(1))
        stream.wait_stream(side)
        gev = []
        for i in range(args.steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            g.replay()
            e1.record(stream)
            gev.append((e0, e1))
        torch.cuda.synchronize(dev)
        graph_ms = sum(x.elapsed_time(y) for x, y in gev) / len(gev)
    except RuntimeError as e:      # graph capture unavailable: report without it
        graph_ms = None
        print(f"graph replay skipped: {e}", file=sys.stderr)
    # end to end: per step the clean loss and the status read back to the host
    l0_host = torch.empty(1, dtype=torch.float64).pin_memory()
    st_host = torch.empty(1, dtype=torch.int32).pin_memory()
    dist_barrier(world, dev)
    t0 = time.perf_counter()
    for i in range(args.steps):
        q.step(W.step_seed(args.warmup + args.steps + i))
        l0_host.copy_(q.losses[0, 2:3], non_blocking=True)
        st_host.copy_(q.status, non_blocking=True)
        stream.synchronize()
        if int(st_host[0]) != 0:
            raise RuntimeError("preconditioner reported non-finite losses")
    e2e_s = max_over_ranks((time.perf_counter() - t0) / args.steps, world, dev)
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return
    peaks, peak_kind = measured_peaks()
    hbm_peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    # bytes the step must move: each weight pass reads and writes theta, each
    # loss reads theta and a (onepass: a pass that perturbs and evaluates
    # reads theta and a and writes theta)
    if schedule == "onepass":
        step_bytes = 2 * K * 3 * d * 4 + 2 * d * 4 + 2 * d * 4
    else:
        passes = 2 * K + 1 if schedule == "fused" else 3 * K + 1
        step_bytes = passes * 2 * d * 4 + (2 * K + 1) * 2 * d * 4
    achieved = step_bytes / (ms_per_step * 1e-3) / 1e9
    # the fused schedule (separate perturbation and loss launches) on the same
    # workload, for comparison with onepass
    other_us = None
    if schedule == "onepass":
        th2 = torch.from_numpy(W.tiny_theta()).to(dev)
        q2 = QuadraticStep(th2, a, K, eps, lr, schedule="fused")
        for s_ in range(args.warmup):
            q2.step(W.step_seed(s_))
        ev2 = []
        for i in range(args.steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            q2.step(W.step_seed(args.warmup + i))
            e1.record(stream)
            ev2.append((e0, e1))
        torch.cuda.synchronize(dev)
        other_us = 1e3 * sum(x.elapsed_time(y) for x, y in ev2) / len(ev2)
    cpu = None if args.no_cpu_baseline or world > 1 else tiny_cpu_baseline(args, K, eps, lr, args.steps)
    line = {
        "metric": METRIC, "value": world * d * K / (ms_per_step * 1e-3) / 1e9, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": tiny_config(ps, args, world),
        "schedule": schedule,
        "roofline": {"bound": "hbm", "kernel": "whole step (launch-bound: every kernel moves 8 MB or less)",
                     "achieved": achieved, "peak": hbm_peak, "unit": "GB/s", "frac": achieved / hbm_peak,
                     "traffic": None, "traffic_source": "not captured for the small workload",
                     "peak_source": f"{peak_kind} hbm_gbs", "bytes_per_step": step_bytes},
        "tiny": {"us_per_step": ms_per_step * 1e3, "library_launches_per_step": launches,
                 "torch_launches_per_step": 1 if K > 1 and schedule != "onepass" else 0,
                 "abi_calls_per_step": calls,
                 "host_us_per_call": host_us_per_call, "host_us_per_step": 1e6 * statistics.median(host_s),
                 "graph_replay_us_per_step": graph_ms * 1e3 if graph_ms is not None else None,
                 "fused_schedule_us_per_step": other_us},
        "e2e": {"value": world * d * K / e2e_s / 1e9, "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 12, "ms_per_step": e2e_s * 1e3},
        "gpu_launches": launches * args.steps,
        "clocks": clk,
        "cpu_baseline": cpu,
        "host": platform.machine(),
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ------------------------------------------------ probe-parallel step
def probe_parallel_step(L, K, rank, world, pair_pass, gather, finish):
    """One probe-parallel step as --probe-parallel runs it (Algorithm 1,
    Sec. 4.3, without the parameter broadcast: the pair passes leave theta
    untouched, so replicas stay identical): this rank's probes k = rank,
    rank + world, ... each get their out-of-place pair pass (pair_pass(k));
    their loss rows -- the seeded triples of L standing in for the forwards
    at theta +- eps z_k and the clean loss -- are all-gathered into the full
    K x 3 table (gather(rows)), and every rank runs the preconditioner and
    the fused update on it (finish(table)). The arithmetic is injected, so
    the rank logic runs on CPU with the oracle. Returns the table."""
    from paper_2609_38095_gb300 import replicas as R
    mine = list(R.probes_of_rank(K, rank, world))
    for k in mine:
        pair_pass(k)
    table = gather(L[mine])
    finish(table)
    return table


# ------------------------------------------------ the other parameter sets
def time_kernels_on_set(key, dev, hbm_peak, alu_peak, view_offset=0):
    """Short CUDA-event timings of the single-op and two-op passes and the
    fused update (with the leading restore, at the set's K) on one parameter
    set: the evidence for the configurations the headline line does not run."""
    import torch

    import paper_2609_38095_gb300 as zo
    ps = W.BY_KEY[key]
    params = W.allocate_params(ps, device=dev, view_offset=view_offset)
    try:
        plist = zo.ParamList(params)
        stream = torch.cuda.current_stream(dev)
        seed, eps, K = W.step_seed(0), ps.eps, ps.K
        c = torch.tensor(W.synthetic_losses(K, 0)[:, 0] - 2.5, dtype=torch.float64, device=dev)

        def ms_of(fn, n):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize(dev)
            e0.record(stream)
            for i in range(n):
                fn(i)
            e1.record(stream)
            torch.cuda.synchronize(dev)
            return e0.elapsed_time(e1) / n

        for i in range(12):                       # the two-op tuner's trials, then its choice
            zo.perturb2(plist, seed, i, eps, i + 1, eps)
        torch.cuda.synchronize(dev)
        zo.perturb2(plist, seed, 0, eps, 1, eps)
        zo.update(plist, seed, c, eps, pre=(K - 1, eps))
        p1 = ms_of(lambda i: zo.perturb(plist, seed, i, eps if i % 2 else -eps), 6)
        p2 = ms_of(lambda i: zo.perturb2(plist, seed, i, eps, i + 1, -eps), 6)
        up = ms_of(lambda i: zo.update(plist, seed + i, c, eps, pre=(K - 1, eps)), 3)
        byt = 2.0 * ps.d * ps.bytes_per_elem
        rate = ps.d * K / (up * 1e-3) / 1e9
        return {"workload": ps.name + (f"+view{view_offset}" if view_offset else ""), "d": ps.d, "K": K,
                "perturb_ms": p1, "perturb_frac_of_measured_hbm": byt / (p1 * 1e-3) / 1e9 / hbm_peak,
                "perturb2_ms": p2, "perturb2_frac_of_measured_hbm": byt / (p2 * 1e-3) / 1e9 / hbm_peak,
                "update_ms": up, "update_gparam_probe_per_s": rate, "update_frac_alu_1instr": rate / alu_peak,
                "update_frac_of_measured_hbm": byt / (up * 1e-3) / 1e9 / hbm_peak}
    finally:
        del params
        torch.cuda.empty_cache()


# ---------------------------------------------------------------- GPU arm
def run_zo(args):
    import torch
    import torch.distributed as dist

    import paper_2609_38095_gb300 as zo

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    zo.set_packing(args.packing)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    def barrier():
        dist_barrier(world, dev)

    def ranks_max(x):
        return max_over_ranks(x, world, dev)

    ps = param_set(args)
    K, eps, d = ps.K, ps.eps, ps.d
    params = W.allocate_params(ps, device=dev, view_offset=args.view_offset)
    plist = zo.ParamList(params)
    shifted = any(t.data_ptr() % 32 for t in params)   # the perturbation passes use perturb_shift_kernel

    def like_param(t):
        """A buffer for theta +- eps z_k laid out like t (same offset into its own allocation)."""
        if not args.view_offset:
            return torch.empty_like(t)
        return torch.empty(t.numel() + args.view_offset, dtype=t.dtype, device=t.device)[args.view_offset:]
    traffic_key = args.config + (f"+view{args.view_offset}" if args.view_offset else "")
    n_steps_total = args.warmup + args.steps + (0 if args.no_e2e else args.steps)
    losses_host = [W.synthetic_losses(K, s) for s in range(n_steps_total)]
    losses_dev = [torch.tensor(L, device=dev) for L in losses_host]
    c = torch.empty(K, dtype=torch.float64, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)
    chunks = (len(params) + 1023) // 1024
    pp = args.probe_parallel
    pair = args.schedule == "pair" or pp
    my_probes = K          # probes whose passes this rank runs
    if pp:
        from paper_2609_38095_gb300 import replicas
        my_probes = len(replicas.probes_of_rank(K, rank, world))
    if pair:
        plus = zo.ParamList([like_param(t) for t in params])
        minus = zo.ParamList([like_param(t) for t in params])

    timing = {"perturb": [], "perturb2": [], "pair": [], "update": [], "precondition": []}
    fused = args.schedule == "fused" and not pp

    def timed(key, record, fn, *a, **kw):
        if not record:
            return fn(*a, **kw)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        fn(*a, **kw)
        e1.record(stream)
        timing[key].append((e0, e1))

    def step(s, losses_d, record):
        """One step; the forward passes (out of scope) would sit after each
        +eps and each -2eps pass. The fused schedule leaves the weights at
        those points, and at the end, bit for bit as Algorithm 1's does."""
        seed = W.step_seed(s)
        if pp:
            def finish(table):
                timed("precondition", record, zo.precondition, table, eps, out=(c, status))
                timed("update", record, zo.update, plist, seed, c, eps, status=status)
            probe_parallel_step(losses_d, K, rank, world,
                                lambda k: timed("pair", record, zo.perturb_pair, plist, plus, minus, seed, k, eps),
                                lambda rows: replicas.all_gather_losses(rows, K), finish)
            return
        if pair:
            for k in range(K):
                timed("pair", record, zo.perturb_pair, plist, plus, minus, seed, k, eps)
        elif fused:
            timed("perturb", record, zo.perturb, plist, seed, 0, eps)
            for k in range(K):
                timed("perturb", record, zo.perturb, plist, seed, k, -2 * eps)
                if k + 1 < K:
                    timed("perturb2", record, zo.perturb2, plist, seed, k, eps, k + 1, eps)
        else:
            for k in range(K):
                for sc in (eps, -2 * eps, eps):
                    timed("perturb", record, zo.perturb, plist, seed, k, sc)
        timed("precondition", record, zo.precondition, losses_d, eps, out=(c, status))
        timed("update", record, zo.update, plist, seed, c, eps, status=status,
              pre=(K - 1, eps) if fused else None)

    for s in range(args.warmup):
        step(s, losses_dev[s], record=False)

    # ---- timed region: inputs resident in HBM
    dev_uuid = None
    try:
        dev_uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        pass
    clocks = ClockSampler(dev_uuid, args.clocks_csv)
    clocks.start()
    barrier()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for i in range(args.steps):
        s = args.warmup + i
        step(s, losses_dev[s], record=True)
    t_end.record(stream)
    barrier()
    clk = clocks.stop()
    elapsed_ms = ranks_max(t_start.elapsed_time(t_end))
    ms_per_step = elapsed_ms / args.steps
    passes = K + 1 if pair else (2 * K + 1 if fused else 3 * K + 1)   # sweeps over the weights, update included
    if pp:
        passes = my_probes + 1                                            # on each rank
        launches = args.steps * (my_probes * chunks + 1 + chunks)
    elif pair:
        launches = args.steps * (K * chunks + 1 + chunks)
    else:
        launches = args.steps * ((passes - 1) * chunks + 1 + chunks)

    def avg_ms(key):
        v = [a.elapsed_time(b) for a, b in timing[key]]
        return sum(v) / len(v) if v else 0.0

    perturb_ms = ranks_max(avg_ms("perturb"))
    perturb2_ms = ranks_max(avg_ms("perturb2"))
    pair_ms = ranks_max(avg_ms("pair"))
    update_ms = ranks_max(avg_ms("update"))
    precond_ms = ranks_max(avg_ms("precondition"))

    # ---- end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        pinned = [torch.from_numpy(L).pin_memory() for L in losses_host]
        c_host = torch.empty(K, dtype=torch.float64).pin_memory()
        st_host = torch.empty(1, dtype=torch.int32).pin_memory()
        staging = torch.empty(K, 3, dtype=torch.float64, device=dev)
        barrier()
        t0 = time.perf_counter()
        for i in range(args.steps):
            s = args.warmup + args.steps + i
            staging.copy_(pinned[s], non_blocking=True)
            step(s, staging, record=False)
            c_host.copy_(c, non_blocking=True)
            st_host.copy_(status, non_blocking=True)
            stream.synchronize()
            if int(st_host[0]) != 0:
                raise RuntimeError("preconditioner reported non-finite losses")
        barrier()
        e2e_s = ranks_max((time.perf_counter() - t0) / args.steps)
        e2e = {"value": whole_job_rate(1 if pp else world, d, K, e2e_s), "unit": UNIT, "h2d_bytes_per_step": K * 3 * 8,
               "d2h_bytes_per_step": K * 8 + 4, "ms_per_step": e2e_s * 1e3}

    # ---- the out-of-place pair schedule on the same weights (two more copies)
    pair_alt = None
    if not pair and not args.no_pair and not pp:
        free, _ = torch.cuda.mem_get_info(dev)
        if free > 2.05 * d * ps.bytes_per_elem:
            plus_a = zo.ParamList([like_param(t) for t in params])
            minus_a = zo.ParamList([like_param(t) for t in params])
            ev = []

            def pair_step(s, record):
                seed = W.step_seed(s)
                e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
                e[0].record(stream)
                for k in range(K):
                    zo.perturb_pair(plist, plus_a, minus_a, seed, k, eps)
                e[1].record(stream)
                zo.precondition(losses_dev[s], eps, out=(c, status))
                zo.update(plist, seed, c, eps, status=status)
                e[2].record(stream)
                if record:
                    ev.append(e)

            pair_step(0, False)
            barrier()
            for i in range(args.steps):
                pair_step(args.warmup + i, True)
            barrier()
            step_ms = ranks_max(sum(e[0].elapsed_time(e[2]) for e in ev) / len(ev))
            pass_ms = ranks_max(sum(e[0].elapsed_time(e[1]) for e in ev) / len(ev) / K)
            pbytes = 3.0 * d * ps.bytes_per_elem
            pair_alt = {"schedule": f"pair ({K + 1} passes: theta +- eps z_k written out of place into two extra "
                                    "copies, then the preconditioner and the fused update)",
                        "value": whole_job_rate(world, d, K, step_ms * 1e-3), "unit": UNIT, "ms_per_step": step_ms,
                        "device_copies_of_weights": 3, "perturb_pair_ms": pass_ms,
                        "perturb_pair_GB/s": pbytes / (pass_ms * 1e-3) / 1e9,
                        "step_hbm_bytes": K * pbytes + 2.0 * d * ps.bytes_per_elem}
            del plus_a, minus_a
            torch.cuda.empty_cache()

    # ---- Algorithm 1's K-pass update against the fused one (same coefficients)
    seq = None
    if not args.no_sequential:
        reps = 1        # the kernels are warm: the sequential passes are zo_perturb's
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        barrier()
        ev[0].record(stream)
        for _ in range(reps):
            zo.update(plist, W.step_seed(0), c, eps, status=status)
        ev[1].record(stream)
        for _ in range(reps):
            zo.update_sequential(plist, W.step_seed(0), c, eps, status=status)
        ev[2].record(stream)
        barrier()
        fused_ms = ev[0].elapsed_time(ev[1]) / reps
        seq_ms = ev[1].elapsed_time(ev[2]) / reps
        seq = {"fused_ms": fused_ms, "sequential_ms": seq_ms, "speedup": seq_ms / fused_ms,
               "sequential_launches": K * chunks,
               "sequential_GB/s": K * 2.0 * d * ps.bytes_per_elem / (seq_ms * 1e-3) / 1e9}

    peaks, peak_kind = measured_peaks()
    hbm_peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    if pair_alt is not None:
        pair_alt["perturb_pair_frac_of_measured_hbm"] = pair_alt["perturb_pair_GB/s"] / hbm_peak
    perturb_bytes = 2.0 * d * ps.bytes_per_elem       # read + write every weight once
    pair_bytes = 3.0 * d * ps.bytes_per_elem          # read theta, write plus and minus
    achieved = perturb_bytes / (perturb_ms * 1e-3) / 1e9 if perturb_ms > 0 else None
    # the roofline is reported for the kernel with the largest share of the step
    n1, n2 = (K + 1, K - 1) if fused else ((0, 0) if pair else (3 * K, 0))
    if pair:
        dom_kernel, dom_ms, dom_launches = ("pair_shift_kernel<*> (tensors off the 32-byte grid)" if shifted
                                            else "perturb_pair_kernel"), pair_ms, my_probes
        traffic, traffic_how = committed_traffic("perturb_pair_kernel", traffic_key)
    elif n2 > 0 and n2 * perturb2_ms > n1 * perturb_ms:
        dom_kernel, dom_ms, dom_launches = ("perturb_shift_kernel<2, *> (zo_perturb2, tensors off the 32-byte grid)"
                                            if shifted else
                                            "perturb_kernel<2, *> (zo_perturb2, configuration tuned per list)",
                                            perturb2_ms, n2)
        traffic, traffic_how = committed_traffic("perturb2_kernel", traffic_key)
    else:
        dom_kernel, dom_ms, dom_launches = ("perturb_shift_kernel<1, *> (zo_perturb, tensors off the 32-byte grid)"
                                            if shifted else "perturb_kernel<1, 0> (zo_perturb)", perturb_ms, n1)
        traffic, traffic_how = committed_traffic("perturb_kernel", traffic_key)
    dom_bytes = pair_bytes if pair else perturb_bytes
    # the update's DRAM bytes (one read and one write of theta, whatever K): the
    # 8-probe-table kernel's committed capture when it is the one this K runs
    if args.packing == 1 and 16 < K <= 384 and not shifted:
        upd_traffic, upd_traffic_how = committed_traffic("update_lut8_kernel", traffic_key)
    else:
        upd_traffic, upd_traffic_how = None, "no capture committed for the update kernel this K runs"
    # algorithmic HBM bytes of one step: every pass reads and writes theta once,
    # except the pair passes (read theta, write two copies)
    step_bytes = my_probes * pair_bytes + perturb_bytes if pair else passes * perturb_bytes
    dom_achieved = dom_bytes / (dom_ms * 1e-3) / 1e9
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    sm_mhz = (clk or {}).get("sm_mhz") or float(peaks.get("sm_max_mhz", 2070.0))
    alu_peak = sms * LANES_PER_SM * sm_mhz * 1e6 / 1e9    # Gparam*probe/s at one instruction per pair
    upd_rate = d * K / (update_ms * 1e-3) / 1e9
    # replicas: every rank does the whole step (d x K each); probe-parallel: the
    # ranks share one step's K probes
    value = whole_job_rate(1 if pp else world, d, K, ms_per_step * 1e-3)

    others = None
    if world == 1 and not args.no_other_sets:
        del params, plist
        if pair:
            del plus, minus
        torch.cuda.empty_cache()
        others = [time_kernels_on_set(k, dev, hbm_peak, alu_peak) for k in ("opt-1.3b", "qwen3-8b", "opt-13b", "opt-30b")
                  if k != args.config]
        others.append(time_kernels_on_set("opt-1.3b", dev, hbm_peak, alu_peak, view_offset=1))
    if rank != 0:
        return
    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        v, dt, M, cores, sample = time_oracle(ps, args.cpu_seconds, packing=args.packing, workers=args.cpu_workers)
        cpu = cpu_baseline_line(ps, args, v, M, cores, sample)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "strong" if pp else "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": stream_config(ps, args, world),
        "schedule": (f"probe-parallel pair schedule ({passes} passes over the weights per step on each "
                     f"of {world} ranks, the K x 3 loss table all-gathered)" if pp else
                     f"{args.schedule} ({passes} passes over the weights per step)"),
        "roofline": {"bound": "hbm", "kernel": dom_kernel, "achieved": dom_achieved, "peak": hbm_peak,
                     "unit": "GB/s", "frac": dom_achieved / hbm_peak, "traffic": traffic, "traffic_source": traffic_how,
                     "peak_source": f"{peak_kind} hbm_gbs", "bytes_per_launch": dom_bytes,
                     "launches_per_step": dom_launches * chunks,
                     "step_share": dom_launches * dom_ms / ms_per_step},
        "kernels": {
            "perturb": ({"ms": perturb_ms, "GB/s": achieved, "frac_of_measured_hbm": achieved / hbm_peak,
                         "frac_of_nominal_hbm": achieved / NOMINAL_HBM_GBS,
                         "launches_per_step": (K + 1 if fused else 3 * K) * chunks} if not pair else None),
            "pair": ({"ms": pair_ms, "GB/s": pair_bytes / (pair_ms * 1e-3) / 1e9,
                      "frac_of_measured_hbm": pair_bytes / (pair_ms * 1e-3) / 1e9 / hbm_peak,
                      "bytes_per_pass": pair_bytes, "launches_per_step": my_probes * chunks} if pair else None),
            "perturb2": ({"ms": perturb2_ms, "GB/s": perturb_bytes / (perturb2_ms * 1e-3) / 1e9,
                          "frac_of_measured_hbm": perturb_bytes / (perturb2_ms * 1e-3) / 1e9 / hbm_peak,
                          "launches_per_step": (K - 1) * chunks} if fused and K > 1 else None),
            "step_hbm": {"passes": passes, "bytes": step_bytes, "ideal_ms": step_bytes / (hbm_peak * 1e9) * 1e3,
                         "frac": step_bytes / (hbm_peak * 1e9) / (ms_per_step * 1e-3)},
            "update": {"ms": update_ms, "gparam_probe_per_s": upd_rate, "bound": "alu",
                       "peak_gparam_probe_per_s_1instr": alu_peak, "frac_alu_1instr": upd_rate / alu_peak,
                       # the two-instruction model (an add and a sign operation per pair)
                       "frac_alu_2instr": upd_rate / (alu_peak / 2),
                       "GB/s": perturb_bytes / (update_ms * 1e-3) / 1e9,
                       "traffic": upd_traffic, "traffic_source": upd_traffic_how},
            "precondition": {"ms": precond_ms},
        },
        "e2e": e2e,
        "sequential": seq,
        "pair_schedule": pair_alt,
        "other_sets": others,
        "gpu_launches": launches,
        "clocks": clk,
        "cpu_baseline": cpu,
        "host": platform.machine(),
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse_args()
    if args.config == "tiny":
        run_tiny(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_zo(args)


if __name__ == "__main__":
    main()
