"""Benchmark of the heterogeneous data-parallel SGD step (arXiv 2110.08941) on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

A step is one synchronous SGD step of the whole hot path through libhs: per-worker forward and
backward over M = 16 compute-proportional segments of a 16384-sample batch (MLP
4096 -> 8192 -> 8192 -> 1000, bf16 tensor cores), softmax cross-entropy, each worker's weight
gradient formed tile by tile in tensor memory and averaged there with the update applied in the
same kernel (biases through per-worker slabs and the reduce + update).  Inputs are seeded
synthetic data already resident in HBM; the working set (over 1 GB of bf16 activations and input
gradients, 0.44 GB of fp32 parameters per step) is far larger than L2, so no explicit L2 flush
is needed between steps.

Prints ONE JSON line (rank 0).  With --gpus N > 1 (launched by torch.distributed.run) every rank
runs an independent replica of the workload (the M workers live on one GPU; there is no cross-GPU
exchange): weak scaling, value = all ranks' samples / max-over-ranks time.

--impl reference times the fp64 CPU oracle on the host cores (bounded samples of the same
workload) as the reference arm.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "samples/sec per synchronous SGD step on 1 GB300"
UNIT = "samples/s"
DEFAULT_WORKLOAD = synth.CFG5


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        d = json.load(open(path))
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"], bf16_sust=d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                    src="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sust=1700.0, src="fallback")


# ------------------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200",
                 "-i", str(self.gpu)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (FileNotFoundError, OSError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for nm, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------------------ workload math
def gemm_flops(wl):
    """Algorithmic flops of the step's products (forward, per-worker weight gradient, input gradient)."""
    n = wl.global_batch
    if wl.arch == synth.MLP:
        dims = wl.dims
        sw = sum(dims[l] * dims[l - 1] for l in range(1, len(dims)))
        sw_dgrad = sum(dims[l] * dims[l - 1] for l in range(2, len(dims)))
        return dict(forward=2.0 * n * sw, wgrad=2.0 * n * sw, dgrad=2.0 * n * sw_dgrad)
    cin, h, w, c1, c2, c3, classes = wl.dims
    per = []                       # (rows per sample x Cout x Cin*9) of each conv
    prev = cin
    for c, s in zip((c1, c2, c3), (1, 2, 2)):
        h, w = (h + 2 - 3) // s + 1, (w + 2 - 3) // s + 1
        per.append(h * w * c * prev * 9)
        prev = c
    fc = classes * c3
    return dict(forward=2.0 * n * (sum(per) + fc), wgrad=2.0 * n * (sum(per) + fc),
                dgrad=2.0 * n * (per[1] + per[2] + fc))


def recorded_traffic(kernel_tag="tc_wgrad_avg_pair"):
    """DRAM bytes per launch of the dominant kernel from the committed ncu summary, or None when the
    kernel sources changed since those counters were taken."""
    import glob
    import hashlib
    files = glob.glob(os.path.join(ROOT, "profiles", kernel_tag + "_*_dram.md"))
    if not files:
        return None
    text = open(files[0]).read()
    vals = {}
    for line in text.splitlines():
        if ":" in line and line.split(":")[0] in ("traffic_bytes_per_launch", "kernel_source_sha256"):
            k, v = line.split(":", 1)
            vals[k] = v.strip()
    csrc = os.path.join(ROOT, "paper_2110_08941_gb300", "csrc")
    h = hashlib.sha256()
    for f in ("gemm_avg.cu", "tc_pair.cuh", "tc_device.cuh", "gemm_tc.cuh"):
        h.update(open(os.path.join(csrc, f), "rb").read())
    if vals.get("kernel_source_sha256") != h.hexdigest():
        return None
    try:
        return float(vals["traffic_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


def straggler_simulation(seed=0, steps=200, every=10):
    """Simulated iteration time of the drifting 8-worker workload (the straggler model of Section 3:
    a synchronous step lasts as long as its slowest worker, X_(M) = max_m n_m / c_m(t)), summed
    over `steps` steps for three schedules: the even split of Sync-SGD, Dynamic Partitioning
    (Algorithm 1, repartitioned every `every` steps from the window's measured throughputs through
    the library's host rule), and the ideal real-valued split n_m proportional to c_m(t).  Host
    only; speeds c_m(t) from the seeded random walk."""
    import paper_2110_08941_gb300 as hs
    wl = synth.WORKLOADS[synth.CFG3]
    m, n = wl.workers, wl.global_batch
    c = synth.drift_walk(m, steps, seed)
    even = hs.hs_partition_sizes([1.0] * m, n)
    sizes = list(even)
    t_even = t_dp = t_ideal = 0.0
    for t in range(steps):
        ct = c[t]
        t_even += max(even[k] / ct[k] for k in range(m))
        t_dp += max(sizes[k] / ct[k] for k in range(m))
        t_ideal += n / float(np.sum(ct))
        if (t + 1) % every == 0:
            sizes = hs.hs_partition_sizes(list(synth.window_throughputs(c[t + 1 - every:t + 1])), n)
    return {"workload": wl.name, "steps": steps, "repartition_every": every,
            "sum_max_time_even": t_even, "sum_max_time_dynamic_partitioning": t_dp,
            "sum_time_ideal_split": t_ideal, "unit": "sample-times (n / speed, speed c_m(0) = 1)"}


def heterogeneity_simulation(per_sample_s: float, seed: int = 0, workers: int = 8, per_worker: int = 128,
                             epochs: int = 15, steps_per_epoch: int = 20, jitter: float = 0.05):
    """Replica of the delay experiments (Section 5.2 / 5.3) on simulated workers.  Every worker
    processes a sample in `per_sample_s` seconds (from the measured GPU step); half of them also
    sleep for a fixed delay each minibatch, 25% ("low") or 50% ("high") of the mean minibatch
    time, with a little multiplicative noise.  Sync-SGD keeps the even split of 128 samples per
    worker (weak scaling); Dynamic Partitioning (Algorithm 1) re-sizes the partitions every epoch
    from the mean measured minibatch times of the last epoch (Eq. 2, the library's host rule).
    A step lasts as long as its slowest worker (Section 3).  Host only."""
    import paper_2110_08941_gb300 as hs
    rng = np.random.default_rng(seed + 5)
    n = workers * per_worker
    base = per_worker * per_sample_s
    out = {}
    for level, frac in (("low", 0.25), ("high", 0.50)):
        delay = np.array([frac * base if k % 2 == 0 else 0.0 for k in range(workers)])
        res = {}
        for sched in ("sync_sgd", "dynamic_partitioning"):
            sizes = [per_worker] * workers
            times = []
            for ep in range(epochs):
                ep_times = np.zeros(workers)
                for _ in range(steps_per_epoch):
                    noise = rng.lognormal(0.0, jitter, workers)
                    x = (np.asarray(sizes) * per_sample_s + delay) * noise
                    ep_times += x
                    times.append(float(x.max()))
                if sched == "dynamic_partitioning":
                    mean_x = ep_times / steps_per_epoch
                    sizes = hs.hs_partition_sizes([sizes[k] / mean_x[k] for k in range(workers)], n)
            t = np.asarray(times)
            res[sched] = {"total_s": float(t.sum()), "mean_step_ms": 1e3 * float(t.mean()),
                          "p50_ms": 1e3 * float(np.percentile(t, 50)), "p90_ms": 1e3 * float(np.percentile(t, 90)),
                          "last_sizes": [int(v) for v in sizes]}
        res["speedup"] = res["sync_sgd"]["total_s"] / res["dynamic_partitioning"]["total_s"]
        out[level] = res
    out["per_sample_ms"] = 1e3 * per_sample_s
    return out


def update_bytes(wl, P):
    # M slab reads + theta read, theta write + bf16 shadow write
    return (wl.workers + 2) * P * 4 + 2 * P


# ------------------------------------------------------------------------------ CPU oracle baseline
def oracle_sample(wl, seconds_target=12.0, max_workers=None):
    """Time the oracle (as it stands) on whole worker segments of the workload: the smallest
    workers first, adding workers until about `seconds_target` of CPU time.  Returns
    (samples/s, description, cores)."""
    from oracle import cnn, mlp, sgd
    from oracle import partition as P

    fn = mlp.worker_loss_grad if wl.arch == synth.MLP else cnn.worker_loss_grad
    try:
        from threadpoolctl import threadpool_info
        threads = max([i.get("num_threads", 1) for i in threadpool_info()] or [1])
    except Exception:
        threads = os.cpu_count()
    x, y = synth.make_batch(wl)
    theta = synth.make_params(wl).astype(np.float64)
    sizes = P.partition_sizes(list(synth.initial_weights(wl)), wl.global_batch)
    off = P.offsets(sizes)
    order = sorted(range(wl.workers), key=lambda m: sizes[m])
    if max_workers:
        order = order[:max_workers]
    done_samples, elapsed, used = 0, 0.0, []
    for m in order:
        xs, ys = x[off[m]:off[m + 1]], y[off[m]:off[m + 1]]
        t0 = time.perf_counter()
        sgd.step(fn, theta, wl.dims, xs, ys, [sizes[m]], wl.lr, sgd.SYNC_CP_WEIGHTED)
        elapsed += time.perf_counter() - t0
        done_samples += sizes[m]
        used.append(m)
        if elapsed >= seconds_target:
            break
    desc = (f"oracle fp64 step (forward, backward, weighted accumulation, update) over the whole segments "
            f"of workers {used} ({done_samples} samples) of {wl.name}")
    return done_samples / elapsed, desc, threads


def blas_name():
    try:
        from threadpoolctl import threadpool_info
        info = [i for i in threadpool_info() if i.get("user_api") == "blas"]
        if info:
            return ", ".join(f"{i.get('internal_api')} {i.get('version')}" for i in info)
    except Exception:
        pass
    try:
        b = np.show_config(mode="dicts")["Build Dependencies"]["blas"]
        return f"{b.get('name')} {b.get('version')}"
    except Exception:
        return None


def _oracle_one_thread_inproc(name, n_samples):
    from oracle import cnn, mlp, sgd
    from oracle import partition as P
    wl = synth.WORKLOADS[name]
    fn = mlp.worker_loss_grad if wl.arch == synth.MLP else cnn.worker_loss_grad
    x, y = synth.make_batch(wl)
    theta = synth.make_params(wl).astype(np.float64)
    sizes = P.partition_sizes(list(synth.initial_weights(wl)), wl.global_batch)
    off = P.offsets(sizes)
    m = min(range(wl.workers), key=lambda k: sizes[k])
    n = min(n_samples, sizes[m])
    xs, ys = x[off[m]:off[m] + n], y[off[m]:off[m] + n]
    t0 = time.perf_counter()
    sgd.step(fn, theta, wl.dims, xs, ys, [n], wl.lr, sgd.SYNC_CP_WEIGHTED)
    dt = time.perf_counter() - t0
    return [n / dt, f"one thread: oracle fp64 step over the first {n} samples of worker {m}'s segment"]


def oracle_one_thread(wl, n_samples=64):
    """The same oracle step on the first `n_samples` rows of the smallest worker's segment, in a child
    process whose BLAS pools are held to one thread.  Returns (samples/s, description) or None."""
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1",
               BLIS_NUM_THREADS="1", CUDA_VISIBLE_DEVICES="")
    code = ("import json, bench; "
            f"print(json.dumps(bench._oracle_one_thread_inproc({wl.name!r}, {int(n_samples)})))")
    try:
        r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True, text=True,
                           timeout=300)
        v, desc = json.loads(r.stdout.strip().splitlines()[-1])
        return float(v), desc
    except Exception:
        return None


# ------------------------------------------------------------------------------ ranks
def max_over_ranks(value: float) -> float:
    """Max of a per-rank number over all ranks of the default process group (identity without one).
    NCCL groups reduce a CUDA tensor, gloo groups a CPU tensor."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    dev = torch.device("cuda", torch.cuda.current_device()) if dist.get_backend() == "nccl" else torch.device("cpu")
    t = torch.tensor([float(value)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.barrier()


# ------------------------------------------------------------------------------ arms
def bench_config(wl, world):
    """The workload description both arms print (same dict, so the two lines compare directly)."""
    return {"workload": wl.name, "global_batch": wl.global_batch, "workers": wl.workers,
            "dims": list(wl.dims), "sync": "cp_weighted", "parallelism": f"replicas{world}",
            "l2": ("working set > L2 (over 1 GB of activations and input gradients, 0.44 GB theta per "
                   "step), no flush" if wl.name == DEFAULT_WORKLOAD else "small workload: working set may sit in L2")}


def run_reference(args, wl, rank, world):
    if rank != 0:
        return
    from oracle import cnn, mlp, sgd
    from oracle import partition as P
    fn = mlp.worker_loss_grad if wl.arch == synth.MLP else cnn.worker_loss_grad
    try:
        from threadpoolctl import threadpool_info
        cores = max([i.get("num_threads", 1) for i in threadpool_info()] or [1])
    except Exception:
        cores = os.cpu_count()
    x, y = synth.make_batch(wl)
    theta = synth.make_params(wl).astype(np.float64)
    sizes = P.partition_sizes(list(synth.initial_weights(wl)), wl.global_batch)
    off = P.offsets(sizes)
    m = min(range(wl.workers), key=lambda k: sizes[k])      # smallest worker segment per step
    xs, ys = x[off[m]:off[m + 1]], y[off[m]:off[m + 1]]

    def one():
        nonlocal theta
        theta, _, _, _, _ = sgd.step(fn, theta, wl.dims, xs, ys, [sizes[m]], wl.lr, sgd.SYNC_CP_WEIGHTED)

    for _ in range(args.warmup):
        one()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        one()
    dt = time.perf_counter() - t0
    value = sizes[m] * args.steps / dt
    sample = (f"each step: oracle fp64 step over worker {m}'s whole segment ({sizes[m]} samples) of {wl.name}")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": bench_config(wl, world),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_ours(args, wl, rank, world, local_rank):
    import torch
    import paper_2110_08941_gb300 as hs

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    precision = hs.HS_BF16 if args.precision == "bf16" else hs.HS_FP32_CHECK
    x, y = synth.make_batch(wl)
    theta0 = synth.make_params(wl)
    w = synth.initial_weights(wl)
    ctx = hs.hs_init(wl.arch, wl.dims, wl.workers, wl.global_batch, compute_weights=w, precision=precision,
                     sync=hs.HS_SYNC_CP_WEIGHTED)
    params = torch.from_numpy(theta0).to(dev)
    xd = torch.from_numpy(x).to(dev)
    yd = torch.from_numpy(y).to(dev)
    stream = torch.cuda.current_stream(dev)
    part = ctx.partition

    for _ in range(args.warmup):
        hs.hs_step(ctx, params, xd, yd, part, wl.lr, stream=stream, want_loss=False)
    torch.cuda.synchronize()

    clocks = ClockSampler(local_rank)
    clocks.start()
    time.sleep(0.3)
    barrier()
    torch.cuda.synchronize()
    # one event after each step: the bracket is the first and last, the step-time spread the rest
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    ev[0].record(stream)
    for i in range(args.steps):
        hs.hs_step(ctx, params, xd, yd, part, wl.lr, stream=stream, want_loss=False)
        ev[i + 1].record(stream)
    torch.cuda.synchronize()
    barrier()
    ms = ev[0].elapsed_time(ev[-1])
    step_ms = np.asarray([ev[i].elapsed_time(ev[i + 1]) for i in range(args.steps)])
    ms = max_over_ranks(ms)
    # The same K steps again with CUDA events around every phase, on the step's stream: the live
    # kernel times behind the roofline.  A second pass because recording (or, on a replayed step,
    # re-pointing) two events per phase costs host time that would show in the small workloads'
    # step time; the library captures the profiled step in the first two of its warm-up steps.
    hs.hs_set_profiling(ctx, True)
    for _ in range(3):
        hs.hs_step(ctx, params, xd, yd, part, wl.lr, stream=stream, want_loss=False)
    torch.cuda.synchronize()
    hs.hs_read_profile(ctx)                 # discard warm-up counts
    pv0, pv1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    pv0.record(stream)
    for _ in range(args.steps):
        hs.hs_step(ctx, params, xd, yd, part, wl.lr, stream=stream, want_loss=False)
    pv1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    prof = hs.hs_read_profile(ctx)
    profiled_ms = pv0.elapsed_time(pv1) / args.steps
    hs.hs_set_profiling(ctx, False)
    loss = hs.hs_step(ctx, params, xd, yd, part, 0.0, stream=stream, want_loss=True)   # finite-loss check

    # the same step replayed from a CUDA graph (captured once, loss not requested): the launch
    # overhead of the step's kernels removed
    graph = None
    try:
        side = torch.cuda.Stream(dev)
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            hs.hs_step(ctx, params, xd, yd, part, wl.lr, stream=side, want_loss=False)
        stream.wait_stream(side)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            hs.hs_step(ctx, params, xd, yd, part, wl.lr, want_loss=False)
        g.replay()
        torch.cuda.synchronize()
        barrier()
        q0, q1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        q0.record(stream)
        for _ in range(args.steps):
            g.replay()
        q1.record(stream)
        torch.cuda.synchronize()
        gms = max_over_ranks(q0.elapsed_time(q1))
        graph = {"ms_per_step": gms / args.steps, "value": world * wl.global_batch * args.steps / (gms * 1e-3),
                 "unit": UNIT, "what": "one hs_step captured in a CUDA graph, replayed"}
        del g
    except Exception as e:   # capture is an optimisation of the launch path; report why it failed
        graph = {"unavailable": f"{type(e).__name__}: {e}"[:200]}

    # the slab-free formulation of the same step (opt-in variant), timed the same way
    fused = None
    if wl.arch == synth.MLP and precision == hs.HS_BF16:
        hs.hs_set_fused_sync(ctx, True)
        for _ in range(args.warmup):
            hs.hs_step(ctx, params, xd, yd, part, wl.lr, stream=stream, want_loss=False)
        barrier()
        torch.cuda.synchronize()
        f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        f0.record(stream)
        for _ in range(args.steps):
            hs.hs_step(ctx, params, xd, yd, part, wl.lr, stream=stream, want_loss=False)
        f1.record(stream)
        torch.cuda.synchronize()
        fms = max_over_ranks(f0.elapsed_time(f1))
        hs.hs_set_fused_sync(ctx, False)
        fused = {"ms_per_step": fms / args.steps, "value": world * wl.global_batch * args.steps / (fms * 1e-3),
                 "unit": UNIT, "what": "slab-free formulation: worker weights folded into the loss-gradient "
                                       "scale, one all-rows weight-gradient product, update of one gradient"}

    # The slab path (HS_TILE_AVERAGE=0: per-worker weight gradients stored as fp32 slabs, then one
    # reduce+update pass) in two further contexts on the same workload and parameters: with the
    # per-layer updates on the step's stream, which times reduce_update_kernel alone, and in its
    # default form, updates on a side stream beside the remaining products.
    def slab_context(overlap):
        env = {"HS_TILE_AVERAGE": "0", "HS_OVERLAP_UPDATE": "1" if overlap else "0"}
        prev = {k: os.environ.get(k) for k in env}
        os.environ.update(env)
        try:
            return hs.hs_init(wl.arch, wl.dims, wl.workers, wl.global_batch, compute_weights=w, precision=precision,
                              sync=hs.HS_SYNC_CP_WEIGHTED)
        finally:
            for k, v in prev.items():
                if v is None:
                    os.environ.pop(k)
                else:
                    os.environ[k] = v

    alone = None
    slab = None
    if wl.arch == synth.MLP and precision == hs.HS_BF16:
        k2 = max(3, min(args.steps, 10))
        for overlap in (False, True):
            ctx2 = slab_context(overlap)
            p2 = params.clone()
            hs.hs_set_profiling(ctx2, not overlap)
            for _ in range(args.warmup):
                hs.hs_step(ctx2, p2, xd, yd, ctx2.partition, wl.lr, stream=stream, want_loss=False)
            torch.cuda.synchronize()
            hs.hs_read_profile(ctx2)
            a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a0.record(stream)
            for _ in range(k2):
                hs.hs_step(ctx2, p2, xd, yd, ctx2.partition, wl.lr, stream=stream, want_loss=False)
            a1.record(stream)
            torch.cuda.synchronize()
            sms = max_over_ranks(a0.elapsed_time(a1)) / k2
            if overlap:
                slab = {"ms_per_step": sms, "value": world * wl.global_batch / (sms * 1e-3), "unit": UNIT,
                        "what": "slab path (HS_TILE_AVERAGE=0): per-worker weight gradients stored as fp32 "
                                "slabs, reduce+update per layer on a side stream beside the remaining products"}
            else:
                prof2 = hs.hs_read_profile(ctx2)
                alone = {"update_ms": prof2["update"][0] / k2, "step_ms": sms}
            ctx2.close()
            del p2

    # end to end through the public API: every step copies its inputs from pinned host memory and
    # reads its loss back.  Pipelined: hs_stage_inputs copies step t + 1's inputs on a copy stream
    # while step t runs (two staging slots); the unpipelined form lets hs_step copy host inputs on
    # its own stream first.
    xh = torch.from_numpy(x).pin_memory()
    yh = torch.from_numpy(y).pin_memory()
    k_e2e = max(3, min(args.steps, 10))
    copy_stream = torch.cuda.Stream(dev)
    for _ in range(3):   # both staging slots' steps captured before the timed loop
        hs.hs_step(ctx, params, hs.hs_stage_inputs(ctx, xh, yh, stream=copy_stream), None, part, wl.lr,
                   stream=stream, want_loss=True)
    barrier()
    t0 = time.perf_counter()
    nxt = hs.hs_stage_inputs(ctx, xh, yh, stream=copy_stream)
    for i in range(k_e2e):
        cur = nxt
        if i + 1 < k_e2e:
            nxt = hs.hs_stage_inputs(ctx, xh, yh, stream=copy_stream)
        hs.hs_step(ctx, params, cur, None, part, wl.lr, stream=stream, want_loss=True)
    e2e_s = time.perf_counter() - t0
    e2e_s = max_over_ranks(e2e_s)
    for _ in range(2):
        hs.hs_step(ctx, params, xh, yh, part, wl.lr, stream=stream, want_loss=True)
    barrier()
    t0 = time.perf_counter()
    for _ in range(k_e2e):
        hs.hs_step(ctx, params, xh, yh, part, wl.lr, stream=stream, want_loss=True)
    e2e_plain_s = max_over_ranks(time.perf_counter() - t0)
    # the host-to-device copy alone (context for the end-to-end figure): one step's inputs, timed
    # on the copy stream after the step that read the slot
    c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    c0.record(copy_stream)
    staged = hs.hs_stage_inputs(ctx, xh, yh, stream=copy_stream)
    c1.record(copy_stream)
    torch.cuda.synchronize()
    h2d_ms = c0.elapsed_time(c1)
    hs.hs_step(ctx, params, staged, None, part, wl.lr, stream=stream, want_loss=True)   # consume the slot

    P = ctx.P
    peaks = _peaks()
    flops = gemm_flops(wl)
    per_step = {k: v[0] / args.steps for k, v in prof.items()}
    launches = sum(v[1] for v in prof.values())
    gemm_phase = max(("forward", "wgrad", "dgrad"), key=lambda k: per_step[k])
    upd_bytes = update_bytes(wl, P)
    candidates = {k: per_step[k] for k in ("forward", "wgrad", "dgrad", "update")}
    dominant = max(candidates, key=candidates.get)

    launches_per_step = {k: max(1, round(v[1] / args.steps)) for k, v in prof.items()}

    # Which bf16 denominator: the burst figure (cuBLAS timed alone, clocks at their maximum) for a
    # short timed region whose SM clock stayed at its maximum; the sustained one (cuBLAS back to
    # back for seconds, at the power cap) once the timed region is long or the clock dropped.
    timed_s = ms * 1e-3
    at_max = bool(clk) and clk["sm_mhz"] >= 0.97 * clk["sm_max_mhz"]
    burst = timed_s < 2.0 and (at_max or not clk)
    bf16_peak = peaks["bf16"] if burst else peaks["bf16_sust"]
    bf16_kind = f"{peaks['src']} bf16 {'burst' if burst else 'sustained'}"

    def tensor_frac(ach):
        frac = ach / bf16_peak
        # a plain cuBLAS GEMM sets the denominator: far above it means the timing is not the work
        assert frac <= 1.2, f"tensor roofline fraction {frac:.3f} > 1.2 against {bf16_kind} {bf16_peak}"
        return frac

    def gemm_roof(name):
        # per launch: the phase's algorithmic flops and time divided by its launches per step
        ach = flops[name] / (per_step[name] * 1e-3) / 1e12
        # the library's rule: the tile-averaged launch for layers with a 256 x 256 weight tile per
        # SM pair (HS_TILE_AVERAGE=0 disables it, =all applies it to every layer)
        pairs = torch.cuda.get_device_properties(dev).multi_processor_count // 2
        env = os.environ.get("HS_TILE_AVERAGE", "1")
        tiles = [-(-wl.dims[i + 1] // 256) * -(-wl.dims[i] // 256) for i in range(len(wl.dims) - 1)]
        tile_layers = [t >= pairs or env == "all" for t in tiles] if env != "0" else [False] * len(tiles)
        tile = (name == "wgrad" and wl.arch == synth.MLP and precision == hs.HS_BF16 and wl.workers <= 32
                and any(tile_layers))
        traffic = recorded_traffic() if (tile and wl.name == DEFAULT_WORKLOAD) else None
        if tile:
            kernel = ("tc_wgrad_avg_pair_kernel (per-worker weight gradients averaged in tensor memory, "
                      "update fused)" + ("" if all(tile_layers) else "; slab-path tc_gemm_pair_kernel on "
                                         f"{tile_layers.count(False)} of {len(tile_layers)} layers"))
        else:
            kernel = f"tc_gemm_pair_kernel ({name})"
        return {"kernel": kernel, "bound": "tensor", "achieved": ach, "peak": bf16_peak,
                "unit": "TFLOP/s", "frac": tensor_frac(ach), "traffic": traffic,
                "flops_per_launch": flops[name] / launches_per_step[name],
                "launches_per_step": launches_per_step[name],
                "peak_kind": bf16_kind,
                "frac_vs_burst": ach / peaks["bf16"], "frac_vs_sustained": ach / peaks["bf16_sust"]}

    upd_ms = alone["update_ms"] if alone else per_step["update"]
    upd_ach = upd_bytes / (upd_ms * 1e-3) / 1e9
    roof_update = {"kernel": "reduce_update", "bound": "hbm", "achieved": upd_ach, "peak": peaks["hbm"],
                   "unit": "GB/s", "frac": upd_ach / peaks["hbm"], "traffic": None,
                   "peak_kind": f"{peaks['src']} copy bandwidth", "algorithmic_bytes": upd_bytes,
                   "timed": ("slab path (HS_TILE_AVERAGE=0), per-layer updates on the step's stream "
                             "(HS_OVERLAP_UPDATE=0), all P parameters" if alone else "inside the step"),
                   "ms_per_step": upd_ms}
    if alone:
        roof_update["step_ms_slab_path_inline_updates"] = alone["step_ms"]
    roofline = roof_update if dominant == "update" else gemm_roof(dominant)
    gemm_ms = per_step["forward"] + per_step["wgrad"] + per_step["dgrad"]
    gemm_total = sum(flops.values())
    out = None
    if rank == 0:
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            v, desc, cores = oracle_sample(wl)
            cpu = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": desc, "blas": blas_name()}
            one = oracle_one_thread(wl)
            if one is not None:
                cpu["one_thread"] = {"value": one[0], "unit": UNIT, "cores": 1, "sample": one[1]}
        value = world * wl.global_batch * args.steps / (ms * 1e-3)
        out = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16" if precision == hs.HS_BF16 else "f32", "data": "synthetic",
            "config": bench_config(wl, world),
            "roofline": roofline,
            "roofline_gemm_phase": {"bound": "tensor", "achieved": gemm_total / (gemm_ms * 1e-3) / 1e12,
                                    "peak": bf16_peak, "unit": "TFLOP/s", "peak_kind": bf16_kind,
                                    "frac": tensor_frac(gemm_total / (gemm_ms * 1e-3) / 1e12),
                                    "frac_vs_burst": gemm_total / (gemm_ms * 1e-3) / 1e12 / peaks["bf16"],
                                    "frac_vs_sustained": gemm_total / (gemm_ms * 1e-3) / 1e12 / peaks["bf16_sust"],
                                    "flops_per_step": gemm_total},
            "roofline_reduce_update": roof_update,
            "step_ms": {"median": float(np.median(step_ms)), "p10": float(np.percentile(step_ms, 10)),
                        "p90": float(np.percentile(step_ms, 90))},
            "phases_ms_per_step": per_step,
            "phases_pass": {"ms_per_step": profiled_ms,
                            "what": "the same steps with CUDA events around every phase, right after the "
                                    "timed region; phase times and the roofline's kernel time come from it"},
            "gpu_launches": int(launches),
            "cpu_baseline": cpu,
            "e2e": {"value": world * wl.global_batch * k_e2e / e2e_s, "unit": UNIT,
                    "h2d_bytes_per_step": int(x.nbytes + y.nbytes), "d2h_bytes_per_step": 12,
                    "pipelined": "hs_stage_inputs on a copy stream, two slots",
                    "unpipelined_value": world * wl.global_batch * k_e2e / e2e_plain_s,
                    "h2d_ms_per_step_alone": h2d_ms,
                    "h2d_gbs_alone": (x.nbytes + y.nbytes) / (h2d_ms * 1e-3) / 1e9},
            "clocks": clk,
            "straggler_sim": straggler_simulation(),
            "fused_sync_variant": fused,
            "slab_path": slab,
            "graph_replay": graph,
            "heterogeneity_sim": heterogeneity_simulation(ms * 1e-3 / args.steps / wl.global_batch),
            "loss_after": loss,
        }
        print(json.dumps(out), flush=True)
    ctx.close()
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(synth.WORKLOADS))
    ap.add_argument("--impl", default="ours", choices=("ours", "reference"))
    ap.add_argument("--precision", default="bf16", choices=("bf16", "fp32"))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--mlp-dims", default=None,
                    help="profiling aid: an MLP of these comma-separated widths in place of the named "
                         "workload's (with --batch and --workers; lognormal compute weights)")
    ap.add_argument("--batch", type=int, default=None)
    ap.add_argument("--workers", type=int, default=None)
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    wl = synth.WORKLOADS[args.workload]
    if args.mlp_dims:
        import dataclasses
        dims = tuple(int(v) for v in args.mlp_dims.split(","))
        n = args.batch or wl.global_batch
        m = args.workers or wl.workers
        wl = dataclasses.replace(wl, name=f"mlp_{'_'.join(map(str, dims))}_b{n}_m{m}", arch=synth.MLP, dims=dims,
                                 n_classes=dims[-1], global_batch=n, workers=m, weights=None,
                                 weight_kind="lognormal", repartition_every=0)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, wl, rank, world)
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    try:
        run_ours(args, wl, rank, world, local_rank)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
