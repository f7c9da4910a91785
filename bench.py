#!/usr/bin/env python
"""Throughput of one ASAP round (Eq. A.1: a minibatch SGD step on every
worker, then the stochastic reduce W <- P W) on GB300.

Workload (default): hashed sparse logistic regression, N = 64 workers,
d = 2^20, 50,000 rows per worker with 100 uniform column ids each, B = 512,
a k = 4 random regular mixing graph drawn anew every round.  A step is one
round over one minibatch per worker; the metric is worker-samples/s
(N * B per round).

Printed JSON line (rank 0):
  value      -- worker-samples/s with the shards resident in HBM, CUDA
                events on the context stream around exactly --steps rounds
  e2e        -- the same metric through the public API with the shards in
                pinned host memory: every round copies its minibatch block
                host->device (overlapped with the previous round) and reads
                the round's metrics back device->host
  roofline   -- the stochastic-reduce kernel (the dominant kernel): 8 N d
                algorithmic bytes per launch / its mean CUDA-event duration
  cpu_baseline -- the CPU oracle as it stands, one full round of the same
                workload on the host cores (rank 0, N = 1 only)
With --impl reference the CPU oracle is timed instead (rank 0 only).
Several GPUs (torchrun) run independent replicas; value sums them.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "worker-samples/s per SGD+reduce round; stochastic-reduce HBM GB/s vs peak"
WORKLOAD = dict(name="sparse_logistic_hashed", N=64, d=1 << 20, rows=50000, nnz=100, B=512, lr=0.1, k=4,
                loss="logistic", graph="random_regular", regenerate=True, graph_seed=0)
PROFILE = os.path.join(ROOT, "profiles", "stochastic_reduce_sparse_logistic_hashed.txt")
MIX_SOURCE = os.path.join(ROOT, "paper_1612_08608_gb300", "csrc", "kernels_mix.cu")


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="asap", choices=["asap", "reference"])
    ap.add_argument("--rows", type=int, default=None, help="rows per worker (default: the workload's)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    return ap.parse_args()


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            j = json.load(f)
        return float(j["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def mix_traffic_per_launch():
    """DRAM bytes per reduce launch from the committed ncu summary, or None
    when the kernel source changed since it was captured."""
    try:
        txt = open(PROFILE).read()
    except OSError:
        return None
    src = hashlib.sha256(open(MIX_SOURCE, "rb").read()).hexdigest()[:16]
    vals = {}
    for line in txt.splitlines():
        if ":" in line:
            k, v = line.split(":", 1)
            vals[k.strip()] = v.strip()
    if vals.get("kernel_source_sha256_16") != src:
        return None
    try:
        return float(vals["dram_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while running."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                 "-lms", "50"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in self.lines:
            p = [x.strip() for x in l.split(",")]
            if len(p) < 8:
                continue
            try:
                sm.append(float(p[0]))
                smax.append(float(p[1]))
            except ValueError:
                continue
            for n, v in zip(names, p[4:8]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def make_shards(rows, seed):
    from paper_1612_08608_gb300 import inputs
    return inputs.sparse_logistic_hashed(seed=seed, N=WORKLOAD["N"], d=WORKLOAD["d"], rows=rows,
                                         nnz=WORKLOAD["nnz"])


def oracle_round_sample(sh, W, t, workers):
    """The oracle on a sample of one round: the local step and the reduce
    row of each listed worker (neighbours' half-steps taken from W when not
    in the sample).  Returns the worker-samples processed."""
    import numpy as np
    from oracle import rounds, sgd
    sched = rounds.graph_schedule(WORKLOAD["graph"], WORKLOAD["N"], WORKLOAD["k"], WORKLOAD["graph_seed"],
                                  WORKLOAD["regenerate"])
    nbr, wgt = sched(t)
    H = {}
    for i in workers:
        H[i], _, _ = sgd.sparse_worker_step(W[i], sh.rowptr[i], sh.col[i], sh.val[i], sh.y[i], t, WORKLOAD["B"],
                                            WORKLOAD["loss"], WORKLOAD["lr"])
    for i in workers:
        acc = np.zeros(W.shape[1])
        for m in range(nbr.shape[1]):
            j = int(nbr[i, m])
            acc += wgt[i, m] * (H[j] if j in H else W[j])
    return len(workers) * WORKLOAD["B"]


def cpu_baseline(sh):
    """One full round of the oracle (rounds.sparse_round) as it stands."""
    import numpy as np
    from oracle import rounds
    sched = rounds.graph_schedule(WORKLOAD["graph"], WORKLOAD["N"], WORKLOAD["k"], WORKLOAD["graph_seed"],
                                  WORKLOAD["regenerate"])
    W = np.zeros((WORKLOAD["N"], WORKLOAD["d"]))
    nbr, wgt = sched(0)
    t0 = time.perf_counter()
    rounds.sparse_round(W, sh, 0, WORKLOAD["B"], WORKLOAD["loss"], WORKLOAD["lr"], nbr, wgt)
    dt = time.perf_counter() - t0
    return {"value": WORKLOAD["N"] * WORKLOAD["B"] / dt, "unit": "worker-samples/s", "cores": 1,
            "kind": "oracle", "sample": "one full round (64 workers' SGD steps, the reduce and both metrics), "
                                        "numpy fp64, single thread; %.1f s" % dt}


def config(rows):
    return {"workload": WORKLOAD["name"], "N_workers": WORKLOAD["N"], "d": WORKLOAD["d"], "B": WORKLOAD["B"],
            "rows_per_worker": rows, "nnz_per_row": WORKLOAD["nnz"], "loss": WORKLOAD["loss"],
            "graph": "random_regular k=4, regenerated every round", "lr": WORKLOAD["lr"],
            "l2_flush": "none: inputs larger than L2 (W 2 x 256 MiB, shards > 5 GB)",
            "parallelism": "independent replicas, one per GPU"}


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def run_reference(args):
    import numpy as np
    world, rank, _ = dist_env()
    if rank != 0:
        return
    rows = args.rows or WORKLOAD["rows"]
    sh = make_shards(rows, seed=0)
    W = np.zeros((WORKLOAD["N"], WORKLOAD["d"]))
    t0 = time.perf_counter()
    oracle_round_sample(sh, W, 0, [0])
    t_one = time.perf_counter() - t0
    budget = 150.0
    per_step = max(1, min(WORKLOAD["N"], int(budget / max(1e-3, (args.steps + args.warmup) * t_one))))
    workers = list(range(per_step))
    for s in range(args.warmup):
        oracle_round_sample(sh, W, s, workers)
    units = 0
    t0 = time.perf_counter()
    for s in range(args.steps):
        units += oracle_round_sample(sh, W, args.warmup + s, workers)
    dt = time.perf_counter() - t0
    value = units / dt
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "worker-samples/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config(rows),
            "cpu_baseline": {"value": value, "unit": "worker-samples/s", "cores": 1, "kind": "oracle",
                             "sample": "per step: %d of 64 workers' SGD step and reduce row (numpy fp64, one "
                                       "thread)" % per_step},
            "e2e": {"value": value, "unit": "worker-samples/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_asap(args):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_1612_08608_gb300 import Context

    world, rank, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev_index = int(os.environ.get("CUDA_VISIBLE_DEVICES", str(local)).split(",")[local]) \
        if os.environ.get("CUDA_VISIBLE_DEVICES") else local
    rows = args.rows or WORKLOAD["rows"]
    sh = make_shards(rows, seed=rank)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    def max_over_ranks(x):
        if world == 1:
            return x
        t = torch.tensor([x], dtype=torch.float64, device="cuda")
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    stream = torch.cuda.Stream()
    ctx = Context(WORKLOAD["N"], WORKLOAD["d"], graph_seed=WORKLOAD["graph_seed"], k=WORKLOAD["k"])
    ctx.set_model(WORKLOAD["loss"], batch=WORKLOAD["B"], lr=WORKLOAD["lr"])
    ctx.set_graph(WORKLOAD["graph"], regenerate=WORKLOAD["regenerate"])
    ctx.set_stream(stream)
    ctx.set_shard_residency("host")
    ctx.load_shards(sh)
    N, B, K, Wm = WORKLOAD["N"], WORKLOAD["B"], args.steps, args.warmup
    units_per_step = N * B

    # ---- end to end: shards in pinned host memory, metrics read back ----
    e2e = None
    if not args.no_e2e:
        h2d = 0
        for s in range(Wm):
            ctx.round(1)
            ctx.read_metrics(s, 1)
        r0 = Wm
        barrier()
        t0 = time.perf_counter()
        for s in range(K):
            h2d += ctx.shard_block_bytes(r0 + s)
            ctx.round(1)
            ctx.read_metrics(r0 + s, 1)
        ctx.sync()
        t_e2e = max_over_ranks(time.perf_counter() - t0)
        graph_bytes = N * (WORKLOAD["k"] + 1) * 8
        e2e = {"value": world * units_per_step * K / t_e2e, "unit": "worker-samples/s",
               "h2d_bytes_per_step": h2d / K + graph_bytes, "d2h_bytes_per_step": 8}

    # ---- device resident: the kernel-level number ----
    ctx.set_shard_residency("device")
    ctx.write_params(np.zeros((N, WORKLOAD["d"]), np.float32), 0)
    with torch.cuda.stream(stream):
        for s in range(Wm):
            ctx.round(1)
        ctx.sync()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        sampler = ClockSampler(dev_index)
        barrier()
        sampler.start()
        time.sleep(0.2)
        l0 = ctx.kernel_launches()
        start.record(stream)
        for s in range(K):
            ctx.local_step()
            ev[s][0].record(stream)
            ctx.stochastic_reduce()
            ev[s][1].record(stream)
        end.record(stream)
        stream.synchronize()
        launches = ctx.kernel_launches() - l0
        clocks = sampler.stop()
        ctx.sync()   # surfaces any device-side protocol error
    elapsed_ms = max_over_ranks(start.elapsed_time(end))
    mix_ms = statistics.fmean(a.elapsed_time(b) for a, b in ev)
    last_loss, last_cons = ctx.read_metrics(ctx.read_params()[1] - 1, 1)
    assert np.isfinite(last_loss[0]) and np.isfinite(last_cons[0])

    peak, peak_kind = peaks()
    alg_bytes = 8.0 * N * WORKLOAD["d"]
    achieved = alg_bytes / (mix_ms * 1e-3) / 1e9
    value = world * units_per_step * K / (elapsed_ms * 1e-3)
    line = {"metric": METRIC, "value": value, "unit": "worker-samples/s", "n_gpus": world, "steps": K,
            "warmup": Wm, "ms_per_step": elapsed_ms / K, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic (seeded; stands in for the paper's "
                                                         "RCV1/webspam/splice-site shards)",
            "config": config(rows),
            "roofline": {"kernel": "stochastic reduce (k_mix)", "bound": "hbm", "achieved": achieved, "peak": peak,
                         "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": mix_traffic_per_launch(), "algorithmic_bytes_per_launch": alg_bytes,
                         "mean_launch_ms": mix_ms},
            "reduce_gbs": achieved,
            "e2e": e2e, "gpu_launches": launches, "clocks": clocks}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(sh)
    ctx.close()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_asap(args)


if __name__ == "__main__":
    main()
