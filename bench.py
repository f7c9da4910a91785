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
                the round's metrics back device->host while the next round
                runs
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
NOMINAL_HBM_GBS = 7900.0        # GB300 HBM3e, nominal (the bench's peak is the measured copy rate)
NOMINAL_BF16_TFLOPS = 2250.0    # dense bf16, nominal
WORKLOADS = {
    # hashed sparse logistic regression (the default, HBM-scale)
    "sparse_logistic_hashed": dict(name="sparse_logistic_hashed", N=64, d=1 << 20, rows=50000, nnz=100, B=512,
                                   lr=0.1, k=4, loss="logistic", graph="random_regular", regenerate=True,
                                   graph_seed=0),
    # RCV1-shaped hinge SVM (L2-resident)
    "sparse_hinge_svm": dict(name="sparse_hinge_svm", N=16, d=47236, rows=20000, B=256, lr=0.1, k=2,
                             loss="hinge", graph="random_regular", regenerate=False, graph_seed=0),
    # dense softmax regression on bf16 features (tensor cores)
    "dense_softmax": dict(name="dense_softmax", N=32, d=2048, C=1000, rows=25600, B=512, lr=0.1, k=2,
                          loss="softmax", graph="root", regenerate=False, graph_seed=0),
}
WORKLOAD = WORKLOADS["sparse_logistic_hashed"]
SCHED = {"tau": 1, "kind": "constant", "gamma": 0.0}   # local steps per round, learning-rate schedule
# (workload, kernel) -> (ncu summary holding its DRAM bytes per launch, kernel source the summary was taken on)
TRAFFIC = {
    ("sparse_logistic_hashed", "reduce"): ("stochastic_reduce_sparse_logistic_hashed.txt", "kernels_mix.cu"),
    ("dense_softmax", "dense_grad"): ("dense_gemms_dense_softmax.txt", "kernels_dense.cu"),
    ("sparse_logistic_hashed", "local_step"): ("local_step_sparse_logistic_hashed.txt", "kernels_sparse.cu"),
}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="asap", choices=["asap", "reference"])
    ap.add_argument("--rows", type=int, default=None, help="rows per worker (default: the workload's)")
    ap.add_argument("--workload", default="sparse_logistic_hashed", choices=sorted(WORKLOADS) + ["mix_sweep", "graph_study"],
                    help="mix_sweep: the stochastic reduce alone over N x d x k, one JSON line each")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--min-time", type=float, default=1.0,
                    help="repeat the timed K rounds until this many seconds (at least 3 repeats)")
    ap.add_argument("--sync-mode", default="bsp", choices=["bsp", "notify_ack"],
                    help="how the reduce meets the local step (sparse models)")
    ap.add_argument("--sweep-only", default="", help="mix_sweep subset: 'N,d,k;N,d,k' (k may be N-1)")
    ap.add_argument("--study-rounds", type=int, default=1000, help="graph_study: rounds per graph")
    ap.add_argument("--study-seeds", type=int, default=3, help="graph_study: data and graph seeds")
    ap.add_argument("--study-lr", type=float, default=2.0, help="graph_study: learning rate")
    ap.add_argument("--label-skew", type=float, default=0.8, help="graph_study: label heterogeneity of the shards")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--local-steps", type=int, default=1, help="minibatch steps per worker per round (sparse)")
    ap.add_argument("--lr-schedule", default="constant", choices=["constant", "inverse"])
    ap.add_argument("--gamma", type=float, default=0.0, help="eta_k = lr / (1 + gamma k) for --lr-schedule inverse")
    return ap.parse_args()


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            j = json.load(f)
        return float(j["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def code_fingerprint(path):
    """sha256 (16 hex digits) of a source file with // comments and blank
    lines removed: a comment edit leaves it, any code change alters it."""
    import re
    lines = []
    for line in open(path, encoding="utf-8").read().splitlines():
        line = re.sub(r"//.*$", "", line).rstrip()
        if line:
            lines.append(line)
    return hashlib.sha256("\n".join(lines).encode()).hexdigest()[:16]


def traffic_per_launch(workload, kernel, key="dram_bytes_per_launch"):
    """DRAM bytes per launch of the kernel (or another `key` of the summary)
    from its committed ncu summary, or None when there is none or the kernel
    source changed since it was taken."""
    if (workload, kernel) not in TRAFFIC:
        return None
    prof, source = TRAFFIC[(workload, kernel)]
    try:
        txt = open(os.path.join(ROOT, "profiles", prof)).read()
    except OSError:
        return None
    src = code_fingerprint(os.path.join(ROOT, "paper_1612_08608_gb300", "csrc", source))
    vals = {}
    for line in txt.splitlines():
        if ":" in line:
            k, v = line.split(":", 1)
            vals[k.strip()] = v.strip()
    if vals.get("kernel_code_sha256_16") != src:
        return None
    try:
        return float(vals[key].split()[0])
    except (KeyError, ValueError, IndexError):
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
    w = WORKLOAD
    if w["name"] == "sparse_logistic_hashed":
        return inputs.sparse_logistic_hashed(seed=seed, N=w["N"], d=w["d"], rows=rows, nnz=w["nnz"])
    if w["name"] == "sparse_hinge_svm":
        return inputs.sparse_hinge_svm(seed=seed, N=w["N"], d=w["d"], rows=rows)
    return inputs.dense_softmax(seed=seed, N=w["N"], d=w["d"], C=w["C"], rows=rows)


def kernel_work(sh):
    """Algorithmic work of one launch of each kernel kind: (unit, amount, bound)
    or (unit, amount, bound, flops) when a memory-bound kernel also runs a
    GEMM.  Sparse byte counts use the mean minibatch over a sample of batches."""
    import numpy as np
    w = WORKLOAD
    N, B, d = w["N"], w["B"], w["d"]
    ld = (d * w.get("C", 1) + 63) // 64 * 64
    out = {}
    if w["loss"] == "softmax":
        C = w["C"]
        out["dense_fwd"] = ("TFLOP/s", 2.0 * N * B * C * d, "tensor")
        # The gradient GEMM carries the fused fp32 master update (read + write
        # 8 B per parameter) plus its bf16 operands R^T and X_b^T: HBM-bound.
        cpad = (C + 255) // 256 * 256
        out["dense_grad"] = ("GB/s", 8.0 * N * C * d + 2.0 * N * B * (cpad + d), "hbm", 2.0 * N * C * d * B)
        out["reduce"] = ("GB/s", 10.0 * N * ld, "hbm")     # fp32 read + write, bf16 copy write
        return out
    rng = np.random.default_rng(0)
    nnz = touched = 0.0
    samples = 16
    for _ in range(samples):
        i = int(rng.integers(N))
        t = int(rng.integers(sh.n_rows(i) // B))
        rp = sh.rowptr[i][t * B:(t + 1) * B + 1]
        nnz += rp[-1] - rp[0]
        touched += np.unique(sh.col[i][rp[0]:rp[-1]]).shape[0]
    nnz, touched = nnz * N / samples, touched * N / samples
    # the fused local step reads every entry once (list position, value,
    # row, segment slot: 12 B), the w value and writes the column sum of
    # every distinct (worker, column) (8 B), and the labels
    out["local_step"] = ("GB/s", 12.0 * nnz + 8.0 * touched + 4.0 * N * B, "hbm")
    out["reduce"] = ("GB/s", 8.0 * N * ld, "hbm")
    # local steps before the round's last: the update scatter and the next gather
    out["apply"] = ("GB/s", 16.0 * touched, "hbm")    # list + column sum read, w read + write per column
    out["gather"] = ("GB/s", 12.0 * touched, "hbm")   # list + w read, w value written per column
    return out


def _sched():
    from oracle import rounds
    w = WORKLOAD
    return rounds.graph_schedule(w["graph"], w["N"], w["k"], w["graph_seed"], w["regenerate"])


def _lr_at(k):
    from oracle import sgd
    return sgd.learning_rate(SCHED["kind"], WORKLOAD["lr"], SCHED["gamma"], k)


def oracle_round_sample(sh, W, t, workers):
    """The oracle on a sample of one round: the local steps and the reduce
    row of each listed worker (neighbours' half-steps taken from W when not
    in the sample).  Returns the worker-samples processed."""
    import numpy as np
    from oracle import sgd
    w = WORKLOAD
    tau = SCHED["tau"]
    nbr, wgt = _sched()(t)
    H = {}
    for i in workers:
        if w["loss"] == "softmax":
            Wm = W[i].astype(np.float32).reshape(w["C"], w["d"])
            H[i] = sgd.softmax_worker_step(Wm, sh.X[i], sh.y[i], t, w["B"], _lr_at(t))[0].reshape(-1)
        else:
            h = W[i]
            for j in range(tau):
                k = t * tau + j
                h, _, _ = sgd.sparse_worker_step(h, sh.rowptr[i], sh.col[i], sh.val[i], sh.y[i], k, w["B"],
                                                 w["loss"], _lr_at(k))
            H[i] = h
    for i in workers:
        acc = np.zeros(W.shape[1])
        for m in range(nbr.shape[1]):
            j = int(nbr[i, m])
            acc += wgt[i, m] * (H[j] if j in H else W[j])
    return len(workers) * w["B"] * (1 if w["loss"] == "softmax" else tau)


def cpu_baseline(sh):
    """One full round of the oracle as it stands."""
    import numpy as np
    from oracle import rounds
    w = WORKLOAD
    P = w["d"] * w.get("C", 1)
    W = np.zeros((w["N"], P))
    nbr, wgt = _sched()(0)
    t0 = time.perf_counter()
    tau = 1 if w["loss"] == "softmax" else SCHED["tau"]
    if w["loss"] == "softmax":
        rounds.softmax_round(W.astype(np.float32), sh, 0, w["B"], w["lr"], nbr, wgt)
    else:
        rounds.sparse_round(W, sh, 0, w["B"], w["loss"], None, nbr, wgt, tau=tau, lr_at=_lr_at)
    dt = time.perf_counter() - t0
    return {"value": w["N"] * w["B"] * tau / dt, "unit": "worker-samples/s", "cores": 1,
            "kind": "oracle", "sample": "one full round (%d workers' SGD steps, the reduce and both metrics), "
                                        "numpy fp64%s; %.1f s" % (w["N"], ", BLAS matmuls" if w["loss"] == "softmax"
                                                                   else ", single thread", dt)}


# ---- the oracle on all host cores (spawned processes; shared-memory W) ----
def _par_attach(name, shape):
    import numpy as np
    from multiprocessing import shared_memory
    shm = shared_memory.SharedMemory(name=name)
    return shm, np.ndarray(shape, dtype=np.float64, buffer=shm.buf)


def _par_step(task):
    """One worker's local SGD step of round 0 (oracle), written into the
    shared half-step matrix H.  The minibatch is passed as its own rows."""
    import numpy as np
    from oracle import sgd
    kind, i, batch, B, lr, loss, hname, shape = task
    shm, H = _par_attach(hname, shape)
    if kind == "softmax":
        Xb, yb, C, d = batch
        h, lval = sgd.softmax_worker_step(np.zeros((C, d), np.float32), Xb, yb, 0, B, lr)
        H[i] = h.reshape(-1)
    else:
        rp, col, val, y = batch
        h, lval, _ = sgd.sparse_worker_step(np.zeros(shape[1]), rp, col, val, y, 0, B, loss, lr)
        H[i] = h
    del H
    shm.close()
    return lval


def _par_reduce(task):
    """Rows r0 .. r1 of W = P H (oracle), written into the shared W."""
    from oracle import reduce
    r0, r1, nbr, wgt, hname, wname, shape = task
    shm_h, H = _par_attach(hname, shape)
    shm_w, W = _par_attach(wname, shape)
    W[r0:r1] = reduce.stochastic_reduce(H, nbr, wgt)
    del H, W
    shm_h.close()
    shm_w.close()
    return r1 - r0


def cpu_baseline_all_cores(sh):
    """One round of the oracle on every host core: the workers' SGD steps in
    parallel, then the rows of the reduce in parallel (a pool of spawned
    processes sharing H and W), the consensus error in the parent.  Same
    arithmetic as the single-thread oracle, each worker's step sequential."""
    import multiprocessing as mp
    import numpy as np
    from multiprocessing import shared_memory
    from oracle import reduce
    w = WORKLOAD
    if w["loss"] != "softmax" and SCHED["tau"] != 1:
        return None
    N, B = w["N"], w["B"]
    P = w["d"] * w.get("C", 1)
    cores = os.cpu_count() or 1
    shape = (N, P)
    shm_h = shared_memory.SharedMemory(create=True, size=8 * N * P)
    shm_w = shared_memory.SharedMemory(create=True, size=8 * N * P)
    try:
        nbr, wgt = _sched()(0)
        tasks = []
        for i in range(N):
            if w["loss"] == "softmax":
                batch = (sh.X[i][:B].copy(), sh.y[i][:B].copy(), w["C"], w["d"])
            else:
                rp = sh.rowptr[i][:B + 1]
                batch = (rp - rp[0], sh.col[i][rp[0]:rp[-1]].copy(), sh.val[i][rp[0]:rp[-1]].copy(), sh.y[i][:B].copy())
            tasks.append((w["loss"], i, batch, B, w["lr"], w["loss"], shm_h.name, shape))
        blk = max(1, -(-N // cores))
        red = [(r0, min(N, r0 + blk), np.asarray(nbr[r0:r0 + blk]), np.asarray(wgt[r0:r0 + blk]), shm_h.name,
                shm_w.name, shape) for r0 in range(0, N, blk)]
        with mp.get_context("spawn").Pool(min(cores, N)) as pool:
            pool.map(_par_step, tasks[:min(cores, N)])          # start-up and imports, untimed
            t0 = time.perf_counter()
            pool.map(_par_step, tasks, chunksize=1)
            pool.map(_par_reduce, red, chunksize=1)
            Wv = np.ndarray(shape, dtype=np.float64, buffer=shm_w.buf)
            reduce.consensus_error(Wv)
            dt = time.perf_counter() - t0
            del Wv
    finally:
        shm_h.close()
        shm_h.unlink()
        shm_w.close()
        shm_w.unlink()
    return {"value": N * B / dt, "unit": "worker-samples/s", "cores": min(cores, N), "kind": "oracle",
            "sample": "one full round on all host cores: %d workers' SGD steps and the reduce rows in %d spawned "
                      "processes, the consensus error in the parent; numpy fp64; %.2f s" % (N, min(cores, N), dt)}


def config(rows):
    w = WORKLOAD
    c = {"workload": w["name"], "N_workers": w["N"], "d": w["d"], "B": w["B"], "rows_per_worker": rows,
         "loss": w["loss"], "lr": w["lr"],
         "graph": "%s k=%d%s" % (w["graph"], w["k"], ", regenerated every round" if w["regenerate"] else ""),
         "parallelism": "independent replicas, one per GPU",
         "sync": SCHED.get("sync", "bsp"),
         "local_steps": SCHED["tau"], "lr_schedule": SCHED["kind"] if SCHED["kind"] == "constant"
         else "lr / (1 + %g k)" % SCHED["gamma"]}
    if "nnz" in w:
        c["nnz_per_row"] = w["nnz"]
    if "C" in w:
        c["classes"] = w["C"]
    c["l2_flush"] = {"sparse_logistic_hashed": "none: inputs larger than L2 (W 2 x 256 MiB, shards > 5 GB)",
                     "dense_softmax": "none: inputs larger than L2 (fp32 W 2 x 262 MB, features 6.7 GB)",
                     "sparse_hinge_svm": "none: the whole working set (~25 MB) stays in L2 by design"}[w["name"]]
    return c


def reduce_max(x, device="cpu"):
    """Max of a per-rank scalar over all ranks (identity without a process
    group).  gloo reduces CPU tensors, NCCL CUDA tensors."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world, units_per_step, steps, seconds_max):
    """Units all ranks processed (each rank runs the same replica workload)
    divided by the slowest rank's time."""
    return world * units_per_step * steps / seconds_max


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
    W = np.zeros((WORKLOAD["N"], WORKLOAD["d"] * WORKLOAD.get("C", 1)))
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
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded)",
            "config": config(rows),
            "cpu_baseline": {"value": value, "unit": "worker-samples/s", "cores": 1, "kind": "oracle",
                             "sample": "per step: %d of %d workers' SGD step and reduce row (numpy fp64)"
                                       % (per_step, WORKLOAD["N"])},
            "e2e": {"value": value, "unit": "worker-samples/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def peaks_all():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            j = json.load(f)
        return {"hbm": (float(j["hbm_gbs"]), "measured"),
                "tensor": (float(j.get("bf16_tflops_sustained", j["bf16_tflops"])), "measured (sustained)")}
    except Exception:
        return {"hbm": (6800.0, "fallback"), "tensor": (1700.0, "fallback (sustained)")}


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
    w = WORKLOAD
    rows = args.rows or w["rows"]
    sh = make_shards(rows, seed=rank)
    dense = w["loss"] == "softmax"

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    def max_over_ranks(x):
        return reduce_max(x, device="cuda")

    stream = torch.cuda.Stream()
    ctx = Context(w["N"], w["d"], graph_seed=w["graph_seed"], k=w["k"])
    ctx.set_model(w["loss"], batch=w["B"], lr=w["lr"], num_classes=w.get("C", 1))
    ctx.set_schedule(local_steps=SCHED["tau"], lr_schedule=SCHED["kind"], gamma=SCHED["gamma"])
    ctx.set_graph(w["graph"], regenerate=w["regenerate"])
    ctx.set_stream(stream)
    if not dense:
        ctx.set_sync_mode(args.sync_mode)
    N, B, K, Wm = w["N"], w["B"], args.steps, args.warmup
    units_per_step = N * B * SCHED["tau"]

    # ---- end to end: shards in pinned host memory, metrics read back ----
    e2e = None
    if dense:
        ctx.load_dense_shards(sh)
        e2e = {"value": None, "unit": "worker-samples/s", "h2d_bytes_per_step": None, "d2h_bytes_per_step": None,
               "note": "dense shards are device-resident only in this version"}
    else:
        ctx.set_shard_residency("host")
        ctx.load_shards(sh)
        if not args.no_e2e:
            h2d = 0
            for s in range(Wm):
                ctx.round(1)
                ctx.read_metrics(s, 1)
            r0 = Wm
            reps = []
            # Repeats of exactly K rounds (at least three, at least one second
            # in all), the median reported.  Round s's loss and consensus
            # error are read back while round s + 1 runs (the read waits for
            # round s only); the last one after the loop, inside the timed
            # region.
            while len(reps) < 3 or (sum(reps) < args.min_time and len(reps) < 5000):
                h2d = 0
                barrier()
                t0 = time.perf_counter()
                for s in range(K):
                    h2d += ctx.shard_block_bytes(r0 + s)
                    ctx.round(1)
                    if s > 0:
                        ctx.read_metrics(r0 + s - 1, 1)
                ctx.read_metrics(r0 + K - 1, 1)
                ctx.sync()
                reps.append(time.perf_counter() - t0)
                r0 += K
            t_e2e = max_over_ranks(statistics.median(reps))
            graph_bytes = N * (w["k"] + 1) * 8 if w["regenerate"] else 0
            # d2h per step: loss and consensus error (8 B) and the device error word (4 B)
            e2e = {"value": whole_job_rate(world, units_per_step, K, t_e2e), "unit": "worker-samples/s",
                   "h2d_bytes_per_step": h2d / K + graph_bytes, "d2h_bytes_per_step": 12, "repeats": len(reps)}
        ctx.set_shard_residency("device")

    # ---- device resident: the kernel-level number ----
    ctx.write_params(np.zeros((N, ctx.P), np.float32), 0)
    for s in range(Wm):
        ctx.round(1)
    ctx.sync()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(dev_index)
    ctx.set_kernel_timing(True)
    barrier()
    sampler.start()
    time.sleep(0.2)
    # Repeats of exactly K rounds each, bracketed by a barrier and a device
    # synchronisation and timed with CUDA events on the context stream; as
    # many repeats as fill at least one second (at least three), and the
    # median repeat is the number reported.
    l0 = ctx.kernel_launches()
    rep_ms = []
    t_wall = time.perf_counter()
    while len(rep_ms) < 3 or (sum(rep_ms) < 1000.0 * args.min_time and len(rep_ms) < 5000):
        barrier()
        start.record(stream)
        for s in range(K):
            ctx.round(1)
        end.record(stream)
        stream.synchronize()
        rep_ms.append(start.elapsed_time(end))
    t_wall = time.perf_counter() - t_wall
    launches = (ctx.kernel_launches() - l0) // len(rep_ms)
    clocks = sampler.stop()
    ctx.sync()   # surfaces any device-side protocol error
    times = ctx.read_kernel_times()
    ctx.set_kernel_timing(False)
    elapsed_ms = max_over_ranks(statistics.median(rep_ms))
    last_loss, last_cons = ctx.read_metrics(ctx.read_params()[1] - 1, 1)
    assert np.isfinite(last_loss[0]) and np.isfinite(last_cons[0])

    pk = peaks_all()
    work = kernel_work(sh)
    kernels = {}
    for name, wk in work.items():
        unit, amount, bound = wk[:3]
        n, ms = times[name]
        if n == 0:
            continue
        mean_ms = ms / n
        scale = 1e12 if unit == "TFLOP/s" else 1e9
        achieved = amount / (mean_ms * 1e-3) / scale
        peak, kind = pk[bound]
        kernels[name] = {"bound": bound, "unit": unit, "achieved": achieved, "peak": peak, "peak_kind": kind,
                         "frac": achieved / peak, "mean_launch_ms": mean_ms, "launches": n,
                         "share": ms / max(1e-9, sum(v[1] for v in times.values())),
                         "algorithmic_per_launch": amount}
        if len(wk) > 3:   # the GEMM inside a memory-bound kernel, against the tensor peak
            tf = wk[3] / (mean_ms * 1e-3) / 1e12
            kernels[name]["tensor_tflops"] = tf
            kernels[name]["tensor_frac"] = tf / pk["tensor"][0]
    dom = max(kernels, key=lambda k: kernels[k]["share"])
    kd = kernels[dom]
    roof = {"kernel": dom, "bound": kd["bound"], "achieved": kd["achieved"], "peak": kd["peak"],
            "peak_kind": kd["peak_kind"], "unit": kd["unit"], "frac": kd["frac"],
            "traffic": traffic_per_launch(w["name"], dom),
            "frac_of_nominal": kd["achieved"] / (NOMINAL_HBM_GBS if kd["unit"] == "GB/s" else NOMINAL_BF16_TFLOPS),
            "ncu_dram_throughput_pct": traffic_per_launch(w["name"], dom, "ncu_dram_throughput_pct"),
            "algorithmic_per_launch": kd["algorithmic_per_launch"], "mean_launch_ms": kd["mean_launch_ms"]}
    value = whole_job_rate(world, units_per_step, K, elapsed_ms * 1e-3)
    line = {"metric": METRIC, "value": value, "unit": "worker-samples/s", "n_gpus": world, "steps": K,
            "warmup": Wm, "ms_per_step": elapsed_ms / K, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16 GEMM inputs, f32 accumulate and master" if dense else "f32",
            "data": "synthetic (seeded; stands in for the paper's %s)" %
                    ("CIFAR-10 CNN workload" if dense else "RCV1/webspam/splice-site shards"),
            "config": config(rows),
            "roofline": roof,
            "reduce_gbs": kernels["reduce"]["achieved"] if "reduce" in kernels else None,
            "kernels": kernels, "e2e": e2e, "gpu_launches": launches, "clocks": clocks,
            "timing": {"repeats": len(rep_ms), "rounds_per_repeat": K, "timed_s": sum(rep_ms) / 1e3,
                       "wall_s": t_wall, "repeat_ms_min_median_max": [min(rep_ms), statistics.median(rep_ms),
                                                                      max(rep_ms)],
                       "rule": "median of repeats of exactly --steps rounds, repeated until >= %g s and >= 3"
                               % args.min_time}}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(sh)
        par = cpu_baseline_all_cores(sh)
        if par is not None:
            line["cpu_baseline"]["all_cores"] = par
    ctx.close()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_mix_sweep(args):
    """The stochastic reduce alone (W <- P W) over the sweep N in {8, 32, 128,
    256} x d in {1e5, 1e6, 1e7} x k in {1, 2, 4, N-1}: per combination the
    mean CUDA-event time of one reduce launch over --steps launches (after
    --warmup), its algorithmic bytes 8 N ld, GB/s against the measured HBM
    peak, and a check of the consensus error: it must contract by at most
    sigma_2(P) per round (Appendix A), and the complete graph reaches
    consensus in one round."""
    import numpy as np
    import torch
    from paper_1612_08608_gb300 import Context, inputs

    torch.cuda.set_device(0)
    peak, kind = peaks()
    only = None if not args.sweep_only else {tuple(int(v) if v != "N-1" else v for v in c.split(","))
                                            for c in args.sweep_only.split(";")}
    for d in (100000, 1000000, 10000000):
        for N in (8, 32, 128, 256):
            for k in (1, 2, 4, "N-1"):
                if only is not None and (N, d, k) not in only:
                    continue
                kk = N - 1 if k == "N-1" else k
                gk = {1: "ring", N - 1: "complete"}.get(kk, "random_regular")
                ctx = Context(N, d, graph_seed=1, k=kk)
                ctx.set_graph(gk)
                W0 = inputs.mixing_params_device(seed=N * 31 + kk, N=N, d=d)
                ctx.write_params_device(W0, 0)
                del W0
                torch.cuda.empty_cache()
                for _ in range(args.warmup):
                    ctx.stochastic_reduce()
                ctx.sync()
                ctx.set_kernel_timing(True)
                for _ in range(args.steps):
                    ctx.stochastic_reduce()
                ctx.sync()
                n, ms = ctx.read_kernel_times()["reduce"]
                ctx.set_kernel_timing(False)
                rounds = args.warmup + args.steps
                _, cons = ctx.read_metrics(0, rounds)
                nbr, wgt = ctx.get_graph(0)
                s2 = sigma2(nbr, wgt)
                ok = bool(np.all(np.isfinite(cons)))
                for t in range(1, rounds):
                    if cons[t - 1] > 1e-5 * cons[0]:
                        ok = ok and cons[t] <= s2 * cons[t - 1] * (1 + 1e-4) + 1e-6 * cons[0]
                if gk == "complete":
                    ok = ok and float(np.max(cons)) == 0.0
                ld = (d + 63) // 64 * 64
                t_ms = ms / max(n, 1)
                gbs = 8.0 * N * ld / (t_ms * 1e-3) / 1e9
                print(json.dumps({"workload": "mix_sweep", "N": N, "d": d, "k": kk, "graph": gk,
                                  "ms_per_reduce": t_ms, "algorithmic_bytes": 8 * N * ld, "GB/s": gbs,
                                  "peak": peak, "peak_kind": kind, "frac": gbs / peak, "launches": n,
                                  "consensus_contracts_by_sigma2": bool(ok)}), flush=True)
                ctx.close()


# ---- graph comparison (Section 6.1): rounds and bytes to a target loss ----
STUDY_GRAPHS = (("complete", "complete", None, False), ("root", "root", 2, False), ("ring", "ring", 1, False),
                ("random_regular_k2", "random_regular", 2, False),
                ("random_regular_k4_regen", "random_regular", 4, True))


def hinge_loss_at(w, rowptr, col, val, y):
    """Mean hinge loss max(0, 1 - y x.w) of a CSR set at w (evaluation)."""
    import numpy as np
    row_of = np.repeat(np.arange(rowptr.shape[0] - 1), np.diff(rowptr))
    m = np.bincount(row_of, weights=val.astype(np.float64) * w[col], minlength=rowptr.shape[0] - 1)
    return float(np.maximum(0.0, 1.0 - y.astype(np.float64) * m).mean())


def study_target(f0, curve, frac=0.9):
    """The loss at which a curve has made `frac` of its total drop from f0
    to its lowest value."""
    return f0 - frac * (f0 - min(curve))


def first_reaching(rounds, curve, target):
    """First round of `rounds` whose value is at or below target (None if none)."""
    for r, v in zip(rounds, curve):
        if v <= target:
            return r
    return None


def sigma2(nbr, wgt):
    """Second singular value of the mixing matrix written out from its rows."""
    import numpy as np
    N = nbr.shape[0]
    P = np.zeros((N, N))
    for i in range(N):
        for m in range(nbr.shape[1]):
            P[i, nbr[i, m]] += wgt[i, m]
    return float(np.linalg.svd(P, compute_uv=False)[1]) if N > 1 else 0.0


def run_graph_study(args):
    """Every graph of STUDY_GRAPHS trains the same RCV1-shaped hinge SVM on
    shards that are heterogeneous by label, from W = 0.  Every `every`
    rounds the average model wbar is evaluated (mean hinge loss on 256
    held-out rows of every worker).  The target is the loss at which the
    complete graph (the all-reduce) has made 90 % of its drop over
    --study-rounds rounds; per graph and seed the rounds to that target, the
    bytes each worker receives to reach it (k d 4 per round), sigma_2 of its
    mixing matrix and the median per-round ratio of its consensus error."""
    import numpy as np
    import torch
    from paper_1612_08608_gb300 import Context, inputs
    torch.cuda.set_device(0)
    N, B, every = 16, 256, 10
    rows, T = args.rows or 4096, args.study_rounds
    summary = {}
    for seed in range(args.study_seeds):
        sh = inputs.sparse_hinge_svm(seed=seed, N=N, rows=rows + 256, label_skew=args.label_skew)
        train = inputs.SparseShards(d=sh.d)
        ev_rp, ev_col, ev_val, ev_y = [np.zeros(1, np.int64)], [], [], []
        for i in range(N):
            rp = sh.rowptr[i]
            train.rowptr.append(rp[:rows + 1].copy())
            train.col.append(sh.col[i][:rp[rows]])
            train.val.append(sh.val[i][:rp[rows]])
            train.y.append(sh.y[i][:rows])
            ev_rp.append(rp[rows + 1:] - rp[rows] + ev_rp[-1][-1])
            ev_col.append(sh.col[i][rp[rows]:])
            ev_val.append(sh.val[i][rp[rows]:])
            ev_y.append(sh.y[i][rows:])
        ev = (np.concatenate(ev_rp), np.concatenate(ev_col), np.concatenate(ev_val), np.concatenate(ev_y))
        curves = {}
        for name, kind, k, regen in STUDY_GRAPHS:
            kk = N - 1 if k is None else k
            ctx = Context(N, sh.d, graph_seed=seed, k=kk)
            ctx.set_model("hinge", batch=B, lr=args.study_lr)
            ctx.set_graph(kind, regenerate=regen)
            ctx.load_shards(train)
            xs, fs = [0], [hinge_loss_at(np.zeros(sh.d), *ev)]
            for t in range(every, T + 1, every):
                ctx.round(every)
                W, _ = ctx.read_params()
                xs.append(t)
                fs.append(hinge_loss_at(W.astype(np.float64).mean(axis=0), *ev))
            _, cons = ctx.read_metrics(0, T)
            nbr, wgt = ctx.get_graph(0)
            ratio = float(np.median(cons[1:] / np.maximum(cons[:-1], 1e-30)))
            curves[name] = (kk, xs, fs, sigma2(nbr, wgt), ratio)
            ctx.close()
        target = study_target(curves["complete"][2][0], curves["complete"][2])
        for name, (kk, xs, fs, s2, ratio) in curves.items():
            hit = first_reaching(xs, fs, target)
            line = {"workload": "graph_study", "seed": seed, "graph": name, "k": kk, "sigma2": s2,
                    "spectral_gap": 1.0 - s2, "target_loss": target, "rounds_to_target": hit,
                    "bytes_per_worker_round": kk * sh.d * 4,
                    "bytes_per_worker_to_target": None if hit is None else kk * sh.d * 4 * hit,
                    "final_loss": fs[-1], "median_consensus_ratio": ratio, "lr": args.study_lr,
                    "label_skew": args.label_skew, "rounds": T}
            print(json.dumps(line), flush=True)
            summary.setdefault(name, []).append(hit)
    print(json.dumps({"workload": "graph_study_summary",
                      "rounds_to_target_per_seed": summary}), flush=True)


def main():
    global WORKLOAD
    args = parse()
    if args.workload == "mix_sweep":
        run_mix_sweep(args)
        return
    if args.workload == "graph_study":
        run_graph_study(args)
        return
    WORKLOAD = WORKLOADS[args.workload]
    SCHED.update(tau=args.local_steps, kind=args.lr_schedule, gamma=args.gamma,
                 sync=args.sync_mode if WORKLOAD["loss"] != "softmax" else "bsp")
    if WORKLOAD["loss"] == "softmax" and args.local_steps != 1:
        raise SystemExit("dense_softmax takes one local step per round")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_asap(args)


if __name__ == "__main__":
    main()
