"""Multi-rank host logic of bench.py on CPU (gloo, world size 2): ranks
time their own replica, the reported rate uses the slowest rank, rank 0
alone prints, and the reference arm runs on rank 0 only."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, elapsed, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    m = bench.reduce_max(elapsed[rank])
    rate = bench.whole_job_rate(world, 64 * 512, 100, m)
    dist.barrier()
    dist.destroy_process_group()
    out.put((rank, m, rate))


def test_max_over_ranks_and_whole_job_rate_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    elapsed = [0.50, 0.75]
    procs = [ctx.Process(target=_worker, args=(r, 2, port, elapsed, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, m, rate in res:
        assert m == pytest.approx(0.75)
        assert rate == pytest.approx(2 * 64 * 512 * 100 / 0.75)


def test_single_process_has_no_collective():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max(0.3) == 0.3
    assert bench.whole_job_rate(1, 10, 5, 2.0) == 25.0


@pytest.mark.parametrize("rank", [0, 1])
def test_reference_arm_prints_on_rank0_only(rank):
    env = dict(os.environ, WORLD_SIZE="2", RANK=str(rank), LOCAL_RANK=str(rank), MASTER_ADDR="127.0.0.1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload",
                        "sparse_hinge_svm", "--rows", "512", "--steps", "2", "--warmup", "1"],
                       capture_output=True, text=True, env=env, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    if rank == 0:
        j = json.loads(lines[-1])
        assert j["impl"] == "reference" and j["value"] > 0 and j["n_gpus"] == 1
        assert j["e2e"]["h2d_bytes_per_step"] == 0 and j["cpu_baseline"]["kind"] == "oracle"
    else:
        assert lines == []
