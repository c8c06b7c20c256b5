"""The multi-rank path of bench.py on CPU: two gloo ranks (127.0.0.1), the
slowest-rank time, the weak-scaling aggregate and the reference arm's launch
contract under torchrun. No GPU."""
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    r, w, _ = bench.dist_setup(world, backend="gloo")
    bench.barrier(w)
    slowest = bench.max_over_ranks(10.0 * (rank + 1), w)  # ranks take 10 and 20 ms
    rate, ms = bench.whole_job(1e9, w, slowest, steps=4)
    q.put((rank, r, w, slowest, rate, ms))
    dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_rank_and_sum_the_work():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, (q_rank, got_rank, w, slowest, rate, ms) in enumerate(res):
        assert q_rank == rank and got_rank == rank and w == 2
        assert slowest == 20.0            # the max over ranks, on every rank
        assert ms == 5.0                   # 20 ms over 4 steps
        assert rate == pytest.approx(2 * 1e9 / 5e-3)  # both ranks' units / slowest time


def test_whole_job_single_rank():
    sys.path.insert(0, ROOT)
    import bench
    rate, ms = bench.whole_job(3.0, 1, 40.0, 8)
    assert ms == 5.0 and rate == pytest.approx(3.0 / 5e-3)


def test_reference_arm_under_torchrun_prints_once():
    port = _free_port()
    env = dict(os.environ, OMP_NUM_THREADS="2")
    out = subprocess.run(
        [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
         "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py",
         "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0"],
        cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1  # rank 0 alone runs and prints
    import json
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
