"""The N > 1 path of bench.py on the CPU: N independent replicas (rows are independent,
so the path has no data-path collective), two gloo ranks on 127.0.0.1.

The whole-job value is the tokens of every rank over the slowest rank's window; the
reference arm runs on rank 0 only and the other ranks exit 0 without output.
"""
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _replica(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r: a window of 10 + r ms, 100 (r + 1) tokens, a generation of 2 (r + 1) s
        out = bench.aggregate_replicas(10.0 + rank, 100.0 * (rank + 1), 2.0 * (rank + 1), dist, "cpu")
        q.put((rank, out))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_replicas_aggregate_max_time_and_summed_tokens(world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_replica, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = dict(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    want = (10.0 + world - 1, 100.0 * world * (world + 1) / 2, 2.0 * world)
    for r in range(world):
        assert got[r] == pytest.approx(want)
    ms, tokens, _ = want
    # the value bench.py prints: whole-job tokens/s, every rank agreeing on it
    assert tokens / (ms / 1e3) == pytest.approx(1e3 * 100.0 * world * (world + 1) / 2 / (10.0 + world - 1))


def test_single_rank_is_the_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.aggregate_replicas(7.5, 123.0, 4.0, None) == (7.5, 123.0, 4.0)


def test_reference_arm_runs_on_rank_zero_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1",
                        "--warmup", "3"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=120)
    assert r.returncode == 0 and r.stdout.strip() == ""
