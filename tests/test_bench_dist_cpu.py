"""The N > 1 host logic of bench.py on CPU: two gloo ranks on 127.0.0.1.

The decode path has no data-path collective (replicas only); what runs across
ranks is the timing aggregation: the slowest replica's time, and the whole-job
time per token over all replicas' calls.  The reference arm runs on rank 0 only.
"""
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


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # each replica timed on its own: rank r took 100 + 10 r ms and its e2e 5 - r us
        got = bench._max_over_ranks([100.0 + 10.0 * rank, 5.0 - rank], world)
        out.put((rank, got))
    finally:
        dist.destroy_process_group()


def test_replica_timing_is_the_max_over_two_gloo_ranks():
    port = _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert res[0] == res[1] == [110.0, 5.0]


def test_us_per_token_counts_every_replica():
    sys.path.insert(0, ROOT)
    import bench
    # 2 replicas x 10 steps x 3 calls = 60 tokens in 6 ms -> 100 us per token for the job
    assert bench._us_per_token(6.0, 10, 3, 2) == pytest.approx(100.0)
    assert bench._us_per_token(6.0, 10, 3, 1) == pytest.approx(200.0)
    assert bench._max_over_ranks([3, 1.5], 1) == [3.0, 1.5]


def test_reference_arm_runs_on_rank_zero_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
                        "--steps", "1", "--warmup", "0"], env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""
