"""The multi-GPU bench path (one replica per rank) on CPU: two gloo ranks on
127.0.0.1 check the slowest-rank reduction, the whole-job rate and that only
rank 0 runs the reference arm."""
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank: int, world: int, port: int, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r took 1 + r seconds of decode and 10 - r ms overall
        got = bench.max_over_ranks([1.0 + rank, 10.0 - rank], world, device="cpu")
        rate = bench.job_tokens_per_s(world, 256, got[0])

        class Args:
            steps, warmup, gpus = 1, 1, world
        ref_rc = bench.run_reference(Args) if rank != 0 else None   # rank != 0 returns at once
        q.put((rank, got, rate, ref_rc, bench.dist_env()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_reduce_to_the_slowest_and_scale_the_rate():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = {}
    for _ in range(world):
        rank, got, rate, ref_rc, env = q.get(timeout=120)
        res[rank] = (got, rate, ref_rc, env)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, (got, rate, ref_rc, env) in res.items():
        assert got == [2.0, 10.0]                  # max over ranks, element-wise
        assert rate == pytest.approx(2 * 256 / 2.0)  # both replicas' tokens over the slowest time
        assert env == (rank, world, rank)
    assert res[1][2] == 0                          # the reference arm: rank 1 exits without work
