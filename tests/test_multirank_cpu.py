"""The N > 1 path of bench.py on the CPU: world_size-2 `gloo` ranks.

A replica run shards sequences across ranks (no data-path collective); the only
exchange is the end-of-run reduction of (time, tokens): the slowest rank's time and
the sum of all ranks' tokens.  The reference arm prints from rank 0 only.
"""
import os
import socket
import subprocess
import sys

import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ids = bench.shard_sequences(rank, 3)
        everyone = [None] * world
        dist.all_gather_object(everyone, ids)
        # rank r took 10 + r ms and emitted 100 * (r + 1) tokens
        ms, tokens = bench.combine_ranks(10.0 + rank, 100 * (rank + 1), world, torch.device("cpu"))
        dist.barrier()
        q.put((rank, everyone, ms, tokens))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_shard_and_combine():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, everyone, ms, tokens in got:
        flat = [i for ids in everyone for i in ids]
        assert sorted(flat) == list(range(6))          # disjoint shards covering every sequence
        assert everyone[rank] == [3 * rank + s for s in range(3)]
        assert ms == 11.0                              # the slowest rank's time
        assert tokens == 300.0                         # every rank's tokens


def test_single_rank_combine_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.combine_ranks(5.0, 7, 1, None) == (5.0, 7)
    assert bench.shard_sequences(0, 2) == [0, 1]


def test_reference_arm_prints_on_rank_zero_only():
    """A non-zero rank of `--impl reference` exits 0 without work or output."""
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1", MASTER_ADDR="127.0.0.1")
    p = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
                        "--steps", "3", "--warmup", "3"], env=env, capture_output=True, text=True, timeout=120)
    assert p.returncode == 0, p.stderr
    assert p.stdout.strip() == ""
