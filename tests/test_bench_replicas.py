"""The N > 1 path of bench.py on the CPU: independent replicas whose timed
region is reduced to the slowest rank, over two gloo ranks; and the
reference arm doing no work on ranks other than 0."""
import os
import socket

import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    dist.barrier()
    got = bench.reduce_max_over_ranks([1.0 + rank, 10.0 - rank, 3.5])
    dist.barrier()
    out.put((rank, got))
    dist.destroy_process_group()


def test_slowest_rank_defines_the_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    results = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert results[0] == results[1] == [2.0, 10.0, 3.5]


def test_single_rank_is_identity():
    assert bench.reduce_max_over_ranks([4.0, 2.0]) == [4.0, 2.0]


def test_reference_arm_idles_on_other_ranks(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    args = bench.argparse.Namespace(steps=1, warmup=3, gpus=2)
    assert bench.run_reference(args) == 0
    assert capsys.readouterr().out == ""
