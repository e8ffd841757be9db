"""The N > 1 host logic of bench.py on CPU: world size 2 over gloo
(replicas only: the step does not shard, ranks only agree on timing)."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    elapsed = [120.0, 150.0][rank]
    committed = [900, 950][rank]
    q.put((rank, bench.reduce_ranks(elapsed, committed, "cpu")))
    dist.barrier()
    dist.destroy_process_group()


def test_reduce_ranks_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in range(2):
        assert res[r] == (150.0, 1850.0)   # max time, summed tokens


def test_reference_arm_nonzero_rank_does_nothing(capsys):
    import bench

    class A:
        pass
    assert bench.run_reference(A(), 2, 1) is None
    assert capsys.readouterr().out == ""
