"""bench.py's multi-rank plumbing on CPU: two gloo ranks, each timing its own independent
problem; the step time reported is the max over ranks and the work is summed (weak scaling)."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench

    r, w, lr = bench.dist_info()
    assert (r, w, lr) == (rank, world, rank)
    bench.barrier()
    ms = bench.reduce_max(1.0 + 2.0 * rank)   # rank 1 is the slow one
    out[rank] = ms
    dist.destroy_process_group()


def test_two_gloo_ranks_reduce_to_the_slowest():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        assert dict(out) == {0: 3.0, 1: 3.0}


def test_work_accounting_per_workload():
    import bench
    import workloads

    w = bench.work(workloads.WORKLOADS["llama8b-5k"])
    assert w["targets"] == 5120 and w["rows"] == 10240
    assert abs(w["gather_bytes"] - 1342177280.0) < 1
    assert abs(w["hash_flops"] - 2 * 10240 * 4096 * 256) < 1
    assert w["match_wordops"] == 5120 * 5120 * 8
