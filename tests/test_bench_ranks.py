"""bench.py's multi-rank logic on CPU (gloo, world size 2): independent
replicas, the timed region is the max over ranks, throughput sums the ranks'
tokens.  No collective touches the data path."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, ws, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    import bench
    assert bench._dist() == (ws, rank, rank)
    local_ms = 100.0 + 50.0 * rank          # rank 1 is slower
    ms, value = bench.aggregate(local_ms, tokens_per_rank=64, ws=ws, device="cpu")
    bench._barrier(ws)
    q.put((rank, ms, value))
    dist.destroy_process_group()


def test_two_rank_aggregation_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for rank, ms, value in res:
        assert ms == pytest.approx(150.0)
        assert value == pytest.approx(2 * 64 / 0.150)
