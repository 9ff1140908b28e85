"""Multi-process path of bench.py on CPU (gloo, world size 2): the timing is the
maximum over ranks, every rank reaches the barriers, and each rank draws its own
independent batch (weak scaling, no collective on the data path)."""
import multiprocessing as mp
import os
import socket

import numpy as np


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, ws, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(ws), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    try:
        import bench
        from paper_2608_06628_gb300 import workloads as wk
        assert bench.dist_info() == (ws, rank, rank)
        slowest = bench.max_over_ranks(1.5 * (rank + 1), ws)
        bench.barrier(ws)
        wl = bench.rank_workload(wk.C3, rank)
        q.put((rank, slowest, wl.seed, wk.prefix_lengths(wl).tolist()))
    finally:
        dist.destroy_process_group()


def test_two_rank_max_and_independent_batches():
    ws, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, ws, port, q)) for r in range(ws)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=5) for _ in range(ws))
    assert [r[0] for r in res] == [0, 1]
    assert all(r[1] == 3.0 for r in res)             # max over ranks, seen by every rank
    assert res[0][2] != res[1][2]                      # independent seeds per rank
    assert not np.array_equal(res[0][3], res[1][3])    # hence independent ragged batches
