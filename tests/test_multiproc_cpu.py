"""The N>1 path on CPU: world-size-2 gloo ranks each simulate their own instance shard (the CPU
oracle stands in for the GPU here), the timing is reduced with MAX, and the results gathered on
rank 0 equal one process simulating both shards."""
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, out_dir):
    import time

    import torch.distributed as dist

    from oracle import plain
    from paper_2508_14544_gb300 import workloads as W
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ids = W.rank_instances("c1", rank)
    w = W.make_workload("c1", ids)
    t0 = time.perf_counter()
    tel = []
    for pol in (0, 1, 2):
        tel.append(int(plain.run_workload(pol, w)["total_latency"].sum()))
    dt = torch.tensor([time.perf_counter() - t0], dtype=torch.float64)
    dist.all_reduce(dt, op=dist.ReduceOp.MAX)
    mine = torch.tensor(tel + [ids.start], dtype=torch.int64)
    gathered = [torch.zeros_like(mine) for _ in range(world)]
    dist.all_gather(gathered, mine)
    if rank == 0:
        np.save(os.path.join(out_dir, "gathered.npy"), torch.stack(gathered).numpy())
        np.save(os.path.join(out_dir, "tmax.npy"), dt.numpy())
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_instance_sharding(tmp_path):
    import torch.multiprocessing as mp

    from oracle import plain
    from paper_2508_14544_gb300 import workloads as W
    port = _free_port()
    mp.spawn(_worker, args=(2, port, str(tmp_path)), nprocs=2, join=True)
    g = np.load(tmp_path / "gathered.npy")
    assert g.shape == (2, 4)
    assert g[0, 3] == 0 and g[1, 3] == 1  # disjoint shards, rank r starts at r * N
    for r in range(2):
        w = W.make_workload("c1", W.rank_instances("c1", r))
        for j, pol in enumerate((0, 1, 2)):
            assert g[r, j] == int(plain.run_workload(pol, w)["total_latency"].sum())
    assert float(np.load(tmp_path / "tmax.npy")[0]) > 0
