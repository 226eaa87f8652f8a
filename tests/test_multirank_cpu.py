"""The multi-GPU path of bench.py on CPU: two gloo ranks. Each rank runs its own
population (no data exchange); whole-job throughput sums the ranks' queries and
divides by the slowest rank's time."""
import os
import socket

import numpy as np
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, ws, port, out):
    import sys
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    import bench
    from paper_2608_27612_gb300 import emr
    from paper_2608_27612_gb300 import workloads as W
    w = bench.rank_workload(W, rank, 5, 40)
    blob = emr.pack_population(w.pop)
    queries = w.P * w.S * emr.grid_build(w.D).n_total
    total, ms, value = bench.aggregate(queries, 10.0 * (rank + 1), ws)
    dist.barrier()
    out[rank] = (int(total), ms, value, int(blob.astype(np.uint64).sum()), w.name)
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_populations_and_aggregate():
    ws = 2
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_rank, args=(ws, _free_port(), out), nprocs=ws, start_method="spawn")
    r0, r1 = out[0], out[1]
    q = 40 * 4 * 5460
    assert r0[0] == r1[0] == ws * q
    assert r0[1] == r1[1] == 20.0
    assert abs(r0[2] - ws * q / 0.020) < 1e-3 * r0[2]
    assert r0[3] != r1[3] and r0[4] != r1[4]  # different populations per rank
