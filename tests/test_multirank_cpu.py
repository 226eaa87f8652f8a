"""Population-parallel discovery on CPU (gloo ranks; every GPU run of this build has one GPU).

One population's genomes are split by packed cost into contiguous ranges
(emr_partition_genomes); each rank packs its own range (the range hook of
emr_pack_population) and produces its lists; the lists are gathered to rank 0
(paper_2608_27612_gb300.dist.gather_lists), where they must equal the whole
population's lists bit for bit. The per-rank lists here come from the float64
oracle on the rank's genome range (this container has no GPU), so the test
checks the partition, the range packing and the gather, not the kernels."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def oracle_lists(w, g0, g1):
    """Per pair of genomes [g0, g1): ascending kept global indices and their fp32 weights."""
    import oracle
    r = oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, g0=g0, g1=g1,
                        fields=("keep_eager", "w"))
    keep = r["keep_eager"].reshape(-1, r["keep_eager"].shape[-1])
    wv = r["w"].reshape(keep.shape)
    idx = [np.flatnonzero(k) for k in keep]
    counts = np.array([len(x) for x in idx], np.int64)
    flat_i = np.concatenate(idx).astype(np.int32) if idx else np.zeros(0, np.int32)
    flat_w = np.concatenate([wv[k][x] for k, x in enumerate(idx)]).astype(np.float32) if idx else np.zeros(0, np.float32)
    return counts, flat_i, flat_w


def test_partition_covers_the_population_and_balances_cost():
    from paper_2608_27612_gb300 import emr
    from paper_2608_27612_gb300 import workloads as W
    w = W.c2(D=5)
    pack = emr.pack_population(w.pop)
    q = emr.make_query(w.sources, device="cpu")
    _, gs, _, _ = emr.pack_records(pack)
    side = np.asarray(w.sources.side)
    cost = np.array([sum(int(gs["cost"][g][s]) + 6 if gs["n_varying"][g][s] else 1 for s in side)
                     for g in range(w.P)])
    for n in (1, 2, 3, 4, 8):
        b = emr.partition_genomes(pack, q, n)
        assert b[0] == 0 and b[-1] == w.P and np.all(np.diff(b) >= 0)
        part = np.array([cost[b[k]:b[k + 1]].sum() for k in range(n)])
        # each boundary is the genome boundary nearest the ideal split, so no part is further
        # from the mean than the heaviest genome
        assert np.abs(part - cost.sum() / n).max() <= cost.max()
    b = emr.partition_genomes(pack, q, 1500)  # more parts than genomes: some parts empty, still a cover
    assert b[0] == 0 and b[-1] == w.P and np.all(np.diff(b) >= 0) and (np.diff(b) == 0).any()
    part = np.array([cost[b[k]:b[k + 1]].sum() for k in range(1500)])
    assert np.abs(part - cost.sum() / 1500).max() <= cost.max()
    with pytest.raises(emr.EmrError):
        emr.partition_genomes(pack, q, 0)


def test_partition_counts_only_used_per_genome_slots():
    """A genome whose per-genome slots are all unused weighs S (1 per slot) whatever its CPPN."""
    from paper_2608_27612_gb300 import emr
    from paper_2608_27612_gb300 import workloads as W
    pop = W.random_population(4, seed=7, h_lo=8, h_hi=12)
    S = 3
    a = np.zeros((4, S), np.float32); b = np.full((4, S), -1.0, np.float32); side = np.zeros((4, S), np.int32)
    heavy = W.Sources(a=a, b=b, side=side, count=np.array([S, S, S, S], np.int32))
    unused = W.Sources(a=a, b=b, side=side, count=np.array([S, 0, 0, 0], np.int32))
    pack = emr.pack_population(pop)
    g_heavy = emr.partition_genomes(pack, emr.make_query(heavy, device="cpu"), 2)
    g_unused = emr.partition_genomes(pack, emr.make_query(unused, device="cpu"), 2)
    assert 1 <= g_heavy[1] <= 3
    assert g_unused[1] == 1  # genome 0 alone outweighs the three empty ones


def test_range_packing_equals_packing_the_subset():
    from paper_2608_27612_gb300 import emr
    from paper_2608_27612_gb300 import workloads as W
    w = W.c2(D=5, P=200)
    for g0, g1 in ((0, 200), (0, 1), (17, 130), (199, 200)):
        assert np.array_equal(emr.pack_population(w.pop, genomes=(g0, g1)),
                              emr.pack_population(w.pop.subset(range(g0, g1))))
    with pytest.raises(ValueError):
        emr.pack_population(w.pop, genomes=(5, 5))


def _rank(rank, ws, port, out):
    import sys
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    import bench
    from paper_2608_27612_gb300 import dist as pdist
    from paper_2608_27612_gb300 import emr
    from paper_2608_27612_gb300 import workloads as W
    from test_multirank_cpu import oracle_lists
    w = W.c2(D=4, P=60)
    pack = emr.pack_population(w.pop)
    g = pdist.genome_ranges(pack, emr.make_query(w.sources, device="cpu"), ws)
    g0, g1 = int(g[rank]), int(g[rank + 1])
    blob = emr.pack_population(w.pop, genomes=(g0, g1))
    counts, idx, wv = oracle_lists(w, g0, g1)
    got = pdist.gather_lists(torch.from_numpy(counts), torch.from_numpy(idx), torch.from_numpy(wv))
    # the benchmark's per-rank workload and its whole-job aggregation
    wr, (b0, b1) = bench.rank_workload(W, emr, rank, ws, 4, 30)
    queries = wr.P * wr.S * emr.grid_build(wr.D).n_total
    total, ms, value = bench.aggregate(queries, 10.0 * (rank + 1), ws)
    dist.barrier()
    res = {"range": (g0, g1), "blob_sum": int(blob.astype(np.uint64).sum()), "bench_range": (b0, b1),
           "bench_P": wr.P, "agg": (total, ms, value)}
    if got is not None:
        res["lists"] = tuple(t.numpy() for t in got)
    out[rank] = res
    dist.destroy_process_group()


def test_two_gloo_ranks_partition_discover_and_gather_equal_one_rank():
    from paper_2608_27612_gb300 import workloads as W
    ws = 2
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_rank, args=(ws, _free_port(), out), nprocs=ws, start_method="spawn")
    r0, r1 = out[0], out[1]
    assert r0["range"][0] == 0 and r0["range"][1] == r1["range"][0] and r1["range"][1] == 60
    assert 0 < r0["range"][1] < 60
    assert "lists" in r0 and "lists" not in r1
    cnt, off, idx, wv = r0["lists"]
    w = W.c2(D=4, P=60)
    c_ref, i_ref, w_ref = oracle_lists(w, 0, 60)
    assert np.array_equal(cnt, c_ref) and np.array_equal(off[1:], np.cumsum(c_ref)) and off[0] == 0
    assert np.array_equal(idx, i_ref) and np.array_equal(wv.view(np.uint32), w_ref.view(np.uint32))
    assert idx.size > 0
    # benchmark: one population of 30 x 2 genomes split by cost, whole-job throughput over the slowest rank
    assert r0["bench_range"][0] == 0 and r0["bench_range"][1] == r1["bench_range"][0] and r1["bench_range"][1] == 60
    assert r0["bench_P"] + r1["bench_P"] == 60
    q = 60 * 4 * 1364
    assert r0["agg"][0] == r1["agg"][0] == q
    assert r0["agg"][1] == r1["agg"][1] == 20.0
    assert abs(r0["agg"][2] - q / 0.020) < 1e-3 * r0["agg"][2]
