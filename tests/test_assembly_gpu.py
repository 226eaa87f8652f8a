"""Substrate network assembly (emr_assemble) and the batched forward pass
(emr_ann_forward) against the oracle's assembly and forward pass."""
import numpy as np
import pytest
import torch

from oracle import assembly as A
from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W

pytestmark = pytest.mark.gpu

X1, Y1, X2, Y2, BIAS, HID, OUT = range(7)
XOR_IN = [(-1.0, -1.0), (1.0, -1.0), (0.0, -1.0)]
XOR_OUT = [(0.0, 1.0)]
XOR_PATTERNS = [[0, 0, 1], [0, 1, 1], [1, 0, 1], [1, 1, 1]]   # two inputs and the bias
ENABLED = {emr.CONN_F: (1, 0, 0, 0), emr.CONN_F | emr.CONN_B: (1, 1, 0, 0), emr.CONN_ALL: (1, 1, 1, 1)}


def gpu_networks(pop, D, types, rounds, mode=emr.EMR_EAGER, slots_max=256):
    pack = emr.pack_population(pop)
    pack_dev = torch.from_numpy(pack).cuda()
    return emr.assemble(pack, pack_dev, XOR_IN, XOR_OUT, emr.grid_build(D), 0.03, 0.3, 0.0, mode, types, rounds,
                        slots_max)


def check_same(nets, ora, unc):
    """Genomes whose queries met no uncertain decision must match exactly; returns how many did."""
    assert nets.P == len(ora)
    n = 0
    for g, (h_o, c_o) in enumerate(ora):
        if unc[g]:
            continue
        n += 1
        h, s, d, w, t = nets.genome(g)
        assert np.array_equal(h.astype(np.int64), h_o), "genome %d hidden nodes" % g
        assert len(s) == len(c_o), "genome %d connections" % g
        if c_o:
            co = np.array([(a, b, ty) for a, b, _, ty in c_o])
            assert np.array_equal(s, co[:, 0]) and np.array_equal(d, co[:, 1]) and np.array_equal(t, co[:, 2])
            wo = np.array([x for _, _, x, _ in c_o])
            assert np.all(np.abs(w - wo) <= 1e-5 + 1e-4 * np.abs(wo)), "genome %d weights" % g
    return n


@pytest.mark.parametrize("types,rounds", [(emr.CONN_F, 0), (emr.CONN_F, 1), (emr.CONN_ALL, 1)])
def test_linear_genome(types, rounds):
    nodes = [(k, k, 0, 0.0) for k in range(5)] + [(5, OUT, 0, 0.0)]
    pop = W.population_from_lists([(nodes, [(X1, 5, 4.0, True), (X2, 5, 4.0, True)])])
    nets = gpu_networks(pop, 4, types, rounds)
    ora, n_unc = A.assemble(pop, XOR_IN, XOR_OUT, 4, 0.03, 0.3, enabled=ENABLED[types], rounds=rounds)
    assert n_unc.sum() == 0
    assert check_same(nets, ora, n_unc) == 1


@pytest.mark.parametrize("types", [emr.CONN_F, emr.CONN_F | emr.CONN_B, emr.CONN_ALL])
@pytest.mark.parametrize("mode", [emr.EMR_EAGER, emr.EMR_GATED])
def test_random_population_networks_and_forward(types, mode):
    pop = W.random_population(12, seed=77)
    D, rounds = 4, 2
    ora, n_unc = A.assemble(pop, XOR_IN, XOR_OUT, D, 0.03, 0.3, gated=mode == emr.EMR_GATED,
                            enabled=ENABLED[types], rounds=rounds)
    nets = gpu_networks(pop, D, types, rounds, mode, slots_max=16)   # several phase-2 batches per round
    n_exact = check_same(nets, ora, n_unc)
    assert n_exact >= 6 and any(len(c) for g, (_, c) in enumerate(ora) if not n_unc[g])
    assert nets.node_off[-1] > 0 and nets.conn_off[-1] > 0
    steps = rounds + 2
    out = emr.ann_forward(nets, XOR_PATTERNS, steps).cpu().numpy()
    for g in range(nets.P):
        h, s, d, w, t = nets.genome(g)
        ref = A.forward(3, 1, h, list(zip(s, d, w.astype(np.float64), t)), XOR_PATTERNS, steps)
        assert np.all(np.abs(out[g] - ref) <= 2e-6), "genome %d" % g


def test_forward_many_networks_and_steps():
    pop = W.random_population(40, seed=78)
    nets = gpu_networks(pop, 5, emr.CONN_ALL, 1)
    pats = np.random.default_rng(3).uniform(-1, 1, (6, 3)).astype(np.float32)
    for steps in (0, 1, 5):
        out = emr.ann_forward(nets, pats, steps).cpu().numpy()
        for g in range(nets.P):
            h, s, d, w, t = nets.genome(g)
            ref = A.forward(3, 1, h, list(zip(s, d, w.astype(np.float64), t)), pats, steps)
            assert np.all(np.abs(out[g] - ref) <= 2e-6), "genome %d steps %d" % (g, steps)


def same_networks(a, b):
    for f in ("node_off", "hidden", "conn_off", "src", "dst", "type"):
        assert np.array_equal(getattr(a, f), getattr(b, f)), f
    assert np.array_equal(a.w.view(np.uint32), b.w.view(np.uint32))


def test_cache_reuses_lists_without_changing_networks():
    pop = W.random_population(24, seed=79)
    pack = emr.pack_population(pop)
    pack_dev = torch.from_numpy(pack).cuda()
    g = emr.grid_build(5)
    args = (pack, pack_dev, XOR_IN, XOR_OUT, g, 0.03, 0.3, 0.0, emr.EMR_EAGER, emr.CONN_ALL, 2, 32)
    ref = emr.assemble(*args)
    cache = emr.Cache()
    first = emr.assemble(*args, cache=cache)
    s1 = cache.stats()
    # genomes that pack to the same records share keys: entries can be fewer than misses
    assert s1["hits"] == 0 and s1["misses"] >= s1["entries"] > 24 * 4
    second = emr.assemble(*args, cache=cache)
    s2 = cache.stats()
    assert s2["misses"] == s1["misses"] and s2["hits"] == s1["misses"]   # every query hit
    same_networks(ref, first)
    same_networks(ref, second)
    # a later population sharing half its genomes hits for those genomes' queries only
    shared = list(range(12, 24))
    pop2 = W.population_from_lists([pop.genome(k) for k in shared] +
                                   [W.random_population(12, seed=80).genome(k) for k in range(12)])
    pack2 = emr.pack_population(pop2)
    nets2 = emr.assemble(pack2, torch.from_numpy(pack2).cuda(), XOR_IN, XOR_OUT, g, 0.03, 0.3, 0.0, emr.EMR_EAGER,
                         emr.CONN_ALL, 2, 32, cache=cache)
    s3 = cache.stats()
    ref2 = emr.assemble(pack2, torch.from_numpy(pack2).cuda(), XOR_IN, XOR_OUT, g, 0.03, 0.3, 0.0, emr.EMR_EAGER,
                        emr.CONN_ALL, 2, 32)
    same_networks(ref2, nets2)
    for k in range(12):   # the shared genomes' networks are those of the first population
        a, b = nets2.genome(k), ref.genome(shared[k])
        for x, y in zip(a, b):
            assert np.array_equal(x, y)
    # at least the shared genomes' four phase-1/3 slots hit; the new genomes miss
    assert s3["hits"] - s2["hits"] >= 12 * 4 and s3["misses"] > s2["misses"]
    # a different parameter is a different key
    emr.assemble(pack, pack_dev, XOR_IN, XOR_OUT, g, 0.03, 0.31, 0.0, emr.EMR_EAGER, emr.CONN_ALL, 2, 32,
                 cache=cache)
    assert cache.stats()["misses"] > s3["misses"]


def test_cache_budget_evicts_but_keeps_results():
    pop = W.random_population(16, seed=81)
    pack = emr.pack_population(pop)
    pack_dev = torch.from_numpy(pack).cuda()
    g = emr.grid_build(5)
    args = (pack, pack_dev, XOR_IN, XOR_OUT, g, 0.03, 0.3, 0.0, emr.EMR_EAGER, emr.CONN_F, 1, 64)
    ref = emr.assemble(*args)
    cache = emr.Cache(max_bytes=64 << 10)
    for _ in range(3):
        same_networks(ref, emr.assemble(*args, cache=cache))
        st = cache.stats()
        assert st["bytes"] <= 64 << 10
    cache.clear()
    assert cache.stats() == {"hits": 0, "misses": 0, "entries": 0, "bytes": 0}
