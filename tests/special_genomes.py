"""Hand-built and mixed test populations of the parity tests (inputs only).

Numpy and the seeded generators only: no CUDA binding and none of the method's
arithmetic, so that both the GPU parity tests and the script storing the oracle's
exclusion counts (tests/golden/make_exclusion_counts.py) can build the same
workloads. Each builder returns a workloads.Workload.
"""
import numpy as np

from paper_2608_27612_gb300 import workloads as W

X1, Y1, X2, Y2, BIAS, HID, OUT = range(7)
IDN, SIG, TNH, GAU, SIN, ABS = range(6)


def edge_cases(D):
    """A constant genome, a hidden-free genome and six random ones, on both query sides."""
    const = ([(k, k, IDN, 0.0) for k in range(5)] + [(5, OUT, SIG, 0.3)], [(X1, 5, 1.0, True)])
    nohid = ([(k, k, IDN, 0.0) for k in range(5)] + [(5, OUT, SIN, 0.0)],
             [(X2, 5, 3.0, True), (Y2, 5, -2.0, True), (BIAS, 5, 0.5, True)])
    rnd = W.random_population(6, seed=9)
    pop = W.population_from_lists([const, nohid] + [rnd.genome(k) for k in range(6)])
    src = W.shared_sources([(0.0, -1.0, W.SIDE_OUT), (0.5, 1.0, W.SIDE_IN)])
    return W.Workload("edge_d%d" % D, pop, src, D, 0.03, 0.3)


def kernel_classes(D):
    """Genomes with 0..30 varying nodes: every kernel class including the interpreter."""
    big = W.random_population(24, seed=31, h_lo=14, h_hi=30, e_max=120)
    small = W.random_population(40, seed=32, h_lo=0, h_hi=12, e_max=40)
    pop = W.population_from_lists([big.genome(k) for k in range(24)] + [small.genome(k) for k in range(40)])
    src = W.shared_sources([(-1.0, -1.0, W.SIDE_OUT), (0.0, 1.0, W.SIDE_IN)])
    return W.Workload("classes_d%d" % D, pop, src, D, 0.03, 0.3)


def weight_filter():
    """100 genomes of the 1000-genome population at depth 5 with the weight filter at 0.1."""
    w = W.c2(D=5, P=100)
    w.w_min = 0.1
    w.name = "c2_d5_p100_wmin"
    return w


def per_genome_slots():
    """5 genomes with 6 per-genome slots each, on random sides, 6/0/3/1/6 of them valid."""
    pop = W.random_population(5, seed=12)
    rng = np.random.default_rng(4)
    S = 6
    a = rng.uniform(-1, 1, (5, S)).astype(np.float32)
    b = rng.uniform(-1, 1, (5, S)).astype(np.float32)
    side = rng.integers(0, 2, (5, S)).astype(np.int32)
    cnt = np.array([6, 0, 3, 1, 6], np.int32)
    return W.Workload("pergenome_d4", pop, W.Sources(a=a, b=b, side=side, count=cnt), 4, 0.03, 0.3)


def _genome(hidden, out_act, conns):
    """hidden: [(id, act)], output id 5; conns: [(src, dst, w)] (all enabled)."""
    nodes = [(k, k, IDN, 0.0) for k in range(5)] + [(5, OUT, out_act, 0.1)]
    nodes += [(i, HID, a, 0.05 * i) for i, a in hidden]
    return nodes, [(s, d, w, True) for s, d, w in conns]


def _chain(n_joint):
    """n_joint joint nodes in a chain (the output last), each fed by x2, y2 and earlier nodes."""
    acts = [SIN, TNH, GAU, SIG, ABS, IDN, SIN, TNH]
    ids = list(range(6, 6 + n_joint - 1)) + [5]
    conns = []
    for k, v in enumerate(ids):
        conns += [(X2, v, 0.7 + 0.1 * k), (Y2, v, -0.5 + 0.2 * k)]
        if k >= 1:
            conns.append((ids[k - 1], v, 0.9))
        if k >= 3:
            conns.append((ids[k - 3], v, -0.6))
    hidden = [(v, acts[k % len(acts)]) for k, v in enumerate(ids[:-1])]
    return _genome(hidden, acts[(n_joint - 1) % len(acts)], conns)


def separable_population():
    """One genome per branch of the separable evaluation (see test_separable_gpu)."""
    g = []
    # x only: a chain of nodes of x2 alone (one table row each), filtered per column
    g.append(_genome([(6, SIN), (7, TNH)], SIG, [(X2, 6, 3.0), (BIAS, 6, 0.2), (6, 7, 2.0), (X2, 7, -0.5),
                                                (7, 5, 1.5)]))
    # y only
    g.append(_genome([(6, GAU)], TNH, [(Y2, 6, 2.0), (6, 5, 1.0), (Y2, 5, 0.7)]))
    # joint output fed by an x node, a y node and x directly
    g.append(_genome([(6, SIN), (7, SIG)], TNH, [(X2, 6, 5.0), (Y2, 7, 4.0), (6, 5, 1.0), (7, 5, 1.0),
                                                 (X2, 5, 0.5)]))
    # joint only through its sources (no grid input of its own)
    g.append(_genome([(6, SIN), (7, GAU)], ABS, [(X2, 6, 3.0), (Y2, 7, 2.0), (6, 5, 1.0), (7, 5, -1.0)]))
    # joint on the incoming side (x1, y1), x only on the outgoing side (x2)
    g.append(_genome([(6, SIN), (7, GAU), (8, SIG)], IDN,
                     [(X1, 6, 3.0), (Y1, 6, 2.0), (X2, 6, 1.0), (6, 7, 1.0), (X1, 7, 1.0), (Y1, 8, 1.0),
                      (7, 5, 1.0), (8, 5, -1.0), (6, 5, 1.0)]))
    # steep joint and steep x-only outputs: their tiles pass the band screen at depths 5 and 6
    g.append(_genome([], SIN, [(X2, 5, 40.0), (Y2, 5, 30.0)]))
    g.append(_genome([], SIN, [(X2, 5, 50.0)]))
    g.append(_genome([(6, SIN)], GAU, [(Y2, 6, 45.0), (6, 5, 1.5)]))
    # parallel connections (0.5 + 0.25 into the output; x2 twice into 6) and a cancelling pair (7 drops out)
    g.append(_genome([(6, SIG), (7, SIN)], TNH, [(X2, 6, 1.0), (X2, 6, 0.5), (6, 5, 0.5), (Y2, 7, 1.0),
                                                 (7, 5, 1.0), (6, 5, 0.25), (7, 5, -1.0)]))
    # 6 and 8 joint nodes (their own kernel classes) and 14 (above the dense limit: the interpreter)
    g += [_chain(6), _chain(8), _chain(14)]
    return W.population_from_lists(g)


def separable(D=6):
    src = W.shared_sources([(0.0, -1.0, W.SIDE_OUT), (0.3, 1.0, W.SIDE_IN), (-0.5, -1.0, W.SIDE_OUT)])
    return W.Workload("separable_d%d" % D, separable_population(), src, D, 0.03, 0.3)
