"""Round-2 query slots of the full-recurrent workload, built from a round-1 keep mask.

Test infrastructure: used by the hidden-to-hidden round's GPU test and by the
script that stores the oracle's exclusion counts. It reads a keep mask given
by the caller (the oracle's, in both places) and converts kept global indices
to grid coordinates by Eq. 1 with the depth-major Morton numbering.
"""
import numpy as np

from paper_2608_27612_gb300 import workloads as W


def dij(p):
    """Depth and grid indices of a global index (depth-major, Morton within a depth)."""
    d = 0
    while (4 ** (d + 2) - 4) // 3 <= p:
        d += 1
    m = p - (4 ** (d + 1) - 4) // 3
    i = sum(((m >> (2 * k)) & 1) << k for k in range(d + 1))
    j = sum(((m >> (2 * k + 1)) & 1) << k for k in range(d + 1))
    return d, i, j


def hidden_sources(w1, keep, S=256):
    """Per genome: the distinct positions its outgoing round-1 slots keep, ascending, first S,
    each queried outgoing from its grid coordinates (Eq. 1). keep: [P, S1, N_total]."""
    P, S1 = keep.shape[0], w1.S
    a = np.zeros((P, S), np.float32); b = np.zeros((P, S), np.float32)
    side = np.zeros((P, S), np.int32); count = np.zeros(P, np.int32)
    for g in range(P):
        rows = [keep[g, s] for s in range(S1) if int(w1.sources.side[s]) == W.SIDE_OUT]
        idx = np.flatnonzero(np.any(rows, axis=0))[:S]
        count[g] = len(idx)
        for k, p in enumerate(idx):
            d, i, j = dij(int(p))
            a[g, k] = (2 * i + 1) / 2.0 ** (d + 1) - 1.0
            b[g, k] = (2 * j + 1) / 2.0 ** (d + 1) - 1.0
    return W.Sources(a=a, b=b, side=side, count=count)


def round2_workload(w1, keep, n_genomes=8, S=256):
    """The second round for the first n_genomes genomes of w1 whose round 1 (keep: [P, S1,
    N_total]) found hidden nodes: their sub-population with those nodes as per-genome slots."""
    src = hidden_sources(w1, keep, S)
    pick = np.flatnonzero(src.count > 0)[:n_genomes]
    src2 = W.Sources(a=src.a[pick], b=src.b[pick], side=src.side[pick], count=src.count[pick])
    return W.Workload("c4_round2_g%d" % len(pick), w1.pop.subset(pick), src2, w1.D, w1.theta, w1.band)
