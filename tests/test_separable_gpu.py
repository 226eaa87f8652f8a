"""GPU parity for CPPNs built to reach every branch of the separable evaluation.

Each genome targets one case: an output of one grid coordinate (x or y,
filtered per column or row), joint nodes fed by nodes of one coordinate, a
joint node with no grid input of its own, chains of 6 and 8 joint nodes (their
own kernel classes), a genome above the dense limit (the interpreter), steep
outputs whose tiles pass the band screen at depths 5 and 6 (the re-evaluated
shared tile and its ring), and parallel or cancelling connections (merged by
the packer). Slots on both query sides swap which inputs are the grid's.
Everything is compared (on the GPU) with the float64 oracle (outputs, halo, planes, lists),
the fused and unfused paths with each other, and the selection path with the
fused lists, bit for bit.
"""
import numpy as np
import pytest
import torch

from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W
from parity_util import full_parity

X1, Y1, X2, Y2, BIAS, HID, OUT = range(7)
IDN, SIG, TNH, GAU, SIN, ABS = range(6)


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


def _workload(D=6):
    src = W.shared_sources([(0.0, -1.0, W.SIDE_OUT), (0.3, 1.0, W.SIDE_IN), (-0.5, -1.0, W.SIDE_OUT)])
    return W.Workload("separable_d%d" % D, separable_population(), src, D, 0.03, 0.3)


def test_classes_cover_every_case():
    """The population reaches the one-coordinate, joint, 6-, 8-joint and interpreter classes (host
    packing only, no GPU)."""
    w = _workload()
    _, gs, nodes, _ = emr.pack_records(emr.pack_population(w.pop))
    nj = gs["n_joint"][:, 0]
    nv = gs["n_varying"][:, 0]
    assert nj[0] == 0 and nj[1] == 0 and nv[0] == 3  # x only, y only (outgoing side)
    assert nj[2] == 1 and nj[3] == 1 and tuple(gs["n_joint"][4]) == (0, 3)
    assert nj[9] == 6 and nj[10] == 8 and nv[11] == 14
    assert gs["n_edges"][8] == 1  # the merged edge 6 -> out; 7 dropped with its cancelling pair


@pytest.mark.gpu
@pytest.mark.parametrize("mode", [emr.EMR_EAGER, emr.EMR_GATED])
def test_separable_population_parity(mode):
    w = _workload()
    gpu, ora, rep = full_parity(w, mode)
    # the steep genomes keep positions at depths 5 and 6 through the band test
    g = gpu["dsc"].grid
    wo = list(g.word_off)
    band = gpu["band_f"].view(np.uint32)
    deep = np.array([bin(int(x)).count("1") for x in band[:, wo[5]:wo[7]].ravel()]).reshape(band.shape[0], -1)
    deep = deep.sum(axis=1)
    S = w.S
    for gi in (5, 6, 7):  # steep joint, steep x-only, steep y chain: outgoing slot 0
        assert deep[gi * S] > 0, "genome %d: no band bits at depths 5..6" % gi
    # the selection path (flagged tiles) gives the fused lists bit for bit
    dsc = gpu["dsc"]
    dsc.idx.zero_(); dsc.w.zero_()
    dsc.run_select()
    torch.cuda.synchronize()
    for (ri, rw), (si, sw) in zip(gpu["lists_f"], dsc.lists()):
        assert np.array_equal(ri, si) and np.array_equal(rw.view(np.uint32), sw.view(np.uint32))
    assert rep["kept"] > 0


@pytest.mark.gpu
def test_separable_population_depth7():
    """Depth 7 (22 tiles per pair, the pyramid tile included): outputs, halo, planes and lists against
    the oracle, and the selection path's lists equal to the fused lists bit for bit."""
    w = _workload(D=7)
    gpu, ora, rep = full_parity(w, emr.EMR_EAGER)
    assert rep["kept"] > 0
    dsc = gpu["dsc"]
    dsc.idx.zero_(); dsc.w.zero_()
    dsc.run_select()
    torch.cuda.synchronize()
    for (ri, rw), (si, sw) in zip(gpu["lists_f"], dsc.lists()):
        assert np.array_equal(ri, si) and np.array_equal(rw.view(np.uint32), sw.view(np.uint32))
