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
from parity_util import assert_stored, full_parity
from special_genomes import separable as _workload

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
    name = "separable_d6_" + ("eager" if mode == emr.EMR_EAGER else "gated")
    gpu, ora, rep = full_parity(w, mode, name=name)
    assert_stored(name)
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
    gpu, ora, rep = full_parity(w, emr.EMR_EAGER, name="separable_d7_eager")
    assert_stored("separable_d7_eager")
    assert rep["kept"] > 0
    dsc = gpu["dsc"]
    dsc.idx.zero_(); dsc.w.zero_()
    dsc.run_select()
    torch.cuda.synchronize()
    for (ri, rw), (si, sw) in zip(gpu["lists_f"], dsc.lists()):
        assert np.array_equal(ri, si) and np.array_equal(rw.view(np.uint32), sw.view(np.uint32))
