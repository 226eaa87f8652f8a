"""Method variants on the device against the oracle: the subtree-leaf variance
split plane (emr_subtree_split) and HyperNEAT weight scaling of the lists
(emr_scale_weights)."""
import numpy as np
import pytest
import torch

import oracle
from oracle import variants as VAR
from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W
from parity_util import unpack_planes

pytestmark = pytest.mark.gpu


def off(d):
    return (4 ** (d + 1) - 4) // 3


@pytest.mark.parametrize("D,P", [(1, 20), (2, 20), (3, 30), (5, 30), (6, 12)])
def test_subtree_split_matches_oracle(D, P):
    w = W.c2(D=D, P=P)
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, materialise=True)
    dsc.run_unfused()
    g = dsc.grid
    split = torch.zeros_like(dsc.split)
    var = torch.full((dsc.n_pairs, g.n_total), -1.0, dtype=torch.float32, device="cuda")
    ws = torch.empty(emr.subtree_workspace_size(g, dsc.n_pairs), dtype=torch.uint8, device="cuda")
    for _ in range(2):   # a second call on the same buffers gives the same planes
        emr.subtree_split(dsc.out, g, dsc.n_pairs, w.theta, split, ws, var)
        torch.cuda.synchronize()
        bits = unpack_planes(split.cpu().numpy(), g)
        v = var.cpu().numpy()
        ora = oracle.discover(w.pop, w.sources, D, w.theta, w.band, fields=("w", "w_err"))
        wo = ora["w"].reshape(-1, g.n_total)
        eo = ora["w_err"].reshape(-1, g.n_total)
        n_dec = n_unc = 0
        for r in range(dsc.n_pairs):
            V, bound, sp, unc = VAR.subtree_split(wo[r], eo[r], D, w.theta)
            n = off(D)
            assert np.all(np.abs(v[r, :n] - V) <= bound + 1e-6), "pair %d variance" % r
            ok = unc == 0
            assert np.array_equal(bits[r, :n][ok], sp[ok]), "pair %d split" % r
            n_dec += int(ok.sum()); n_unc += int((~ok).sum())
        assert n_dec > 0 and n_unc <= 0.01 * (n_dec + n_unc)
    # the same plane feeds the mask combine: keep = band and not split
    mask = torch.zeros_like(dsc.mask)
    emr.mask_combine(split, dsc.band_bits, g, dsc.n_pairs, emr.EMR_EAGER, mask)
    m = unpack_planes(mask.cpu().numpy(), g)
    band_pm = torch.zeros_like(dsc.mask)                 # band bits, position-major (no split)
    emr.mask_combine(torch.zeros_like(split), dsc.band_bits, g, dsc.n_pairs, emr.EMR_EAGER, band_pm)
    b = unpack_planes(band_pm.cpu().numpy(), g)
    s = bits.copy()
    s[:, off(D):] = 0                                    # depth D never splits
    assert np.array_equal(m, b & (1 - s))


def test_weight_scaling_of_lists():
    w = W.c2(D=6, P=50)
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band)
    dsc.run_fused()
    torch.cuda.synchronize()
    total = int(dsc.offsets[-1])
    raw = dsc.w[:total].cpu().numpy().astype(np.float64)
    assert total > 100
    for thr, wm in [(0.1, 3.0), (0.3, 1.0), (0.0, 5.0)]:
        wv = dsc.w.clone()
        emr.scale_weights(wv, dsc.offsets, dsc.n_pairs, dsc.cap, thr, wm)
        got = wv[:total].cpu().numpy()
        want = VAR.scale_weights(raw, np.float32(thr), wm)
        assert np.all(np.abs(got - want) <= 4e-7 * wm), (thr, wm)
        assert np.array_equal(got == 0, np.abs(raw.astype(np.float32)) <= np.float32(thr))
