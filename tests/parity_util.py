"""Comparison helpers for the GPU-vs-oracle parity tests.

Tolerance (fp32 device vs fp64 oracle): |gpu - oracle| <= 1e-5 + 1e-4 |oracle| for
every CPPN output whose fp32 error bound (computed by the oracle) is within that
tolerance; outputs above it are "ill-conditioned" and counted. Masks and
compacted indices are compared bit for bit wherever the oracle reports the
decision as certain (its margin to the threshold exceeds 1e-6 plus the
decision's own error bound); the uncertain positions are counted.
"""
import numpy as np
import torch

import oracle
from paper_2608_27612_gb300 import emr

TOL_ABS, TOL_REL = 1e-5, 1e-4


def tol(ref):
    return TOL_ABS + TOL_REL * np.abs(ref)


def unpack_planes(planes, grid):
    """[n_pairs, n_words] uint32/int32 bit planes -> [n_pairs, n_total] uint8 by global index."""
    p = np.ascontiguousarray(planes).view(np.uint32)
    bits = np.unpackbits(p.view(np.uint8), axis=1, bitorder="little")
    parts = []
    for d in range(grid.D + 1):
        w0 = grid.word_off[d]
        parts.append(bits[:, 32 * w0: 32 * w0 + 4 ** (d + 1)])
    return np.concatenate(parts, axis=1)


def check_outputs(gpu_w, ora_w, ora_err, what="w"):
    """Outputs within tolerance wherever the oracle's bound is within tolerance."""
    gpu_w = np.asarray(gpu_w, np.float64)
    t = tol(ora_w)
    ill = ~(ora_err <= t)
    diff = np.abs(gpu_w - ora_w)
    bad = (~(diff <= t)) & ~ill
    if bad.any():
        k = np.argwhere(bad)[0]
        raise AssertionError("%s: %d outputs outside tolerance, first at %s: gpu %r oracle %r (bound %r)" % (
            what, int(bad.sum()), tuple(k), gpu_w[tuple(k)], ora_w[tuple(k)], ora_err[tuple(k)]))
    ok = ~ill
    return {"n": int(gpu_w.size), "ill_conditioned": int(ill.sum()),
            "max_abs_err": float(diff[ok].max()) if ok.any() else 0.0}


def check_bits(gpu_bits, ora_bits, ora_unc, what="mask"):
    """Bit-exact wherever the oracle's decision is certain."""
    mism = (gpu_bits.astype(bool) != ora_bits.astype(bool)) & ~ora_unc.astype(bool)
    if mism.any():
        k = np.argwhere(mism)[0]
        raise AssertionError("%s: %d certain positions differ, first at %s (gpu %d oracle %d)" % (
            what, int(mism.sum()), tuple(k), gpu_bits[tuple(k)], ora_bits[tuple(k)]))
    return {"n": int(gpu_bits.size), "uncertain": int(ora_unc.astype(bool).sum()),
            "kept": int(gpu_bits.astype(bool).sum())}


def check_lists(lists, gpu_mask, ora_w=None, ora_err=None):
    """Compacted lists: exactly the ascending set bits of the device mask, with
    weights equal to the oracle's CPPN outputs within tolerance."""
    n_pairs = gpu_mask.shape[0]
    assert len(lists) == n_pairs
    total = 0
    for r, (idx, w) in enumerate(lists):
        want = np.flatnonzero(gpu_mask[r])
        assert np.array_equal(idx.astype(np.int64), want), "pair %d: indices differ from the mask" % r
        if len(idx):
            assert np.all(np.diff(idx) > 0)
        if ora_w is not None and len(idx):
            check_outputs(w, ora_w[r][idx], ora_err[r][idx], what="list w pair %d" % r)
        total += len(idx)
    return total


# ---- the GPU path and the oracle on one workload ------------------------------------

def run_gpu(w, mode=emr.EMR_EAGER, unfused=True, fused=True, cap=None, lists=True):
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, mode, cap=cap, materialise=unfused)
    g = dsc.grid
    res = {"dsc": dsc}
    if unfused:
        dsc.run_unfused(with_var=True)
        torch.cuda.synchronize()
        res["out"] = dsc.out.cpu().numpy()
        res["halo"] = dsc.out_halo.cpu().numpy()
        res["var"] = dsc.var_dbg.cpu().numpy()
        res["mask_u"] = unpack_planes(dsc.mask.cpu().numpy(), g)
        res["split_u"] = dsc.split.cpu().numpy()
        res["band_u"] = dsc.band_bits.cpu().numpy()
        res["lists_u"] = dsc.lists()
    if fused:
        dsc.mask.zero_(); dsc.split.zero_(); dsc.band_bits.zero_()
        dsc.run_fused()
        torch.cuda.synchronize()
        res["mask_f"] = unpack_planes(dsc.mask.cpu().numpy(), g)
        res["split_f"] = dsc.split.cpu().numpy()
        res["band_f"] = dsc.band_bits.cpu().numpy()
        res["lists_f"] = dsc.lists() if lists else None
        if unfused and lists:
            # the fused kernel's own sparse outputs, read by emr_compact
            dsc.out.zero_()
            dsc.run_fused(sparse_out=True)
            res["lists_s"] = dsc.lists()
    return res


def run_oracle(w, g1=None):
    r = oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, g1=g1)
    return {k: v.reshape(-1, v.shape[-1]) for k, v in r.items()}


def full_parity(w, mode=emr.EMR_EAGER, n_oracle=None):
    gpu = run_gpu(w, mode)
    ora = run_oracle(w, g1=n_oracle)
    n = ora["w"].shape[0]
    keep, unc = ("keep_eager", "unc_eager") if mode == emr.EMR_EAGER else ("keep_gated", "unc_gated")
    rep = {}
    rep["out"] = check_outputs(gpu["out"][:n], ora["w"], ora["w_err"])
    rep["halo"] = check_outputs(gpu["halo"][:n], ora["w_halo"], ora["halo_err"], "halo")
    dv = np.abs(gpu["var"][:n] - ora["var"])
    assert np.all((dv <= ora["var_err"] + 1e-12) | ~np.isfinite(ora["var_err"]))
    rep["mask_u"] = check_bits(gpu["mask_u"][:n], ora[keep], ora[unc], "unfused mask")
    rep["mask_f"] = check_bits(gpu["mask_f"][:n], ora[keep], ora[unc], "fused mask")
    # fused and unfused paths compute the same fp32 decisions
    assert np.array_equal(gpu["split_u"], gpu["split_f"])
    assert np.array_equal(gpu["band_u"], gpu["band_f"])
    assert np.array_equal(gpu["mask_u"], gpu["mask_f"])
    rep["kept"] = check_lists(gpu["lists_f"][:n], gpu["mask_f"][:n], ora["w"], ora["w_err"])
    check_lists(gpu["lists_u"][:n], gpu["mask_u"][:n], ora["w"], ora["w_err"])
    # weights recomputed from the records at compaction, and those the fused kernel
    # stores itself, equal the materialised outputs bit for bit
    for (i_u, w_u), (i_f, w_f), (i_s, w_s) in zip(gpu["lists_u"], gpu["lists_f"], gpu["lists_s"]):
        assert np.array_equal(i_u, i_f) and np.array_equal(i_u, i_s)
        assert np.array_equal(w_u.view(np.uint32), w_f.view(np.uint32))
        assert np.array_equal(w_u.view(np.uint32), w_s.view(np.uint32))
    return gpu, ora, rep
