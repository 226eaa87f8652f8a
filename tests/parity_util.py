"""Comparison helpers for the GPU-vs-oracle parity tests.

Tolerance (fp32 device vs fp64 oracle): |gpu - oracle| <= 1e-5 + 1e-4 |oracle| for
every CPPN output whose fp32 error bound (computed by the oracle) is within that
tolerance; outputs above it are "ill-conditioned" and counted. Masks and
compacted indices are compared bit for bit wherever the oracle reports the
decision as certain (its margin to the threshold exceeds 1e-6 plus the
decision's own error bound); the uncertain positions are counted.
"""
import numpy as np

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
