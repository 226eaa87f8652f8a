"""Comparison helpers for the GPU-vs-oracle parity tests.

Tolerance (fp32 device vs fp64 oracle): every CPPN output must satisfy
|gpu - oracle| <= max(1e-5 + 1e-4 |oracle|, bound), where bound is the oracle's
forward error bound for the device's fp32 evaluation. Outputs whose bound exceeds
the plain tolerance are "ill-conditioned": they are still compared, against their
bound, and counted. Masks and compacted indices are compared bit for bit wherever
the oracle reports the decision as certain (its margin to the threshold exceeds
1e-6 plus the decision's own error bound); the uncertain positions are counted,
with how many of them the device decided as the oracle did.

Every comparison adds its counts to a session-wide report (record()); the
terminal summary prints it per workload, and where a workload has stored oracle
counts (tests/golden/exclusion_counts.json) the run's counts must stay within
them (a small margin allows libm differences between hosts).
"""
import json
import os

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
    """Every output within max(tolerance, the oracle's fp32 bound); a NaN never passes."""
    gpu_w = np.asarray(gpu_w, np.float64)
    t = tol(ora_w)
    ill = ~(ora_err <= t)
    lim = np.where(ill, ora_err, t)
    diff = np.abs(gpu_w - ora_w)
    bad = ~(diff <= lim)
    if bad.any():
        k = np.argwhere(bad)[0]
        raise AssertionError("%s: %d outputs outside tolerance, first at %s: gpu %r oracle %r (bound %r)" % (
            what, int(bad.sum()), tuple(k), gpu_w[tuple(k)], ora_w[tuple(k)], ora_err[tuple(k)]))
    ok = ~ill
    fin = ill & np.isfinite(ora_err) & (ora_err > 0)
    return {"outputs": int(gpu_w.size), "ill_conditioned": int(ill.sum()),
            "unbounded": int((~np.isfinite(ora_err)).sum()),
            "max_abs_err": float(diff[ok].max()) if ok.any() else 0.0,
            "max_err_over_bound_ill": float((diff[fin] / ora_err[fin]).max()) if fin.any() else 0.0}


def check_bits(gpu_bits, ora_bits, ora_unc, what="mask"):
    """Bit-exact wherever the oracle's decision is certain; uncertain ones counted."""
    g = gpu_bits.astype(bool)
    o = ora_bits.astype(bool)
    u = ora_unc.astype(bool)
    mism = (g != o) & ~u
    if mism.any():
        k = np.argwhere(mism)[0]
        raise AssertionError("%s: %d certain positions differ, first at %s (gpu %d oracle %d)" % (
            what, int(mism.sum()), tuple(k), gpu_bits[tuple(k)], ora_bits[tuple(k)]))
    return {"decisions": int(gpu_bits.size), "uncertain": int(u.sum()),
            "uncertain_agree": int((u & (g == o)).sum()), "kept": int((g & ~u).sum())}


def check_lists(lists, gpu_mask, ora_w=None, ora_err=None):
    """Compacted lists: exactly the ascending set bits of the device mask, with
    weights equal to the oracle's CPPN outputs within max(tolerance, bound)."""
    n_pairs = gpu_mask.shape[0]
    assert len(lists) == n_pairs
    total = 0
    ws, refs, errs = [], [], []
    for r, (idx, w) in enumerate(lists):
        want = np.flatnonzero(gpu_mask[r])
        assert np.array_equal(idx.astype(np.int64), want), "pair %d: indices differ from the mask" % r
        if len(idx):
            assert np.all(np.diff(idx) > 0)
        if ora_w is not None and len(idx):
            ws.append(w); refs.append(ora_w[r][idx]); errs.append(ora_err[r][idx])
        total += len(idx)
    rep = {"entries": total}
    if ws:
        o = check_outputs(np.concatenate(ws), np.concatenate(refs), np.concatenate(errs), "list weights")
        rep.update(kept_weights=o["outputs"], kept_ill_conditioned=o["ill_conditioned"])
    return rep


# ---- the session report ------------------------------------------------------------

REPORT = {}
_GOLD = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "exclusion_counts.json")
CEILING_KEYS = ("ill_conditioned", "unbounded", "uncertain", "kept_ill_conditioned")


def stored_counts():
    try:
        with open(_GOLD) as f:
            return json.load(f)
    except OSError:
        return {}


def ceiling(stored):
    return stored + max(4, stored // 50)


def record(name, *parts, compare_stored=True):
    """Sum the counts of the given check results under `name`; where the oracle's counts for
    `name` are stored, assert the exclusion counts stay within them and the compared totals
    equal them."""
    tot = REPORT.setdefault(name, {})
    for p in parts:
        for k, v in p.items():
            if k.startswith("max_"):
                tot[k] = max(tot.get(k, 0.0), v)
            else:
                tot[k] = tot.get(k, 0) + v
    return tot


def assert_stored(name):
    """The run's totals for `name` against the stored oracle counts."""
    tot = REPORT[name]
    gold = stored_counts().get(name)
    assert gold is not None, "no stored oracle counts for %s" % name
    for k in ("outputs", "decisions"):
        if k in tot:
            assert tot[k] == gold[k], "%s: %s compared %d, stored %d" % (name, k, tot[k], gold[k])
    for k in CEILING_KEYS:
        if k in tot:
            assert tot[k] <= ceiling(gold[k]), "%s: %s = %d above the stored %d" % (name, k, tot[k], gold[k])
    return tot


def report_lines():
    cols = ("outputs", "ill_conditioned", "unbounded", "max_err_over_bound_ill", "decisions", "uncertain",
            "uncertain_agree", "kept", "kept_weights", "kept_ill_conditioned")
    lines = ["parity exclusions per workload: " + " | ".join(cols)]
    for name in sorted(REPORT):
        r = REPORT[name]
        cells = []
        for c in cols:
            v = r.get(c)
            cells.append("-" if v is None else ("%.3g" % v if isinstance(v, float) else str(v)))
        lines.append("  %s: %s" % (name, " | ".join(cells)))
    return lines


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


def oracle_blocks(w, block, gated=False):
    """The oracle's outputs, bounds and keep decisions over genome blocks of w:
    yields (g0, g1, {field: [pairs of the block, N_total]})."""
    keep, unc = ("keep_gated", "unc_gated") if gated else ("keep_eager", "unc_eager")
    for g0 in range(0, w.P, block):
        g1 = min(w.P, g0 + block)
        r = oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, g0=g0, g1=g1,
                            fields=("w", "w_err", keep, unc))
        yield g0, g1, {k: v.reshape(-1, v.shape[-1]) for k, v in r.items()}


def mask_from_lists(lists, n_total):
    m = np.zeros((len(lists), n_total), np.uint8)
    for r, (idx, _) in enumerate(lists):
        m[r, idx] = 1
    return m


def full_parity(w, mode=emr.EMR_EAGER, n_oracle=None, name=None):
    """Outputs, halo, variance, masks of both paths and lists against the oracle; with a
    name, the counts go into the session report."""
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
    rep["lists"] = check_lists(gpu["lists_f"][:n], gpu["mask_f"][:n], ora["w"], ora["w_err"])
    rep["kept"] = rep["lists"]["entries"]
    check_lists(gpu["lists_u"][:n], gpu["mask_u"][:n], ora["w"], ora["w_err"])
    # weights recomputed from the records at compaction, and those the fused kernel
    # stores itself, equal the materialised outputs bit for bit
    for (i_u, w_u), (i_f, w_f), (i_s, w_s) in zip(gpu["lists_u"], gpu["lists_f"], gpu["lists_s"]):
        assert np.array_equal(i_u, i_f) and np.array_equal(i_u, i_s)
        assert np.array_equal(w_u.view(np.uint32), w_f.view(np.uint32))
        assert np.array_equal(w_u.view(np.uint32), w_s.view(np.uint32))
    if name:
        record(name, rep["out"], rep["mask_f"], rep["lists"])
    return gpu, ora, rep
