"""Write tests/golden/exclusion_counts.json: the oracle's own exclusion counts per workload.

Calls only the float64 oracle (oracle/) and the seeded input generators. For each
workload it records how many CPPN outputs are ill-conditioned (the oracle's fp32 error
bound exceeds the 1e-5 + 1e-4 |w| tolerance; the parity tests compare those against
their bound instead), how many have no finite bound, and how many keep decisions are
uncertain (the margin to a threshold is within 1e-6 plus the decision's own bound;
the parity tests count those and compare every other decision bit for bit). The GPU
parity tests recompute the same counts from the oracle in the run and assert they do
not exceed these figures by more than a small margin (libm differences between hosts),
so that a change that widened the oracle's bounds, and so exempted more cells, fails.

Run: python tests/golden/make_exclusion_counts.py [names to recompute; default all]
"""
import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)
sys.path.insert(0, os.path.dirname(HERE))

import oracle  # noqa: E402
from paper_2608_27612_gb300 import workloads as W  # noqa: E402

TOL_ABS, TOL_REL = 1e-5, 1e-4


def block_counts(r, keep="keep_eager", unc="unc_eager"):
    w, err = r["w"], r["w_err"]
    tol = TOL_ABS + TOL_REL * np.abs(w)
    ill = ~(err <= tol)
    kept = r[keep].astype(bool)
    return {"outputs": int(w.size), "ill_conditioned": int(ill.sum()),
            "unbounded": int((~np.isfinite(err)).sum()), "decisions": int(w.size),
            "uncertain": int(r[unc].astype(bool).sum()), "kept": int((kept & ~r[unc].astype(bool)).sum()),
            "kept_ill_conditioned": int((kept & ill).sum())}


def add(a, b):
    return {k: a.get(k, 0) + b[k] for k in b}


def counts(w, g0=0, g1=None, block=50, gated=False):
    g1 = w.P if g1 is None else g1
    tot = {}
    keep, unc = ("keep_gated", "unc_gated") if gated else ("keep_eager", "unc_eager")
    for b0 in range(g0, g1, block):
        r = oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, g0=b0, g1=min(g1, b0 + block),
                            fields=("w", "w_err", keep, unc))
        tot = add(tot, block_counts(r, keep, unc))
    return tot


def c4_round2(n_genomes=8):
    """Round 2 of the first 8 of the first 40 genomes whose round 1 (by the oracle) found hidden nodes."""
    from hh_sources import round2_workload
    w1 = W.c4_round1(P=40)
    r1 = oracle.discover(w1.pop, w1.sources, w1.D, w1.theta, w1.band, fields=("keep_eager",))
    return round2_workload(w1, r1["keep_eager"], n_genomes)


def cases():
    import special_genomes as SG
    for D in (0, 1, 2, 3):
        yield "edge_d%d" % D, lambda D=D: counts(SG.edge_cases(D))
    for D in (4, 6):
        yield "classes_d%d" % D, lambda D=D: counts(SG.kernel_classes(D))
    yield "c2_d5_p100_wmin_eager", lambda: counts(SG.weight_filter())
    yield "c2_d5_p100_wmin_gated", lambda: counts(SG.weight_filter(), gated=True)
    yield "pergenome_d4", lambda: counts(SG.per_genome_slots())
    yield "separable_d6_eager", lambda: counts(SG.separable(6))
    yield "separable_d6_gated", lambda: counts(SG.separable(6), gated=True)
    yield "separable_d7_eager", lambda: counts(SG.separable(7))
    yield "c1_d4_eager", lambda: counts(W.c1())
    yield "c1_d4_gated", lambda: counts(W.c1(), gated=True)
    yield "c2_d5", lambda: counts(W.c2(D=5), block=250)
    yield "c2_d7", lambda: counts(W.c2(D=7))
    yield "c3_d6", lambda: counts(W.c3(D=6), block=32)
    yield "c4_r1_d8", lambda: counts(W.c4_round1(), block=10)
    yield "c4_r2_d8_g8", lambda: counts(c4_round2(), block=1)


def main():
    only = set(sys.argv[1:])
    try:
        with open(os.path.join(HERE, "exclusion_counts.json")) as f:
            old = json.load(f)
    except OSError:
        old = {}
    out = {"_about": "oracle exclusion counts per workload (tests/golden/make_exclusion_counts.py); "
                     "outputs are grid positions (halo excluded), decisions are eager keep decisions "
                     "unless the name says gated"}
    for name, fn in cases():
        if only and name not in only and name in old:
            out[name] = old[name]
            continue
        out[name] = fn()
        print(name, out[name], flush=True)
    with open(os.path.join(HERE, "exclusion_counts.json"), "w") as f:
        json.dump(out, f, indent=1, sort_keys=True)
        f.write("\n")


if __name__ == "__main__":
    main()
