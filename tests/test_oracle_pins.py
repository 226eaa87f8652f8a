"""Pins for the float64 oracle: values the paper prints, closed forms, library
routines, brute force and Theorem 1. No GPU is involved."""
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2608_27612_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
X1, Y1, X2, Y2, BIAS, HID, OUT = range(7)
IDN, SIG, TNH, GAU, SIN, ABS = range(6)


def golden(name):
    vals = {}
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if line and not line.startswith("#"):
            k, v, _cite = line.split()
            vals[k] = float(v)
    return vals


def inputs_nodes():
    return [(k, k, IDN, 0.0) for k in range(5)]


def genome(nodes, conns):
    return W.population_from_lists([(inputs_nodes() + nodes, conns)])


def coord(d, i):
    return (2 * i + 1) / 2 ** (d + 1) - 1


# ---- grid (Eq. 1) ------------------------------------------------------------

def test_paper_printed_grid_sizes():
    g = golden("paper_grid_values.txt")
    assert oracle.n_total(4) == g["n_total_d4"]
    assert oracle.n_total(7) == g["n_total_d7"]
    assert round(oracle.n_total(13) / 1e6) == g["n_total_d13_millions"]
    # two fp32 coordinates per position: 87,380 * 8 B = 682.7 KiB ~ "683 KB"
    assert round(oracle.n_total(7) * 8 / 1024) == g["grid_kb_d7"]
    # depth 4 has (4^5 - 1)/3 = 341 quadtree cells, each owning 4 child positions
    assert 4 * (4 ** 5 - 1) // 3 == oracle.n_total(4)


@pytest.mark.parametrize("D", [0, 1, 3, 5])
def test_index_is_a_bijection_with_children_rule(D):
    seen = set()
    for d in range(D + 1):
        n = 2 ** (d + 1)
        for i in range(n):
            for j in range(n):
                p = oracle.index(d, i, j)
                seen.add(p)
                if d < D:
                    base = oracle.index(d, i, j) - oracle.index(d, 0, 0)
                    for a in (0, 1):
                        for b in (0, 1):
                            c = oracle.index(d + 1, 2 * i + a, 2 * j + b) - oracle.index(d + 1, 0, 0)
                            assert c == 4 * base + a + 2 * b
    assert seen == set(range(oracle.n_total(D)))


def test_grid_positions_exact_and_disjoint_across_depths():
    pts = set()
    for d in range(8):
        n = 2 ** (d + 1)
        for i in range(n):
            x = Fraction(2 * i + 1, n) - 1
            assert float(x) == coord(d, i) and float(np.float32(x)) == float(x)
            pts.add((d, x))
    xs = {}
    for d, x in pts:
        assert x not in xs, "a coordinate repeats across depths"
        xs[x] = d


# ---- CPPN evaluation -----------------------------------------------------------

def test_cppn_identity_single_edge_is_linear():
    pop = genome([(9, OUT, IDN, 0.0)], [(X2, 9, 1.75, True)])
    xs = np.array([[0.3, -0.2, x, 0.9, 1.0] for x in np.linspace(-1, 1, 9)])
    out, err = oracle.cppn(pop, 0, xs)
    assert np.array_equal(out, 1.75 * xs[:, 2])
    assert np.all(err <= 1e-6 * (1 + np.abs(out)))


@pytest.mark.parametrize("act,ref", [
    (IDN, lambda z: z), (SIG, lambda z: 1 / (1 + math.exp(-z))), (TNH, math.tanh),
    (GAU, lambda z: math.exp(-z * z)), (SIN, math.sin), (ABS, abs)])
def test_cppn_activation_of_bias_matches_c_library(act, ref):
    for b in (0.0, -1.25, 0.5, 2.0):
        pop = genome([(7, OUT, act, b)], [])
        out, _ = oracle.cppn(pop, 0, np.array([[0.1, 0.2, 0.3, 0.4, 1.0]]))
        assert out[0] == pytest.approx(ref(np.float32(b)), abs=1e-15)
    assert oracle.cppn(genome([(7, OUT, SIG, 0.0)], []), 0, np.zeros((1, 5)))[0][0] == 0.5
    assert oracle.cppn(genome([(7, OUT, GAU, 0.0)], []), 0, np.zeros((1, 5)))[0][0] == 1.0
    assert oracle.cppn(genome([(7, OUT, TNH, 0.0)], []), 0, np.zeros((1, 5)))[0][0] == 0.0


def test_cppn_chain_closed_form_and_id_order_independence():
    # hidden ids deliberately not in topological order: 12 -> 10 -> out(5)
    nodes = [(5, OUT, IDN, 0.25), (10, HID, SIN, 0.0), (12, HID, GAU, 0.5)]
    conns = [(12, 10, -1.5, True), (X2, 12, 2.0, True), (10, 5, 3.0, True), (Y1, 5, -0.5, True),
             (BIAS, 10, 0.75, True), (Y2, 5, 9.0, False)]
    pop = genome(nodes, conns)
    rng = np.random.default_rng(1)
    xs = np.column_stack([rng.uniform(-1, 1, (20, 4)), np.ones(20)])
    out, _ = oracle.cppn(pop, 0, xs)
    h12 = np.exp(-(0.5 + 2.0 * xs[:, 2]) ** 2)
    h10 = np.sin(-1.5 * h12 + 0.75)
    np.testing.assert_allclose(out, 0.25 + 3.0 * h10 - 0.5 * xs[:, 1], rtol=0, atol=1e-14)


def test_cppn_dead_node_and_disabled_edges_do_not_change_output():
    base = [(5, OUT, TNH, 0.0), (6, HID, SIG, 0.0)]
    conns = [(X2, 6, 1.0, True), (6, 5, 2.0, True)]
    p1 = genome(base, conns)
    p2 = genome(base + [(7, HID, SIN, 0.3)], conns + [(Y2, 7, 4.0, True), (6, 7, 1.0, True),
                                                     (7, 5, 5.0, False)])
    xs = np.column_stack([np.random.default_rng(2).uniform(-1, 1, (16, 4)), np.ones(16)])
    assert np.array_equal(oracle.cppn(p1, 0, xs)[0], oracle.cppn(p2, 0, xs)[0])


def test_cppn_rejects_cycles_and_malformed_genomes():
    cyc = genome([(5, OUT, IDN, 0.0), (6, HID, SIG, 0.0), (7, HID, SIG, 0.0)],
                 [(X2, 6, 1.0, True), (6, 7, 1.0, True), (7, 6, 1.0, True), (7, 5, 1.0, True)])
    assert oracle.check_population(cyc) == (oracle.ORA_ERR_CYCLE, 0)
    # the same loop with one edge disabled is acyclic
    ok = genome([(5, OUT, IDN, 0.0), (6, HID, SIG, 0.0), (7, HID, SIG, 0.0)],
                [(X2, 6, 1.0, True), (6, 7, 1.0, True), (7, 6, 1.0, False), (7, 5, 1.0, True)])
    assert oracle.check_population(ok) == (0, -1)
    two_out = genome([(5, OUT, IDN, 0.0), (6, OUT, IDN, 0.0)], [])
    assert oracle.check_population(two_out)[0] == oracle.ORA_ERR_ARG
    into_input = genome([(5, OUT, IDN, 0.0)], [(5, X2, 1.0, True)])
    assert oracle.check_population(into_input)[0] == oracle.ORA_ERR_ARG


def test_cppn_bound_covers_float32_evaluation():
    """The error bound must cover an independent float32 evaluation (numpy)."""
    pop = W.random_population(60, seed=11, h_lo=0, h_hi=12, e_max=40)
    rng = np.random.default_rng(3)
    f32 = np.float32
    acts = {IDN: lambda z: z, SIG: lambda z: f32(1) / (f32(1) + np.exp(-z)), TNH: np.tanh,
            GAU: lambda z: np.exp(-z * z), SIN: np.sin, ABS: np.abs}
    for g in range(pop.P):
        nodes, conns = pop.genome(g)
        xs = np.column_stack([rng.uniform(-1, 1, (64, 4)), np.ones(64)]).astype(np.float32)
        ref, err = oracle.cppn(pop, g, xs.astype(np.float64))
        val = {i: xs[:, k] for (i, k, a, b) in nodes if k < 5}
        pending = [(i, a, b) for (i, k, a, b) in nodes if k >= 5]
        while pending:
            for t, (i, a, b) in enumerate(pending):
                ins = [(s, w) for (s, d, w, e) in conns if e and d == i]
                if all(s in val for s, _ in ins):
                    z = np.full(64, f32(b))
                    for s, w in ins:
                        z = z + f32(w) * val[s]
                    val[i] = acts[a](z.astype(f32)).astype(f32)
                    pending.pop(t)
                    break
        out_id = [i for (i, k, a, b) in nodes if k == OUT][0]
        assert np.all(np.abs(val[out_id].astype(np.float64) - ref) <= err + 1e-300)


# ---- variance, band, keep: closed forms -------------------------------------

def linear(alpha, beta, gamma, side=W.SIDE_OUT):
    xs, ys = (X2, Y2) if side == W.SIDE_OUT else (X1, Y1)
    return genome([(5, OUT, IDN, 0.0)], [(xs, 5, alpha, True), (ys, 5, beta, True), (BIAS, 5, gamma, True)])


@pytest.mark.parametrize("alpha,beta,gamma", [(4.0, 0.0, 0.0), (0.0, 4.0, 0.25), (3.0, -1.0, -0.5),
                                              (-0.75, 2.5, 1.0)])
@pytest.mark.parametrize("side", [W.SIDE_OUT, W.SIDE_IN])
def test_linear_genome_variance_and_band_closed_forms(alpha, beta, gamma, side):
    """f = alpha x + beta y + gamma: V at depth d = (alpha^2 + beta^2) 4^-(d+2) (0 at depth D),
    B at depth d = max(|alpha|, |beta|) 2^-d, at every position including the border."""
    D = 5
    src = W.shared_sources([(0.5, -1.0, side)])
    r = oracle.discover(linear(alpha, beta, gamma, side), src, D, 0.03, 0.3)
    for d in range(D + 1):
        lo, hi = oracle.index(d, 0, 0), oracle.n_total(d)
        V = r["var"][0, 0, lo:hi]
        Vd = 0.0 if d == D else (alpha ** 2 + beta ** 2) * 4.0 ** -(d + 2)
        np.testing.assert_allclose(V, Vd, rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["bnd"][0, 0, lo:hi], max(abs(alpha), abs(beta)) * 2.0 ** -d,
                                   rtol=1e-12, atol=1e-15)


def test_worked_example_depth4_keeps_exactly_grid3():
    """alpha=4, beta=0, D=4, theta=0.03, band=0.3: V_d = 4^-d and B_d = 4 * 2^-d, so depths
    0..2 split, depth 3 is a low-variance leaf with B = 0.5 > 0.3 and depth 4 has B = 0.25:
    eager, gated and lazy all keep exactly Grid_3 (256 positions)."""
    pop, D = linear(4.0, 0.0, 0.0), 4
    src = W.shared_sources([(0.0, -1.0, W.SIDE_OUT)])
    r = oracle.discover(pop, src, D, 0.03, 0.3)
    lz, _ = oracle.lazy(pop, src, D, 0.03, 0.3)
    want = np.zeros(oracle.n_total(D), np.uint8)
    want[oracle.index(3, 0, 0):oracle.n_total(3)] = 1
    for m in (r["keep_eager"], r["keep_gated"], lz):
        assert np.array_equal(m[0, 0], want)
    assert want.sum() == 256
    assert r["unc_eager"].sum() == 0 and r["unc_gated"].sum() == 0


def test_strict_inequalities_at_exact_ties():
    """A cell splits when V > theta (Eq. 2), a position passes the band test when B > band and
    the weight filter when |w| > w_min, all strictly. For f = 4x at D = 4, V_d = 4^-d, B_d =
    4 * 2^-d and the depth-3 outputs are odd multiples of 1/4, all exact in binary, so each
    threshold can be met exactly."""
    pop, D = linear(4.0, 0.0, 0.0), 4
    src = W.shared_sources([(0.0, -1.0, W.SIDE_OUT)])
    lo = lambda d: oracle.index(d, 0, 0)
    # theta = V_1 = 1/4: depth 1 does not split. Eager keeps depths 1..3 (B = 2, 1, 1/2 > 0.3);
    # gated and lazy keep depth 1 only (depth 2's parents did not split).
    r = oracle.discover(pop, src, D, 0.25, 0.3)
    lz, _ = oracle.lazy(pop, src, D, 0.25, 0.3)
    want_e = np.zeros(oracle.n_total(D), np.uint8)
    want_e[lo(1):oracle.n_total(3)] = 1
    want_g = np.zeros(oracle.n_total(D), np.uint8)
    want_g[lo(1):oracle.n_total(1)] = 1
    assert np.array_equal(r["keep_eager"][0, 0], want_e)
    assert np.array_equal(r["keep_gated"][0, 0], want_g) and np.array_equal(lz[0, 0], want_g)
    # band = B_3 = 1/2: the depth-3 leaves fail the band test and nothing is kept
    r = oracle.discover(pop, src, D, 0.03, 0.5)
    lz, _ = oracle.lazy(pop, src, D, 0.03, 0.5)
    assert r["keep_eager"].sum() == 0 and r["keep_gated"].sum() == 0 and lz.sum() == 0
    # w_min = 1/4: the 2 x 16 depth-3 positions with f = -1/4, +1/4 drop out of the 256
    r = oracle.discover(pop, src, D, 0.03, 0.3, 0.25)
    lz, _ = oracle.lazy(pop, src, D, 0.03, 0.3, 0.25)
    keep = r["keep_eager"][0, 0]
    assert keep.sum() == 224 and np.all(np.abs(r["w"][0, 0][keep == 1]) > 0.25)
    assert np.array_equal(lz[0, 0], r["keep_gated"][0, 0]) and np.array_equal(keep, r["keep_gated"][0, 0])


@pytest.mark.parametrize("axis", ["x", "y"])
def test_separable_gauss_variance_and_band(axis):
    """f = gauss(x2) (or gauss(y2)): the four children of a cell at (x, y) sit at x +- h,
    so V = ((g(x+h) - g(x-h)) / 2)^2; B = min(|g(x) - g(x-s)|, |g(x) - g(x+s)|) along the
    varying axis (the other axis contributes 0)."""
    D = 4
    src = W.shared_sources([(0.0, -1.0, W.SIDE_OUT)])
    pop = genome([(5, OUT, GAU, 0.0)], [((X2 if axis == "x" else Y2), 5, 1.3, True)])
    r = oracle.discover(pop, src, D, 0.03, 0.3)
    k = float(np.float32(1.3))  # weights are stored in fp32
    g = lambda t: math.exp(-(k * t) ** 2)
    for d in range(D + 1):
        n = 2 ** (d + 1)
        h, s = 2.0 ** -(d + 2), 2.0 ** -d
        for i in range(n):
            for j in range(n):
                p = oracle.index(d, i, j)
                t = coord(d, i) if axis == "x" else coord(d, j)
                V = 0.0 if d == D else ((g(t + h) - g(t - h)) / 2) ** 2
                B = min(abs(g(t) - g(t - s)), abs(g(t) - g(t + s)))
                assert r["var"][0, 0, p] == pytest.approx(V, abs=1e-15)
                assert r["bnd"][0, 0, p] == pytest.approx(B, abs=1e-15)


@pytest.mark.parametrize("inp", [X2, Y2])
@pytest.mark.parametrize("edge", [-1.0, 1.0])
def test_band_zero_where_the_halo_mirrors_the_border(inp, edge):
    """f = |u - edge| for the grid coordinate u (x or y) is linear inside the domain, but the
    halo neighbour beyond that edge (distance 2^-d from a border position at distance 2^-(d+1)
    from the edge) mirrors the border position: the band value is exactly 0 on the border row or
    column at the edge and 2^-d everywhere else (the halo beyond the other edge continues the
    line), and the variance is 4^-(d+2) below depth D. Pins which halo side each neighbour
    of a border position reads."""
    D = 4
    pop = genome([(5, OUT, ABS, 0.0)], [(inp, 5, 1.0, True), (BIAS, 5, -edge, True)])
    r = oracle.discover(pop, W.shared_sources([(0.0, -1.0, W.SIDE_OUT)]), D, 0.03, 0.3)
    for d in range(D + 1):
        n = 2 ** (d + 1)
        for i in range(n):
            for j in range(n):
                u = i if inp == X2 else j
                border = u == (0 if edge < 0 else n - 1)
                p = oracle.index(d, i, j)
                assert r["bnd"][0, 0, p] == (0.0 if border else 2.0 ** -d)
                assert r["var"][0, 0, p] == (0.0 if d == D else 4.0 ** -(d + 2))


def test_constant_genome_keeps_nothing():
    # depends only on the source coordinates (OUT side): constant over the grid
    pop = genome([(5, OUT, SIG, 0.2), (6, HID, SIN, 0.0)],
                 [(X1, 6, 2.0, True), (Y1, 5, 1.0, True), (6, 5, -3.0, True)])
    src = W.shared_sources([(0.3, -1.0, W.SIDE_OUT), (-0.7, 0.4, W.SIDE_OUT)])
    r = oracle.discover(pop, src, 4, 0.03, 0.3)
    assert np.all(r["var"] == 0) and np.all(r["bnd"] == 0)
    assert r["keep_eager"].sum() == 0 and r["keep_gated"].sum() == 0


def test_reflection_symmetry_of_x_only_genome():
    pop = genome([(5, OUT, SIN, 0.0), (6, HID, TNH, 0.1)],
                 [(X2, 6, 2.5, True), (6, 5, 4.0, True), (X2, 5, 3.0, True)])
    src = W.shared_sources([(0.0, -1.0, W.SIDE_OUT)])
    D = 5
    r = oracle.discover(pop, src, D, 0.03, 0.3)
    assert r["keep_eager"].sum() > 0
    for d in range(D + 1):
        n = 2 ** (d + 1)
        for i in range(n):
            for j in range(n):
                a, b = oracle.index(d, i, j), oracle.index(d, i, n - 1 - j)
                assert r["keep_eager"][0, 0, a] == r["keep_eager"][0, 0, b]
                assert r["w"][0, 0, a] == r["w"][0, 0, b]


def test_in_side_equals_out_side_of_swapped_genome():
    pop = W.random_population(8, seed=21)
    swapped = []
    swap = {X1: X2, Y1: Y2, X2: X1, Y2: Y1}
    for g in range(pop.P):
        nodes, conns = pop.genome(g)
        nodes = [(i, swap.get(k, k) if k < 5 else k, a, b) for (i, k, a, b) in nodes]
        swapped.append((nodes, conns))
    pop_sw = W.population_from_lists(swapped)
    D = 4
    o = oracle.discover(pop, W.shared_sources([(0.25, -1.0, W.SIDE_OUT)]), D, 0.03, 0.3)
    i = oracle.discover(pop_sw, W.shared_sources([(0.25, -1.0, W.SIDE_IN)]), D, 0.03, 0.3)
    assert np.array_equal(o["w"], i["w"]) and np.array_equal(o["keep_eager"], i["keep_eager"])


def test_per_genome_slots_address_like_shared_slots():
    """Per-genome query slots (a [P, S] slot table with a count per genome, as the hidden-to-hidden
    round uses): over the genome range [1, 5), genome g's slot s is evaluated exactly like the same
    point given as a shared slot, and a slot at or past the genome's count keeps nothing and holds
    zeros; the lazy tree reads the same slots."""
    pop = W.random_population(5, seed=31)
    rng = np.random.default_rng(7)
    P, S, D = 5, 3, 4
    a = rng.uniform(-1, 1, (P, S)).astype(np.float32)
    b = rng.uniform(-1, 1, (P, S)).astype(np.float32)
    side = rng.integers(0, 2, (P, S)).astype(np.int32)
    count = np.array([3, 1, 0, 2, 3], np.int32)
    per = W.Sources(a=a, b=b, side=side, count=count)
    r = oracle.discover(pop, per, D, 0.03, 0.3, g0=1, g1=5)
    lz, _ = oracle.lazy(pop, per, D, 0.03, 0.3, g0=1, g1=5)
    assert np.array_equal(lz, r["keep_gated"])
    used = 0
    for gl, g in enumerate(range(1, 5)):
        for k in range(S):
            if k < count[g]:
                ref = oracle.discover(pop, W.shared_sources([(float(a[g, k]), float(b[g, k]), int(side[g, k]))]),
                                      D, 0.03, 0.3, g0=g, g1=g + 1)
                for f in ("w", "w_halo", "var", "bnd", "keep_eager", "keep_gated"):
                    assert np.array_equal(r[f][gl, k], ref[f][0, 0]), (g, k, f)
                used += 1
            else:
                assert not r["w"][gl, k].any() and not r["keep_eager"][gl, k].any() and not lz[gl, k].any()
    assert used == 6


# ---- brute force: re-evaluation at Eq. 1 coordinates ------------------------

def test_discover_matches_direct_evaluation_at_grid_and_halo_points():
    w = W.c2(D=5, P=6)
    D = w.D
    r = oracle.discover(w.pop, w.sources, D, w.theta, w.band)
    rng = np.random.default_rng(5)
    for g in range(w.P):
        for s in range(w.S):
            a, b, side = float(w.sources.a[s]), float(w.sources.b[s]), int(w.sources.side[s])
            pts, idx = [], []
            for _ in range(40):
                d = int(rng.integers(0, D + 1)); n = 2 ** (d + 1)
                i, j = int(rng.integers(0, n)), int(rng.integers(0, n))
                pts.append((d, i, j)); idx.append(oracle.index(d, i, j))
            def q(x, y):
                return [a, b, x, y, 1.0] if side == W.SIDE_OUT else [x, y, a, b, 1.0]
            ins = [q(coord(d, i), coord(d, j)) for (d, i, j) in pts]
            ref, _ = oracle.cppn(w.pop, g, np.array(ins))
            assert np.array_equal(ref, r["w"][g, s, idx])
            # variance from numpy over the 4 children, band from the 4 neighbours
            for (d, i, j), p in zip(pts, idx):
                s_ = 2.0 ** -d
                x, y = coord(d, i), coord(d, j)
                nb = oracle.cppn(w.pop, g, np.array([q(x - s_, y), q(x + s_, y), q(x, y - s_), q(x, y + s_)]))[0]
                c0 = r["w"][g, s, p]
                dl, dr, db, dt = np.abs(c0 - nb)
                assert r["bnd"][g, s, p] == pytest.approx(max(min(dt, db), min(dl, dr)), abs=1e-14)
                if d < D:
                    ch = [q(coord(d + 1, 2 * i + (k & 1)), coord(d + 1, 2 * j + (k >> 1))) for k in range(4)]
                    v = np.var(oracle.cppn(w.pop, g, np.array(ch))[0])
                    assert r["var"][g, s, p] == pytest.approx(v, abs=1e-14)
            # halo layout: side 0 (i=-1), 1 (i=n), 2 (j=-1), 3 (j=n)
            d = int(rng.integers(0, D + 1)); n = 2 ** (d + 1); t = int(rng.integers(0, n))
            hoff = 8 * (2 ** d - 1)
            hp = [(-1, t), (n, t), (t, -1), (t, n)]
            ref, _ = oracle.cppn(w.pop, g, np.array([q(coord(d, i), coord(d, j)) for i, j in hp]))
            assert np.array_equal(ref, r["w_halo"][g, s, [hoff + k * n + t for k in range(4)]])


def test_eq2_active_mask_by_recursion():
    """Gated keep = eager keep AND every ancestor split (Eq. 2), checked by walking up."""
    w = W.c2(D=4, P=20)
    r = oracle.discover(w.pop, w.sources, w.D, w.theta, w.band)
    for g in range(w.P):
        for s in range(w.S):
            for d in range(w.D + 1):
                n = 2 ** (d + 1)
                for i in range(n):
                    for j in range(n):
                        act, (pi, pj) = True, (i, j)
                        for dd in range(d - 1, -1, -1):
                            pi, pj = pi >> 1, pj >> 1
                            act = act and r["var"][g, s, oracle.index(dd, pi, pj)] > w.theta
                        p = oracle.index(d, i, j)
                        assert r["keep_gated"][g, s, p] == (r["keep_eager"][g, s, p] and act)


# ---- Theorem 1 ----------------------------------------------------------------

def _theorem1(w, g1=None):
    r = oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, g1=g1,
                        fields=("keep_eager", "keep_gated", "unc_gated"))
    lz, evals = oracle.lazy(w.pop, w.sources, w.D, w.theta, w.band, g1=g1)
    assert np.all(lz <= r["keep_eager"]), "lazy must be a subset of eager"
    assert np.array_equal(lz, r["keep_gated"]), "lazy must equal the gated mask"
    return r, lz, evals


def test_theorem1_single_genome():
    _theorem1(W.c1())


def test_theorem1_population_depth5():
    r, lz, _ = _theorem1(W.c2(D=5))
    assert lz.sum() > 0 and r["keep_eager"].sum() > lz.sum()


@pytest.mark.slow
def test_theorem1_population_depth7_50_genomes():
    _theorem1(W.c2(D=7), g1=50)


def test_weight_filter_variant():
    w = W.c2(D=4, P=30)
    r0 = oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, 0.0)
    r1 = oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, 0.1)
    assert np.all(r1["keep_eager"] <= r0["keep_eager"])
    want = r0["keep_eager"] & (np.abs(r0["w"]) > 0.1)
    assert np.array_equal(r1["keep_eager"], want)
    lz, _ = oracle.lazy(w.pop, w.sources, w.D, w.theta, w.band, 0.1)
    assert np.array_equal(lz, r1["keep_gated"])


def test_keep_at_matches_whole_grid_decisions():
    """Per-position decisions by direct queries equal the whole-grid definition."""
    w = W.c2(D=5, P=12)
    r = oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, fields=("w", "var", "bnd", "keep_eager", "unc_eager"))
    pts = [(d, i, j) for d in range(w.D + 1) for i in range(2 ** (d + 1)) for j in range(2 ** (d + 1))]
    d, i, j = (np.array(x) for x in zip(*pts))
    idx = np.array([oracle.index(*p) for p in pts])
    for g in range(w.P):
        for s in range(w.S):
            o = oracle.keep_at(w.pop, g, float(w.sources.a[s]), float(w.sources.b[s]), int(w.sources.side[s]),
                               w.D, w.theta, w.band, 0.0, d, i, j)
            assert np.array_equal(o["w"], r["w"][g, s, idx])
            np.testing.assert_allclose(o["var"], r["var"][g, s, idx], rtol=0, atol=1e-15)
            np.testing.assert_allclose(o["bnd"], r["bnd"][g, s, idx], rtol=0, atol=1e-15)
            assert np.array_equal(o["keep"], r["keep_eager"][g, s, idx])
            assert np.array_equal(o["unc"], r["unc_eager"][g, s, idx])
