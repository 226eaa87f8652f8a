"""Pins for the oracle's method variants (oracle/variants.py)."""
import numpy as np

import oracle
from oracle import variants as VAR
from paper_2608_27612_gb300 import workloads as W


def test_weight_scaling_closed_values():
    thr, wm = 0.2, 3.0
    w = np.array([0.2, -0.2, 0.1, -0.05, 1.0, -1.0, 0.6, -0.6, 1.7, -4.0, 0.0])
    want = np.array([0.0, 0.0, 0.0, 0.0, 3.0, -3.0, 1.5, -1.5, 3.0, -3.0, 0.0])
    assert np.allclose(VAR.scale_weights(w, thr, wm), want, rtol=0, atol=1e-15)
    # monotone above the threshold, odd in w
    x = np.linspace(0.21, 1.0, 50)
    s = VAR.scale_weights(x, thr, wm)
    assert np.all(np.diff(s) > 0) and np.array_equal(VAR.scale_weights(-x, thr, wm), -s)

X2, Y2, BIAS, OUT = 2, 3, 4, 6


def linear(alpha, beta, gamma):
    nodes = [(k, k, 0, 0.0) for k in range(5)] + [(5, OUT, 0, 0.0)]
    conns = [(X2, 5, alpha, True), (Y2, 5, beta, True), (BIAS, 5, gamma, True)]
    return W.population_from_lists([(nodes, conns)])


def test_subtree_variance_linear_closed_form():
    D = 5
    for alpha, beta, gamma in [(4.0, 0.0, 0.0), (1.5, -2.0, 0.5), (0.0, 0.75, -1.0)]:
        r = oracle.discover(linear(alpha, beta, gamma), W.shared_sources([(0.0, -1.0, W.SIDE_OUT)]), D, 0.03, 0.3,
                            fields=("w", "w_err", "var"))
        V, bound, split, unc = VAR.subtree_split(r["w"][0, 0], r["w_err"][0, 0], D, 0.03)
        h = 2.0 ** -D
        for d in range(D):
            k = 2 ** (D - d)
            want = (alpha ** 2 + beta ** 2) * h * h * (k * k - 1) / 12
            seg = V[(4 ** (d + 1) - 4) // 3:(4 ** (d + 2) - 4) // 3]
            assert np.allclose(seg, want, rtol=1e-12, atol=1e-15)
        # one level above the leaves the subtree variance is the four-children variance
        lo, hi = (4 ** D - 4) // 3, (4 ** (D + 1) - 4) // 3
        assert np.allclose(V[lo:hi], r["var"][0, 0][lo:hi], rtol=1e-12, atol=1e-15)
        assert np.all(bound >= 0)


def test_subtree_variance_constant_genome_is_zero():
    r = oracle.discover(linear(0.0, 0.0, 0.7), W.shared_sources([(0.0, -1.0, W.SIDE_OUT)]), 4, 0.03, 0.3,
                        fields=("w", "w_err"))
    V, bound, split, unc = VAR.subtree_split(r["w"][0, 0], r["w_err"][0, 0], 4, 0.03)
    assert np.all(V == 0) and not split.any()



def test_subtree_split_is_strict_at_an_exact_tie():
    """One level above the leaves a cell's subtree is its four children: for f = 4x its variance
    is 4^2 * 4^-(d+2) = 4^-(D-1) at d = D - 1, exact in binary. With theta equal to it those
    cells do not split (V > theta is strict), while every cell above (more leaves, larger
    variance) does."""
    D = 3
    r = oracle.discover(linear(4.0, 0.0, 0.0), W.shared_sources([(0.0, -1.0, W.SIDE_OUT)]), D, 0.03, 0.3,
                        fields=("w", "w_err"))
    theta = 4.0 ** -(D - 1)
    V, bound, split, unc = VAR.subtree_split(r["w"][0, 0], r["w_err"][0, 0], D, theta)
    lo, hi = (4 ** D - 4) // 3, (4 ** (D + 1) - 4) // 3
    assert np.all(V[lo:hi] == theta) and not split[lo:hi].any() and split[:lo].all()
