"""Variants of the method that the paper does not use by default (float64, oracle side).

TEST INFRASTRUCTURE ONLY, like the rest of oracle/. It shares no code with the
CUDA path.

  scale_weights   HyperNEAT's expression threshold and weight scaling (the
                  indirect encoding of Section 2): an output of magnitude at
                  most thr is not expressed (0); a larger one keeps its sign and
                  has its magnitude, clamped to 1, mapped linearly from
                  (thr, 1] onto (0, w_max].

  subtree_split   ES-HyperNEAT's reading of a cell's variance: the population
                  variance of the outputs at all depth-D descendants of a cell
                  of depth d < D (4^(D-d) leaves), against theta (Section 3.2
                  uses the four children instead; this is the alternative).
                  Each value carries a bound for the device's fp32 evaluation:
                  the leaves' own error bounds propagated through the
                  variance, plus rounding of a level-by-level merge.

Parity status: scale_weights pinned (tests/test_variants_oracle.py) by its
values at the threshold, at +-1, at the midpoint, beyond 1 and below the
threshold. subtree_split pinned by the closed form for a linear genome
(variance of a k x k grid of spacing h: (alpha^2 + beta^2) h^2 (k^2 - 1) / 12),
by equality with the four-children variance one level above the leaves, by
zero for a constant genome, and by its strict split at an exact tie.
"""
from __future__ import annotations

import numpy as np


def scale_weights(w, thr, w_max):
    w = np.asarray(w, np.float64)
    a = np.abs(w)
    out = np.sign(w) * w_max * (np.minimum(a, 1.0) - thr) / (1.0 - thr)
    return np.where(a > thr, out, 0.0)


U32 = 2.0 ** -24


def _off(d):
    return (4 ** (d + 1) - 4) // 3


def subtree_split(w, w_err, D, theta, margin=1e-6):
    """One pair's outputs w (and error bounds) over the whole grid (global index): per position of
    depths 0..D-1 the subtree-leaf variance V, its bound, the split decision V > theta and whether
    that decision is uncertain (|V - theta| within margin + bound). Arrays of length off(D)."""
    w = np.asarray(w, np.float64)
    e = np.asarray(w_err, np.float64)
    X0, E0 = w[_off(D):_off(D + 1)], e[_off(D):_off(D + 1)]
    n = _off(D)
    V = np.zeros(n); bound = np.zeros(n)
    for d in range(D):
        k = 4 ** (D - d)
        X, E = X0.reshape(-1, k), E0.reshape(-1, k)      # Morton: a cell's leaves are contiguous
        mu = X.mean(axis=1)
        dev = X - mu[:, None]
        v = (dev ** 2).mean(axis=1)
        ee = E + E.mean(axis=1)[:, None]                 # bound on |error of x_i - error of the mean|
        prop = 2.0 * (np.abs(dev) * ee).mean(axis=1) + (ee ** 2).mean(axis=1)
        rnd = (24 * (D - d) + 16) * U32 * (v + prop + (np.abs(X) + E).max(axis=1) ** 2)
        V[_off(d):_off(d + 1)] = v
        bound[_off(d):_off(d + 1)] = 2.0 * (prop + rnd)
    split = (V > theta).astype(np.uint8)
    unc = (np.abs(V - theta) <= margin + bound).astype(np.uint8)
    return V, bound, split, unc
