"""Pins for the oracle's substrate network assembly and forward pass
(oracle/assembly.py): a linear genome whose every query keeps exactly Grid_3
gives connection counts per substrate configuration and weights in closed
form; a genome whose incoming query keeps nothing is pruned to nothing; hand
networks give the synchronous update's outputs step by step."""
import math

import numpy as np
import pytest

from oracle import assembly as A
from paper_2608_27612_gb300 import workloads as W

X1, Y1, X2, Y2, BIAS, HID, OUT = range(7)
IDN = 0
XOR_IN = [(-1.0, -1.0), (1.0, -1.0), (0.0, -1.0)]   # two inputs and the bias node
XOR_OUT = [(0.0, 1.0)]


def genome(conns):
    nodes = [(k, k, IDN, 0.0) for k in range(5)] + [(5, OUT, IDN, 0.0)]
    return W.population_from_lists([(nodes, conns)])


def grid3():
    """Global indices of Grid_3 and their coordinates."""
    base = (4 ** 4 - 4) // 3
    out = []
    for m in range(256):
        i = sum(((m >> (2 * k)) & 1) << k for k in range(4))
        j = sum(((m >> (2 * k + 1)) & 1) << k for k in range(4))
        out.append((base + m, (2 * i + 1) / 16 - 1, (2 * j + 1) / 16 - 1))
    return out


@pytest.mark.parametrize("enabled,rounds,n_phase2", [
    ((1, 0, 0, 0), 0, 0),            # feedforward: no hidden rounds
    ((1, 0, 0, 0), 1, 16 * 16 * 120),  # forward pairs of Grid_3: the target's row above the source's
    ((1, 1, 0, 0), 1, 2 * 16 * 16 * 120),
    ((1, 0, 1, 0), 1, 16 * 16 * 120 + 16 * 16 * 15),
    ((1, 0, 0, 1), 1, 16 * 16 * 120 + 256),
    ((1, 1, 1, 1), 1, 256 * 256)])
def test_linear_genome_networks_in_closed_form(enabled, rounds, n_phase2):
    # f = 4 x1 + 4 x2 (identity output): every outgoing query from (a, b) sees 4a + 4x and the incoming
    # query toward (0, 1) sees 4x, so each keeps exactly Grid_3 (V_3 = 1/64 < 0.03 < V_2, B_3 = 0.5 > 0.3 > B_4)
    pop = genome([(X1, 5, 4.0, True), (X2, 5, 4.0, True)])
    nets, n_unc = A.assemble(pop, XOR_IN, XOR_OUT, 4, 0.03, 0.3, enabled=enabled, rounds=rounds)
    assert n_unc.sum() == 0
    hidden, conns = nets[0]
    g3 = grid3()
    assert np.array_equal(hidden, sorted(p for p, _, _ in g3))
    assert len(conns) == 3 * 256 + 256 + n_phase2
    xy = {k + 4: (x, y) for k, (_, x, y) in enumerate(sorted(g3))}
    for s, d, w, t in conns:
        if s < 3:                           # input -> hidden: 4 a + 4 x_t, forward
            assert w == 4 * XOR_IN[s][0] + 4 * xy[d][0] and t == A.F
        elif d == 3:                        # hidden -> output: 4 x_s, forward
            assert w == 4 * xy[s][0] and t == A.F
        else:                               # hidden -> hidden: 4 x_s + 4 x_t
            assert w == 4 * xy[s][0] + 4 * xy[d][0]
            ys, yt = xy[s][1], xy[d][1]
            assert t == (A.S if s == d else A.F if ys < yt else A.B if ys > yt else A.L)
            assert enabled[t]
    # sorted by destination, then source
    keys = [(d, s) for s, d, _, _ in conns]
    assert keys == sorted(keys)


def test_genome_without_output_connections_prunes_everything():
    # f = 4 x2: the incoming query toward (0, 1) sees the constant 0 and keeps nothing
    pop = genome([(X2, 5, 4.0, True)])
    nets, n_unc = A.assemble(pop, XOR_IN, XOR_OUT, 4, 0.03, 0.3, rounds=1)
    assert n_unc.sum() == 0
    hidden, conns = nets[0]
    assert len(hidden) == 0 and conns == []


def sig(z):
    return 1.0 / (1.0 + math.exp(-z))


def test_forward_single_connection():
    for x in (0.0, 1.0, -0.5):
        for steps in (1, 3):
            out = A.forward(1, 1, [], [(0, 1, 2.5, 0)], [[x]], steps)
            assert abs(out[0, 0] - sig(2.5 * x)) < 1e-15
    assert A.forward(1, 1, [], [(0, 1, 2.5, 0)], [[1.0]], 0)[0, 0] == 0.0


def test_forward_chain_and_self_loop_step_by_step():
    w1, w2, ws = 1.5, -2.0, 0.75
    chain = [(0, 2, w1, 0), (2, 1, w2, 0)]
    x = 0.8
    assert abs(A.forward(1, 1, [9], chain, [[x]], 1)[0, 0] - 0.5) < 1e-15           # output saw hidden = 0
    assert abs(A.forward(1, 1, [9], chain, [[x]], 2)[0, 0] - sig(w2 * sig(w1 * x))) < 1e-15
    loop = chain + [(2, 2, ws, 3)]
    h1 = sig(w1 * x)
    h2 = sig(w1 * x + ws * h1)
    assert abs(A.forward(1, 1, [9], loop, [[x]], 3)[0, 0] - sig(w2 * h2)) < 1e-15
    # patterns are independent columns
    two = A.forward(1, 1, [9], loop, [[x], [-x]], 3)
    assert abs(two[1, 0] - A.forward(1, 1, [9], loop, [[-x]], 3)[0, 0]) < 1e-15
