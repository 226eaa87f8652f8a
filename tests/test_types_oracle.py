"""Pins for the oracle's connection-type classification (Section 6 taxonomy:
forward when the source lies below the target, backward above, lateral on the
same row, self-loop when source and target coincide) and for the six substrate
configurations of Section 6's table as the library exports them."""
import numpy as np
import pytest

import oracle
from paper_2608_27612_gb300 import emr

F, B, L, S = oracle.TYPE_F, oracle.TYPE_B, oracle.TYPE_L, oracle.TYPE_S


def n_total(D):
    return (4 ** (D + 2) - 4) // 3


def depth_of(gidx):
    d = np.zeros(len(gidx), np.int64)
    for e in range(1, 15):
        d += gidx >= (4 ** (e + 1) - 4) // 3
    return d


def rows_of(gidx):
    """Grid row j of each global index (Morton decode, written with integer shifts)."""
    d = depth_of(gidx)
    m = gidx - (4 ** (d + 1) - 4) // 3
    j = np.zeros_like(m)
    for k in range(15):
        j |= ((m >> (2 * k + 1)) & 1) << k
    return d, j


def test_slots_off_every_row_are_all_forward_or_all_backward():
    D = 5
    g = np.arange(n_total(D))
    # the substrate's input row y = -1 and output row y = +1 lie off every grid row
    assert np.all(oracle.conn_types(0.0, -1.0, 0, g) == F)   # input -> position: upward
    assert np.all(oracle.conn_types(0.0, 1.0, 1, g) == F)    # position -> output: upward
    assert np.all(oracle.conn_types(0.3, 1.0, 0, g) == B)    # from above the grid
    assert np.all(oracle.conn_types(-0.7, -1.0, 1, g) == B)  # into a node below the grid


@pytest.mark.parametrize("ds,is_,js", [(0, 1, 0), (2, 3, 5), (3, 0, 15), (4, 17, 9)])
def test_on_grid_slot_counts_match_closed_form(ds, is_, js):
    D = 5
    a = (2 * is_ + 1) / 2.0 ** (ds + 1) - 1.0
    b = (2 * js + 1) / 2.0 ** (ds + 1) - 1.0
    g = np.arange(n_total(D))
    t = oracle.conn_types(a, b, 0, g)
    d, j = rows_of(g)
    for e in range(D + 1):
        n = 2 ** (e + 1)
        te = t[d == e]
        # rows strictly above the slot: (2j+1) / 2^(e+1) > (2 js + 1) / 2^(ds+1), cross-multiplied
        above = sum(1 for jj in range(n) if (2 * jj + 1) * 2 ** (ds + 1) > (2 * js + 1) * 2 ** (e + 1))
        same = sum(1 for jj in range(n) if (2 * jj + 1) * 2 ** (ds + 1) == (2 * js + 1) * 2 ** (e + 1))
        assert same == (1 if e == ds else 0)
        assert np.sum(te == F) == n * above
        assert np.sum(te == S) == (1 if e == ds else 0)
        assert np.sum(te == L) == (n - 1 if e == ds else 0)
        assert np.sum(te == B) == n * (n - above - same)
    # the self-loop is the slot's own position
    p = (4 ** (ds + 1) - 4) // 3 + sum((((is_ >> k) & 1) << (2 * k)) | (((js >> k) & 1) << (2 * k + 1))
                                       for k in range(ds + 1))
    assert t[p] == S and np.sum(t == S) == 1


def test_incoming_side_reverses_forward_and_backward():
    rng = np.random.default_rng(7)
    D = 4
    g = np.arange(n_total(D))
    for _ in range(6):
        ds = int(rng.integers(0, D + 1))
        i, j = (int(v) for v in rng.integers(0, 2 ** (ds + 1), 2))
        a = (2 * i + 1) / 2.0 ** (ds + 1) - 1.0
        b = (2 * j + 1) / 2.0 ** (ds + 1) - 1.0
        out, inn = oracle.conn_types(a, b, 0, g), oracle.conn_types(a, b, 1, g)
        swap = np.array([B, F, L, S], np.uint8)
        assert np.array_equal(inn, swap[out])


def test_substrate_configurations_match_the_table():
    # Section 6's table: F, H(idden rounds), B, L, S per configuration
    table = {emr.SUBSTRATE_FEEDFORWARD: ("F", False), emr.SUBSTRATE_HH: ("F", True),
             emr.SUBSTRATE_BACKWARD: ("FB", True), emr.SUBSTRATE_LATERAL: ("FL", True),
             emr.SUBSTRATE_SELF: ("FS", True), emr.SUBSTRATE_FULL: ("FBLS", True)}
    bit = {"F": emr.CONN_F, "B": emr.CONN_B, "L": emr.CONN_L, "S": emr.CONN_S}
    for cfg, (letters, hh) in table.items():
        types, rounds = emr.substrate_config(cfg)
        assert types == sum(bit[c] for c in letters)
        assert rounds == (1 if hh else 0)
    with pytest.raises(emr.EmrError):
        emr.substrate_config(6)
