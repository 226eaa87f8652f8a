"""Strength of the oracle's pins: a plausible mistake planted in a copy of the
oracle's C source (a dropped term, a wrong divisor, sign, index or operand, a
non-strict comparison) must make at least one pin of test_oracle_pins.py fail.

Each mutant is compiled into a temporary directory and exercised in a child
process (a mutant that crashed could not take the test run with it); the
installed oracle is never touched. No GPU is involved.
"""
import os
import subprocess
import sys
import tempfile

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
SRC = os.path.join(ROOT, "oracle", "emr_oracle.c")

# name: (text in emr_oracle.c, its replacement[, the pins to run instead of PINS]).
# Every mutant stays memory-safe (indices stay within the buffers the unmutated
# oracle sizes).
MUTATIONS = {
    # Section 3.2: population variance of the four children
    "variance_divides_by_3": ("v += dq * dq / 4.0;", "v += dq * dq / 3.0;"),
    "variance_drops_a_child": ("for (int q = 0; q < 4; q++) {\n                            double dq = c[q] - m;",
                               "for (int q = 0; q < 3; q++) {\n                            double dq = c[q] - m;"),
    "variance_wrong_mean": ("\n                            m += c[q] / 4.0;", "\n                            m += c[q] / 2.0;"),
    "children_drop_row_offset": ("int64_t ch = level_offset(d + 1) + morton(2 * i + (q & 1), 2 * j + (q >> 1));",
                                 "int64_t ch = level_offset(d + 1) + morton(2 * i + (q & 1), 2 * j);"),
    # band: max over axes of the min over the two neighbours along each axis
    "band_min_max_swapped": ("double B = fmax(fmin(dt, db), fmin(dl, dr));",
                             "double B = fmin(fmax(dt, db), fmax(dl, dr));"),
    "band_axes_mixed": ("double B = fmax(fmin(dt, db), fmin(dl, dr));",
                        "double B = fmax(fmin(dt, dl), fmin(db, dr));"),
    "band_neighbours_two_apart": ("int64_t ni[4] = {i - 1, i + 1, i, i};", "int64_t ni[4] = {i - 2, i + 2, i, i};"),
    "halo_sides_swapped": ("int sd = ni[q] < 0 ? 0 : ni[q] >= n ? 1 : nj[q] < 0 ? 2 : 3;",
                           "int sd = ni[q] < 0 ? 0 : ni[q] >= n ? 1 : nj[q] < 0 ? 3 : 2;"),
    # decisions (strict inequalities) and Eq. 2
    "split_not_strict": ("int sp64 = d < D && pv[p] > theta;", "int sp64 = d < D && pv[p] >= theta;"),
    "band_not_strict": ("int ke64 = !sp64 && B > band &&", "int ke64 = !sp64 && B >= band &&"),
    "weight_filter_not_strict": ("int ke64 = !sp64 && B > band && (w_min <= 0.0 || fabs(pw[p]) > w_min);",
                                 "int ke64 = !sp64 && B > band && (w_min <= 0.0 || fabs(pw[p]) >= w_min);"),
    "eager_keeps_split_cells": ("int ke64 = !sp64 && B > band &&", "int ke64 = B > band &&"),
    "eq2_uses_own_variance": ("ac64 = act64[par] && pv[par] > theta;", "ac64 = act64[par] && pv[p] > theta;"),
    "eq2_ignores_ancestors": ("ac64 = act64[par] && pv[par] > theta;", "ac64 = pv[par] > theta;"),
    # grid and numbering (Eq. 1)
    "coordinate_off_centre": ("return (2.0 * (double)i + 1.0) / (double)side_len(d) - 1.0;",
                              "return (2.0 * (double)i) / (double)side_len(d) - 1.0;"),
    "morton_bits_transposed": ("m |= ((i >> k) & 1) << (2 * k);\n        m |= ((j >> k) & 1) << (2 * k + 1);",
                               "m |= ((i >> k) & 1) << (2 * k + 1);\n        m |= ((j >> k) & 1) << (2 * k);"),
    "level_offset_off_by_one": ("return (((int64_t)1 << (2 * (d + 1))) - 4) / 3;",
                                "return (((int64_t)1 << (2 * (d + 1))) - 1) / 3;"),
    # query sides
    "out_side_x_y_transposed": ("if (side == 0) { in[0] = a; in[1] = b; in[2] = x; in[3] = y; }",
                                "if (side == 0) { in[0] = a; in[1] = b; in[2] = y; in[3] = x; }"),
    "in_side_as_out_side": ("else { in[0] = x; in[1] = y; in[2] = a; in[3] = b; }",
                            "else { in[0] = a; in[1] = b; in[2] = x; in[3] = y; }"),
    # CPPN evaluation
    "bias_dropped": ("double z = (double)G->bias[v];", "double z = 0.0;"),
    "edge_weight_dropped": ("z += G->w[e] * val[s];", "z += val[s];"),
    "sigmoid_sign": ("case 1: return 1.0 / (1.0 + exp(-z));", "case 1: return 1.0 / (1.0 + exp(z));"),
    "tanh_as_sin": ("case 2: return tanh(z);", "case 2: return sin(z);"),
    "gauss_not_squared": ("case 3: return exp(-z * z);", "case 3: return exp(-fabs(z));"),
    # the lazy quadtree (Theorem 1's other side)
    "lazy_split_not_strict": ("if (d < c->D && lazy_var(c, d, i, j) > c->theta) {",
                              "if (d < c->D && lazy_var(c, d, i, j) >= c->theta) {"),
    "lazy_band_half_distance": ("s = 1.0 / (double)((int64_t)1 << d);", "s = 0.5 / (double)((int64_t)1 << d);"),
    "lazy_variance_divides_by_3": ("s += (v[q] - m) * (v[q] - m) / 4.0;", "s += (v[q] - m) * (v[q] - m) / 3.0;"),
    # decisions at individual positions (checked against the whole-grid definition)
    "keep_at_band_axes_mixed": ("double B = fmax(fmin(dt, db), fmin(dl, dr)), Be = 0.0,",
                                "double B = fmax(fmin(dt, dl), fmin(db, dr)), Be = 0.0,",
                                ["test_keep_at_matches_whole_grid_decisions"]),
}

# Pins run against each mutant (the quick ones; parametrized pins over all their cases).
PINS = [
    "test_paper_printed_grid_sizes",
    "test_index_is_a_bijection_with_children_rule",
    "test_cppn_identity_single_edge_is_linear",
    "test_cppn_activation_of_bias_matches_c_library",
    "test_cppn_chain_closed_form_and_id_order_independence",
    "test_linear_genome_variance_and_band_closed_forms",
    "test_worked_example_depth4_keeps_exactly_grid3",
    "test_strict_inequalities_at_exact_ties",
    "test_separable_gauss_variance_and_band",
    "test_band_zero_where_the_halo_mirrors_the_border",
    "test_constant_genome_keeps_nothing",
    "test_reflection_symmetry_of_x_only_genome",
    "test_in_side_equals_out_side_of_swapped_genome",
    "test_eq2_active_mask_by_recursion",
    "test_theorem1_single_genome",
]

RUNNER = r"""
import itertools, sys
root, here, lib, src = sys.argv[1:5]
sys.path[:0] = [root, here]
import oracle
oracle._LIB, oracle._SRC, oracle._lib = lib, src, None
import test_oracle_pins as P

def cases(f):
    marks = [m for m in getattr(f, "pytestmark", []) if m.name == "parametrize"]
    axes = []
    for m in marks:
        names = [n.strip() for n in m.args[0].split(",")]
        axes.append([dict(zip(names, v if len(names) > 1 else (v,))) for v in m.args[1]])
    for combo in itertools.product(*axes):
        kw = {}
        for part in combo:
            kw.update(part)
        yield kw

caught = []
for name in sys.argv[5:]:
    f = getattr(P, name)
    for kw in cases(f):
        try:
            f(**kw)
        except Exception:
            caught.append(name)
            break
print("CAUGHT " + " ".join(caught))
"""


def _build(tmp, name, old, new):
    text = open(SRC).read()
    assert text.count(old) == 1, "mutation %s: its target text must occur exactly once" % name
    src = os.path.join(tmp, name + ".c")
    lib = os.path.join(tmp, "lib" + name + ".so")
    with open(src, "w") as f:
        f.write(text.replace(old, new))
    subprocess.run(["gcc", "-O1", "-std=c99", "-fPIC", "-shared", "-o", lib, src, "-lm"], check=True,
                   capture_output=True)
    return src, lib


def _caught(src, lib, pins):
    p = subprocess.run([sys.executable, "-c", RUNNER, ROOT, HERE, lib, src] + pins, capture_output=True,
                       text=True, timeout=600)
    lines = [l for l in p.stdout.splitlines() if l.startswith("CAUGHT")]
    if p.returncode != 0 or not lines:  # a mutant that crashes the process is caught too
        return ["(crash)"]
    return lines[-1].split()[1:]


@pytest.fixture(scope="module")
def tmpdir_mut():
    with tempfile.TemporaryDirectory() as d:
        yield d


def test_unmutated_oracle_passes_every_pin(tmpdir_mut):
    """The harness itself: the oracle source compiled the same way fails no pin."""
    src = os.path.join(tmpdir_mut, "unmutated.c")
    lib = os.path.join(tmpdir_mut, "libunmutated.so")
    with open(src, "w") as f:
        f.write(open(SRC).read())
    subprocess.run(["gcc", "-O1", "-std=c99", "-fPIC", "-shared", "-o", lib, src, "-lm"], check=True,
                   capture_output=True)
    assert _caught(src, lib, PINS) == []


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_fails_a_pin(name, tmpdir_mut):
    old, new, *pins = MUTATIONS[name]
    src, lib = _build(tmpdir_mut, name, old, new)
    assert _caught(src, lib, pins[0] if pins else PINS), "no pin catches the planted mistake %r" % name
