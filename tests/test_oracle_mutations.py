"""Strength of the oracle's pins: a plausible mistake planted in a copy of the
oracle (a dropped term, a wrong divisor, sign, index or operand, a non-strict
comparison) must make at least one pin fail.

Each mutant is a copy of the oracle package in a temporary directory with one
passage of one file changed (the C source is compiled there); a child process
puts that copy ahead of the real package, so a mutant that crashed could not
take the test run with it, and runs the pins. The installed oracle is never
touched. No GPU is involved.
"""
import os
import shutil
import subprocess
import sys
import tempfile

import pytest

import oracle

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
PKG = os.path.join(ROOT, "oracle")

C_PINS = [  # the quick pins of test_oracle_pins.py (parametrized pins over all their cases)
    "test_oracle_pins." + n for n in (
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
        "test_per_genome_slots_address_like_shared_slots",
        "test_eq2_active_mask_by_recursion",
        "test_theorem1_single_genome",
    )]
KEEP_AT_PINS = ["test_oracle_pins.test_keep_at_matches_whole_grid_decisions"]
TYPE_PINS = ["test_types_oracle.*"]
VARIANT_PINS = ["test_variants_oracle.*"]
ASSEMBLY_PINS = ["test_assembly_oracle.*"]

# name: (file of the oracle package, its text, the replacement, the pins to run).
# Every mutant stays memory-safe (indices stay within the buffers the unmutated
# oracle sizes).
C = "emr_oracle.c"
MUTATIONS = {
    # Section 3.2: population variance of the four children
    "variance_divides_by_3": (C, "v += dq * dq / 4.0;", "v += dq * dq / 3.0;", C_PINS),
    "variance_drops_a_child": (C, "for (int q = 0; q < 4; q++) {\n                            double dq = c[q] - m;",
                               "for (int q = 0; q < 3; q++) {\n                            double dq = c[q] - m;", C_PINS),
    "variance_wrong_mean": (C, "\n                            m += c[q] / 4.0;", "\n                            m += c[q] / 2.0;",
                            C_PINS),
    "children_drop_row_offset": (C, "int64_t ch = level_offset(d + 1) + morton(2 * i + (q & 1), 2 * j + (q >> 1));",
                                 "int64_t ch = level_offset(d + 1) + morton(2 * i + (q & 1), 2 * j);", C_PINS),
    # band: max over axes of the min over the two neighbours along each axis
    "band_min_max_swapped": (C, "double B = fmax(fmin(dt, db), fmin(dl, dr));",
                             "double B = fmin(fmax(dt, db), fmax(dl, dr));", C_PINS),
    "band_axes_mixed": (C, "double B = fmax(fmin(dt, db), fmin(dl, dr));",
                        "double B = fmax(fmin(dt, dl), fmin(db, dr));", C_PINS),
    "band_neighbours_two_apart": (C, "int64_t ni[4] = {i - 1, i + 1, i, i};", "int64_t ni[4] = {i - 2, i + 2, i, i};",
                                  C_PINS),
    "halo_sides_swapped": (C, "int sd = ni[q] < 0 ? 0 : ni[q] >= n ? 1 : nj[q] < 0 ? 2 : 3;",
                           "int sd = ni[q] < 0 ? 0 : ni[q] >= n ? 1 : nj[q] < 0 ? 3 : 2;", C_PINS),
    # decisions (strict inequalities) and Eq. 2
    "split_not_strict": (C, "int sp64 = d < D && pv[p] > theta;", "int sp64 = d < D && pv[p] >= theta;", C_PINS),
    "band_not_strict": (C, "int ke64 = !sp64 && B > band &&", "int ke64 = !sp64 && B >= band &&", C_PINS),
    "weight_filter_not_strict": (C, "int ke64 = !sp64 && B > band && (w_min <= 0.0 || fabs(pw[p]) > w_min);",
                                 "int ke64 = !sp64 && B > band && (w_min <= 0.0 || fabs(pw[p]) >= w_min);", C_PINS),
    "eager_keeps_split_cells": (C, "int ke64 = !sp64 && B > band &&", "int ke64 = B > band &&", C_PINS),
    "eq2_uses_own_variance": (C, "ac64 = act64[par] && pv[par] > theta;", "ac64 = act64[par] && pv[p] > theta;",
                              C_PINS),
    "eq2_ignores_ancestors": (C, "ac64 = act64[par] && pv[par] > theta;", "ac64 = pv[par] > theta;", C_PINS),
    # grid and numbering (Eq. 1)
    "coordinate_off_centre": (C, "return (2.0 * (double)i + 1.0) / (double)side_len(d) - 1.0;",
                              "return (2.0 * (double)i) / (double)side_len(d) - 1.0;", C_PINS),
    "morton_bits_transposed": (C, "m |= ((i >> k) & 1) << (2 * k);\n        m |= ((j >> k) & 1) << (2 * k + 1);",
                               "m |= ((i >> k) & 1) << (2 * k + 1);\n        m |= ((j >> k) & 1) << (2 * k);", C_PINS),
    "level_offset_off_by_one": (C, "return (((int64_t)1 << (2 * (d + 1))) - 4) / 3;",
                                "return (((int64_t)1 << (2 * (d + 1))) - 1) / 3;", C_PINS),
    # query sides
    "out_side_x_y_transposed": (C, "if (side == 0) { in[0] = a; in[1] = b; in[2] = x; in[3] = y; }",
                                "if (side == 0) { in[0] = a; in[1] = b; in[2] = y; in[3] = x; }", C_PINS),
    "in_side_as_out_side": (C, "else { in[0] = x; in[1] = y; in[2] = a; in[3] = b; }",
                            "else { in[0] = a; in[1] = b; in[2] = x; in[3] = y; }", C_PINS),
    # per-genome query slots (the hidden-to-hidden round)
    "per_genome_slot_relative_to_range": (C, "            int64_t si = per_genome ? (int64_t)g * S + s : s;\n            double a",
                                          "            int64_t si = per_genome ? (int64_t)gl * S + s : s;\n            double a",
                                          C_PINS),
    "unused_slots_evaluated": (C, "            if (per_genome && src_count && s >= src_count[g]) continue;\n            int64_t si",
                               "            int64_t si", C_PINS),
    "lazy_unused_slots_evaluated": (C, "        if (per_genome && src_count && s >= src_count[g]) continue;\n        int64_t si",
                                    "        int64_t si", C_PINS),
    # CPPN evaluation
    "bias_dropped": (C, "double z = (double)G->bias[v];", "double z = 0.0;", C_PINS),
    "edge_weight_dropped": (C, "z += G->w[e] * val[s];", "z += val[s];", C_PINS),
    "sigmoid_sign": (C, "case 1: return 1.0 / (1.0 + exp(-z));", "case 1: return 1.0 / (1.0 + exp(z));", C_PINS),
    "tanh_as_sin": (C, "case 2: return tanh(z);", "case 2: return sin(z);", C_PINS),
    "gauss_not_squared": (C, "case 3: return exp(-z * z);", "case 3: return exp(-fabs(z));", C_PINS),
    # the lazy quadtree (Theorem 1's other side)
    "lazy_split_not_strict": (C, "if (d < c->D && lazy_var(c, d, i, j) > c->theta) {",
                              "if (d < c->D && lazy_var(c, d, i, j) >= c->theta) {", C_PINS),
    "lazy_band_half_distance": (C, "s = 1.0 / (double)((int64_t)1 << d);", "s = 0.5 / (double)((int64_t)1 << d);",
                                C_PINS),
    "lazy_variance_divides_by_3": (C, "s += (v[q] - m) * (v[q] - m) / 4.0;", "s += (v[q] - m) * (v[q] - m) / 3.0;",
                                   C_PINS),
    # decisions at individual positions (checked against the whole-grid definition)
    "keep_at_band_axes_mixed": (C, "double B = fmax(fmin(dt, db), fmin(dl, dr)), Be = 0.0,",
                                "double B = fmax(fmin(dt, dl), fmin(db, dr)), Be = 0.0,", KEEP_AT_PINS),
    # connection types (Section 6's taxonomy)
    "types_ignore_the_query_side": (C, "    double xs = side == 0 ? a : x, ys = side == 0 ? b : y;   /* source */\n"
                                       "    double xt = side == 0 ? x : a, yt = side == 0 ? y : b;   /* target */",
                                    "    double xs = a, ys = b;\n    double xt = x, yt = y;", TYPE_PINS),
    "lateral_typed_forward_in_types": (C, "if (ys < yt) return 0;", "if (ys <= yt) return 0;", TYPE_PINS),
    "self_loop_typed_lateral": (C, "    if (xs == xt && ys == yt) return 3;\n", "", TYPE_PINS),
    # method variants (HyperNEAT weight scaling, subtree-leaf variance)
    "scaling_without_clamp": ("variants.py", "(np.minimum(a, 1.0) - thr) / (1.0 - thr)", "(a - thr) / (1.0 - thr)",
                              VARIANT_PINS),
    "scaling_drops_sign": ("variants.py", "out = np.sign(w) * w_max *", "out = w_max *", VARIANT_PINS),
    "subtree_variance_ddof_1": ("variants.py", "v = (dev ** 2).mean(axis=1)", "v = (dev ** 2).sum(axis=1) / (k - 1)",
                                VARIANT_PINS),
    "subtree_split_not_strict": ("variants.py", "split = (V > theta)", "split = (V >= theta)", VARIANT_PINS),
    # network assembly and the substrate ANN
    "forward_weights_transposed": ("assembly.py", "W[d_, s_] += w", "W[s_, d_] += w", ASSEMBLY_PINS),
    "forward_sigmoid_sign": ("assembly.py", "nv = 1.0 / (1.0 + np.exp(-z))", "nv = 1.0 / (1.0 + np.exp(z))",
                             ASSEMBLY_PINS),
    "forward_inputs_not_held": ("assembly.py", "        nv[:n_in] = pat.T\n", "", ASSEMBLY_PINS),
    "prune_ignores_outputs": ("assembly.py", "kept = sorted(p for p in hidden[g] if p in fwd and p in bwd)",
                              "kept = sorted(p for p in hidden[g] if p in fwd)", ASSEMBLY_PINS),
    "lateral_typed_forward": ("assembly.py", "return F if ys < yt else B if ys > yt else L",
                              "return F if ys <= yt else B", ASSEMBLY_PINS),
    "one_hidden_round_too_many": ("assembly.py", "for _ in range(rounds):", "for _ in range(rounds + 1):",
                                  ASSEMBLY_PINS),
}

RUNNER = r"""
import importlib, itertools, os, sys
pkg, here, root = sys.argv[1:4]
sys.path[:0] = [pkg, here, root]  # the mutated oracle package ahead of the real one
import oracle
assert os.path.dirname(oracle.__file__) == os.path.join(pkg, "oracle"), oracle.__file__

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

pins = []
for spec in sys.argv[4:]:
    mod, name = spec.split(".")
    m = importlib.import_module(mod)
    names = sorted(n for n in dir(m) if n.startswith("test_")) if name == "*" else [name]
    pins += [(mod + "." + n, getattr(m, n)) for n in names]
caught = []
for name, f in pins:
    for kw in cases(f):
        try:
            f(**kw)
        except Exception:
            caught.append(name)
            break
print("CAUGHT " + " ".join(caught))
"""


def _package(tmp, name, fname=None, old=None, new=None):
    """A copy of the oracle package under tmp/name/oracle, with `old` replaced by `new` in
    `fname` (the C library rebuilt there when its source changes)."""
    oracle.build()  # the copy starts from a built library
    dst = os.path.join(tmp, name, "oracle")
    shutil.copytree(PKG, dst, ignore=shutil.ignore_patterns("__pycache__"))
    if fname is not None:
        path = os.path.join(dst, fname)
        text = open(path).read()
        assert text.count(old) == 1, "mutation %s: its target text must occur exactly once" % name
        with open(path, "w") as f:
            f.write(text.replace(old, new))
        if fname.endswith(".c"):
            lib = os.path.join(dst, "libemr_oracle.so")
            subprocess.run(["gcc", "-O1", "-std=c99", "-fPIC", "-shared", "-o", lib, path, "-lm"], check=True,
                           capture_output=True)
    return os.path.join(tmp, name)


def _caught(pkg, pins):
    p = subprocess.run([sys.executable, "-c", RUNNER, pkg, HERE, ROOT] + pins, capture_output=True, text=True,
                       timeout=600)
    lines = [l for l in p.stdout.splitlines() if l.startswith("CAUGHT")]
    if p.returncode != 0 or not lines:  # a mutant that crashes the process is caught too
        return ["(crash)"]
    return lines[-1].split()[1:]


@pytest.fixture(scope="module")
def tmpdir_mut():
    with tempfile.TemporaryDirectory() as d:
        yield d


def test_unmutated_oracle_passes_every_pin(tmpdir_mut):
    """The harness itself: an unchanged copy of the package fails no pin."""
    pkg = _package(tmpdir_mut, "unmutated")
    assert _caught(pkg, C_PINS + KEEP_AT_PINS + TYPE_PINS + VARIANT_PINS + ASSEMBLY_PINS) == []


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_fails_a_pin(name, tmpdir_mut):
    fname, old, new, pins = MUTATIONS[name]
    pkg = _package(tmpdir_mut, name, fname, old, new)
    assert _caught(pkg, pins), "no pin catches the planted mistake %r" % name
