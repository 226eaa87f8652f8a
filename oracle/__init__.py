"""Python driver for the float64 CPU oracle (oracle/emr_oracle.c).

TEST INFRASTRUCTURE ONLY: imported by the tests, by the smoke check and by the
benchmark's CPU-baseline leg, never by the library. It shares no code with the
CUDA path; both sides are fed the same seeded inputs from
paper_2608_27612_gb300.workloads, which holds none of the method's arithmetic.

Parity status of each oracle function (what pins it, in tests/test_oracle_pins.py):
  ora_n_total / ora_index   pinned: the paper's printed N_total values (Eq. 1),
                            the 683 KB grid size, cell counts, disjointness.
  ora_cppn                  pinned: hand-computed genomes, closed forms, the C
                            library's activations at special points.
  ora_discover              pinned: closed-form variance and band of linear and
                            separable genomes, the worked depth-4 example,
                            constant genomes, symmetry, Theorem 1 against the
                            lazy tree, a direct re-evaluation at sampled points,
                            the strict inequalities at exact ties, the band of
                            genomes the halo mirrors at one edge, per-genome
                            slots against the same points as shared slots. Planted
                            mistakes (tests/test_oracle_mutations.py) each fail
                            one of these pins.
  ora_lazy                  pinned: Theorem 1 (lazy subset of eager, lazy equal to
                            the gated mask) and the closed-form worked example.
  ora_keep_at               pinned: equal to ora_discover's outputs, variance, band
                            value, decisions and uncertainty at every position.
  ora_conn_type(s)          pinned: sources off every grid row (all forward or all
                            backward), per-depth counts of forward / backward /
                            lateral targets against closed forms for sources on the
                            grid, exactly one self-loop per on-grid source, and the
                            outgoing / incoming reversal.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "emr_oracle.c")
_LIB = os.path.join(_HERE, "libemr_oracle.so")
_lib = None

ORA_OK, ORA_ERR_ARG, ORA_ERR_CYCLE, ORA_ERR_ALLOC = 0, 1, 2, 3


def build(force: bool = False) -> str:
    """Compile the oracle with the system C compiler (OpenMP when available)."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    base = ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-o", _LIB + ".tmp", _SRC, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(_LIB + ".tmp", _LIB)
    return _LIB


def lib():
    global _lib
    if _lib is None:
        build()
        _lib = C.CDLL(_LIB)
        _lib.ora_n_total.restype = C.c_int64
        _lib.ora_n_halo.restype = C.c_int64
        _lib.ora_index.restype = C.c_int64
        _lib.ora_index.argtypes = [C.c_int, C.c_int64, C.c_int64]
    return _lib


def _p(a):
    return a.ctypes.data_as(C.c_void_p) if a is not None else None


def _pop_args(pop):
    return [_p(pop.node_ptr), _p(pop.node_id), _p(pop.node_kind), _p(pop.node_act), _p(pop.node_bias),
            _p(pop.conn_ptr), _p(pop.conn_src), _p(pop.conn_dst), _p(pop.conn_w), _p(pop.conn_enabled)]


def n_total(D: int) -> int:
    return int(lib().ora_n_total(D))


def n_halo(D: int) -> int:
    return int(lib().ora_n_halo(D))


def index(d: int, i: int, j: int) -> int:
    return int(lib().ora_index(d, i, j))


def threads() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def check_population(pop):
    bad = np.zeros(1, np.int32)
    rc = lib().ora_check_population(C.c_int(pop.P), *_pop_args(pop), _p(bad))
    return int(rc), int(bad[0])


def cppn(pop, g: int, inputs):
    """CPPN output and fp32 error bound of genome g at inputs [n, 5] = (x1,y1,x2,y2,bias)."""
    x = np.ascontiguousarray(inputs, np.float64).reshape(-1, 5)
    out = np.zeros(len(x)); err = np.zeros(len(x))
    rc = lib().ora_cppn(C.c_int(g), *_pop_args(pop), C.c_int64(len(x)), _p(x), _p(out), _p(err))
    if rc != ORA_OK:
        raise ValueError("oracle: genome %d rejected (code %d)" % (g, rc))
    return out, err


def _src_args(sources):
    a = np.ascontiguousarray(sources.a, np.float32)
    b = np.ascontiguousarray(sources.b, np.float32)
    s = np.ascontiguousarray(sources.side, np.int32)
    cnt = None if sources.count is None else np.ascontiguousarray(sources.count, np.int32)
    return a, b, s, cnt


ALL_FIELDS = ("w", "w_err", "w_halo", "halo_err", "var", "var_err", "bnd", "bnd_err",
              "keep_eager", "unc_eager", "keep_gated", "unc_gated", "split")


def discover(pop, sources, D: int, theta: float, band: float, w_min: float = 0.0,
             g0: int = 0, g1: int | None = None, fields=ALL_FIELDS, nthreads: int | None = None):
    """Eager discovery by definition for genomes [g0, g1). Returns {field: array}
    with arrays shaped [G, S, N_total] ([G, S, N_halo] for the halo fields)."""
    g1 = pop.P if g1 is None else g1
    G, S = g1 - g0, sources.S
    NT, NH = n_total(D), n_halo(D)
    out = {}
    for f in ALL_FIELDS:
        if f in fields:
            n = NH if "halo" in f else NT
            dt = np.uint8 if f in ("keep_eager", "unc_eager", "keep_gated", "unc_gated", "split") else np.float64
            out[f] = np.zeros((G, S, n), dt)
    a, b, s, cnt = _src_args(sources)
    rc = lib().ora_discover(
        *_pop_args(pop), C.c_int(g0), C.c_int(g1), C.c_int(S), _p(a), _p(b), _p(s),
        C.c_int(1 if sources.per_genome else 0), _p(cnt), C.c_int(D), C.c_double(theta),
        C.c_double(band), C.c_double(w_min), *[_p(out.get(f)) for f in ALL_FIELDS],
        C.c_int(nthreads or threads()))
    if rc != ORA_OK:
        raise ValueError("oracle: discover failed (code %d)" % rc)
    return out


def lazy(pop, sources, D: int, theta: float, band: float, w_min: float = 0.0,
         g0: int = 0, g1: int | None = None, nthreads: int | None = None):
    """Lazy ES-HyperNEAT quadtree: keep [G, S, N_total] (uint8) and CPPN query counts [G, S]."""
    g1 = pop.P if g1 is None else g1
    G, S = g1 - g0, sources.S
    keep = np.zeros((G, S, n_total(D)), np.uint8)
    evals = np.zeros((G, S), np.int64)
    a, b, s, cnt = _src_args(sources)
    rc = lib().ora_lazy(*_pop_args(pop), C.c_int(g0), C.c_int(g1), C.c_int(S), _p(a), _p(b), _p(s),
                        C.c_int(1 if sources.per_genome else 0), _p(cnt), C.c_int(D),
                        C.c_double(theta), C.c_double(band), C.c_double(w_min), _p(keep), _p(evals),
                        C.c_int(nthreads or threads()))
    if rc != ORA_OK:
        raise ValueError("oracle: lazy failed (code %d)" % rc)
    return keep, evals


TYPE_F, TYPE_B, TYPE_L, TYPE_S = 0, 1, 2, 3


def conn_types(a: float, b: float, side: int, gidx):
    """Connection type codes (0 forward, 1 backward, 2 lateral, 3 self) of the connections between
    slot (a, b) on `side` and the grid positions gidx (Section 6 taxonomy)."""
    g = np.ascontiguousarray(gidx, np.int64)
    out = np.zeros(len(g), np.uint8)
    rc = lib().ora_conn_types(C.c_double(a), C.c_double(b), C.c_int(side), C.c_int64(len(g)), _p(g), _p(out))
    if rc != ORA_OK:
        raise ValueError("oracle: conn_types failed (code %d)" % rc)
    return out


def keep_at(pop, g: int, a: float, b: float, side: int, D: int, theta: float, band: float, w_min: float,
            d, i, j, nthreads: int | None = None):
    """Eager keep decision (fp64) and its uncertainty at listed positions (d, i, j) of genome g's
    query from slot (a, b, side), by direct CPPN queries. Returns dict of arrays."""
    d = np.ascontiguousarray(d, np.int32)
    i = np.ascontiguousarray(i, np.int64)
    j = np.ascontiguousarray(j, np.int64)
    n = len(d)
    out = {k: np.zeros(n) for k in ("w", "w_err", "var", "bnd")}
    keep = np.zeros(n, np.uint8)
    unc = np.zeros(n, np.uint8)
    rc = lib().ora_keep_at(C.c_int(g), *_pop_args(pop), C.c_float(a), C.c_float(b), C.c_int(side), C.c_int(D),
                           C.c_double(theta), C.c_double(band), C.c_double(w_min), C.c_int64(n), _p(d), _p(i), _p(j),
                           _p(out["w"]), _p(out["w_err"]), _p(out["var"]), _p(out["bnd"]), _p(keep), _p(unc),
                           C.c_int(nthreads or threads()))
    if rc != ORA_OK:
        raise ValueError("oracle: keep_at failed (code %d)" % rc)
    out["keep"], out["unc"] = keep, unc
    return out
