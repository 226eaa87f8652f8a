"""The roofline's work model (bench.algorithmic_work: fp32 lane-ops and MUFU ops per query, the
separable evaluation's minimum) on hand-built genomes, against counts made by hand from its
definition. No GPU: the model reads the host-side packed genomes only."""
import numpy as np
import pytest

import bench
from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W

X1, Y1, X2, Y2, BIAS, HID, OUT = range(7)
IDN, SIG, TNH, GAU, SIN, ABS = range(6)
SHARE = 66 / 4096    # a one-coordinate value is evaluated at 66 coordinates of a 64 x 64 tile
FILTER = 4.5 + 1.0   # variance (six squared differences, their sum, a compare) + band screen, per query
FP32 = {IDN: 0, SIG: 2, TNH: 3, GAU: 2, SIN: 4, ABS: 0}  # the documented activation costs
MUFU = {IDN: 0, SIG: 2, TNH: 2, GAU: 1, SIN: 1, ABS: 0}


def work(nodes, conns, side):
    base = [(k, k, IDN, 0.0) for k in range(5)]
    pop = W.population_from_lists([(base + nodes, [(s, d, w, True) for s, d, w in conns])])
    q = emr.make_query(W.shared_sources([(0.25, -1.0, side)]), device="cpu")
    return bench.algorithmic_work(emr.pack_population(pop), q, emr)[0, 0]


def test_cost_table_is_the_documented_one():
    assert bench.ACT_FP32 == FP32 and bench.ACT_MUFU == MUFU
    assert (bench.VAR_OPS, bench.BAND_OPS) == (4.5, 1.0) and bench.TILE_SIDE == 64


def test_one_coordinate_output():
    """sin(1.5 x2 + 0.2): one node of x alone (first-layer FMA + sin), once per tile column. A dead
    hidden node adds nothing; on the incoming side x2 is the slot's coordinate: constant, no work."""
    nodes = [(5, OUT, SIN, 0.2), (6, HID, TNH, 0.0)]
    conns = [(X2, 5, 1.5), (Y2, 6, 1.0)]
    F, M = work(nodes, conns, W.SIDE_OUT)
    assert F == pytest.approx(SHARE * (1 + FP32[SIN]) + FILTER) and M == pytest.approx(SHARE * MUFU[SIN])
    assert tuple(work(nodes, conns, W.SIDE_IN)) == (0.0, 0.0)


def test_joint_output_of_both_coordinates():
    """tanh(0.7 x2 - 1.2 y2): per query the x + y add and tanh; per tile column and row the two
    first-layer products."""
    F, M = work([(5, OUT, TNH, 0.0)], [(X2, 5, 0.7), (Y2, 5, -1.2)], W.SIDE_OUT)
    assert F == pytest.approx(1 + FP32[TNH] + SHARE * 2 + FILTER) and M == pytest.approx(MUFU[TNH])


def test_joint_node_fed_by_one_coordinate_nodes():
    """sin(gauss(x2) + sigmoid(y2) + 0.5 x2): the gauss node (x) and the sigmoid node (y) are table
    work, and so are the output's two first-layer products and its two one-coordinate sources;
    per query only its add and sin."""
    nodes = [(5, OUT, SIN, 0.0), (6, HID, GAU, 0.0), (7, HID, SIG, 0.0)]
    conns = [(X2, 6, 1.0), (Y2, 7, 1.0), (6, 5, 1.0), (7, 5, 1.0), (X2, 5, 0.5)]
    F, M = work(nodes, conns, W.SIDE_OUT)
    table = (1 + FP32[GAU]) + (1 + FP32[SIG]) + (2 + 2)
    assert F == pytest.approx(1 + FP32[SIN] + SHARE * table + FILTER)
    assert M == pytest.approx(MUFU[SIN] + SHARE * (MUFU[GAU] + MUFU[SIG]))


def test_joint_chain():
    """abs(2 tanh(x2 + y2) + x2): two joint nodes; the output's edge from the joint tanh node is per
    query work, its own x product table work."""
    nodes = [(5, OUT, ABS, 0.0), (6, HID, TNH, 0.0)]
    conns = [(X2, 6, 1.0), (Y2, 6, 1.0), (6, 5, 2.0), (X2, 5, 1.0)]
    F, M = work(nodes, conns, W.SIDE_OUT)
    assert F == pytest.approx((1 + FP32[TNH]) + (1 + 1 + FP32[ABS]) + SHARE * (2 + 2) + FILTER)
    assert M == pytest.approx(MUFU[TNH])


def test_constant_output_counts_nothing():
    nodes = [(5, OUT, SIG, 0.3), (6, HID, SIN, 0.0)]
    conns = [(X1, 6, 2.0), (6, 5, 1.0), (Y1, 5, -1.0)]
    assert tuple(work(nodes, conns, W.SIDE_OUT)) == (0.0, 0.0)


def test_launch_count_matches_the_profiled_launch_list():
    """bench.py's gpu_launches claim for the 1000-genome depth-7 step equals the kernels per step
    in the committed ncu launch list (profiles/launches_c2_pop1000_d7.md: launches over 16 steps)."""
    import os
    import types
    path = os.path.join(os.path.dirname(bench.__file__), "profiles", "launches_c2_pop1000_d7.md")
    rows = [l.split("|") for l in open(path) if l.startswith("| ") and not l.startswith("| kernel")]
    per_step = sum(int(r[2]) for r in rows) / 16
    w = W.c2(D=7, P=1000)
    dsc = types.SimpleNamespace(pack=emr.pack_population(w.pop), grid=emr.grid_build(7),
                                query=emr.make_query(w.sources, device="cpu"))
    assert bench.launches_in_step(emr, dsc) == per_step == 11


def test_reference_arm_prints_the_contract_line():
    """bench.py --impl reference (the oracle on the host cores, a bounded sample of the same
    workload) prints one JSON line with the benchmark's metric and the reference arm's keys."""
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(bench.__file__)
    p = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "1"], capture_output=True, text=True, timeout=600, cwd=root)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [l for l in p.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    j = json.loads(lines[0])
    assert j["impl"] == "reference" and j["metric"] == bench.METRIC and j["unit"] == bench.UNIT
    assert j["value"] > 0 and j["higher_is_better"] is True and j["steps"] == 1 and j["warmup"] == 1
    assert j["cpu_baseline"]["kind"] == "oracle" and j["cpu_baseline"]["value"] == j["value"]
    assert j["cpu_baseline"]["cores"] >= 1 and j["cpu_baseline"]["sample"]
    assert j["e2e"] == {"value": j["value"], "unit": j["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert j["config"]["workload"] == "c2_xor_pop1000_d7"


def test_reference_arm_under_torchrun_prints_from_rank_0_only():
    """Launched the way the driver launches N > 1 (torchrun, one process per rank), the reference
    arm runs on rank 0 alone, which prints the one JSON line; the other rank exits 0 without work."""
    import json
    import os
    import socket
    import subprocess
    import sys
    root = os.path.dirname(bench.__file__)
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    p = subprocess.run([sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
                        "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(root, "bench.py"),
                        "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "1"],
                       capture_output=True, text=True, timeout=600, cwd=root)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [l for l in p.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    j = json.loads(lines[0])
    assert j["impl"] == "reference" and j["n_gpus"] == 2 and j["value"] > 0


def survey(nodes, conns, side):
    base = [(k, k, IDN, 0.0) for k in range(5)]
    pop = W.population_from_lists([(base + nodes, [(s, d, w, True) for s, d, w in conns])])
    q = emr.make_query(W.shared_sources([(0.25, -1.0, side)]), device="cpu")
    return bench.survey_work(emr.pack_population(pop), q, emr)[0, 0]


def test_survey_model_counts_every_node_at_every_position():
    """The survey model (every varying node evaluated per query): tanh(2 x2 - y2 + h), h = sin(x2 + 0.3)
    on the outgoing side: h has 1 varying in-connection + sin (4 FP32, 1 sin); the output 3 (x2, y2,
    h) + tanh (3 FP32, ex2 + rcp); plus 3.25 + 8 of filter. On the incoming side nothing varies."""
    nodes = [(5, OUT, TNH, 0.0), (6, HID, SIN, 0.0)]
    conns = [(X2, 6, 1.0), (BIAS, 6, 0.3), (X2, 5, 2.0), (Y2, 5, -1.0), (6, 5, 1.0)]
    F, ex2, rcp, sn = survey(nodes, conns, W.SIDE_OUT)
    assert F == pytest.approx(1 + 4 + 3 + 3 + 3.25 + 8) and (ex2, rcp, sn) == (1, 1, 1)
    assert tuple(survey(nodes, conns, W.SIDE_IN)) == (11.25, 0, 0, 0)


def test_survey_roofline_takes_the_slower_pipe():
    work = np.array([[[20.0, 1.0, 1.0, 0.0]]])
    probe = {"ex2_Gops": 1e3, "rcp_Gops": 5e2, "sin_Gops": 5e2}
    r = bench.survey_roofline(work, 1000, 152, probe, 1e-6)
    t_fp32 = 20.0 * 1000 / (152 * 128 * 2070e6)
    t_mufu = 1000 * (1 / 1e12 + 1 / 5e11)
    assert r["t_fp32_ms"] == pytest.approx(t_fp32 * 1e3) and r["t_mufu_ms"] == pytest.approx(t_mufu * 1e3)
    assert r["frac"] == pytest.approx(max(t_fp32, t_mufu) / 1e-6)


def test_level_ij_inverts_the_oracle_numbering():
    import oracle
    rng = np.random.default_rng(3)
    d = rng.integers(0, 10, 500)
    i = np.array([rng.integers(0, 2 ** (k + 1)) for k in d])
    j = np.array([rng.integers(0, 2 ** (k + 1)) for k in d])
    p = [oracle.index(int(a), int(b), int(c)) for a, b, c in zip(d, i, j)]
    dd, ii, jj = bench.level_ij(p)
    assert np.array_equal(dd, d) and np.array_equal(ii, i) and np.array_equal(jj, j)


class _FakeDiscovery:
    """Lists held like emr.Discovery's (host tensors), filled from the oracle."""

    def __init__(self, w, keep, ws):
        import torch
        from types import SimpleNamespace
        rows = keep.reshape(-1, keep.shape[-1])
        idx = [np.flatnonzero(r) for r in rows]
        off = np.concatenate([[0], np.cumsum([len(x) for x in idx])])
        self.grid = SimpleNamespace(n_total=keep.shape[-1])
        self.offsets = torch.from_numpy(off.astype(np.int64))
        self.idx = torch.from_numpy(np.concatenate(idx).astype(np.int32))
        self.w = torch.from_numpy(np.concatenate([ws.reshape(len(rows), -1)[r][x] for r, x in enumerate(idx)])
                                  .astype(np.float32))


def test_lists_parity_counts_agreement_and_planted_errors():
    """bench.lists_parity on oracle-made lists: no mismatch; a dropped entry and a wrong weight are
    each counted."""
    import oracle
    w = W.c2(D=4, P=6)
    r = oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, fields=("keep_eager", "unc_eager", "w"))
    ora = {"keep_eager": r["keep_eager"], "unc_eager": r["unc_eager"]}
    fake = _FakeDiscovery(w, r["keep_eager"], r["w"])
    rep = bench.lists_parity(w, fake, ora, w.P)
    assert rep["mismatches"] == 0 and rep["weight_mismatches"] == 0 and rep["kept"] > 0
    fake.w[0] += 0.01
    assert bench.lists_parity(w, fake, ora, w.P)["weight_mismatches"] == 1
    keep = r["keep_eager"].copy()
    k = np.flatnonzero(keep.reshape(-1))[0]
    keep.reshape(-1)[k] = 0
    fake = _FakeDiscovery(w, keep, r["w"])
    assert bench.lists_parity(w, fake, ora, w.P)["mismatches"] == 1
