"""GPU parity: libemr's kernels (through the C ABI) against the float64 oracle.

Bars: CPPN outputs within 1e-5 + 1e-4 |oracle| (positions whose fp32 error
bound exceeds that are counted as ill-conditioned); masks and compacted indices
bit-exact wherever the oracle's decision is certain (uncertain ones counted).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W
from parity_util import check_bits, check_lists, check_outputs, full_parity, run_gpu, run_oracle, unpack_planes

pytestmark = pytest.mark.gpu
X1, Y1, X2, Y2, BIAS, HID, OUT = range(7)
IDN, SIG, TNH, GAU, SIN, ABS = range(6)


def test_single_genome_depth4_both_modes():
    for mode in (emr.EMR_EAGER, emr.EMR_GATED):
        _, _, rep = full_parity(W.c1(), mode)
        assert rep["out"]["ill_conditioned"] == 0


def test_population_depth5_all_genomes():
    w = W.c2(D=5)
    _, ora, rep = full_parity(w)
    assert rep["kept"] > 0
    print("c2 d5:", rep)


def test_population_depth5_gated_matches_lazy_tree():
    w = W.c2(D=5, P=200)
    gpu = run_gpu(w, emr.EMR_GATED, unfused=False)
    ora = run_oracle(w)
    lz, _ = oracle.lazy(w.pop, w.sources, w.D, w.theta, w.band)
    lz = lz.reshape(-1, lz.shape[-1])
    check_bits(gpu["mask_f"], lz, ora["unc_gated"], "gated vs lazy")


def test_wide_input_depth6_subset():
    w = W.c3(D=6)
    gpu = run_gpu(w, unfused=True, fused=True)
    n_gen = 12
    ora = run_oracle(w, g1=n_gen)
    n = ora["w"].shape[0]
    check_outputs(gpu["out"][:n], ora["w"], ora["w_err"])
    check_bits(gpu["mask_f"][:n], ora["keep_eager"], ora["unc_eager"])
    check_lists(gpu["lists_f"][:n], gpu["mask_f"][:n], ora["w"], ora["w_err"])
    assert np.array_equal(gpu["mask_u"], gpu["mask_f"])


def test_bench_configuration_depth7_sampled():
    """The benchmark's workload (1000 genomes, 4 slots, depth 7) in its launch
    configuration: full masks and lists for 16 genomes, outputs at sampled
    positions of every genome."""
    w = W.c2(D=7)
    gpu = run_gpu(w, unfused=True, fused=True)
    ora = run_oracle(w, g1=16)
    n = ora["w"].shape[0]
    check_outputs(gpu["out"][:n], ora["w"], ora["w_err"])
    check_bits(gpu["mask_f"][:n], ora["keep_eager"], ora["unc_eager"])
    check_lists(gpu["lists_f"][:n], gpu["mask_f"][:n], ora["w"], ora["w_err"])
    assert np.array_equal(gpu["mask_u"], gpu["mask_f"])
    rng = np.random.default_rng(7)
    g = emr.grid_build(7)
    for gi in rng.choice(w.P, 40, replace=False):
        for s in range(w.S):
            pos = rng.integers(0, g.n_total, 64)
            ins = []
            for p in pos:
                d, i, j = emr.index_to_ij(int(p))
                x, y = (2 * i + 1) / 2 ** (d + 1) - 1, (2 * j + 1) / 2 ** (d + 1) - 1
                a, b = float(w.sources.a[s]), float(w.sources.b[s])
                ins.append([a, b, x, y, 1.0] if w.sources.side[s] == W.SIDE_OUT else [x, y, a, b, 1.0])
            ref, err = oracle.cppn(w.pop, int(gi), np.array(ins))
            check_outputs(gpu["out"][gi * w.S + s, pos], ref, err)
    # the benchmark step's own path (emr_eval_filter_tiles + emr_select): the same lists for every pair,
    # and its keep decisions at sampled positions of every genome against the oracle's
    dsc = gpu["dsc"]
    dsc.idx.zero_(); dsc.w.zero_()
    dsc.run_select()
    torch.cuda.synchronize()
    sel = dsc.lists()
    for (ri, rw), (si, sw) in zip(gpu["lists_f"], sel):
        assert np.array_equal(ri, si) and np.array_equal(rw.view(np.uint32), sw.view(np.uint32))
    n_checked = 0
    for gi in rng.choice(w.P, 60, replace=False):
        for s in range(w.S):
            r = gi * w.S + s
            kept = sel[r][0]
            # every kept position, plus random others
            pos = np.unique(np.concatenate([kept[:32], rng.integers(0, g.n_total, 32)])).astype(np.int64)
            d = np.zeros(len(pos), np.int32); ii = np.zeros(len(pos), np.int64); jj = np.zeros(len(pos), np.int64)
            for k, p in enumerate(pos):
                d[k], ii[k], jj[k] = emr.index_to_ij(int(p))
            ko = oracle.keep_at(w.pop, int(gi), float(w.sources.a[s]), float(w.sources.b[s]),
                                int(w.sources.side[s]), w.D, w.theta, w.band, w.w_min, d, ii, jj)
            ok = ko["unc"] == 0
            got = np.isin(pos, kept)
            assert np.array_equal(got[ok], ko["keep"][ok].astype(bool)), "pair %d" % r
            n_checked += int(ok.sum())
    assert n_checked > 8000


def test_linear_worked_example_keeps_grid3():
    pop = W.population_from_lists([([(k, k, IDN, 0.0) for k in range(5)] + [(5, OUT, IDN, 0.0)],
                                     [(X2, 5, 4.0, True)])])
    w = W.Workload("linear", pop, W.shared_sources([(0.0, -1.0, W.SIDE_OUT)]), 4, 0.03, 0.3)
    for mode in (emr.EMR_EAGER, emr.EMR_GATED):
        gpu = run_gpu(w, mode)
        want = np.zeros((1, oracle.n_total(4)), np.uint8)
        want[0, oracle.index(3, 0, 0):oracle.n_total(3)] = 1
        assert np.array_equal(gpu["mask_f"], want) and np.array_equal(gpu["mask_u"], want)
        assert len(gpu["lists_f"][0][0]) == 256


def test_edge_cases_small_depths_constant_and_hidden_free_genomes():
    const = ([(k, k, IDN, 0.0) for k in range(5)] + [(5, OUT, SIG, 0.3)], [(X1, 5, 1.0, True)])
    nohid = ([(k, k, IDN, 0.0) for k in range(5)] + [(5, OUT, SIN, 0.0)],
             [(X2, 5, 3.0, True), (Y2, 5, -2.0, True), (BIAS, 5, 0.5, True)])
    rnd = W.random_population(6, seed=9)
    pop = W.population_from_lists([const, nohid] + [rnd.genome(k) for k in range(6)])
    src = W.shared_sources([(0.0, -1.0, W.SIDE_OUT), (0.5, 1.0, W.SIDE_IN)])
    for D in (0, 1, 2, 3):
        w = W.Workload("edge", pop, src, D, 0.03, 0.3)
        full_parity(w)


def test_every_kernel_class_including_interpreter():
    """Genomes with 0..30 varying nodes: the constant, dense-4, dense-8, dense-12
    and interpreter (more than 12 varying nodes) classes in one population."""
    big = W.random_population(24, seed=31, h_lo=14, h_hi=30, e_max=120)
    small = W.random_population(40, seed=32, h_lo=0, h_hi=12, e_max=40)
    pop = W.population_from_lists([big.genome(k) for k in range(24)] + [small.genome(k) for k in range(40)])
    h, gs, _, _ = emr.pack_records(emr.pack_population(pop))
    assert gs["n_varying"][:, 0].max() > 12 and (gs["n_varying"][:, 0] == 0).any()
    src = W.shared_sources([(-1.0, -1.0, W.SIDE_OUT), (0.0, 1.0, W.SIDE_IN)])
    for D in (4, 6):
        w = W.Workload("classes", pop, src, D, 0.03, 0.3)
        full_parity(w)


def test_weight_filter_and_gated_mode():
    w = W.c2(D=5, P=100)
    w.w_min = 0.1
    full_parity(w, emr.EMR_EAGER)
    full_parity(w, emr.EMR_GATED)


def test_per_genome_slots_with_counts():
    pop = W.random_population(5, seed=12)
    rng = np.random.default_rng(4)
    S = 6
    a = rng.uniform(-1, 1, (5, S)).astype(np.float32)
    b = rng.uniform(-1, 1, (5, S)).astype(np.float32)
    side = rng.integers(0, 2, (5, S)).astype(np.int32)
    cnt = np.array([6, 0, 3, 1, 6], np.int32)
    w = W.Workload("pergenome", pop, W.Sources(a=a, b=b, side=side, count=cnt), 4, 0.03, 0.3)
    gpu, ora, _ = full_parity(w)
    for g in range(5):
        for s in range(cnt[g], S):
            assert gpu["mask_f"][g * S + s].sum() == 0 and len(gpu["lists_f"][g * S + s][0]) == 0


def test_compaction_capacity_overflow_drops_tail_and_reports_total():
    w = W.c2(D=5, P=50)
    full = run_gpu(w, unfused=False)
    total = sum(len(i) for i, _ in full["lists_f"])
    cap = total // 2
    small = run_gpu(w, unfused=False, cap=cap, lists=False)
    dsc = small["dsc"]
    assert int(dsc.offsets[-1]) == total
    with pytest.raises(emr.EmrError):
        dsc.lists()
    all_idx = np.concatenate([i for i, _ in full["lists_f"]])
    assert np.array_equal(dsc.idx[:cap].cpu().numpy(), all_idx[:cap])


def _morton(i, j):
    m = np.zeros_like(i, dtype=np.int64)
    for k in range(16):
        m |= ((i >> k) & 1) << (2 * k)
        m |= ((j >> k) & 1) << (2 * k + 1)
    return m


ACT_FN = {SIG: lambda z: 1 / (1 + np.exp(-z)), TNH: np.tanh, GAU: lambda z: np.exp(-z * z), SIN: np.sin,
          ABS: np.abs, IDN: lambda z: z}


@pytest.mark.parametrize("act,wx", [(SIG, 40.0), (TNH, 20.0), (GAU, 6.0), (SIN, 40.0), (SIN, 3000.0),
                                    (ABS, 5.0), (IDN, 5.0)])
def test_activation_accuracy_budget(act, wx):
    """Device activations against fp64 at the device's own fp32 pre-activation:
    within 2^-20 + u|v| (sigmoid, tanh, gauss), 2^-19 + u|v| (sin, |z| <= 8192), exact (abs, identity)."""
    pop = W.population_from_lists([([(k, k, IDN, 0.0) for k in range(5)] + [(5, OUT, act, 0.0)],
                                     [(X2, 5, wx, True), (BIAS, 5, 0.3125, True)])])
    D = 9
    w = W.Workload("act", pop, W.shared_sources([(0.0, 0.0, W.SIDE_OUT)]), D, 0.03, 0.3)
    gpu = run_gpu(w, fused=False)
    out = gpu["out"][0]
    g = emr.grid_build(D)
    for d in range(D + 1):
        n = 2 ** (d + 1)
        ii, jj = np.meshgrid(np.arange(n), np.arange(n), indexing="ij")
        ii, jj = ii.ravel(), jj.ravel()
        gidx = g.level_off[d] + _morton(ii, jj)
        x = (2 * ii + 1) / 2 ** (d + 1) - 1
        z = (np.float64(np.float32(wx)) * x + 0.3125).astype(np.float32).astype(np.float64)
        v = ACT_FN[act](z)
        budget = {IDN: 0.0, ABS: 0.0, SIN: 2.0 ** -19}.get(act, 2.0 ** -20) + 2.0 ** -24 * np.abs(v)
        err = np.abs(out[gidx] - v)
        assert np.all(err <= budget), (act, float(err.max()))
    # the deepest level against CUDA's own single-precision functions at the same fp32 inputs
    zt = torch.from_numpy(z.astype(np.float32)).cuda()
    ref = {SIG: torch.sigmoid, TNH: torch.tanh, GAU: lambda t: torch.exp(-t * t), SIN: torch.sin,
           ABS: torch.abs, IDN: lambda t: t}[act](zt).double().cpu().numpy()
    assert np.all(np.abs(out[gidx] - ref) <= budget + 4 * 2.0 ** -24 * (1 + np.abs(ref)))
