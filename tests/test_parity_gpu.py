"""GPU parity: libemr's kernels (through the C ABI) against the float64 oracle.

Bars: CPPN outputs within max(1e-5 + 1e-4 |oracle|, the oracle's fp32 error bound)
(outputs whose bound exceeds the plain tolerance are counted as ill-conditioned);
masks and compacted indices bit-exact wherever the oracle's decision is certain
(uncertain ones counted). The single-genome, 1000-genome (depths 5 and 7) and
wide-input workloads are compared over every genome; their counts must stay within
the oracle's stored counts.
"""
import numpy as np
import pytest
import torch

import oracle
import special_genomes as SG
from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W
from parity_util import (assert_stored, check_bits, check_lists, check_outputs, full_parity, mask_from_lists,
                         oracle_blocks, record, run_gpu, run_oracle, unpack_planes)

pytestmark = pytest.mark.gpu
X1, Y1, X2, Y2, BIAS, HID, OUT = range(7)
IDN, SIG, TNH, GAU, SIN, ABS = range(6)


def test_single_genome_depth4_both_modes():
    for mode, name in ((emr.EMR_EAGER, "c1_d4_eager"), (emr.EMR_GATED, "c1_d4_gated")):
        _, _, rep = full_parity(W.c1(), mode, name=name)
        assert rep["out"]["ill_conditioned"] == 0
        assert_stored(name)


def test_population_depth5_all_genomes():
    w = W.c2(D=5)
    _, ora, rep = full_parity(w, name="c2_d5")
    assert rep["kept"] > 0
    assert_stored("c2_d5")


def test_population_depth5_gated_matches_lazy_tree():
    w = W.c2(D=5, P=200)
    gpu = run_gpu(w, emr.EMR_GATED, unfused=False)
    ora = run_oracle(w)
    lz, _ = oracle.lazy(w.pop, w.sources, w.D, w.theta, w.band)
    lz = lz.reshape(-1, lz.shape[-1])
    check_bits(gpu["mask_f"], lz, ora["unc_gated"], "gated vs lazy")


def test_wide_input_depth6_all_genomes():
    """All 256 genomes x 33 slots: materialised outputs, fused and unfused masks, lists."""
    w = W.c3(D=6)
    gpu = run_gpu(w, unfused=True, fused=True)
    assert np.array_equal(gpu["mask_u"], gpu["mask_f"])
    S = w.S
    for g0, g1, ora in oracle_blocks(w, 32):
        rows = slice(g0 * S, g1 * S)
        o = check_outputs(gpu["out"][rows], ora["w"], ora["w_err"])
        b = check_bits(gpu["mask_f"][rows], ora["keep_eager"], ora["unc_eager"])
        l = check_lists(gpu["lists_f"][rows], gpu["mask_f"][rows], ora["w"], ora["w_err"])
        record("c3_d6", o, b, l)
    assert_stored("c3_d6")


def test_bench_configuration_depth7_all_genomes():
    """The benchmark's workload (1000 genomes, 4 slots, depth 7) over every genome: the
    materialised outputs (emr_eval), and the keep decisions and lists of the benchmark
    step's own launch path (emr_eval_prepare + emr_eval_filter_tiles + emr_select)."""
    w = W.c2(D=7)
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, emr.EMR_EAGER, materialise=True)
    g = dsc.grid
    dsc.run_unfused()
    torch.cuda.synchronize()
    out = dsc.out.cpu().numpy()
    mask_u = unpack_planes(dsc.mask.cpu().numpy(), g)
    dsc.idx.zero_(); dsc.w.zero_(); dsc.counts.zero_(); dsc.offsets.zero_()
    dsc.run_select()
    torch.cuda.synchronize()
    sel = dsc.lists()
    S = w.S
    for g0, g1, ora in oracle_blocks(w, 100):
        rows = slice(g0 * S, g1 * S)
        o = check_outputs(out[rows], ora["w"], ora["w_err"])
        mask = mask_from_lists(sel[rows], g.n_total)
        assert np.array_equal(mask, mask_u[rows]), "genomes %d..%d: step lists differ from the unfused mask" % (g0, g1)
        b = check_bits(mask, ora["keep_eager"], ora["unc_eager"])
        l = check_lists(sel[rows], mask, ora["w"], ora["w_err"])
        record("c2_d7", o, b, l)
    tot = assert_stored("c2_d7")
    assert tot["entries"] == int(dsc.offsets[-1]) > 0


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
    for D in (0, 1, 2, 3):
        w = SG.edge_cases(D)
        full_parity(w, name=w.name)
        assert_stored(w.name)


def test_every_kernel_class_including_interpreter():
    """Genomes with 0..30 varying nodes: the constant, dense-4, dense-8, dense-12
    and interpreter (more than 12 varying nodes) classes in one population."""
    for D in (4, 6):
        w = SG.kernel_classes(D)
        if D == 4:
            h, gs, _, _ = emr.pack_records(emr.pack_population(w.pop))
            assert gs["n_varying"][:, 0].max() > 12 and (gs["n_varying"][:, 0] == 0).any()
        full_parity(w, name=w.name)
        assert_stored(w.name)


def test_weight_filter_and_gated_mode():
    w = SG.weight_filter()
    for mode, name in ((emr.EMR_EAGER, w.name + "_eager"), (emr.EMR_GATED, w.name + "_gated")):
        full_parity(w, mode, name=name)
        assert_stored(name)


def test_per_genome_slots_with_counts():
    w = SG.per_genome_slots()
    cnt, S = w.sources.count, w.S
    gpu, ora, _ = full_parity(w, name=w.name)
    assert_stored(w.name)
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
