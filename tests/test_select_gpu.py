"""emr_eval_filter_tiles + emr_select (combine, compaction and kept weights over
the tiles whose flag shows band bits) give exactly the lists of emr_eval_filter +
emr_mask_combine(_types) + emr_compact_records, and the flags are exactly the
tiles holding band bits."""
import numpy as np
import pytest
import torch

from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def tile_word_ranges(g):
    D = g.D
    wo = list(g.word_off)
    ranges = [(0, wo[min(D, 4) + 1])]
    for k in range(emr.dense_tiles(D) - 1):
        b = wo[5] + 128 * k
        ranges.append((b, b + 128))
    return ranges


def compare(w, mode=emr.EMR_EAGER, types=emr.CONN_ALL):
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, mode, types=types)
    dsc.run_fused()
    torch.cuda.synchronize()
    ref = dsc.lists()
    ref_counts = dsc.counts.cpu().numpy().copy()
    band_ref = dsc.band_bits.cpu().numpy().copy()
    dsc.idx.zero_(); dsc.w.zero_(); dsc.counts.zero_(); dsc.offsets.zero_()
    dsc.run_select()
    torch.cuda.synchronize()
    got = dsc.lists()
    assert np.array_equal(dsc.counts.cpu().numpy(), ref_counts)
    for (ri, rw), (gi, gw) in zip(ref, got):
        assert np.array_equal(ri, gi) and np.array_equal(rw.view(np.uint32), gw.view(np.uint32))
    band = dsc.band_bits.cpu().numpy()
    assert np.array_equal(band, band_ref)  # same fused evaluation
    # the one-call path gives the same lists
    dsc.idx.zero_(); dsc.w.zero_(); dsc.counts.zero_(); dsc.offsets.zero_()
    dsc.run_discover()
    torch.cuda.synchronize()
    one = dsc.lists()
    for (ri, rw), (gi, gw) in zip(ref, one):
        assert np.array_equal(ri, gi) and np.array_equal(rw.view(np.uint32), gw.view(np.uint32))
    flags = dsc.tile_flags.cpu().numpy()
    want = np.stack([band[:, b:e].any(axis=1) for b, e in tile_word_ranges(dsc.grid)], axis=1)
    assert np.array_equal(flags.astype(bool), want)
    return sum(len(i) for i, _ in ref), flags.mean()


@pytest.mark.parametrize("D", [0, 1, 2, 3, 4, 5, 6])
def test_select_small_depths(D):
    w = W.c2(D=D, P=60)
    compare(w)


def test_select_c2_depth7_modes_and_types():
    w = W.c2(D=7, P=80)
    kept, frac = compare(w)
    assert kept > 0 and frac < 0.5
    compare(w, emr.EMR_GATED)
    compare(w, emr.EMR_EAGER, emr.CONN_F | emr.CONN_L)


def test_select_interpreter_class_and_sharp_genomes():
    big = W.random_population(6, seed=31, h_lo=14, h_hi=30, e_max=120)
    rest = W.c5(D=7).pop
    pop = W.population_from_lists([big.genome(k) for k in range(6)] + [rest.genome(k) for k in range(10)])
    w = W.Workload("mixed_d7", pop, W.c5().sources, 7, 0.03, 0.3)
    compare(w)
    compare(w, emr.EMR_GATED)


def test_select_weight_filter_and_c1():
    w = W.c2(D=6, P=50)
    compare(W.Workload("c2_wmin", w.pop, w.sources, 6, w.theta, w.band, 0.1))
    compare(W.c1())


def test_select_per_genome_slots():
    w = W.c4_round2_random(D=6, P=20, S=32)
    compare(w)
    compare(w, emr.EMR_EAGER, emr.CONN_F | emr.CONN_B)


def test_copy_async_round_trip():
    """emr_copy_async moves bytes host -> device -> host (pinned buffers) on a stream."""
    src = torch.arange(1 << 16, dtype=torch.int32).pin_memory()
    dev = torch.empty_like(src, device="cuda")
    back = torch.zeros_like(src).pin_memory()
    stream = torch.cuda.Stream()
    emr.copy_async(dev, src, src.numel() * 4, stream)
    emr.copy_async(back, dev, src.numel() * 4, stream)
    stream.synchronize()
    assert torch.equal(back, src)
    emr.copy_async(back, dev, 0, stream)  # nothing to copy
