"""Chunked streaming (emr_stream): identical lists to the whole-grid path at
every chunk size, the depth-13 workload checked against the oracle at sampled
positions, and the capacity / timeout failure paths."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W
from parity_util import check_outputs

pytestmark = pytest.mark.gpu


def run_stream(w, chunk, chunk_cap=1 << 22, cap=1 << 24, timeout_ms=0):
    pack = emr.pack_population(w.pop)
    pack_dev = torch.from_numpy(pack).cuda()
    q = emr.make_query(w.sources)
    g = emr.grid_build(w.D, chunk)
    ws = torch.empty(emr.stream_workspace_size(pack, q, g, chunk_cap), dtype=torch.uint8, device="cuda")
    n_pairs = w.P * q.S
    h_idx = torch.zeros(cap, dtype=torch.int32).pin_memory()
    h_w = torch.zeros(cap, dtype=torch.float32).pin_memory()
    counts = np.zeros(n_pairs, np.int64)
    offsets = np.zeros(n_pairs + 1, np.int64)
    keep = (pack, pack_dev, q, ws, h_idx, h_w)
    try:
        emr.stream(pack, pack_dev, q, g, w.theta, w.band, w.w_min, ws, chunk_cap, h_idx, h_w, counts, offsets,
                   timeout_ms)
    finally:
        torch.cuda.synchronize()
        del keep
    idx, wv = h_idx.numpy(), h_w.numpy()
    return [(idx[offsets[r]:offsets[r + 1]].copy(), wv[offsets[r]:offsets[r + 1]].copy())
            for r in range(n_pairs)], counts


def whole_grid(w):
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, w.w_min)
    dsc.run_fused()
    torch.cuda.synchronize()
    return dsc.lists()


@pytest.mark.parametrize("chunk", [0, 1 << 12, 1 << 14, 1 << 16])
def test_stream_lists_equal_whole_grid_lists(chunk):
    w = W.c2(D=7, P=150)
    ref = whole_grid(w)
    got, counts = run_stream(w, chunk)
    assert [len(i) for i, _ in ref] == list(counts)
    for (ri, rw), (gi, gw) in zip(ref, got):
        assert np.array_equal(ri, gi) and np.array_equal(rw, gw)


def test_stream_mixed_kernel_classes_and_depth10():
    big = W.random_population(6, seed=31, h_lo=14, h_hi=30, e_max=120)
    rest = W.c5(D=10).pop
    pop = W.population_from_lists([big.genome(k) for k in range(6)] + [rest.genome(k) for k in range(10)])
    w = W.Workload("mixed_d10", pop, W.c5().sources, 10, 0.03, 0.3)
    ref = whole_grid(w)
    got, _ = run_stream(w, 1 << 16)
    for (ri, rw), (gi, gw) in zip(ref, got):
        assert np.array_equal(ri, gi) and np.array_equal(rw, gw)


def _sample_check(w, lists, n_kept=400, n_random=3000, seed=0):
    """Oracle decisions at sampled kept positions and random positions of each pair."""
    rng = np.random.default_rng(seed)
    g = emr.grid_build(w.D)
    unc_total = 0
    for r, (idx, wv) in enumerate(lists):
        gen, s = divmod(r, w.S)
        a, b, side = float(w.sources.a[s]), float(w.sources.b[s]), int(w.sources.side[s])
        pick = rng.choice(len(idx), min(n_kept, len(idx)), replace=False) if len(idx) else np.zeros(0, int)
        rand = rng.integers(0, g.n_total, n_random)
        pos = np.concatenate([idx[pick].astype(np.int64), rand])
        dij = np.array([emr.index_to_ij(int(p)) for p in pos]).reshape(-1, 3)
        o = oracle.keep_at(w.pop, gen, a, b, side, w.D, w.theta, w.band, w.w_min, dij[:, 0], dij[:, 1], dij[:, 2])
        gpu_keep = np.isin(pos, idx)
        certain = o["unc"] == 0
        bad = certain & (gpu_keep != o["keep"].astype(bool))
        assert not bad.any(), "pair %d: %d sampled decisions differ" % (r, int(bad.sum()))
        unc_total += int((~certain).sum())
        check_outputs(wv[pick], o["w"][:len(pick)], o["w_err"][:len(pick)], "pair %d weights" % r)
    return unc_total


def test_stream_depth13_workload_sampled_against_oracle():
    w = W.c5()  # 16 genomes x 4 slots, depth 13 (357,913,940 positions per pair), chunks of 2^26
    lists, counts = run_stream(w, w.chunk, chunk_cap=1 << 24, cap=1 << 26)
    assert counts.sum() > 0
    for idx, _ in lists:
        assert np.all(np.diff(idx) > 0)
    _sample_check(w, lists)


def test_stream_capacity_errors_report_true_totals():
    w = W.c2(D=7, P=100)
    full, counts = run_stream(w, 1 << 14)
    total = int(counts.sum())
    with pytest.raises(emr.EmrError) as e:
        run_stream(w, 1 << 14, cap=total // 2)
    assert e.value.status == emr.EMR_ERR_CAPACITY
    with pytest.raises(emr.EmrError) as e:
        run_stream(w, 1 << 14, chunk_cap=8)
    assert e.value.status == emr.EMR_ERR_CAPACITY


def test_stream_host_wait_times_out_and_device_stays_usable():
    w = W.c5(D=12)
    with pytest.raises(emr.EmrError) as e:
        run_stream(w, 1 << 22, timeout_ms=1)
    assert e.value.status == emr.EMR_ERR_TIMEOUT
    torch.cuda.synchronize()
    x = torch.ones(16, device="cuda")
    assert float(x.sum()) == 16.0


def test_eval_chunks_equal_the_whole_grid_evaluation():
    """emr_eval_chunk over every chunk of a depth-7 grid (chunks of 2^14 positions) gives emr_eval's
    outputs and halo bit for bit."""
    w = W.c2(D=7, P=60)
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, materialise=True)
    dsc.prepare()
    emr.eval(dsc.pack, dsc.query, dsc.grid, dsc.out, dsc.out_halo, dsc.ws)
    gc = emr.grid_build(7, 1 << 14)
    n = emr.grid_chunk(gc)[0]
    assert n == 6
    halo = torch.full_like(dsc.out_halo, float("nan"))
    for k in range(n):
        _, lo, hi = emr.grid_chunk(gc, k)
        out = torch.full((dsc.n_pairs, hi - lo), float("nan"), device="cuda")
        emr.eval_chunk(dsc.pack, dsc.query, gc, k, out, halo, dsc.ws)
        torch.cuda.synchronize()
        assert torch.equal(out.view(torch.int32), dsc.out[:, lo:hi].view(torch.int32)), "chunk %d" % k
    assert torch.equal(halo.view(torch.int32), dsc.out_halo.view(torch.int32))


def test_eval_chunk_at_depth_13_against_the_oracle():
    """One depth-13 chunk (2^26 positions) of one deep-grid genome's four slots, materialised, against the
    oracle's CPPN at sampled positions of the chunk."""
    w = W.c5(P=1)
    pack = emr.pack_population(w.pop)
    pack_dev = torch.from_numpy(pack).cuda()
    q = emr.make_query(w.sources)
    g = emr.grid_build(13, 1 << 26)
    ws = torch.zeros(emr.eval_workspace_size(pack, q), dtype=torch.uint8, device="cuda")
    emr.eval_prepare(pack, pack_dev, q, ws)
    n, lo, hi = emr.grid_chunk(g, 3)
    out = torch.empty(q.S, hi - lo, device="cuda")
    emr.eval_chunk(pack, q, g, 3, out, None, ws)
    torch.cuda.synchronize()
    rng = np.random.default_rng(11)
    pos = np.sort(rng.integers(lo, hi, 300))
    for s in range(q.S):
        ins = []
        for p in pos:
            d, i, j = emr.index_to_ij(int(p))
            x, y = (2 * i + 1) / 2 ** (d + 1) - 1, (2 * j + 1) / 2 ** (d + 1) - 1
            ins.append([float(w.sources.a[s]), float(w.sources.b[s]), x, y, 1.0])
        ref, err = oracle.cppn(w.pop, 0, np.array(ins))
        check_outputs(out[s, torch.from_numpy(pos - lo).cuda()].cpu().numpy(), ref, err, "slot %d" % s)
