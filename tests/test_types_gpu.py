"""Connection-type filtering (Section 6 taxonomy and its six substrate
configurations) on the h->h round, where query slots sit on grid positions so
that every type occurs; type codes of the compacted lists; GATED and typed
chunked streaming against the whole-grid path. Round-2 slots come from the
oracle's round-1 result."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W
from parity_util import check_bits, unpack_planes
from hh_sources import hidden_sources

pytestmark = pytest.mark.gpu

ENABLED = {emr.CONN_F: (1, 0, 0, 0), emr.CONN_F | emr.CONN_B: (1, 1, 0, 0), emr.CONN_F | emr.CONN_L: (1, 0, 1, 0),
           emr.CONN_F | emr.CONN_S: (1, 0, 0, 1), emr.CONN_ALL: (1, 1, 1, 1)}


@pytest.fixture(scope="module")
def round2():
    w1 = W.c4_round1(P=8)
    w1 = W.Workload("c4_round1_d6", w1.pop, w1.sources, 6, w1.theta, w1.band)
    r1 = oracle.discover(w1.pop, w1.sources, w1.D, w1.theta, w1.band, fields=("keep_eager",))
    src2 = hidden_sources(w1, r1["keep_eager"], S=64)
    w2 = W.Workload("c4_round2_d6", w1.pop, src2, w1.D, w1.theta, w1.band)
    g = int(np.argmax(src2.count))
    ora = oracle.discover(w2.pop, src2, w2.D, w2.theta, w2.band, g0=g, g1=g + 1,
                          fields=("keep_eager", "unc_eager", "keep_gated", "unc_gated"))
    ora = {k: v.reshape(-1, v.shape[-1]) for k, v in ora.items()}
    types = np.stack([oracle.conn_types(float(src2.a[g, s]), float(src2.b[g, s]), int(src2.side[g, s]),
                                        np.arange(ora["keep_eager"].shape[1])) for s in range(src2.S)])
    return w2, g, ora, types


@pytest.mark.parametrize("types", sorted(ENABLED))
@pytest.mark.parametrize("mode", [emr.EMR_EAGER, emr.EMR_GATED])
def test_typed_mask_matches_oracle(round2, types, mode):
    w2, g, ora, ty = round2
    dsc = emr.Discovery(w2.pop, w2.sources, w2.D, w2.theta, w2.band, 0.0, mode, types=types)
    dsc.run_fused()
    torch.cuda.synchronize()
    S = w2.sources.S
    mask = unpack_planes(dsc.mask.cpu().numpy(), dsc.grid)[g * S:(g + 1) * S]
    keep, unc = ("keep_eager", "unc_eager") if mode == emr.EMR_EAGER else ("keep_gated", "unc_gated")
    want = ora[keep] & np.asarray(ENABLED[types], np.uint8)[ty]
    check_bits(mask, want, ora[unc], "typed mask")
    if types == emr.CONN_ALL:  # every type occurs in this round
        kept_types = np.unique(ty[ora[keep].astype(bool)])
        assert set(kept_types.tolist()) >= {0, 1}
    # the lists hold exactly the typed mask, in order
    lists = dsc.lists()
    for s in range(S):
        assert np.array_equal(lists[g * S + s][0], np.flatnonzero(mask[s]))


def test_list_type_codes_match_oracle(round2):
    w2, g, ora, ty = round2
    dsc = emr.Discovery(w2.pop, w2.sources, w2.D, w2.theta, w2.band)
    dsc.run_fused()
    codes = dsc.conn_types().cpu().numpy()
    off = dsc.offsets.cpu().numpy()
    idx = dsc.idx[:int(off[-1])].cpu().numpy()
    src = w2.sources
    n_checked = 0
    for r in range(dsc.n_pairs):
        gg, s = divmod(r, src.S)
        sl = slice(off[r], off[r + 1])
        if off[r + 1] == off[r]:
            continue
        want = oracle.conn_types(float(src.a[gg, s]), float(src.b[gg, s]), int(src.side[gg, s]), idx[sl])
        assert np.array_equal(codes[sl], want), "pair %d" % r
        n_checked += off[r + 1] - off[r]
    assert n_checked == off[-1] > 0
    # on the checked genome the codes are those of the oracle's positions
    S = src.S
    for s in range(S):
        r = g * S + s
        assert np.array_equal(codes[off[r]:off[r + 1]], ty[s][idx[off[r]:off[r + 1]]])


def stream_lists(w, mode, types, chunk):
    pack = emr.pack_population(w.pop)
    q = emr.make_query(w.sources)
    gr = emr.grid_build(w.D, chunk)
    ws = torch.empty(emr.stream_workspace_size(pack, q, gr, 1 << 20), dtype=torch.uint8, device="cuda")
    n_pairs = w.P * q.S
    cap = 1 << 22
    h_idx = torch.zeros(cap, dtype=torch.int32).pin_memory()
    h_w = torch.zeros(cap, dtype=torch.float32).pin_memory()
    counts = np.zeros(n_pairs, np.int64)
    offsets = np.zeros(n_pairs + 1, np.int64)
    emr.stream(pack, torch.from_numpy(pack).cuda(), q, gr, w.theta, w.band, w.w_min, ws, 1 << 20, h_idx, h_w,
               counts, offsets, mode=mode, types=types)
    torch.cuda.synchronize()
    idx, wv = h_idx.numpy(), h_w.numpy()
    assert offsets[-1] == counts.sum()
    return [(idx[offsets[r]:offsets[r + 1]].copy(), wv[offsets[r]:offsets[r + 1]].copy()) for r in range(n_pairs)]


@pytest.mark.parametrize("mode,types", [(emr.EMR_GATED, emr.CONN_ALL), (emr.EMR_EAGER, emr.CONN_F | emr.CONN_L),
                                        (emr.EMR_GATED, emr.CONN_F | emr.CONN_B)])
@pytest.mark.parametrize("which", ["c2", "round2"])
def test_stream_mode_equals_whole_grid(round2, mode, types, which):
    w = W.c2(D=7, P=40) if which == "c2" else round2[0]
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, mode, types=types)
    dsc.run_fused()
    torch.cuda.synchronize()
    ref = dsc.lists()
    got = stream_lists(w, mode, types, 1 << 12)
    assert sum(len(i) for i, _ in ref) > 0
    for (ri, rw), (gi, gw) in zip(ref, got):
        assert np.array_equal(ri, gi) and np.array_equal(rw.view(np.uint32), gw.view(np.uint32))
