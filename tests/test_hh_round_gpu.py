"""The full-recurrent workload's two discovery rounds (Section 2 Phase 2; Table 1
"h->h query"): round 1 from the substrate inputs and outputs, round 2 from every
hidden node round 1 discovered, as per-genome query slots. Round-2 slots are
built from the oracle's round-1 result, so no oracle input comes from the GPU."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W
from parity_util import check_bits, check_lists, unpack_planes

pytestmark = pytest.mark.gpu


def fused(w):
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, w.w_min)
    dsc.run_fused()
    torch.cuda.synchronize()
    return dsc, dsc.lists()


def dij(p, D):
    """Depth and grid indices of a global index (depth-major, Morton within a depth)."""
    d = 0
    while (4 ** (d + 2) - 4) // 3 <= p:
        d += 1
    m = p - (4 ** (d + 1) - 4) // 3
    i = sum(((m >> (2 * k)) & 1) << k for k in range(d + 1))
    j = sum(((m >> (2 * k + 1)) & 1) << k for k in range(d + 1))
    return d, i, j


def hidden_sources(w1, keep, S=256):
    """Per genome: the distinct positions its outgoing round-1 slots keep, ascending, first S,
    each queried outgoing from its grid coordinates (Eq. 1)."""
    P, S1 = w1.P, w1.S
    a = np.zeros((P, S), np.float32); b = np.zeros((P, S), np.float32)
    side = np.zeros((P, S), np.int32); count = np.zeros(P, np.int32)
    for g in range(P):
        rows = [keep[g, s] for s in range(S1) if int(w1.sources.side[s]) == W.SIDE_OUT]
        idx = np.flatnonzero(np.any(rows, axis=0))[:S]
        count[g] = len(idx)
        for k, p in enumerate(idx):
            d, i, j = dij(int(p), w1.D)
            a[g, k] = (2 * i + 1) / 2.0 ** (d + 1) - 1.0
            b[g, k] = (2 * j + 1) / 2.0 ** (d + 1) - 1.0
    return W.Sources(a=a, b=b, side=side, count=count)


def test_round1_depth8_against_oracle():
    w = W.c4_round1()
    dsc, lists = fused(w)
    mask = unpack_planes(dsc.mask.cpu().numpy(), dsc.grid)
    n_gen = 6
    ora = oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, g1=n_gen,
                          fields=("w", "w_err", "keep_eager", "unc_eager"))
    ora = {k: v.reshape(-1, v.shape[-1]) for k, v in ora.items()}
    n = n_gen * w.S
    check_bits(mask[:n], ora["keep_eager"], ora["unc_eager"])
    check_lists(lists[:n], mask[:n], ora["w"], ora["w_err"])


def test_round2_hidden_sources_against_oracle_and_stream():
    w1 = W.c4_round1(P=8)
    r1 = oracle.discover(w1.pop, w1.sources, w1.D, w1.theta, w1.band, fields=("keep_eager",))
    src2 = hidden_sources(w1, r1["keep_eager"], S=256)
    assert src2.count.max() > 0
    w2 = W.Workload("c4_round2", w1.pop, src2, w1.D, w1.theta, w1.band)
    dsc, lists2 = fused(w2)
    mask = unpack_planes(dsc.mask.cpu().numpy(), dsc.grid)
    S = src2.S
    g = int(np.argmax(src2.count > 0))
    ora = oracle.discover(w2.pop, src2, w2.D, w2.theta, w2.band, g0=g, g1=g + 1,
                          fields=("w", "w_err", "keep_eager", "unc_eager"))
    ora = {k: v.reshape(-1, v.shape[-1]) for k, v in ora.items()}
    rows = slice(g * S, (g + 1) * S)
    check_bits(mask[rows], ora["keep_eager"], ora["unc_eager"])
    check_lists(lists2[rows], mask[rows], ora["w"], ora["w_err"])
    for r in range(w2.P * S):
        if r % S >= src2.count[r // S]:
            assert len(lists2[r][0]) == 0
    # the same round streamed in chunks gives the same lists
    pack = emr.pack_population(w2.pop)
    q = emr.make_query(src2)
    gr = emr.grid_build(w2.D, 1 << 14)
    ws = torch.empty(emr.stream_workspace_size(pack, q, gr, 1 << 22), dtype=torch.uint8, device="cuda")
    cap = 1 << 24
    h_idx = torch.zeros(cap, dtype=torch.int32).pin_memory()
    h_w = torch.zeros(cap, dtype=torch.float32).pin_memory()
    counts = np.zeros(w2.P * S, np.int64)
    offsets = np.zeros(w2.P * S + 1, np.int64)
    emr.stream(pack, torch.from_numpy(pack).cuda(), q, gr, w2.theta, w2.band, 0.0, ws, 1 << 22, h_idx, h_w, counts,
               offsets)
    idx = h_idx.numpy()
    for r in range(w2.P * S):
        assert np.array_equal(idx[offsets[r]:offsets[r + 1]], lists2[r][0])
