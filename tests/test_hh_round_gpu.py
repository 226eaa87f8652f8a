"""The full-recurrent workload's two discovery rounds (Section 2 Phase 2; Table 1
"h->h query"): round 1 from the substrate inputs and outputs, round 2 from every
hidden node round 1 discovered, as per-genome query slots. Round-2 slots are
built from the oracle's round-1 result, so no oracle input comes from the GPU."""
import numpy as np
import pytest
import torch

import oracle
from hh_sources import round2_workload
from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W
from parity_util import assert_stored, check_bits, check_lists, oracle_blocks, record, unpack_planes

pytestmark = pytest.mark.gpu


def fused(w):
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, w.w_min)
    dsc.run_fused()
    torch.cuda.synchronize()
    return dsc, dsc.lists()


def test_round1_depth8_all_genomes_against_oracle():
    """All 150 genomes x 12 slots at depth 8 (629 M decisions)."""
    w = W.c4_round1()
    dsc, lists = fused(w)
    planes = dsc.mask.cpu().numpy()
    S = w.S
    for g0, g1, ora in oracle_blocks(w, 10):
        rows = slice(g0 * S, g1 * S)
        mask = unpack_planes(planes[rows], dsc.grid)
        b = check_bits(mask, ora["keep_eager"], ora["unc_eager"])
        l = check_lists(lists[rows], mask, ora["w"], ora["w_err"])
        record("c4_r1_d8", b, l)
    assert_stored("c4_r1_d8")


def test_round2_hidden_sources_against_oracle_and_stream():
    """Round 2 of the first 8 genomes (of 40) whose round 1, by the oracle, found hidden nodes: those
    nodes as per-genome slots (up to 256 per genome), every genome compared; then the same round
    streamed in chunks."""
    w1 = W.c4_round1(P=40)
    r1 = oracle.discover(w1.pop, w1.sources, w1.D, w1.theta, w1.band, fields=("keep_eager",))
    w2 = round2_workload(w1, r1["keep_eager"], 8)
    src2 = w2.sources
    assert w2.P == 8 and src2.count.min() > 0 and src2.count.max() == 256
    dsc, lists2 = fused(w2)
    planes = dsc.mask.cpu().numpy()
    S = src2.S
    for g0, g1, ora in oracle_blocks(w2, 1):
        rows = slice(g0 * S, g1 * S)
        mask = unpack_planes(planes[rows], dsc.grid)
        b = check_bits(mask, ora["keep_eager"], ora["unc_eager"])
        l = check_lists(lists2[rows], mask, ora["w"], ora["w_err"])
        record("c4_r2_d8_g8", b, l)
    assert_stored("c4_r2_d8_g8")
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
