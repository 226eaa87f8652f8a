"""emr_eval_filter_noalloc: the fused evaluation for callers that cannot
allocate device memory (its scratch is a static array inside libemr). Checked
through the C ABI against emr_eval_prepare + emr_eval_filter on two calls in a
row. Both run the same specialisation and tile kernels on the same inputs, so the
check is exact equality (planes and every output word), not a tolerance. The
file is collected last so that a failure here never hides another test."""
import numpy as np
import pytest
import torch

from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _buffers(dsc):
    z = lambda n: torch.zeros(dsc.n_pairs, n, dtype=torch.int32, device="cuda")
    return z(dsc.grid.n_words), z(dsc.grid.n_words), torch.zeros(dsc.n_pairs, dsc.grid.n_total, device="cuda")


def test_noalloc_matches_workspace_entry_point_on_two_calls():
    w = W.c2(D=6, P=300)
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, emr.EMR_EAGER)
    assert emr.eval_workspace_size(dsc.pack, dsc.query) <= (16 << 20)
    split_ref, band_ref, out_ref = _buffers(dsc)
    dsc.prepare()
    emr.eval_filter(dsc.pack, dsc.query, dsc.grid, w.theta, w.band, w.w_min, split_ref, band_ref, out_ref, dsc.ws)
    torch.cuda.synchronize()
    passed = out_ref != 0
    for call in range(2):
        split, band_bits, out = _buffers(dsc)
        emr.eval_filter_noalloc(dsc.pack, dsc.pack_dev, dsc.query, dsc.grid, w.theta, w.band, w.w_min, split,
                                band_bits, out)
        torch.cuda.synchronize()
        assert torch.equal(split, split_ref), "call %d: split plane differs" % call
        assert torch.equal(band_bits, band_ref), "call %d: band plane differs" % call
        assert torch.equal(out.view(torch.int32), out_ref.view(torch.int32)), "call %d: outputs differ" % call
        assert torch.equal(out != 0, passed)


def test_noalloc_rejects_populations_beyond_the_static_area():
    w = W.c3(D=6)
    src = W.shared_sources(W.evenly_spaced(64, -1.0, W.SIDE_OUT))  # 256 x 64 pairs
    pack = emr.pack_population(w.pop)
    q = emr.make_query(src)
    assert emr.eval_workspace_size(pack, q) > (16 << 20)
    g = emr.grid_build(4)
    n_pairs = w.P * q.S
    split = torch.zeros(n_pairs, g.n_words, dtype=torch.int32, device="cuda")
    band_bits = torch.zeros_like(split)
    with pytest.raises(emr.EmrError) as e:
        emr.eval_filter_noalloc(pack, torch.from_numpy(pack).cuda(), q, g, 0.03, 0.3, 0.0, split, band_bits, None)
    assert e.value.status == emr.EMR_ERR_RANGE
