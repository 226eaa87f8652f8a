"""Host-side checks of libemr's C ABI (no GPU): the library loads and exports
every declared entry point; the grid descriptor, index inverse and genome packer
behave as documented. The packer's results are compared with the oracle's
independent genome handling where both apply."""
import ctypes as C
import os
import re

import numpy as np
import pytest

import oracle
from paper_2608_27612_gb300 import emr
from paper_2608_27612_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
X1, Y1, X2, Y2, BIAS, HID, OUT = range(7)
IDN, SIG, TNH, GAU, SIN, ABS = range(6)


def declared_symbols():
    names = set()
    inc = os.path.join(ROOT, "include")
    for f in os.listdir(inc):
        if f.endswith(".h"):
            txt = open(os.path.join(inc, f)).read()
            names |= set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(emr_\w+)\s*\(", txt, re.M))
    return names


def test_library_exports_every_declared_symbol():
    L = emr.lib()
    names = declared_symbols()
    assert {"emr_grid_build", "emr_pack_population", "emr_eval", "emr_variance_filter", "emr_eval_filter",
            "emr_compact"} <= names
    for n in sorted(names):
        assert hasattr(L, n), n
    assert emr.strerror(emr.EMR_ERR_CYCLE).startswith("genome has a cycle")


@pytest.mark.parametrize("D", [0, 1, 4, 7, 13, 14])
def test_grid_descriptor_matches_eq1_counts(D):
    g = emr.grid_build(D)
    assert g.n_total == oracle.n_total(D) and g.n_halo == oracle.n_halo(D)
    for d in range(D + 1):
        assert g.level_off[d] == oracle.index(d, 0, 0)
        assert g.halo_off[d] == 8 * (2 ** d - 1)
        assert g.word_off[d + 1] - g.word_off[d] == -(-(4 ** (d + 1)) // 32)
    assert g.level_off[D + 1] == g.n_total and g.word_off[D + 1] == g.n_words
    for d in range(D + 1, 16):  # entries past D + 1 repeat the totals
        assert (g.level_off[d], g.halo_off[d], g.word_off[d]) == (g.n_total, g.n_halo, g.n_words)


def test_grid_descriptor_errors():
    with pytest.raises(emr.EmrError) as e:
        emr.grid_build(15)
    assert e.value.status == emr.EMR_ERR_RANGE
    with pytest.raises(emr.EmrError):
        emr.grid_build(-1)
    for bad in (1000, 4095, 6000):
        with pytest.raises(emr.EmrError) as e:
            emr.grid_build(5, bad)
        assert e.value.status == emr.EMR_ERR_ARG
    assert emr.grid_build(13, 1 << 26).chunk == 1 << 26


def test_index_to_ij_inverts_the_numbering():
    rng = np.random.default_rng(0)
    for _ in range(2000):
        d = int(rng.integers(0, 15))
        n = 2 ** (d + 1)
        i, j = int(rng.integers(0, n)), int(rng.integers(0, n))
        assert emr.index_to_ij(oracle.index(d, i, j)) == (d, i, j)
    with pytest.raises(emr.EmrError):
        emr.index_to_ij(-1)
    with pytest.raises(emr.EmrError):
        emr.index_to_ij(oracle.n_total(14))


def _genome(nodes, conns):
    return W.population_from_lists([([(k, k, IDN, 0.0) for k in range(5)] + nodes, conns)])


def _pack_records(blob):
    """Decode the blob (layout of csrc/emr_internal.h) for white-box checks."""
    h = np.frombuffer(blob[:72].tobytes(), dtype=np.dtype([
        ("magic", "<u4"), ("version", "<u4"), ("P", "<i4"), ("max_nodes", "<i4"), ("max_varying", "<i4", 2),
        ("max_vedges", "<i4", 2), ("max_edges", "<i4"), ("reserved", "<i4"), ("off_genomes", "<u8"),
        ("off_nodes", "<u8"), ("off_edges", "<u8"), ("total", "<u8")]))[0]
    gdt = np.dtype([("node_beg", "<u4"), ("edge_beg", "<u4"), ("n_nodes", "<u2"), ("n_edges", "<u2"),
                    ("n_varying", "<u2", 2), ("n_vedges", "<u2", 2), ("cost", "<u4", 2), ("n_joint", "<u2", 2)])
    ndt = np.dtype([("act", "u1"), ("vary", "u1"), ("axes", "u1"), ("r", "u1"), ("edge_beg", "<u2"), ("edge_cnt", "<u2"),
                    ("bias", "<f4"), ("w_in", "<f4", 5)])
    P = int(h["P"])
    gs = np.frombuffer(blob.tobytes(), gdt, P, int(h["off_genomes"]))
    nn = int(gs["n_nodes"].astype(np.int64).sum())
    nodes = np.frombuffer(blob.tobytes(), ndt, nn, int(h["off_nodes"]))
    return h, gs, nodes


def test_pack_topological_order_dead_nodes_and_variation_flags():
    # hidden 12 (x2) -> 10 (sin) -> out; hidden 7 depends only on the source (x1) -> out;
    # hidden 9 is dead (feeds nothing that reaches the output).
    nodes = [(5, OUT, TNH, 0.0), (10, HID, SIN, 0.5), (12, HID, GAU, 0.0), (7, HID, SIG, 0.0), (9, HID, ABS, 0.0)]
    conns = [(12, 10, 1.0, True), (X2, 12, 2.0, True), (10, 5, 3.0, True), (X1, 7, 1.5, True), (7, 5, -1.0, True),
             (Y2, 9, 1.0, True), (12, 9, 1.0, True), (Y1, 5, 0.25, False)]
    pop = _genome(nodes, conns)
    blob = emr.pack_population(pop)
    h, gs, nd = _pack_records(blob)
    assert h["magic"] == 0x504D5245 and h["P"] == 1
    g = gs[0]
    assert g["n_nodes"] == 4  # 9 dropped
    # Kahn with ties by id: 7 and 12 are ready first (7 < 12), then 10, then the output
    assert list(nd["act"]) == [SIG, GAU, SIN, TNH]
    assert nd["w_in"][0][X1] == np.float32(1.5) and nd["w_in"][1][X2] == np.float32(2.0)
    # OUT side: x2/y2 vary -> 12, 10, out vary, 7 is constant; IN side: x1/y1 vary -> 7 and out vary
    assert [int(v) & 1 for v in nd["vary"]] == [0, 1, 1, 1]
    assert [(int(v) >> 1) & 1 for v in nd["vary"]] == [1, 0, 0, 1]
    assert tuple(g["n_varying"]) == (3, 2)
    assert emr.pack_info(blob) == (1, 3, 2)
    # grid coordinates per side (bits 2 s: x, 2 s + 1: y): OUT side 12, 10, out follow x2 only;
    # IN side 7 and the output follow x1 only; no node depends on both coordinates
    assert [int(a) for a in nd["axes"]] == [4, 1, 1, 5]
    assert tuple(g["n_joint"]) == (0, 0)


def test_pack_merges_parallel_connections_and_drops_zero_weights():
    # 6 -> out twice (0.5 + 0.25 = 0.75); 7 -> out cancels (1 - 1 = 0), so 7 is dropped with its
    # edge; x2 -> 8 twice with weights summing to 0 leaves 8 with the y2 input only
    nodes = [(5, OUT, IDN, 0.0), (6, HID, SIG, 0.0), (7, HID, SIN, 0.0), (8, HID, TNH, 0.0)]
    conns = [(X2, 6, 1.0, True), (Y2, 6, 1.0, True), (6, 5, 0.5, True), (7, 5, 1.0, True), (X2, 7, 1.0, True),
             (6, 5, 0.25, True), (7, 5, -1.0, True), (X2, 8, 2.0, True), (Y2, 8, 1.0, True), (X2, 8, -2.0, True),
             (8, 5, 1.0, True)]
    blob = emr.pack_population(_genome(nodes, conns))
    h, gs, nd = _pack_records(blob)
    g = gs[0]
    assert g["n_nodes"] == 3 and g["n_edges"] == 2  # 6, 8, out; edges 6 -> out, 8 -> out
    _, _, _, ed = emr.pack_records(blob)
    ed = ed[int(g["edge_beg"]):int(g["edge_beg"]) + int(g["n_edges"])]
    assert sorted(float(e["w"]) for e in ed) == [0.75, 1.0]
    # OUT side: 6 joint (x2, y2), 8 y only (its x2 inputs cancel), the output joint
    assert [int(a) & 3 for a in nd["axes"]] == [3, 2, 3]
    assert tuple(g["n_joint"]) == (2, 0) and tuple(g["n_varying"]) == (3, 0)
    assert nd["w_in"][1][X2] == 0.0 and nd["w_in"][1][Y2] == 1.0


def test_pack_rejects_like_the_oracle():
    cyc = _genome([(5, OUT, IDN, 0.0), (6, HID, SIG, 0.0), (7, HID, SIG, 0.0)],
                  [(X2, 6, 1.0, True), (6, 7, 1.0, True), (7, 6, 1.0, True), (7, 5, 1.0, True)])
    good = W.random_population(3, seed=1)
    pop = W.population_from_lists([good.genome(0), good.genome(1), cyc.genome(0), good.genome(2)])
    with pytest.raises(emr.EmrError) as e:
        emr.pack_population(pop)
    assert e.value.status == emr.EMR_ERR_CYCLE and e.value.bad_genome == 2
    assert oracle.check_population(pop) == (oracle.ORA_ERR_CYCLE, 2)
    for bad in ([(5, OUT, IDN, 0.0), (6, OUT, IDN, 0.0)], [(5, HID, IDN, 0.0)]):
        with pytest.raises(emr.EmrError) as e:
            emr.pack_population(_genome(bad, []))
        assert e.value.status == emr.EMR_ERR_ARG
    with pytest.raises(emr.EmrError) as e:
        emr.pack_population(_genome([(5, OUT, IDN, 0.0)], [(5, X2, 1.0, True)]))
    assert e.value.status == emr.EMR_ERR_ARG
    with pytest.raises(emr.EmrError) as e:  # unknown connection endpoint
        emr.pack_population(_genome([(5, OUT, IDN, 0.0)], [(77, 5, 1.0, True)]))
    assert e.value.status == emr.EMR_ERR_ARG


def test_pack_capacity_and_varying_limit():
    pop = W.random_population(4, seed=3)
    L = emr.lib()
    used, bad = C.c_size_t(), C.c_int32()
    small = np.zeros(64, np.uint8)
    st = L.emr_pack_population(pop.P, emr._ptr(pop.node_ptr), emr._ptr(pop.node_id), emr._ptr(pop.node_kind),
                               emr._ptr(pop.node_act), emr._ptr(pop.node_bias), emr._ptr(pop.conn_ptr),
                               emr._ptr(pop.conn_src), emr._ptr(pop.conn_dst), emr._ptr(pop.conn_w),
                               emr._ptr(pop.conn_enabled), emr._ptr(small), C.c_size_t(64), C.byref(used),
                               C.byref(bad))
    assert st == emr.EMR_ERR_CAPACITY and used.value > 64
    # a chain of 70 varying hidden nodes exceeds the 64-node limit
    nodes = [(5, OUT, IDN, 0.0)] + [(100 + k, HID, IDN, 0.0) for k in range(70)]
    conns = [(X2, 100, 1.0, True)] + [(100 + k, 101 + k, 1.0, True) for k in range(69)] + [(169, 5, 1.0, True)]
    with pytest.raises(emr.EmrError) as e:
        emr.pack_population(_genome(nodes, conns))
    assert e.value.status == emr.EMR_ERR_RANGE


@pytest.mark.parametrize("cfg", ["c2", "c3", "c5"])
def test_workload_populations_pack(cfg):
    w = {"c2": lambda: W.c2(D=5), "c3": lambda: W.c3(), "c5": lambda: W.c5()}[cfg]()
    blob = emr.pack_population(w.pop)
    P, mo, mi = emr.pack_info(blob)
    assert P == w.P and 1 <= mo <= 64 and 0 <= mi <= 64
    assert oracle.check_population(w.pop) == (0, -1)
    _, gs, _ = _pack_records(blob)
    assert gs["n_varying"].max() <= 64 and gs["n_vedges"].max() <= 512


def test_cache_handle_host_only():
    c = emr.Cache(1 << 20)
    assert c.stats() == {"hits": 0, "misses": 0, "entries": 0, "bytes": 0}
    c.clear()
    assert c.stats()["entries"] == 0
    del c
    # the raw entry points' documented errors on NULL handles
    L = emr.lib()
    assert L.emr_cache_create(C.c_size_t(1 << 20), None) == emr.EMR_ERR_ARG
    assert L.emr_cache_clear(None) == emr.EMR_ERR_ARG
    assert L.emr_cache_stats(None, None, None, None, None) == emr.EMR_ERR_ARG
    assert L.emr_cache_destroy(None) == emr.EMR_OK


def test_discover_and_copy_reject_arguments_before_device_work():
    """emr_discover checks its arguments, and its workspace size against the host pack and
    query, before any CUDA call; emr_copy_async treats 0 bytes as nothing to do and null
    pointers as an argument error. On a machine without a GPU these come back as the status
    codes the header documents (the buffers are host memory standing in for device memory:
    nothing reads them)."""
    import types
    import torch
    w = W.c1()
    pack = emr.pack_population(w.pop)
    q = emr.make_query(w.sources, device="cpu")
    g = emr.grid_build(w.D)
    need = emr.discover_workspace_size(pack, q, g)
    assert need > 0
    n = w.P * q.S
    st = types.SimpleNamespace(cuda_stream=0)
    ws = torch.zeros(need, dtype=torch.uint8)
    idx, wv = torch.zeros(64, dtype=torch.int32), torch.zeros(64)
    counts, offsets = torch.zeros(n, dtype=torch.int64), torch.zeros(n + 1, dtype=torch.int64)

    def status(**kw):
        args = dict(theta=w.theta, band=w.band, w_min=0.0, mode=emr.EMR_EAGER, types=emr.CONN_ALL,
                    ws=ws, cap=64)
        args.update(kw)
        with pytest.raises(emr.EmrError) as e:
            emr.discover(pack, pack, q, g, args["theta"], args["band"], args["w_min"], args["mode"], args["types"],
                         args["ws"], idx, wv, args["cap"], counts, offsets, stream=st)
        return e.value.status

    assert status(ws=ws[:need - 1]) == emr.EMR_ERR_CAPACITY
    assert status(mode=7) == emr.EMR_ERR_ARG
    assert status(types=emr.CONN_ALL + 1) == emr.EMR_ERR_ARG
    assert status(theta=float("nan")) == emr.EMR_ERR_ARG
    assert status(band=-0.3) == emr.EMR_ERR_ARG
    assert status(cap=-1) == emr.EMR_ERR_ARG
    emr.copy_async(None, None, 0, stream=st)  # nothing to copy
    for dst, src in ((None, ws), (ws, None)):
        with pytest.raises(emr.EmrError) as e:
            emr.copy_async(dst, src, 8, stream=st)
        assert e.value.status == emr.EMR_ERR_ARG


def test_every_entry_point_rejects_zero_arguments():
    """Every status-returning entry point checks its arguments before it reads a pointer or calls
    CUDA: with every argument zero (null pointers, zero sizes and counts) it returns an argument or
    range error, except where zero arguments are a valid call (index 0, destroying a null cache,
    copying 0 bytes, the feedforward substrate configuration), which returns EMR_OK."""
    L = emr.lib()
    zero_ok = {"emr_index_to_ij", "emr_cache_destroy", "emr_copy_async", "emr_substrate_config"}
    pointer_types = (C.c_void_p, C.c_char_p)
    tested = 0
    for name in sorted(declared_symbols()):
        f = getattr(L, name)
        if f.restype is not C.c_int32 or not f.argtypes:  # emr_strerror, emr_version
            continue
        args = [None if (t in pointer_types or issubclass(t, C._Pointer)) else t(0) for t in f.argtypes]
        rc = f(*args)
        if name in zero_ok:
            assert rc == emr.EMR_OK, name
        else:
            assert rc in (emr.EMR_ERR_ARG, emr.EMR_ERR_RANGE), (name, rc)
        tested += 1
    assert tested >= 35


def test_stream_workspace_holds_the_split_plane_and_two_chunks():
    """emr_stream_workspace_size (host only): the resident split plane of every pair plus the
    records and two chunk buffers, growing with the chunk and with the device list capacity; 5.3 GB
    for the depth-13 configuration with the benchmark's chunk (2^26) and list capacity (2^24)."""
    w = W.c5()
    pack = emr.pack_population(w.pop)
    q = emr.make_query(w.sources, device="cpu")
    size = lambda chunk, cap: emr.stream_workspace_size(pack, q, emr.grid_build(w.D, chunk), cap)
    split_plane = w.P * q.S * emr.grid_build(w.D).n_words * 4
    big = size(1 << 26, 1 << 24)
    assert split_plane < size(1 << 20, 1 << 20) < size(1 << 26, 1 << 20) < big
    assert size(1 << 26, 1 << 20) < big and round(big / 1e9, 1) == 5.3


def test_pack_release_joins_workers_and_the_next_pack_is_identical():
    """emr_pack_release joins the packer's worker threads (the process's native thread count drops)
    and frees its buffers; packing again starts them afresh and gives the same blob (host only)."""
    tasks = lambda: len(os.listdir("/proc/self/task"))
    w = W.c2(D=5)
    first = emr.pack_population(w.pop)
    with_pool = tasks()
    emr.pack_release()
    without = tasks()
    emr.pack_release()  # idempotent
    assert tasks() == without
    if (os.cpu_count() or 1) > 1:
        assert without < with_pool
    again = emr.pack_population(w.pop)
    assert np.array_equal(first, again) and tasks() == with_pool


def test_pack_writes_every_byte_and_each_genome_in_its_own_slot():
    """The blob's bytes do not depend on what the buffer held before (every byte written: records,
    zeroed slot tails, section gaps), and each genome's records start at its input's offsets
    (node_ptr[g] - node_ptr[0], conn_ptr[g] - conn_ptr[0]) with room for its input (host only)."""
    w = W.c2(D=5)
    n = emr.pack_size(w.pop)
    a = emr.pack_population(w.pop, out=np.zeros(n, np.uint8)).copy()
    b = emr.pack_population(w.pop, out=np.full(n, 0xA5, np.uint8)).copy()
    assert len(a) <= n and np.array_equal(a, b)
    h, gs, nodes, edges = emr.pack_records(a)
    nptr, cptr = np.asarray(w.pop.node_ptr), np.asarray(w.pop.conn_ptr)
    assert np.array_equal(gs["node_beg"], nptr[:-1] - nptr[0])
    assert np.array_equal(gs["edge_beg"], cptr[:-1] - cptr[0])
    assert np.all(gs["n_nodes"] <= np.diff(nptr)) and np.all(gs["n_edges"] <= np.diff(cptr))
    used_n = np.zeros(len(nodes), bool)
    for g in range(int(h["P"])):
        used_n[int(gs["node_beg"][g]):int(gs["node_beg"][g]) + int(gs["n_nodes"][g])] = True
    assert not nodes[~used_n].view(np.uint8).any()  # the slots' unused records are zero


def test_pack_from_several_threads_at_once_gives_the_sequential_blobs():
    """emr_pack_population called from several host threads at once (ctypes releases the GIL):
    one call gets the worker pool and the shared scratch, the others pack on their own; every
    result equals the blob of a call made alone, back-to-back calls included (host only)."""
    import threading
    pops = [W.c2(D=5).pop, W.c3(D=6).pop, W.c4_round1().pop, W.random_population(300, seed=4)]
    ref = [emr.pack_population(p).copy() for p in pops]
    out = [[None] * 6 for _ in pops]
    errs = []

    def run(i):
        try:
            for k in range(6):
                out[i][k] = emr.pack_population(pops[i]).copy()
        except Exception as e:  # noqa: BLE001 - reported below
            errs.append(e)

    ts = [threading.Thread(target=run, args=(i,)) for i in range(len(pops))]
    for t in ts:
        t.start()
    for t in ts:
        t.join()
    assert not errs
    for i in range(len(pops)):
        assert all(np.array_equal(o, ref[i]) for o in out[i])


def test_pack_large_and_small_genome_paths_agree():
    """Genomes of up to 64 nodes take the packer's bit-mask Kahn order and reachability, larger ones
    the adjacency-list path. The same genomes with 60 isolated hidden nodes added (interleaved ids;
    isolated nodes never reach the output, and Kahn's smallest-id order of the other nodes is
    unchanged by them) go through the large path and must give the same records (host only)."""
    base = W.random_population(200, seed=11)
    padded = []
    for g in range(base.P):
        nodes, conns = base.genome(g)
        top = max(i for i, _, _, _ in nodes)
        extra = [(top + 1 + 2 * k if k % 2 else -(k + 1), W.KIND_HIDDEN, W.ACT_SIGMOID, 0.5) for k in range(60)]
        padded.append((nodes + extra, conns))
    pop_pad = W.population_from_lists(padded)
    a, b = emr.pack_population(base), emr.pack_population(pop_pad)
    ha, ga, na, ea = emr.pack_records(a)
    hb, gb, nb, eb = emr.pack_records(b)
    assert int(W.np.diff(pop_pad.node_ptr).min()) > 64
    for f in ("max_nodes", "max_varying", "max_vedges", "max_edges"):
        assert W.np.array_equal(ha[f], hb[f])
    for g in range(base.P):
        for f in ("n_nodes", "n_edges", "n_varying", "n_vedges", "cost", "n_joint"):
            assert W.np.array_equal(ga[g][f], gb[g][f]), (g, f)
        x0, x1, n = int(ga[g]["node_beg"]), int(gb[g]["node_beg"]), int(ga[g]["n_nodes"])
        assert na[x0:x0 + n].tobytes() == nb[x1:x1 + n].tobytes()
        y0, y1, m = int(ga[g]["edge_beg"]), int(gb[g]["edge_beg"]), int(ga[g]["n_edges"])
        assert ea[y0:y0 + m].tobytes() == eb[y1:y1 + m].tobytes()


def test_grid_chunks_cover_the_grid_in_whole_tiles():
    """emr_grid_chunk: chunks in ascending global index, contiguous, covering [0, N_total), every
    boundary but the first a 64 x 64 tile boundary past depth 4, the same count emr_stream uses."""
    for D, chunk in ((0, 0), (5, 4096), (7, 0), (7, 1 << 14), (10, 1 << 16), (13, 1 << 26)):
        g = emr.grid_build(D, chunk)
        n = emr.grid_chunk(g)[0]
        r = [emr.grid_chunk(g, k)[1:] for k in range(n)]
        assert r[0][0] == 0 and r[-1][1] == g.n_total
        assert all(a[1] == b[0] for a, b in zip(r, r[1:]))
        lo5 = oracle.n_total(4) if D >= 5 else g.n_total
        assert all(b[0] >= lo5 and (b[0] - lo5) % 4096 == 0 for b in r[1:])
        if chunk:
            assert all(hi - lo <= max(chunk, lo5 + chunk) for lo, hi in r)
        with pytest.raises(emr.EmrError) as e:
            emr.grid_chunk(g, n)
        assert e.value.status == emr.EMR_ERR_RANGE
    g = emr.grid_build(13, 1 << 26)
    assert emr.grid_chunk(g)[0] == 6  # depth 13 in chunks of 2^26: 5.33 chunks, the remainder in the lowest
