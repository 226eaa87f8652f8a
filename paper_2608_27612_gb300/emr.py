"""Thin ctypes binding of libemr's C ABI (include/emr.h), same names, no compute.

Device buffers are torch tensors (passed by data_ptr); streams are torch
streams. Every step of the path runs in libemr's kernels: this module only
marshals arguments, allocates caller-owned buffers for the convenience
wrappers and turns status codes into exceptions. There is no fallback: if the
library has not been built, loading it raises.
"""
from __future__ import annotations

import ctypes as C
import os
from dataclasses import dataclass

import numpy as np
import torch

from . import _build

EMR_OK, EMR_ERR_ARG, EMR_ERR_CYCLE, EMR_ERR_RANGE, EMR_ERR_CAPACITY, EMR_ERR_CUDA, EMR_ERR_TIMEOUT, \
    EMR_ERR_ALLOC = range(8)
EMR_MAX_DEPTH = 14
EMR_EAGER, EMR_GATED = 0, 1
CONN_F, CONN_B, CONN_L, CONN_S, CONN_ALL = 1, 2, 4, 8, 15
SUBSTRATE_FEEDFORWARD, SUBSTRATE_HH, SUBSTRATE_BACKWARD, SUBSTRATE_LATERAL, SUBSTRATE_SELF, SUBSTRATE_FULL = range(6)
TYPE_CODES = ("forward", "backward", "lateral", "self")
_M = EMR_MAX_DEPTH + 2

_lib = None


class EmrError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__("%s: %s (status %d)" % (what, strerror(status) if _lib else "?", status))


class Grid(C.Structure):
    _fields_ = [("D", C.c_int32), ("reserved", C.c_int32), ("n_total", C.c_int64), ("n_halo", C.c_int64),
                ("n_words", C.c_int64), ("chunk", C.c_int64), ("level_off", C.c_int64 * _M),
                ("halo_off", C.c_int64 * _M), ("word_off", C.c_int64 * _M)]


class QueryC(C.Structure):
    _fields_ = [("S", C.c_int32), ("per_genome", C.c_int32), ("a_host", C.c_void_p), ("b_host", C.c_void_p),
                ("side_host", C.c_void_p), ("count_host", C.c_void_p), ("a_dev", C.c_void_p),
                ("b_dev", C.c_void_p), ("side_dev", C.c_void_p), ("count_dev", C.c_void_p)]


def lib() -> C.CDLL:
    """Load libemr (after torch, so both share one CUDA runtime). Raises if it is not built."""
    global _lib
    if _lib is None:
        if not os.path.exists(_build.LIB):
            raise RuntimeError("libemr is not built (%s missing): run __graft_entry__.build()" % _build.LIB)
        _lib = C.CDLL(_build.LIB)
        vp, i32, i64, f32, sz = C.c_void_p, C.c_int32, C.c_int64, C.c_float, C.c_size_t
        sig = {
            "emr_grid_build": [i32, i64, vp],
            "emr_index_to_ij": [i64, vp, vp, vp],
            "emr_pack_size": [i32, vp, vp, vp],
            "emr_pack_population": [i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp, vp],
            "emr_pack_info": [vp, vp, vp, vp],
            "emr_partition_genomes": [vp, vp, i32, vp],
            "emr_eval_workspace_size": [vp, vp, vp],
            "emr_eval_prepare": [vp, vp, vp, vp, sz, vp],
            "emr_eval": [vp, vp, vp, vp, vp, vp, sz, vp],
            "emr_grid_chunk": [vp, i64, vp, vp, vp],
            "emr_eval_chunk": [vp, vp, vp, i64, vp, vp, vp, sz, vp],
            "emr_variance_filter": [vp, vp, vp, i32, i32, f32, f32, f32, i32, vp, vp, vp, vp, vp],
            "emr_mask_combine": [vp, vp, vp, i32, i32, vp, vp],
            "emr_eval_filter": [vp, vp, vp, f32, f32, f32, vp, vp, vp, vp, sz, vp],
            "emr_eval_filter_noalloc": [vp, vp, vp, vp, f32, f32, f32, vp, vp, vp, vp],
            "emr_stream_workspace_size": [vp, vp, vp, i64, vp],
            "emr_stream": [vp, vp, vp, vp, f32, f32, f32, vp, sz, i64, vp, vp, i64, vp, vp, i64, vp],
            "emr_stream_mode": [vp, vp, vp, vp, f32, f32, f32, i32, i32, vp, sz, i64, vp, vp, i64, vp, vp, i64, vp],
            "emr_mask_combine_types": [vp, vp, vp, vp, i32, i32, i32, vp, vp],
            "emr_conn_types": [vp, vp, vp, vp, i32, i64, vp, vp],
            "emr_scale_weights": [vp, vp, i32, i64, f32, f32, vp],
            "emr_subtree_workspace_size": [vp, i32, vp],
            "emr_subtree_split": [vp, vp, i32, f32, vp, vp, vp, sz, vp],
            "emr_eval_filter_tiles": [vp, vp, vp, f32, f32, f32, vp, vp, vp, vp, sz, vp],
            "emr_select": [vp, vp, vp, vp, vp, vp, sz, vp, i32, i32, vp, vp, i64, vp, vp, vp, sz, vp],
            "emr_select_workspace_size": [vp, i32, vp],
            "emr_discover_workspace_size": [vp, vp, vp, vp],
            "emr_discover": [vp, vp, vp, vp, f32, f32, f32, i32, i32, vp, sz, vp, vp, i64, vp, vp, vp],
            "emr_copy_async": [vp, vp, sz, vp],
            "emr_substrate_config": [i32, vp, vp],
            "emr_assemble_workspace_size": [vp, i32, i32, i32, vp, i64, vp],
            "emr_assemble": [vp, vp, i32, vp, vp, i32, vp, vp, vp, f32, f32, f32, i32, i32, i32, i32, vp, sz, i64,
                             vp, vp, i64, vp, vp, vp, vp, vp, i64, vp, vp],
            "emr_cache_create": [sz, vp],
            "emr_cache_destroy": [vp],
            "emr_cache_clear": [vp],
            "emr_cache_stats": [vp, vp, vp, vp, vp],
            "emr_ann_forward": [i32, i32, i32, i32, vp, vp, vp, vp, vp, i32, vp, i32, vp, vp],
            "emr_compact_workspace_size": [vp, i32, vp],
            "emr_compact": [vp, vp, vp, i32, vp, vp, i64, vp, vp, vp, sz, vp],
            "emr_compact_records": [vp, vp, vp, vp, sz, vp, vp, vp, i64, vp, vp, vp, sz, vp],
            "emr_version": [],
            "emr_probe_alu": [i32, i32, i32, vp, vp, vp, vp],
        }
        for name, args in sig.items():
            f = getattr(_lib, name)
            f.argtypes = args
            f.restype = C.c_int32
        _lib.emr_pack_release.argtypes = []
        _lib.emr_pack_release.restype = None
        _lib.emr_strerror.argtypes = [C.c_int32]
        _lib.emr_strerror.restype = C.c_char_p
    return _lib


def strerror(status: int) -> str:
    return lib().emr_strerror(status).decode()


def _check(status: int, what: str):
    if status != EMR_OK:
        raise EmrError(status, what)


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, torch.Tensor):
        return C.c_void_p(x.data_ptr())
    if isinstance(x, np.ndarray):
        return x.ctypes.data_as(C.c_void_p)
    return x


def _stream(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return C.c_void_p(s.cuda_stream)


# ---- a1 -----------------------------------------------------------------------

def grid_build(D: int, chunk: int = 0) -> Grid:
    g = Grid()
    _check(lib().emr_grid_build(D, chunk, C.byref(g)), "emr_grid_build")
    return g


def index_to_ij(gidx: int):
    d, i, j = C.c_int32(), C.c_int32(), C.c_int32()
    _check(lib().emr_index_to_ij(gidx, C.byref(d), C.byref(i), C.byref(j)), "emr_index_to_ij")
    return d.value, i.value, j.value


# ---- a2 -----------------------------------------------------------------------

def _pop_ptrs(pop):
    """Addresses of a Population's ten arrays, kept on the object together with the arrays
    themselves (so an address never outlives its array); a field that now holds another
    array is looked up again."""
    arrays = (pop.node_ptr, pop.node_id, pop.node_kind, pop.node_act, pop.node_bias, pop.conn_ptr,
              pop.conn_src, pop.conn_dst, pop.conn_w, pop.conn_enabled)
    cache = getattr(pop, "_emr_ptrs", None)
    if cache is None or any(a is not b for a, b in zip(cache[0], arrays)):
        cache = (arrays, tuple(int(a.ctypes.data) for a in arrays))
        try:
            object.__setattr__(pop, "_emr_ptrs", cache)
        except AttributeError:
            pass
    return cache[1]


def _range_ptrs(pop, genomes):
    """P and the ten array addresses for genomes [g0, g1) of pop (the whole population when
    genomes is None): node_ptr and conn_ptr offset to g0, the other arrays unchanged."""
    ptr = _pop_ptrs(pop)
    if genomes is None:
        return pop.P, ptr
    g0, g1 = int(genomes[0]), int(genomes[1])
    if not 0 <= g0 < g1 <= pop.P:
        raise ValueError("genome range [%d, %d) outside [0, %d)" % (g0, g1, pop.P))
    return g1 - g0, (ptr[0] + 8 * g0,) + ptr[1:5] + (ptr[5] + 8 * g0,) + ptr[6:]


def pack_size(pop, genomes=None) -> int:
    """Upper bound of the packed blob's bytes for a workloads.Population (emr_pack_size)."""
    n = C.c_size_t()
    P, ptr = _range_ptrs(pop, genomes)
    _check(lib().emr_pack_size(P, ptr[0], ptr[5], C.byref(n)), "emr_pack_size")
    return int(n.value)


def pack_population(pop, out=None, genomes=None) -> np.ndarray:
    """Packed blob (numpy uint8) of a workloads.Population, or of its genomes [g0, g1) when
    genomes = (g0, g1); written into `out` (a contiguous uint8 array, e.g. a view of pinned
    memory) when given, else into a new array."""
    L = lib()
    n = C.c_size_t()
    P, ptr = _range_ptrs(pop, genomes)
    _check(L.emr_pack_size(P, ptr[0], ptr[5], C.byref(n)), "emr_pack_size")
    if out is not None:
        if out.dtype != np.uint8 or not out.flags.c_contiguous or len(out) < n.value:
            raise ValueError("out: contiguous uint8 array of at least %d bytes" % n.value)
        buf = out
    else:
        buf = np.empty(n.value + 16, np.uint8)   # the packer clears what it uses
    used, bad = C.c_size_t(), C.c_int32()
    st = L.emr_pack_population(P, *ptr, int(buf.ctypes.data), len(buf), C.byref(used), C.byref(bad))
    if st != EMR_OK:
        e = EmrError(st, "emr_pack_population (genome %d)" % bad.value)
        e.bad_genome = bad.value
        raise e
    return buf[:used.value]


def pack_release() -> None:
    """Join the packer's worker threads and free its kept buffers (emr_pack_release)."""
    lib().emr_pack_release()


def partition_genomes(pack: np.ndarray, query, n_parts: int) -> np.ndarray:
    """Contiguous genome ranges of balanced cost (emr_partition_genomes): int32 [n_parts + 1],
    part k = genomes [g[k], g[k+1])."""
    g = np.zeros(n_parts + 1, np.int32)
    q = query.c
    _check(lib().emr_partition_genomes(_ptr(pack), C.byref(q), n_parts, _ptr(g)), "emr_partition_genomes")
    return g


def pack_info(pack: np.ndarray):
    P, mo, mi = C.c_int32(), C.c_int32(), C.c_int32()
    _check(lib().emr_pack_info(_ptr(pack), C.byref(P), C.byref(mo), C.byref(mi)), "emr_pack_info")
    return P.value, mo.value, mi.value


@dataclass
class Query:
    """Host and device copies of the query slots (workloads.Sources)."""
    a: np.ndarray
    b: np.ndarray
    side: np.ndarray
    count: np.ndarray | None
    a_dev: torch.Tensor
    b_dev: torch.Tensor
    side_dev: torch.Tensor
    count_dev: torch.Tensor | None
    S: int
    per_genome: bool

    @property
    def c(self) -> QueryC:
        q = QueryC()
        q.S, q.per_genome = self.S, 1 if self.per_genome else 0
        q.a_host, q.b_host, q.side_host = (self.a.ctypes.data, self.b.ctypes.data, self.side.ctypes.data)
        q.count_host = self.count.ctypes.data if self.count is not None else None
        q.a_dev, q.b_dev, q.side_dev = (self.a_dev.data_ptr(), self.b_dev.data_ptr(), self.side_dev.data_ptr())
        q.count_dev = self.count_dev.data_ptr() if self.count_dev is not None else None
        return q


def make_query(sources, device="cuda") -> Query:
    a = np.ascontiguousarray(sources.a, np.float32)
    b = np.ascontiguousarray(sources.b, np.float32)
    s = np.ascontiguousarray(sources.side, np.int32)
    cnt = None if sources.count is None else np.ascontiguousarray(sources.count, np.int32)
    dev = lambda x: torch.from_numpy(x).to(device) if x is not None else None
    return Query(a, b, s, cnt, dev(a), dev(b), dev(s), dev(cnt), int(a.shape[-1]), a.ndim == 2)


# ---- workspace sizes ------------------------------------------------------------

def eval_workspace_size(pack: np.ndarray, query: Query) -> int:
    n = C.c_size_t()
    q = query.c
    _check(lib().emr_eval_workspace_size(_ptr(pack), C.byref(q), C.byref(n)), "emr_eval_workspace_size")
    return n.value


def compact_workspace_size(grid: Grid, n_pairs: int) -> int:
    n = C.c_size_t()
    _check(lib().emr_compact_workspace_size(C.byref(grid), n_pairs, C.byref(n)), "emr_compact_workspace_size")
    return n.value


# ---- a3..a6 -----------------------------------------------------------------------

def eval_prepare(pack, pack_dev, query: Query, ws, stream=None):
    q = query.c
    _check(lib().emr_eval_prepare(_ptr(pack), _ptr(pack_dev), C.byref(q), _ptr(ws), C.c_size_t(ws.numel()),
                                  _stream(stream)), "emr_eval_prepare")


def eval(pack, query: Query, grid: Grid, out, out_halo, ws, stream=None):
    q = query.c
    _check(lib().emr_eval(_ptr(pack), C.byref(q), C.byref(grid), _ptr(out), _ptr(out_halo), _ptr(ws),
                          C.c_size_t(ws.numel()), _stream(stream)), "emr_eval")


def grid_chunk(grid: Grid, chunk_idx: int = 0):
    """(number of chunks, first global index, end global index) of chunk chunk_idx (emr_grid_chunk)."""
    n, lo, hi = C.c_int64(), C.c_int64(), C.c_int64()
    _check(lib().emr_grid_chunk(C.byref(grid), chunk_idx, C.byref(n), C.byref(lo), C.byref(hi)), "emr_grid_chunk")
    return n.value, lo.value, hi.value


def eval_chunk(pack, query: Query, grid: Grid, chunk_idx: int, out, out_halo, ws, stream=None):
    """emr_eval_chunk: CPPN outputs of one chunk, out [pairs, chunk positions]."""
    q = query.c
    _check(lib().emr_eval_chunk(_ptr(pack), C.byref(q), C.byref(grid), chunk_idx, _ptr(out), _ptr(out_halo),
                                _ptr(ws), ws.numel(), _stream(stream)), "emr_eval_chunk")

def variance_filter(out, out_halo, grid: Grid, P: int, S: int, theta: float, band: float, w_min: float, mode: int,
                    mask, split, band_bits, var_dbg=None, stream=None):
    _check(lib().emr_variance_filter(_ptr(out), _ptr(out_halo), C.byref(grid), P, S, theta, band, w_min, mode,
                                     _ptr(mask), _ptr(split), _ptr(band_bits), _ptr(var_dbg), _stream(stream)),
           "emr_variance_filter")


def mask_combine(split, band_bits, grid: Grid, n_pairs: int, mode: int, mask, stream=None):
    _check(lib().emr_mask_combine(_ptr(split), _ptr(band_bits), C.byref(grid), n_pairs, mode, _ptr(mask),
                                  _stream(stream)), "emr_mask_combine")


def eval_filter(pack, query: Query, grid: Grid, theta: float, band: float, w_min: float, split, band_bits, out, ws,
                stream=None):
    q = query.c
    _check(lib().emr_eval_filter(_ptr(pack), C.byref(q), C.byref(grid), theta, band, w_min, _ptr(split),
                                 _ptr(band_bits), _ptr(out), _ptr(ws), C.c_size_t(ws.numel()), _stream(stream)),
           "emr_eval_filter")


def eval_filter_noalloc(pack, pack_dev, query: Query, grid: Grid, theta: float, band: float, w_min: float, split,
                        band_bits, out, stream=None):
    """emr_eval_filter_noalloc: prepare + fused evaluation in libemr's static device scratch."""
    q = query.c
    _check(lib().emr_eval_filter_noalloc(_ptr(pack), _ptr(pack_dev), C.byref(q), C.byref(grid), theta, band, w_min,
                                         _ptr(split), _ptr(band_bits), _ptr(out), _stream(stream)),
           "emr_eval_filter_noalloc")


def stream_workspace_size(pack, query: Query, grid: Grid, chunk_cap: int) -> int:
    n = C.c_size_t()
    q = query.c
    _check(lib().emr_stream_workspace_size(_ptr(pack), C.byref(q), C.byref(grid), chunk_cap, C.byref(n)),
           "emr_stream_workspace_size")
    return n.value


def stream(pack, pack_dev, query: Query, grid: Grid, theta: float, band: float, w_min: float, ws, chunk_cap: int,
           h_idx, h_w, counts, offsets, timeout_ms: int = 0, stream=None, mode: int = EMR_EAGER,
           types: int = CONN_ALL):
    """emr_stream (eager, every type) or emr_stream_mode: chunked discovery; lists land in the
    (pinned) host tensors h_idx / h_w."""
    q = query.c
    if mode == EMR_EAGER and types == CONN_ALL:
        _check(lib().emr_stream(_ptr(pack), _ptr(pack_dev), C.byref(q), C.byref(grid), theta, band, w_min, _ptr(ws),
                                C.c_size_t(ws.numel()), chunk_cap, _ptr(h_idx), _ptr(h_w), h_idx.numel(),
                                _ptr(counts), _ptr(offsets), timeout_ms, _stream(stream)), "emr_stream")
        return
    _check(lib().emr_stream_mode(_ptr(pack), _ptr(pack_dev), C.byref(q), C.byref(grid), theta, band, w_min, mode,
                                 types, _ptr(ws), C.c_size_t(ws.numel()), chunk_cap, _ptr(h_idx), _ptr(h_w),
                                 h_idx.numel(), _ptr(counts), _ptr(offsets), timeout_ms, _stream(stream)),
           "emr_stream_mode")


def dense_tiles(D: int) -> int:
    """Dense tiles of a depth-D grid: one for depths 0..4, then the 64 x 64 blocks of depths 5..D."""
    return 1 + sum(4 ** (d - 5) for d in range(5, D + 1))


def eval_filter_tiles(pack, query: Query, grid: Grid, theta: float, band: float, w_min: float, split, band_bits,
                      tile_flags, ws, stream=None):
    q = query.c
    _check(lib().emr_eval_filter_tiles(_ptr(pack), C.byref(q), C.byref(grid), theta, band, w_min, _ptr(split),
                                       _ptr(band_bits), _ptr(tile_flags), _ptr(ws), C.c_size_t(ws.numel()),
                                       _stream(stream)), "emr_eval_filter_tiles")


def select_workspace_size(grid: Grid, n_pairs: int) -> int:
    n = C.c_size_t()
    _check(lib().emr_select_workspace_size(C.byref(grid), n_pairs, C.byref(n)), "emr_select_workspace_size")
    return n.value


def select(split, band_bits, tile_flags, pack, query: Query, eval_ws, grid: Grid, mode: int, types: int, idx, w,
           cap: int, counts, offsets, ws, stream=None):
    """emr_select: combine + compaction + kept weights over the flagged tiles only."""
    q = query.c
    _check(lib().emr_select(_ptr(split), _ptr(band_bits), _ptr(tile_flags), _ptr(pack), C.byref(q), _ptr(eval_ws),
                            C.c_size_t(eval_ws.numel()), C.byref(grid), mode, types, _ptr(idx), _ptr(w), cap,
                            _ptr(counts), _ptr(offsets), _ptr(ws), C.c_size_t(ws.numel()), _stream(stream)),
           "emr_select")


def discover_workspace_size(pack, query: Query, grid: Grid) -> int:
    n = C.c_size_t()
    q = query.c
    _check(lib().emr_discover_workspace_size(_ptr(pack), C.byref(q), C.byref(grid), C.byref(n)),
           "emr_discover_workspace_size")
    return n.value


def discover(pack, pack_dev, query: Query, grid: Grid, theta: float, band: float, w_min: float, mode: int,
             types: int, ws, idx, w, cap: int, counts, offsets, stream=None, qc=None):
    """emr_discover: the whole path (records, fused evaluation and filter, selection) in one call.
    qc: a QueryC from query.c, to reuse across calls."""
    q = qc if qc is not None else query.c
    _check(lib().emr_discover(_ptr(pack), _ptr(pack_dev), C.byref(q), C.byref(grid), theta, band, w_min, mode, types,
                              _ptr(ws), C.c_size_t(ws.numel()), _ptr(idx), _ptr(w), cap, _ptr(counts),
                              _ptr(offsets), _stream(stream)), "emr_discover")


def copy_async(dst, src, nbytes: int, stream=None):
    """emr_copy_async: nbytes from src to dst (tensors, numpy arrays or addresses; host buffers
    pinned) on the stream."""
    _check(lib().emr_copy_async(_ptr(dst), _ptr(src), C.c_size_t(nbytes), _stream(stream)), "emr_copy_async")


def mask_combine_types(split, band_bits, query: Query, grid: Grid, n_pairs: int, mode: int, types: int, mask,
                       stream=None):
    q = query.c
    _check(lib().emr_mask_combine_types(_ptr(split), _ptr(band_bits), C.byref(q), C.byref(grid), n_pairs, mode,
                                        types, _ptr(mask), _stream(stream)), "emr_mask_combine_types")


def subtree_workspace_size(grid: Grid, n_pairs: int) -> int:
    n = C.c_size_t()
    _check(lib().emr_subtree_workspace_size(C.byref(grid), n_pairs, C.byref(n)), "emr_subtree_workspace_size")
    return n.value


def subtree_split(out, grid: Grid, n_pairs: int, theta: float, split, ws, var_out=None, stream=None):
    """emr_subtree_split: split plane from the variance over each cell's depth-D descendants."""
    _check(lib().emr_subtree_split(_ptr(out), C.byref(grid), n_pairs, theta, _ptr(split), _ptr(var_out), _ptr(ws),
                                   C.c_size_t(ws.numel()), _stream(stream)), "emr_subtree_split")


def scale_weights(w, offsets, n_pairs: int, cap: int, w_thr: float, w_max: float, stream=None):
    """emr_scale_weights: HyperNEAT's thresholded linear weight scaling of list weights, in place."""
    _check(lib().emr_scale_weights(_ptr(w), _ptr(offsets), n_pairs, cap, w_thr, w_max, _stream(stream)),
           "emr_scale_weights")


def conn_types(idx, offsets, query: Query, grid: Grid, n_pairs: int, cap: int, type_out, stream=None):
    """emr_conn_types: type code (0 F, 1 B, 2 L, 3 S) of every list entry into the device uint8 tensor."""
    q = query.c
    _check(lib().emr_conn_types(_ptr(idx), _ptr(offsets), C.byref(q), C.byref(grid), n_pairs, cap, _ptr(type_out),
                                _stream(stream)), "emr_conn_types")


def substrate_config(config: int):
    """(enabled EMR_CONN_* bits, hidden-to-hidden rounds on) of a Section 6 substrate configuration."""
    t, h = C.c_int32(), C.c_int32()
    _check(lib().emr_substrate_config(config, C.byref(t), C.byref(h)), "emr_substrate_config")
    return t.value, h.value


def compact(mask, out, grid: Grid, n_pairs: int, idx, w, cap: int, counts, offsets, ws, stream=None):
    _check(lib().emr_compact(_ptr(mask), _ptr(out), C.byref(grid), n_pairs, _ptr(idx), _ptr(w), cap, _ptr(counts),
                             _ptr(offsets), _ptr(ws), C.c_size_t(ws.numel()), _stream(stream)), "emr_compact")


def compact_records(mask, pack, query: Query, eval_ws, grid: Grid, idx, w, cap: int, counts, offsets, ws,
                    stream=None):
    """emr_compact_records: lists with the kept weights recomputed from the prepared records."""
    q = query.c
    _check(lib().emr_compact_records(_ptr(mask), _ptr(pack), C.byref(q), _ptr(eval_ws),
                                     C.c_size_t(eval_ws.numel()), C.byref(grid), _ptr(idx), _ptr(w), cap,
                                     _ptr(counts), _ptr(offsets), _ptr(ws), C.c_size_t(ws.numel()),
                                     _stream(stream)), "emr_compact_records")


# ---- network assembly and the substrate ANN ----------------------------------------------

@dataclass
class Networks:
    """Assembled substrate networks (host arrays, layout of emr_assemble)."""
    n_in: int
    n_out: int
    node_off: np.ndarray   # int64 [P + 1]
    hidden: np.ndarray     # int32 global grid indices
    conn_off: np.ndarray   # int64 [P + 1]
    src: np.ndarray        # int32
    dst: np.ndarray        # int32
    w: np.ndarray          # float32
    type: np.ndarray       # uint8
    _dev: tuple | None = None  # device copies made by ann_forward

    @property
    def P(self) -> int:
        return len(self.node_off) - 1

    def genome(self, g: int):
        """(hidden positions, src, dst, w, type) of genome g."""
        h = self.hidden[self.node_off[g]:self.node_off[g + 1]]
        c = slice(self.conn_off[g], self.conn_off[g + 1])
        return h, self.src[c], self.dst[c], self.w[c], self.type[c]


class Cache:
    """emr_cache: connection lists reused across emr_assemble calls (owned handle)."""

    def __init__(self, max_bytes: int = 1 << 30):
        h = C.c_void_p()
        _check(lib().emr_cache_create(max_bytes, C.byref(h)), "emr_cache_create")
        self.handle = h

    def stats(self):
        v = [C.c_int64() for _ in range(4)]
        _check(lib().emr_cache_stats(self.handle, *[C.byref(x) for x in v]), "emr_cache_stats")
        return dict(zip(("hits", "misses", "entries", "bytes"), (x.value for x in v)))

    def clear(self):
        _check(lib().emr_cache_clear(self.handle), "emr_cache_clear")

    def __del__(self):
        if getattr(self, "handle", None) and _lib is not None:
            _lib.emr_cache_destroy(self.handle)
            self.handle = None


def assemble(pack, pack_dev, in_xy, out_xy, grid: Grid, theta: float, band: float, w_min: float = 0.0,
             mode: int = EMR_EAGER, types: int = CONN_ALL, rounds: int = 1, slots_max: int = 256,
             list_cap: int = 1 << 24, hidden_cap: int = 1 << 22, conn_cap: int = 1 << 24, stream=None,
             cache: Cache | None = None) -> Networks:
    """emr_assemble: substrate networks of every genome (device workspace allocated here)."""
    in_xy = np.ascontiguousarray(in_xy, np.float32).reshape(-1, 2)
    out_xy = np.ascontiguousarray(out_xy, np.float32).reshape(-1, 2)
    ix, iy = np.ascontiguousarray(in_xy[:, 0]), np.ascontiguousarray(in_xy[:, 1])
    ox, oy = np.ascontiguousarray(out_xy[:, 0]), np.ascontiguousarray(out_xy[:, 1])
    n = C.c_size_t()
    _check(lib().emr_assemble_workspace_size(_ptr(pack), len(ix), len(ox), slots_max, C.byref(grid), list_cap,
                                             C.byref(n)), "emr_assemble_workspace_size")
    ws = torch.empty(n.value, dtype=torch.uint8, device="cuda")
    P = pack_info(pack)[0]
    node_off = np.zeros(P + 1, np.int64)
    conn_off = np.zeros(P + 1, np.int64)
    hidden = np.zeros(hidden_cap, np.int32)
    src = np.zeros(conn_cap, np.int32)
    dst = np.zeros(conn_cap, np.int32)
    w = np.zeros(conn_cap, np.float32)
    ty = np.zeros(conn_cap, np.uint8)
    _check(lib().emr_assemble(_ptr(pack), _ptr(pack_dev), len(ix), _ptr(ix), _ptr(iy), len(ox), _ptr(ox), _ptr(oy),
                              C.byref(grid), theta, band, w_min, mode, types, rounds, slots_max, _ptr(ws),
                              C.c_size_t(ws.numel()), list_cap, _ptr(node_off), _ptr(hidden), hidden_cap,
                              _ptr(conn_off), _ptr(src), _ptr(dst), _ptr(w), _ptr(ty), conn_cap,
                              cache.handle if cache is not None else None, _stream(stream)),
           "emr_assemble")
    nh, nc = int(node_off[-1]), int(conn_off[-1])
    return Networks(len(ix), len(ox), node_off, hidden[:nh].copy(), conn_off, src[:nc].copy(), dst[:nc].copy(),
                    w[:nc].copy(), ty[:nc].copy())


def ann_forward(nets: Networks, patterns, steps: int, device="cuda", stream=None, out=None):
    """emr_ann_forward: outputs [P, K, n_out] (device tensor) of every network on patterns [K, n_in].
    The networks' arrays are copied to the device once and kept with them."""
    dev = torch.device(device)
    if getattr(nets, "_dev", None) is None or nets._dev[0] != dev:
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
        nets._dev = (dev, t(nets.node_off), t(nets.conn_off), t(nets.src), t(nets.dst), t(nets.w))
    _, node_off, conn_off, src, dst, w = nets._dev
    pat = patterns if isinstance(patterns, torch.Tensor) else \
        torch.as_tensor(np.ascontiguousarray(patterns, np.float32).reshape(-1, nets.n_in), device=dev)
    K = pat.shape[0]
    if out is None:
        out = torch.zeros(nets.P, K, nets.n_out, dtype=torch.float32, device=dev)
    max_hidden = int(np.max(np.diff(nets.node_off))) if nets.P else 0
    _check(lib().emr_ann_forward(nets.P, nets.n_in, nets.n_out, max_hidden, _ptr(node_off), _ptr(conn_off),
                                 _ptr(src), _ptr(dst), _ptr(w), K, _ptr(pat), steps, _ptr(out), _stream(stream)),
           "emr_ann_forward")
    return out


# ---- ALU probes (roofline denominators) -------------------------------------------------

PROBE_FFMA, PROBE_EX2, PROBE_RCP, PROBE_SIN = range(4)


def probe_alu(op: int, blocks: int, iters: int, stream=None):
    """(operations, milliseconds) of one probe launch (include/emr_probe.h)."""
    sink = torch.zeros(blocks, dtype=torch.float32, device="cuda")
    ops, ms = C.c_double(), C.c_float()
    _check(lib().emr_probe_alu(op, blocks, iters, C.byref(ops), C.byref(ms), _ptr(sink), _stream(stream)),
           "emr_probe_alu")
    return ops.value, ms.value


# ---- convenience: the whole path on caller-visible buffers --------------------------

class Discovery:
    """Buffers and calls for one (population, query, depth) configuration.

    run_fused(): CPPN outputs never materialised; the kept weights are recomputed at compaction
    (or, with sparse_out=True, written by the fused kernel where the band test passed).
    run_unfused(): CPPN outputs materialised, then filtered.
    """

    def __init__(self, pop, sources, D: int, theta: float, band: float, w_min: float = 0.0,
                 mode: int = EMR_EAGER, cap: int | None = None, materialise: bool = False, device="cuda",
                 types: int = CONN_ALL):
        self.device = torch.device(device)
        self.pack = pack_population(pop)
        self.pack_dev = torch.from_numpy(self.pack).to(self.device)
        self.query = make_query(sources, self.device)
        self.grid = grid_build(D)
        self.P, self.S = pop.P, self.query.S
        self.n_pairs = self.P * self.S
        self.theta, self.band, self.w_min, self.mode, self.types = theta, band, w_min, mode, types
        g = self.grid
        u32 = dict(dtype=torch.int32, device=self.device)
        self.mask = torch.zeros(self.n_pairs, g.n_words, **u32)
        self.split = torch.zeros(self.n_pairs, g.n_words, **u32)
        self.band_bits = torch.zeros(self.n_pairs, g.n_words, **u32)
        self.out = (torch.zeros(self.n_pairs, g.n_total, dtype=torch.float32, device=self.device)
                    if materialise else None)
        self.out_halo = (torch.zeros(self.n_pairs, g.n_halo, dtype=torch.float32, device=self.device)
                         if materialise else None)
        self.var_dbg = None
        self.ws = torch.zeros(eval_workspace_size(self.pack, self.query), dtype=torch.uint8, device=self.device)
        self.cws = torch.zeros(compact_workspace_size(g, self.n_pairs), dtype=torch.uint8, device=self.device)
        self.cap = int(cap if cap is not None else min(self.n_pairs * g.n_total, 1 << 27))
        self.idx = torch.zeros(self.cap, dtype=torch.int32, device=self.device)
        self.w = torch.zeros(self.cap, dtype=torch.float32, device=self.device)
        self.counts = torch.zeros(self.n_pairs, dtype=torch.int64, device=self.device)
        self.offsets = torch.zeros(self.n_pairs + 1, dtype=torch.int64, device=self.device)

    def prepare(self, stream=None):
        eval_prepare(self.pack, self.pack_dev, self.query, self.ws, stream)

    def _materialise(self):
        if self.out is None:
            self.out = torch.zeros(self.n_pairs, self.grid.n_total, dtype=torch.float32, device=self.device)
        if self.out_halo is None:
            self.out_halo = torch.zeros(self.n_pairs, self.grid.n_halo, dtype=torch.float32, device=self.device)

    def run_fused(self, sparse_out: bool = False, stream=None):
        """emr_eval_prepare, emr_eval_filter, emr_mask_combine, emr_compact_records
        (sparse_out: emr_eval_filter writes band-passing outputs, emr_compact reads them)."""
        self.prepare(stream)
        if sparse_out:
            self._materialise()
        eval_filter(self.pack, self.query, self.grid, self.theta, self.band, self.w_min, self.split,
                    self.band_bits, self.out if sparse_out else None, self.ws, stream)
        self.combine(stream)
        if sparse_out:
            compact(self.mask, self.out, self.grid, self.n_pairs, self.idx, self.w, self.cap, self.counts,
                    self.offsets, self.cws, stream)
        else:
            compact_records(self.mask, self.pack, self.query, self.ws, self.grid, self.idx, self.w, self.cap,
                            self.counts, self.offsets, self.cws, stream)

    def run_select(self, stream=None):
        """emr_eval_prepare, emr_eval_filter_tiles, emr_select (no mask plane)."""
        if getattr(self, "tile_flags", None) is None:
            self.tile_flags = torch.zeros(self.n_pairs, dense_tiles(self.grid.D), dtype=torch.uint8,
                                          device=self.device)
            self.sws = torch.zeros(select_workspace_size(self.grid, self.n_pairs), dtype=torch.uint8,
                                   device=self.device)
        self.prepare(stream)
        eval_filter_tiles(self.pack, self.query, self.grid, self.theta, self.band, self.w_min, self.split,
                          self.band_bits, self.tile_flags, self.ws, stream)
        select(self.split, self.band_bits, self.tile_flags, self.pack, self.query, self.ws, self.grid, self.mode,
               self.types, self.idx, self.w, self.cap, self.counts, self.offsets, self.sws, stream)

    def run_discover(self, stream=None):
        """emr_discover: the whole path in one call on its own workspace."""
        if getattr(self, "dws", None) is None:
            self.dws = torch.zeros(discover_workspace_size(self.pack, self.query, self.grid), dtype=torch.uint8,
                                   device=self.device)
        discover(self.pack, self.pack_dev, self.query, self.grid, self.theta, self.band, self.w_min, self.mode,
                 self.types, self.dws, self.idx, self.w, self.cap, self.counts, self.offsets, stream)

    def combine(self, stream=None):
        """emr_mask_combine, or emr_mask_combine_types when a connection-type filter is set."""
        if self.types == CONN_ALL:
            mask_combine(self.split, self.band_bits, self.grid, self.n_pairs, self.mode, self.mask, stream)
        else:
            mask_combine_types(self.split, self.band_bits, self.query, self.grid, self.n_pairs, self.mode,
                               self.types, self.mask, stream)

    def conn_types(self, stream=None):
        """Type codes of the current lists (device uint8 tensor of cap entries)."""
        t = torch.zeros(self.cap, dtype=torch.uint8, device=self.device)
        conn_types(self.idx, self.offsets, self.query, self.grid, self.n_pairs, self.cap, t, stream)
        return t

    def run_unfused(self, with_var: bool = False, stream=None):
        """emr_eval_prepare, emr_eval, emr_variance_filter, emr_compact."""
        self._materialise()
        if with_var and self.var_dbg is None:
            self.var_dbg = torch.zeros(self.n_pairs, self.grid.n_total, dtype=torch.float32, device=self.device)
        self.prepare(stream)
        eval(self.pack, self.query, self.grid, self.out, self.out_halo, self.ws, stream)
        variance_filter(self.out, self.out_halo, self.grid, self.P, self.S, self.theta, self.band, self.w_min,
                        self.mode, self.mask, self.split, self.band_bits, self.var_dbg if with_var else None,
                        stream)
        if self.types != CONN_ALL:
            self.combine(stream)
        compact(self.mask, self.out, self.grid, self.n_pairs, self.idx, self.w, self.cap, self.counts,
                self.offsets, self.cws, stream)

    def lists(self):
        """Host copies: per pair (idx, w) arrays, ascending global index."""
        off = self.offsets.cpu().numpy()
        total = int(off[-1])
        if total > self.cap:
            raise EmrError(EMR_ERR_CAPACITY, "compaction capacity %d < %d" % (self.cap, total))
        idx = self.idx[:total].cpu().numpy()
        w = self.w[:total].cpu().numpy()
        return [(idx[off[r]:off[r + 1]], w[off[r]:off[r + 1]]) for r in range(self.n_pairs)]


# ---- inspection of a packed blob (layout of csrc/emr_internal.h) ----------------------

_HDR = np.dtype([("magic", "<u4"), ("version", "<u4"), ("P", "<i4"), ("max_nodes", "<i4"),
                 ("max_varying", "<i4", 2), ("max_vedges", "<i4", 2), ("max_edges", "<i4"), ("reserved", "<i4"),
                 ("off_genomes", "<u8"), ("off_nodes", "<u8"), ("off_edges", "<u8"), ("total", "<u8")])
_GEN = np.dtype([("node_beg", "<u4"), ("edge_beg", "<u4"), ("n_nodes", "<u2"), ("n_edges", "<u2"),
                 ("n_varying", "<u2", 2), ("n_vedges", "<u2", 2), ("cost", "<u4", 2), ("n_joint", "<u2", 2)])
_NODE = np.dtype([("act", "u1"), ("vary", "u1"), ("axes", "u1"), ("reserved", "u1"), ("edge_beg", "<u2"), ("edge_cnt", "<u2"),
                  ("bias", "<f4"), ("w_in", "<f4", 5)])
_EDGE = np.dtype([("src", "<u2"), ("reserved", "<u2"), ("w", "<f4")])


def pack_records(pack: np.ndarray):
    """(header, genome table, node records, edge records) of a packed blob, as numpy views. The node
    and edge arrays are the blob's whole sections: genome g's records start at its node_beg and
    edge_beg (the slots past its n_nodes and n_edges are zero)."""
    raw = np.ascontiguousarray(pack).tobytes()
    h = np.frombuffer(raw[:_HDR.itemsize], _HDR)[0]
    P = int(h["P"])
    gs = np.frombuffer(raw, _GEN, P, int(h["off_genomes"]))
    nn = (int(h["off_edges"]) - int(h["off_nodes"])) // _NODE.itemsize
    ne = (int(h["total"]) - int(h["off_edges"])) // _EDGE.itemsize
    return h, gs, np.frombuffer(raw, _NODE, nn, int(h["off_nodes"])), np.frombuffer(raw, _EDGE, ne,
                                                                                    int(h["off_edges"]))
