#!/usr/bin/env python3
"""Benchmark of the eager multi-resolution substrate-discovery hot path on GB300.

Metric: CPPN queries/sec = genomes x query slots x N_total(D) / seconds, on the
1000-genome XOR-shaped population at depth 7 (4 slots: 3 outgoing substrate
inputs, 1 incoming output), 349.5 M queries per step. A step is one pass of the
whole path through libemr's C ABI: the per-pair records and pair schedule
(emr_eval_prepare), fused evaluation + variance + band filter of every tile
(emr_eval_filter_tiles), and the keep mask, ordered lists and kept weights from
the flagged tiles (emr_select).

`value` is device time with inputs resident in HBM (CUDA events, L2 flushed
between steps); `e2e` is the same metric through the host-buffer path: packing
on the host into pinned memory, the H2D copy of the packed genomes and slots,
emr_discover (the same three stages in one call), and the D2H read of the
offsets and connection lists, each step's copies overlapping its neighbours'
kernels, timed by the wall clock. Steps alternate between two compute streams
(each with its own workspace), so one step's latency-bound preparation and
selection overlap the next step's tile kernels; the figure with every step on
one stream is reported beside it (`e2e.one_stream`).

--impl reference times the float64 CPU oracle on a bounded sample of the same
workload (the only other place this script runs the oracle).
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "CPPN queries/sec (genomes x positions) at pop 1000 depth 7"
UNIT = "queries/s"

# Per-activation algorithmic cost per query (fp32 lane ops, MUFU ops).
ACT_FP32 = {0: 0, 1: 2, 2: 3, 3: 2, 4: 4, 5: 0}
ACT_MUFU = {0: 0, 1: 2, 2: 2, 3: 1, 4: 1, 5: 0}
VAR_OPS, BAND_OPS = 4.5, 1.0
MUFU_PER_SM_CLK = 16          # nominal MUFU lanes per SM per clock
FP32_PER_SM_CLK = 128         # FP32 lanes per SM per clock
SM_MAX_MHZ = 2070.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="emr", choices=["emr", "reference"])
    ap.add_argument("--depth", type=int, default=7)
    ap.add_argument("--pop", type=int, default=1000)
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--cpu-genomes", type=int, default=1000, help="oracle baseline sample (genomes)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extra", action="store_true", help="skip the streamed depth-13 and h->h round measurements")
    return ap.parse_args()


def dist_init():
    import torch
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    return rank, ws, local


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def allreduce(x, ws, op="max"):
    """All-reduce a float over the ranks (max or sum); works on the nccl and gloo backends."""
    if ws == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX if op == "max" else dist.ReduceOp.SUM)
    return float(t.item())


def allreduce_max(x, ws):
    return allreduce(x, ws, "max")


def rank_workload(W, emr, rank, ws, depth, pop):
    """This rank's share of one population: pop x ws genomes of the 1000-genome recipe (same
    generator, so at one rank it is that population), split by packed cost into ws contiguous
    genome ranges (emr_partition_genomes); about pop genomes per rank, so the work per GPU stays
    fixed as ranks are added (weak scaling). Returns the rank's workload and its genome range."""
    w = W.c2(D=depth, P=pop * ws)
    if ws == 1:
        return w, (0, w.P)
    from paper_2608_27612_gb300 import dist as pdist
    g = pdist.genome_ranges(emr.pack_population(w.pop), emr.make_query(w.sources, device="cpu"), ws)
    g0, g1 = int(g[rank]), int(g[rank + 1])
    full = w.pop
    w.pop = full.subset(range(g0, g1))
    w.name = "%s_genomes%d-%d" % (w.name, g0, g1)
    w.extra["full_population"] = full
    return w, (g0, g1)


def aggregate(local_queries, local_ms, ws):
    """Whole-job throughput: queries of all ranks over the slowest rank's time per step."""
    total = allreduce(float(local_queries), ws, "sum")
    ms = allreduce(float(local_ms), ws, "max")
    return total, ms, total / (ms / 1e3)


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""
    FIELDS = ["clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
              "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
              "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]

    def __init__(self, index):
        self.index, self.proc, self.lines = index, None, []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + ",".join(self.FIELDS),
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            p = [x.strip() for x in ln.split(",")]
            if len(p) < 8:
                continue
            try:
                sm.append(float(p[0])); mx.append(float(p[1]))
            except ValueError:
                continue
            for nm, v in zip(names, p[4:8]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


TILE_SIDE = 64


def algorithmic_work(pack, query, emr):
    """Per pair: fp32 lane ops and MUFU ops per query, for the evaluation as the tile
    kernels organise it, counted at its minimum on the packed DAG (dead nodes removed,
    constants folded). A node that depends on the grid x (or y) coordinate alone has one
    value per tile column (row): it is evaluated at the 66 distinct coordinates of a
    64 x 64 tile (ring included), a 66/4096 share per query (its first-layer FMA, its
    in-edges, its activation); so are the x part and the y part of a joint node's input
    (one first-layer operation each, plus the edges from sources of that one coordinate).
    Per query: each joint node's x + y add, its edges from joint sources and its
    activation; plus the filter at its minimum: per parent the six squared pairwise child
    differences, their sum and one compare (4.5 per query), and per quad the band
    screen's four compares on the sibling differences (1 per query; the full band test
    of the few quads the screen lets through is not counted). The pyramid tile (depths
    0..4, 0.4% of the positions at depth 7) is counted like the 64 x 64 tiles. A pair
    whose output is constant over the grid (no varying node) has variance and band value
    0 everywhere and counts no work."""
    h, gs, nodes, edges = emr.pack_records(pack)
    share = (TILE_SIDE + 2) / (TILE_SIDE * TILE_SIDE)
    per = np.zeros((len(gs), 2, 2))
    for g in range(len(gs)):
        nb, n, eb = int(gs["node_beg"][g]), int(gs["n_nodes"][g]), int(gs["edge_beg"][g])
        for side in (0, 1):
            F = M = F1 = M1 = 0.0
            for t in range(n):
                nd = nodes[nb + t]
                ax = (int(nd["axes"]) >> (2 * side)) & 3
                if ax == 0:
                    continue
                sax = [(int(nodes[nb + int(edges[eb + int(nd["edge_beg"]) + e]["src"])]["axes"]) >> (2 * side)) & 3
                       for e in range(int(nd["edge_cnt"]))]
                a = int(nd["act"])
                if ax == 3:
                    F += 1 + sum(1 for x in sax if x == 3) + ACT_FP32[a]
                    M += ACT_MUFU[a]
                    F1 += 2 + sum(1 for x in sax if x in (1, 2))
                else:
                    F1 += 1 + sum(1 for x in sax if x) + ACT_FP32[a]
                    M1 += ACT_MUFU[a]
            varying = F1 > 0 or F > 0
            per[g, side] = (F + share * F1 + VAR_OPS + BAND_OPS, M + share * M1) if varying else (0.0, 0.0)
    side = np.broadcast_to(query.side, (len(gs), query.S))
    return per[np.arange(len(gs))[:, None], side]  # [P, S, 2]


ACT_EX2 = {0: 0, 1: 1, 2: 1, 3: 1, 4: 0, 5: 0}   # MUFU ops per activation, by unit
ACT_RCP = {0: 0, 1: 1, 2: 1, 3: 0, 4: 0, 5: 0}
ACT_SIN = {0: 0, 1: 0, 2: 0, 3: 0, 4: 1, 5: 0}
SURVEY_VAR_OPS, SURVEY_BAND_OPS = 3.25, 8.0


def survey_work(pack, query, emr):
    """Per pair: the per-query work of the hot path as the method defines it, counted on
    the packed DAG (dead nodes removed, constants folded, parallel connections merged)
    with every node evaluated at every position. FP32 ops F = sum over the nodes that
    vary over the grid of (in-connections whose source varies: the grid's two inputs of
    the query side and varying nodes; plus the activation's FP32 ops) + 3.25 (4-child
    variance, amortised) + 8 (band test); MUFU ops counted per unit (ex2, rcp, sin).
    A pair whose output is constant still counts its filter (11.25). Returns [P, S, 4]:
    (F, ex2, rcp, sin) per query."""
    h, gs, nodes, edges = emr.pack_records(pack)
    per = np.zeros((len(gs), 2, 4))
    for g in range(len(gs)):
        nb, n, eb = int(gs["node_beg"][g]), int(gs["n_nodes"][g]), int(gs["edge_beg"][g])
        for side in (0, 1):
            grid_in = (2, 3) if side == 0 else (0, 1)   # outgoing: x2, y2 vary; incoming: x1, y1
            F = SURVEY_VAR_OPS + SURVEY_BAND_OPS
            ex2 = rcp = sn = 0.0
            for t in range(n):
                nd = nodes[nb + t]
                if not (int(nd["vary"]) >> side) & 1:
                    continue
                e_var = sum(1 for k in grid_in if float(nd["w_in"][k]) != 0.0)
                for e in range(int(nd["edge_cnt"])):
                    src = int(edges[eb + int(nd["edge_beg"]) + e]["src"])
                    if (int(nodes[nb + src]["vary"]) >> side) & 1:
                        e_var += 1
                a = int(nd["act"])
                F += e_var + ACT_FP32[a]
                ex2 += ACT_EX2[a]; rcp += ACT_RCP[a]; sn += ACT_SIN[a]
            per[g, side] = (F, ex2, rcp, sn)
    side = np.broadcast_to(query.side, (len(gs), query.S))
    return per[np.arange(len(gs))[:, None], side]


def survey_roofline(work, n_total, sms, probe, seconds):
    """Fraction of the FP32/MUFU roofline under the survey work model: the bound is the
    larger of the FP32 time (sum F over SMs x 128 lanes x max clock) and the MUFU time
    (each unit's ops over its measured throughput; the MUFU ops share one pipe)."""
    peak = sms * FP32_PER_SM_CLK * SM_MAX_MHZ * 1e6
    t_fp32 = float(work[..., 0].sum()) * n_total / peak
    t_mufu = n_total * (float(work[..., 1].sum()) / (probe["ex2_Gops"] * 1e9) +
                        float(work[..., 2].sum()) / (probe["rcp_Gops"] * 1e9) +
                        float(work[..., 3].sum()) / (probe["sin_Gops"] * 1e9))
    t_roof = max(t_fp32, t_mufu)
    return {"frac": t_roof / seconds, "t_roof_ms": t_roof * 1e3, "t_fp32_ms": t_fp32 * 1e3,
            "t_mufu_ms": t_mufu * 1e3, "achieved": t_roof * peak / seconds / 1e12,
            "fp32_ops_per_query": float(work[..., 0].mean()),
            "mufu_ops_per_query": float(work[..., 1:].sum(axis=-1).mean())}


def roofline_entry(emr, dsc, g, sms, probe, tile_s):
    """The tile kernels' ALU roofline under both work models. frac (= frac_survey_model)
    counts the method's per-query work with every node evaluated at every position (the
    model the 60% target is set on); frac_executed counts the separable evaluation's own
    minimum (what the kernels must issue)."""
    sv = survey_roofline(survey_work(dsc.pack, dsc.query, emr), g.n_total, sms, probe, tile_s)
    work = algorithmic_work(dsc.pack, dsc.query, emr)
    ratio = probe["ffma_per_mufu"]
    work_eq = float(np.maximum(work[..., 0], ratio * work[..., 1]).sum()) * g.n_total
    peak = sms * FP32_PER_SM_CLK * SM_MAX_MHZ * 1e6
    return {"bound": "alu", "achieved": sv["achieved"], "peak": peak / 1e12, "unit": "Tlane-op/s",
            "frac": sv["frac"], "frac_survey_model": sv["frac"],
            "survey_model": {k: v for k, v in sv.items() if k != "frac"},
            "survey_model_definition": "per query F = sum over grid-varying nodes of (varying in-connections + "
                                       "activation FP32 ops) + 3.25 (variance) + 8 (band), every node at every "
                                       "position; MUFU ex2/rcp/sin ops at their measured throughputs; "
                                       "T_roof = max(FP32 time at %d SMs x 128 lanes x %.0f MHz, MUFU time)"
                                       % (sms, SM_MAX_MHZ),
            "frac_executed": work_eq / tile_s / peak, "achieved_executed": work_eq / tile_s / 1e12,
            "executed_model_definition": "the separable evaluation's minimum: joint nodes per position, "
                                         "one-coordinate nodes per tile column/row (66/4096 per query), 4.5 "
                                         "variance + 1 band-screen ops, constant pairs 0; a MUFU op weighs the "
                                         "measured FFMA:MUFU ratio %.2f" % ratio,
            "fp32_ops_per_query_executed": float(work[..., 0].mean()),
            "mufu_ops_per_query_executed": float(work[..., 1].mean()),
            "kernel": "tile kernels of emr_eval_filter_tiles (tile_kernel_pyramid, tile_kernel_warp, "
                      "tile_kernel_one_axis; tile_kernel_dense up to depth 5)", "kernel_ms": tile_s * 1e3,
            "peak_basis": "%d SMs x %d FP32 lanes x %.0f MHz (max SM clock, nominal unit counts)"
                          % (sms, FP32_PER_SM_CLK, SM_MAX_MHZ)}


def alu_probe(emr, sms):
    """Measured FFMA and MUFU (ex2, rcp, sin) throughput in ops/s, and the FFMA:MUFU ratio."""
    out = {}
    names = {emr.PROBE_FFMA: "ffma", emr.PROBE_EX2: "ex2", emr.PROBE_RCP: "rcp", emr.PROBE_SIN: "sin"}
    for op, nm in names.items():
        iters = 4000 if op == emr.PROBE_FFMA else 500
        emr.probe_alu(op, sms * 8, 50)
        ops, ms = emr.probe_alu(op, sms * 8, iters)
        out[nm + "_Gops"] = ops / (ms * 1e-3) / 1e9
    mufu = min(out["ex2_Gops"], out["rcp_Gops"])
    out["ffma_per_mufu"] = out["ffma_Gops"] / mufu
    return out


def profiled_traffic():
    """DRAM bytes per step of the dense tile kernels from the committed ncu summary, if that
    summary was taken on the current kernel source (else None)."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "tile_kernels_c2_pop300_d7.md")
    src = os.path.join(ROOT, "paper_2608_27612_gb300", "csrc", "emr_kernels.cu")
    try:
        fields = dict(l.split(":", 1) for l in open(path).read().splitlines() if l.startswith(("traffic_", "kernel_")))
        sha = hashlib.sha256(open(src, "rb").read()).hexdigest()
        if fields.get("kernel_source_sha256", "").strip() == sha:
            return int(fields["traffic_bytes_per_step"])
    except (OSError, ValueError, KeyError):
        pass
    return None


def streamed_run(emr, torch, w, chunk, chunk_cap, cap, reps, mode=0, types=15, label=None):
    """Queries/sec of emr_stream (emr_stream_mode when a mode or type filter is given) on
    workload w (lists copied to pinned host memory)."""
    pack = emr.pack_population(w.pop)
    pack_dev = torch.from_numpy(pack).cuda()
    q = emr.make_query(w.sources)
    g = emr.grid_build(w.D, chunk)
    ws = torch.empty(emr.stream_workspace_size(pack, q, g, chunk_cap), dtype=torch.uint8, device="cuda")
    n_pairs = w.P * q.S
    h_idx = torch.empty(cap, dtype=torch.int32).pin_memory()
    h_w = torch.empty(cap, dtype=torch.float32).pin_memory()
    counts = np.zeros(n_pairs, np.int64)
    offsets = np.zeros(n_pairs + 1, np.int64)
    queries = float(n_pairs) * g.n_total
    if w.sources.count is not None:
        queries = float(w.sources.count.sum()) * g.n_total
    times = []
    for k in range(reps + 1):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        emr.stream(pack, pack_dev, q, g, w.theta, w.band, w.w_min, ws, chunk_cap, h_idx, h_w, counts, offsets,
                   mode=mode, types=types)
        if k:
            times.append(time.perf_counter() - t0)
    del ws
    torch.cuda.empty_cache()
    s = statistics.median(times)
    return {"workload": label or w.name, "queries": queries, "seconds": s, "value": queries / s, "unit": UNIT,
            "chunk_positions": chunk, "kept": int(offsets[-1]), "mode": "gated" if mode else "eager",
            "connection_types": types,
            "timing": "host wall clock per emr_stream call (synchronous, lists on the host), median of %d" % reps}


def networks_run(emr, torch, W, D=5, P=1000, config=None, reps=20):
    """Substrate networks of the XOR population (c2 genomes, inputs (-1,-1), (1,-1), bias (0,-1),
    output (0,1)): emr_assemble wall time, then emr_ann_forward on the four XOR patterns
    (CUDA events, networks resident on the device)."""
    config = emr.SUBSTRATE_HH if config is None else config
    w = W.c2(D=D, P=P)
    types, rounds = emr.substrate_config(config)
    pack = emr.pack_population(w.pop)
    pack_dev = torch.from_numpy(pack).cuda()
    grid = emr.grid_build(D)
    xor_in, xor_out = [(-1.0, -1.0), (1.0, -1.0), (0.0, -1.0)], [(0.0, 1.0)]
    times = []
    for k in range(3):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        nets = emr.assemble(pack, pack_dev, xor_in, xor_out, grid, w.theta, w.band, 0.0, emr.EMR_EAGER, types,
                            rounds)
        times.append(time.perf_counter() - t0)
    t_asm = statistics.median(times[1:])
    cache = emr.Cache(8 << 30)
    emr.assemble(pack, pack_dev, xor_in, xor_out, grid, w.theta, w.band, 0.0, emr.EMR_EAGER, types, rounds,
                 cache=cache)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    emr.assemble(pack, pack_dev, xor_in, xor_out, grid, w.theta, w.band, 0.0, emr.EMR_EAGER, types, rounds,
                 cache=cache)
    t_cached = time.perf_counter() - t0
    cst = cache.stats()
    del cache
    patterns = torch.tensor([[0, 0, 1], [0, 1, 1], [1, 0, 1], [1, 1, 1]], dtype=torch.float32, device="cuda")
    steps = rounds + 2
    out = emr.ann_forward(nets, patterns, steps)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        emr.ann_forward(nets, patterns, steps, out=out)
    e1.record()
    torch.cuda.synchronize()
    t_fwd = e0.elapsed_time(e1) / 1e3 / reps
    n_conn = int(nets.conn_off[-1])
    return {"workload": "c2_xor_networks_pop%d_d%d_%s" % (P, D, ["feedforward", "hh", "backward", "lateral",
                                                              "self", "full"][config]),
            "assemble_seconds": t_asm, "networks_per_s": P / t_asm,
            "assemble_seconds_cached": t_cached, "cache": cst,
            "hidden_nodes": int(nets.node_off[-1]), "connections": n_conn,
            "forward_seconds": t_fwd, "forward_steps": steps, "patterns": 4,
            "forward_connection_updates_per_s": n_conn * 4 * steps / t_fwd,
            "timing": "assembly: host wall clock per emr_assemble call (all query rounds, lists to the host, "
                      "pruning), median of 2 after one warm-up; forward: CUDA events, mean of %d" % reps}


def hbm_peak():
    """Measured copy bandwidth (GB/s) of the GB300s, or the stated fallback."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "of measured"
    except (OSError, ValueError, KeyError):
        return 6800.0, "of fallback"


def variants_run(emr, torch, W, D=7, P=1000, reps=10):
    """The subtree-leaf variance split (memory-bound over materialised outputs) and HyperNEAT weight
    scaling of the lists, on the c2 workload; CUDA events."""
    w = W.c2(D=D, P=P)
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, materialise=True)
    dsc.run_unfused()
    g = dsc.grid
    split = torch.zeros_like(dsc.split)
    ws = torch.empty(emr.subtree_workspace_size(g, dsc.n_pairs), dtype=torch.uint8, device="cuda")
    ev = lambda: torch.cuda.Event(enable_timing=True)
    emr.subtree_split(dsc.out, g, dsc.n_pairs, w.theta, split, ws)
    torch.cuda.synchronize()
    e0, e1 = ev(), ev()
    e0.record()
    for _ in range(reps):
        emr.subtree_split(dsc.out, g, dsc.n_pairs, w.theta, split, ws)
    e1.record()
    torch.cuda.synchronize()
    t_sub = e0.elapsed_time(e1) / 1e3 / reps
    leaves = dsc.n_pairs * 4 ** (D + 1)
    alg_bytes = 4 * leaves + 4 * dsc.n_pairs * int(g.word_off[D])   # leaves read, split words of depths < D written
    peak, basis = hbm_peak()
    dsc.run_fused()
    total = int(dsc.offsets[-1])
    wv = dsc.w.clone()
    torch.cuda.synchronize()
    e0.record()
    for _ in range(reps):
        emr.scale_weights(wv, dsc.offsets, dsc.n_pairs, dsc.cap, 0.1, 3.0)
    e1.record()
    torch.cuda.synchronize()
    t_scale = e0.elapsed_time(e1) / 1e3 / reps
    del ws, dsc
    torch.cuda.empty_cache()
    return {"subtree_split": {"workload": "c2_pop%d_d%d_materialised" % (P, D), "seconds": t_sub,
                              "leaves": leaves, "leaves_per_s": leaves / t_sub,
                              "roofline": {"bound": "hbm", "achieved": alg_bytes / t_sub / 1e9, "peak": peak,
                                           "unit": "GB/s", "frac": alg_bytes / t_sub / 1e9 / peak,
                                           "peak_basis": basis,
                                           "traffic_note": "algorithmic bytes: 4 B per depth-D output read, the "
                                                           "split words of depths < D written; the level "
                                                           "aggregates (about 1.8 B more per leaf) are scratch"}},
            "scale_weights": {"entries": total, "seconds": t_scale},
            "timing": "CUDA events, mean of %d" % reps}


def _events_mean(torch, fn, reps, flush):
    """Mean CUDA-event time (s) of fn() over reps runs, L2 flushed before each; the runs are
    queued back to back (one synchronisation at the end), so the host's calls overlap the
    device's work wherever the host is the faster of the two."""
    for _ in range(2):  # warm-up
        fn()
    evs = []
    for _ in range(reps):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        fn()
        e1.record()
        evs.append((e0, e1))
    torch.cuda.synchronize()
    return statistics.mean(e0.elapsed_time(e1) for e0, e1 in evs) / 1e3


def config_table(emr, torch, W, sms, probe, flush, reps=10, oracle_seconds=2.0):
    """Per workload: the step's device throughput (emr_discover: prepare + tiles + select, L2
    flushed, CUDA events), the tile kernels' ALU roofline under both work models (their time from
    a pass of the three calls with events around the tile launches), and the float64 oracle's
    throughput on a sample of about oracle_seconds (cores stated); the lazy ES-HyperNEAT tree
    timed on the single-genome and 1000-genome workloads."""
    import oracle
    oracle.build()
    rows = []
    specs = [("c1_single_d4", W.c1(), True), ("c2_xor_pop1000_d5", W.c2(D=5), True),
             ("c2_xor_pop1000_d6", W.c2(D=6), True), ("c2_xor_pop1000_d7", W.c2(D=7), True),
             ("c3_wide_pop256_d6", W.c3(D=6), False), ("c4_recurrent_r1_pop150_d8", W.c4_round1(), False)]
    for name, w, lazy in specs:
        dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, emr.EMR_EAGER)
        g = dsc.grid
        q = dsc.n_pairs * g.n_total
        dsc.run_select()
        torch.cuda.synchronize()
        tile = {}

        dws = torch.zeros(emr.discover_workspace_size(dsc.pack, dsc.query, g), dtype=torch.uint8, device="cuda")
        qc = dsc.query.c

        def step():
            emr.discover(dsc.pack, dsc.pack_dev, dsc.query, g, dsc.theta, dsc.band, dsc.w_min, dsc.mode,
                         dsc.types, dws, dsc.idx, dsc.w, dsc.cap, dsc.counts, dsc.offsets, qc=qc)

        def staged():  # the three calls, events around the tile launches
            dsc.prepare()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            emr.eval_filter_tiles(dsc.pack, dsc.query, g, dsc.theta, dsc.band, dsc.w_min, dsc.split,
                                  dsc.band_bits, dsc.tile_flags, dsc.ws)
            b.record()
            emr.select(dsc.split, dsc.band_bits, dsc.tile_flags, dsc.pack, dsc.query, dsc.ws, g, dsc.mode,
                       dsc.types, dsc.idx, dsc.w, dsc.cap, dsc.counts, dsc.offsets, dsc.sws)
            tile.setdefault("ev", []).append((a, b))

        t_step = _events_mean(torch, step, reps, flush)
        _events_mean(torch, staged, reps, flush)
        t_tile = statistics.mean(a.elapsed_time(b) for a, b in tile["ev"][-reps:]) / 1e3
        roof = roofline_entry(emr, dsc, g, sms, probe, t_tile)
        row = {"workload": name, "queries": q, "gpu_step_ms": t_step * 1e3, "gpu_value": q / t_step,
               "tile_kernels_ms": t_tile * 1e3, "frac_survey_model": roof["frac_survey_model"],
               "frac_executed": roof["frac_executed"], "kept": int(dsc.offsets[-1])}
        # oracle: whole genomes until about oracle_seconds have passed
        n_g, t_o = 0, 0.0
        while n_g < w.P and t_o < oracle_seconds:
            k = max(1, min(w.P - n_g, 8))
            t0 = time.perf_counter()
            oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, g0=n_g, g1=n_g + k,
                            fields=("keep_eager",))
            t_o += time.perf_counter() - t0
            n_g += k
        qo = n_g * w.S * g.n_total
        row["oracle"] = {"value": qo / t_o, "cores": oracle.threads(),
                         "sample": "%d of %d genomes x %d slots (%.3g queries + halo), %.2f s"
                                   % (n_g, w.P, w.S, qo, t_o)}
        if lazy:
            n_l = min(w.P, n_g)
            t0 = time.perf_counter()
            _, evals = oracle.lazy(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, g0=0, g1=n_l)
            t_l = time.perf_counter() - t0
            ql = n_l * w.S * g.n_total
            row["lazy"] = {"seconds": t_l, "cppn_evaluations": int(evals.sum()),
                           "evaluations_per_s": float(evals.sum()) / t_l,
                           "grid_equivalent_value": ql / t_l, "cores": oracle.threads(),
                           "sample": "%d genomes x %d slots, the lazy float64 quadtree (the ES-HyperNEAT order): "
                                     "grid_equivalent_value = the grid's queries of the sample / its time"
                                     % (n_l, w.S)}
        rows.append(row)
        del dsc
        torch.cuda.empty_cache()
    return rows


def hbm_rates(emr, torch, W, flush, reps=10):
    """Achieved bandwidth of the materialised evaluation (emr_eval: 4 B written per position and
    halo point) and of the compaction of a materialised mask (emr_compact: the mask plane read,
    8 B per kept entry and 16 B per pair written), 1000 genomes x 4 slots at depth 7, against the
    measured copy bandwidth."""
    w = W.c2(D=7)
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, emr.EMR_EAGER, materialise=True)
    g = dsc.grid
    peak, basis = hbm_peak()
    dsc.prepare()
    t_eval = _events_mean(torch, lambda: emr.eval(dsc.pack, dsc.query, g, dsc.out, dsc.out_halo, dsc.ws), reps,
                          flush)
    b_eval = 4 * dsc.n_pairs * (g.n_total + g.n_halo)
    dsc.run_unfused()
    torch.cuda.synchronize()
    kept = int(dsc.offsets[-1])
    t_cmp = _events_mean(torch, lambda: emr.compact(dsc.mask, dsc.out, g, dsc.n_pairs, dsc.idx, dsc.w, dsc.cap,
                                                    dsc.counts, dsc.offsets, dsc.cws), reps, flush)
    b_cmp = 4 * dsc.n_pairs * g.n_words + 8 * kept + 16 * dsc.n_pairs
    del dsc
    torch.cuda.empty_cache()
    ent = lambda b, t, what: {"bytes": b, "ms": t * 1e3, "achieved_gbs": b / t / 1e9, "peak_gbs": peak,
                              "frac": b / t / 1e9 / peak, "peak_basis": basis, "bytes_counted": what}
    return {"emr_eval_materialised": ent(b_eval, t_eval, "4 B per position and halo point written"),
            "emr_compact": ent(b_cmp, t_cmp, "mask plane read, 8 B per kept entry and 16 B per pair written"),
            "workload": "c2_xor_pop1000_d7", "timing": "CUDA events, L2 flushed, mean of %d" % reps}


def oracle_samples(W):
    """The float64 oracle on stated samples of the two workloads too large to run whole: the
    hidden-to-hidden round (2 genomes x 256 slots at depth 8) and the streamed depth-13 grid
    (the oracle's per-position keep decision, by direct CPPN queries, at 2^18 sampled positions
    of each of the 64 pairs)."""
    import oracle
    oracle.build()
    out = {}
    w = W.c4_round2_random()
    t0 = time.perf_counter()
    oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, g0=0, g1=2, fields=("keep_eager",))
    t = time.perf_counter() - t0
    q = 2 * w.S * oracle.n_total(w.D)
    out["c4_round2_hh_d8"] = {"value": q / t, "cores": oracle.threads(),
                              "sample": "2 of %d genomes x %d slots at depth %d (%.3g queries + halo), %.2f s"
                                        % (w.P, w.S, w.D, q, t)}
    w = W.c5()
    rng = np.random.default_rng(13)
    n = 1 << 14
    N = oracle.n_total(w.D)
    t = 0.0
    for gen in range(w.P):
        for s in range(w.S):
            d, i, j = level_ij(rng.integers(0, N, n))
            t0 = time.perf_counter()
            oracle.keep_at(w.pop, gen, float(w.sources.a[s]), float(w.sources.b[s]), int(w.sources.side[s]), w.D,
                           w.theta, w.band, w.w_min, d, i, j)
            t += time.perf_counter() - t0
    q = w.P * w.S * n
    out["c5_streamed_d13"] = {"value": q / t, "cores": oracle.threads(),
                              "sample": "%d positions of each of the %d pairs at depth %d, each position's keep "
                                        "decision from direct CPPN queries (itself, its 4 children, its 4 band "
                                        "neighbours), %.2f s" % (n, w.P * w.S, w.D, t)}
    return out


def launches_in_step(emr, dsc):
    """Kernel launches of one step: prepare (records, with the schedule in the last CTA); the
    tiles; selection (count, scan, write, kept weights). From depth 6 on, the tiles take one
    block launch for the depths 0..4 tile of every pair up to 8 joint nodes and of the
    one-coordinate pairs (one more for 9..12 joint nodes), then a warp-per-tile launch for the
    64 x 64 tiles of each non-empty class; up to depth 5, a block launch per class, the 1..2
    and 3..4 joint classes sharing one. The interpreter class takes one launch; constant-output
    pairs none (their tiles hold no band bit). Memsets are not kernels."""
    _, gs, _, _ = emr.pack_records(dsc.pack)
    side = np.asarray(dsc.query.side)
    def per_pair(field):
        f = gs[field][:, side] if not dsc.query.per_genome else \
            np.take_along_axis(gs[field], side.reshape(gs.shape[0], -1), axis=1)
        return f.astype(np.int64)
    nv, nj = per_pair("n_varying"), per_pair("n_joint")
    cls = np.where(nv > 12, 0, np.where(nj > 8, 1, np.where(nj > 6, 2, np.where(nj > 4, 3, np.where(
        nj > 2, 4, np.where(nj > 0, 5, 6))))))
    present = set(np.unique(cls[nv > 0]).tolist())
    if dsc.grid.D >= 6:
        tiles = len(present) + (1 if 1 in present else 0) + (1 if present & {2, 3, 4, 5, 6} else 0)
    else:
        tiles = len(present) - (1 if {4, 5} <= present else 0)
    return 1 + tiles + 4


def oracle_baseline(w, genomes):
    """The float64 oracle, as it stands, on the first `genomes` genomes (timed), with the
    keep decisions and their uncertainty flags it returns."""
    import oracle
    oracle.build()
    t0 = time.perf_counter()
    r = oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, g0=0, g1=genomes,
                        fields=("keep_eager", "unc_eager"))
    dt = time.perf_counter() - t0
    q = genomes * w.S * oracle.n_total(w.D)
    return {"value": q / dt, "unit": UNIT, "cores": oracle.threads(), "kind": "oracle",
            "sample": "%d of %d genomes x %d slots at depth %d (%.3g queries + halo), %.2f s"
                      % (genomes, w.P, w.S, w.D, q, dt)}, r


def level_ij(p):
    """Depth and grid indices (i, j) of global indices (depth-major, Morton within a depth)."""
    p = np.asarray(p, np.int64)
    d = np.zeros(len(p), np.int64)
    for k in range(1, 16):
        d += p >= (4 ** (k + 1) - 4) // 3
    m = p - (4 ** (d + 1) - 4) // 3
    i = np.zeros_like(m); j = np.zeros_like(m)
    for k in range(16):
        i |= ((m >> (2 * k)) & 1) << k
        j |= ((m >> (2 * k + 1)) & 1) << k
    return d.astype(np.int32), i, j


def lists_parity(w, dsc, ora, genomes):
    """The timed step's lists against the oracle: every certain keep decision of the first
    `genomes` genomes bit for bit, and every kept weight within max(1e-5 + 1e-4|w|, the
    oracle's fp32 bound) (the oracle re-evaluated at the kept positions)."""
    import oracle
    S, N = w.S, dsc.grid.n_total
    n_pairs = genomes * S
    off = dsc.offsets.cpu().numpy()
    n = int(off[n_pairs])
    idx = dsc.idx[:n].cpu().numpy().astype(np.int64)
    wv = dsc.w[:n].cpu().numpy().astype(np.float64)
    cnt = np.diff(off[:n_pairs + 1])
    rows = np.repeat(np.arange(n_pairs), cnt)
    keep = ora["keep_eager"].reshape(n_pairs, N).astype(bool)
    unc = ora["unc_eager"].reshape(n_pairs, N).astype(bool)
    gpu = np.zeros((n_pairs, N), bool)
    gpu[rows, idx] = True
    mism = (gpu != keep) & ~unc
    w_bad = ill = 0
    for r in np.flatnonzero(cnt):
        g, s = divmod(int(r), S)
        sl = slice(int(off[r]), int(off[r + 1]))
        d, i, j = level_ij(idx[sl])
        o = oracle.keep_at(w.pop, g, float(w.sources.a[s]), float(w.sources.b[s]), int(w.sources.side[s]), w.D,
                           w.theta, w.band, w.w_min, d, i, j, nthreads=1)
        t = 1e-5 + 1e-4 * np.abs(o["w"])
        lim = np.where(o["w_err"] > t, o["w_err"], t)
        w_bad += int((~(np.abs(wv[sl] - o["w"]) <= lim)).sum())
        ill += int((o["w_err"] > t).sum())
    return {"genomes": genomes, "decisions": int(keep.size), "mismatches": int(mism.sum()),
            "uncertain": int(unc.sum()), "uncertain_agree": int((unc & (gpu == keep)).sum()),
            "kept": n, "weights_checked": n, "weight_mismatches": w_bad, "ill_conditioned": ill,
            "rule": "keep decisions bit-exact where the oracle's margin exceeds 1e-6 + its fp32 bound "
                    "(the rest counted as uncertain); kept weights within max(1e-5 + 1e-4|w|, bound); "
                    "ill_conditioned counts kept weights whose bound exceeds the plain tolerance"}


def run_reference(args):
    rank, ws, _ = int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), 0
    if rank != 0:
        return
    from paper_2608_27612_gb300 import workloads as W
    import oracle
    oracle.build()
    w = W.c2(D=args.depth, P=args.pop)
    per_step = 4  # genomes per step: a bounded sample of the workload
    q = per_step * w.S * oracle.n_total(w.D)
    ts = []
    for k in range(args.warmup + args.steps):
        g0 = (k * per_step) % w.P
        t0 = time.perf_counter()
        oracle.discover(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, g0=g0, g1=g0 + per_step,
                        fields=("keep_eager",))
        if k >= args.warmup:
            ts.append(time.perf_counter() - t0)
    ms = 1e3 * statistics.mean(ts)
    val = q / (ms / 1e3)
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": val, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "genomes": w.P, "slots": w.S, "depth": w.D,
                   "queries_per_step_full": w.P * w.S * oracle.n_total(w.D), "sample_genomes_per_step": per_step},
        "cpu_baseline": {"value": val, "unit": UNIT, "cores": oracle.threads(), "kind": "oracle",
                         "sample": "%d genomes x %d slots per step at depth %d" % (per_step, w.S, w.D)},
        "e2e": {"value": val, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    import torch
    rank, ws, local = dist_init()
    torch.cuda.set_device(local)
    from paper_2608_27612_gb300 import emr
    from paper_2608_27612_gb300 import workloads as W

    # One population split by cost over the ranks (no collective on the data path; the lists are
    # gathered to rank 0 after the timed region).
    w, g_range = rank_workload(W, emr, rank, ws, args.depth, args.pop)
    dsc = emr.Discovery(w.pop, w.sources, w.D, w.theta, w.band, w.w_min, emr.EMR_EAGER)
    g = dsc.grid
    queries = dsc.n_pairs * g.n_total
    stream = torch.cuda.current_stream()
    flush = torch.empty(64 << 20, dtype=torch.float32, device="cuda")  # 256 MB > 129 MB L2

    ev = lambda: torch.cuda.Event(enable_timing=True)
    tile_flags = torch.zeros(dsc.n_pairs, emr.dense_tiles(w.D), dtype=torch.uint8, device="cuda")
    sws = torch.zeros(emr.select_workspace_size(g, dsc.n_pairs), dtype=torch.uint8, device="cuda")

    dws = torch.zeros(emr.discover_workspace_size(dsc.pack, dsc.query, g), dtype=torch.uint8, device="cuda")
    qc = dsc.query.c

    def step():
        """One pass through the one-call entry point (emr_discover), inputs resident on the device."""
        emr.discover(dsc.pack, dsc.pack_dev, dsc.query, g, dsc.theta, dsc.band, dsc.w_min, dsc.mode, dsc.types,
                     dws, dsc.idx, dsc.w, dsc.cap, dsc.counts, dsc.offsets, qc=qc)

    def staged(evs):
        """The same pass in its three calls, CUDA events between them (the phase pass)."""
        dsc.prepare()
        evs[0].record(stream)
        emr.eval_filter_tiles(dsc.pack, dsc.query, g, dsc.theta, dsc.band, dsc.w_min, dsc.split, dsc.band_bits,
                              tile_flags, dsc.ws)
        evs[1].record(stream)
        emr.select(dsc.split, dsc.band_bits, tile_flags, dsc.pack, dsc.query, dsc.ws, g, dsc.mode, dsc.types,
                   dsc.idx, dsc.w, dsc.cap, dsc.counts, dsc.offsets, sws)

    launches_per_step = launches_in_step(emr, dsc)
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.2)
    starts, ends = [ev() for _ in range(args.steps)], [ev() for _ in range(args.steps)]
    barrier(ws)
    torch.cuda.synchronize()
    wall0 = time.perf_counter()
    for k in range(args.steps):
        flush.zero_()
        starts[k].record(stream)
        step()
        ends[k].record(stream)
    torch.cuda.synchronize()
    barrier(ws)
    wall = time.perf_counter() - wall0
    # the phase pass: right after the timed region, same inputs, L2 flushed before each pass, the
    # clock sampler still running; its tile time is the roofline's kernel time
    for _ in range(3):
        staged((ev(), ev()))
    pstarts, pends, tiles = [ev() for _ in range(args.steps)], [ev() for _ in range(args.steps)], []
    torch.cuda.synchronize()
    for k in range(args.steps):
        flush.zero_()
        te = (ev(), ev())
        pstarts[k].record(stream)
        staged(te)
        pends[k].record(stream)
        tiles.append(te)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    tile_ms = [a.elapsed_time(b) for a, b in tiles]
    phases = {"prepare_ms": statistics.mean(s.elapsed_time(t[0]) for s, t in zip(pstarts, tiles)),
              "tiles_ms": statistics.mean(tile_ms),
              "select_ms": statistics.mean(t[1].elapsed_time(e) for t, e in zip(tiles, pends)),
              "staged_step_ms": statistics.mean(s.elapsed_time(e) for s, e in zip(pstarts, pends)),
              "note": "phase pass after the timed region: the same step in its three calls (emr_eval_prepare, "
                      "emr_eval_filter_tiles, emr_select) with CUDA events between them, which keep the calls "
                      "from overlapping; the timed steps run the one-call emr_discover"}
    _, ms, value = aggregate(queries, statistics.mean(step_ms), ws)

    # roofline of the dominant kernel (fused eval + variance + band)
    props = torch.cuda.get_device_properties(local)
    sms = props.multi_processor_count
    probe = alu_probe(emr, sms)
    tile_s = statistics.mean(tile_ms) / 1e3
    roofline = roofline_entry(emr, dsc, g, sms, probe, tile_s)
    roofline["traffic"] = profiled_traffic() if args.pop == 1000 and args.depth == 7 else None
    roofline["traffic_note"] = ("DRAM bytes of the tile launches per step, from profiles/"
                                "tile_kernels_c2_pop300_d7.md (300-genome capture scaled by pairs, x10/3); null "
                                "when the kernel source changed since")
    roofline["kernel_ms_source"] = ("CUDA events around emr_eval_filter_tiles in the phase pass right after the "
                                    "timed region (same inputs, L2 flushed before each step, same clocks sampled)")
    roofline["alu_probe"] = probe
    if clocks:
        roofline["frac_at_sampled_clock"] = roofline["frac"] * SM_MAX_MHZ / clocks["sm_mhz"]
        roofline["frac_executed_at_sampled_clock"] = roofline["frac_executed"] * SM_MAX_MHZ / clocks["sm_mhz"]

    # end to end through host buffers and the one-call entry point (emr_discover), pipelined: each
    # step packs its population into pinned memory, copies it and the query slots to the device and
    # reads its lists back (offsets first, then the entries they count). Input and output sets
    # alternate: step k + 1's inputs are copied while step k computes, and step k's lists are read
    # on a second stream while step k + 1 computes. Measured with every step on one compute stream,
    # and with steps alternating between two compute streams (the reported figure).
    e2e = None
    if args.e2e_steps > 0:
        # each rank packs its genome range of the whole population through the range hook
        full_pop = w.extra.get("full_population", w.pop)
        pack_range = g_range if full_pop is not w.pop else None
        # one pinned input buffer per step in flight, [a | b | side | packed population], and one
        # device copy of it: a single host-to-device copy a step of the bytes in use; the packer
        # writes in place
        S = dsc.query.S
        ob = (12 * S + 255) // 256 * 256
        in_bytes = ob + emr.pack_size(full_pop, genomes=pack_range)
        in_pinned = [torch.empty(in_bytes, dtype=torch.uint8).pin_memory() for _ in range(2)]
        for buf in in_pinned:
            q_h = buf[:12 * S].numpy()
            q_h[:4 * S] = np.ascontiguousarray(dsc.query.a, np.float32).view(np.uint8)
            q_h[4 * S:8 * S] = np.ascontiguousarray(dsc.query.b, np.float32).view(np.uint8)
            q_h[8 * S:12 * S] = np.ascontiguousarray(dsc.query.side, np.int32).view(np.uint8)
        # two device input buffers: step k + 1's inputs are copied (on their own stream) while
        # step k's kernels run
        in_dev = [torch.empty(in_bytes, dtype=torch.uint8, device="cuda") for _ in range(2)]
        pack_dev = [t[ob:] for t in in_dev]
        q_e2e = [emr.Query(dsc.query.a, dsc.query.b, dsc.query.side, None, t[:4 * S].view(torch.float32),
                           t[4 * S:8 * S].view(torch.float32), t[8 * S:12 * S].view(torch.int32), None, S, False)
                 for t in in_dev]
        qc = [q.c for q in q_e2e]
        outs = [(dsc.idx, dsc.w, dsc.counts, dsc.offsets),
                (torch.empty_like(dsc.idx), torch.empty_like(dsc.w), torch.empty_like(dsc.counts),
                 torch.empty_like(dsc.offsets))]
        res_off = [torch.empty(dsc.n_pairs + 1, dtype=torch.int64).pin_memory() for _ in range(2)]
        idx_h = torch.empty(dsc.cap, dtype=torch.int32).pin_memory()
        w_h = torch.empty(dsc.cap, dtype=torch.float32).pin_memory()
        res_off_np = [t.numpy() for t in res_off]
        ws_bytes = emr.discover_workspace_size(dsc.pack, dsc.query, g)

        def e2e_run(n_compute):
            """Wall-clock steps through emr_discover with n_compute compute streams (1: every step on
            the benchmark's stream; 2: steps alternate between two streams and workspaces, so that
            one step's latency-bound preparation and selection overlap the other's tile kernels)."""
            cstreams = [stream] if n_compute == 1 else [torch.cuda.Stream() for _ in range(2)]
            dws = [torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda") for _ in range(len(cstreams))]
            copy_in = torch.cuda.Stream()
            inputs_in = [torch.cuda.Event(), torch.cuda.Event()]  # step k's inputs are on the device
            done = [torch.cuda.Event(), torch.cuda.Event()]       # step k's offsets are on the host
            read = [torch.cuda.Event(), torch.cuda.Event()]       # step k's lists are on the host
            copy = torch.cuda.Stream()
            h2d = d2h = 0
            n_warm, n_steps = 2, args.e2e_steps

            def read_lists(k):
                b = k & 1
                done[b].synchronize()
                n = min(int(res_off_np[b][-1]), dsc.cap)
                copy.wait_event(done[b])
                emr.copy_async(idx_h, outs[b][0], 4 * n, copy)
                emr.copy_async(w_h, outs[b][1], 4 * n, copy)
                read[b].record(copy)
                return 8 * (dsc.n_pairs + 1) + 8 * n

            torch.cuda.synchronize()
            for k in range(n_warm + n_steps):
                if k == n_warm:
                    t0 = time.perf_counter()
                b = k & 1
                cs, wsp = cstreams[k % len(cstreams)], dws[k % len(cstreams)]
                buf = in_pinned[b]
                # this input set's last user, step k - 2, has finished (its offsets were synchronised
                # on in the previous iteration), so the packer and the copy may overwrite it
                blob = emr.pack_population(full_pop, out=buf[ob:].numpy(), genomes=pack_range)
                h2d = ob + len(blob)
                emr.copy_async(in_dev[b], buf, h2d, copy_in)
                inputs_in[b].record(copy_in)
                cs.wait_event(inputs_in[b])
                if k >= 2:
                    cs.wait_event(read[b])  # step k - 2's lists have left this output set
                idx_o, w_o, cnt_o, off_o = outs[b]
                emr.discover(blob, pack_dev[b], q_e2e[b], g, dsc.theta, dsc.band, dsc.w_min, dsc.mode, dsc.types,
                             wsp, idx_o, w_o, dsc.cap, cnt_o, off_o, stream=cs, qc=qc[b])
                emr.copy_async(res_off[b], off_o, 8 * (dsc.n_pairs + 1), cs)
                done[b].record(cs)
                if k >= 1:
                    d2h = read_lists(k - 1)
            d2h = read_lists(n_warm + n_steps - 1)
            torch.cuda.synchronize()
            elapsed = time.perf_counter() - t0
            _, e2e_ms, e2e_value = aggregate(queries, elapsed / n_steps * 1e3, ws)
            return {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "ms_per_step": e2e_ms, "compute_streams": n_compute,
                    "pipeline": "two input and two output sets: each step packs into pinned memory on the host, "
                                "copies its inputs on a copy stream while the previous step computes, and its "
                                "lists are read on a second copy stream after step k+1 is queued; %s; wall "
                                "clock over %d steps"
                                % ("every step on one compute stream" if n_compute == 1 else
                                   "steps alternate between two compute streams, each with its own workspace",
                                   n_steps)}

        # output set 0 is dsc's own buffers: the parity check below reads the lists an even step left there
        one = e2e_run(1)
        e2e = e2e_run(2)
        e2e["one_stream"] = {"value": one["value"], "ms_per_step": one["ms_per_step"]}

    gather = None
    if ws > 1:
        # the lists of every rank's genome range to rank 0 (the rank that assembles networks)
        from paper_2608_27612_gb300 import dist as pdist
        n_loc = min(int(dsc.offsets[-1]), dsc.cap)
        torch.cuda.synchronize()
        barrier(ws)
        t0 = time.perf_counter()
        got = pdist.gather_lists(dsc.counts, dsc.idx[:n_loc], dsc.w[:n_loc])
        torch.cuda.synchronize()
        g_ms = allreduce((time.perf_counter() - t0) * 1e3, ws, "max")
        gather = {"ms": g_ms, "entries_local": n_loc,
                  "entries_total": int(got[1][-1]) if got is not None else None,
                  "pairs_total": int(got[0].numel()) if got is not None else None,
                  "how": "torch.distributed all_gather of sizes, then gather of padded counts, indices and "
                         "weights to rank 0 (NCCL); wall clock, max over ranks; outside the timed steps"}

    extra = None
    if rank == 0 and ws == 1 and not args.no_extra:
        c4r2 = W.c4_round2_random()
        extra = {"c5_streamed_d13": streamed_run(emr, torch, W.c5(), 1 << 26, 1 << 24, 1 << 26, 3),
                 "c5_streamed_d13_gated": streamed_run(emr, torch, W.c5(), 1 << 26, 1 << 24, 1 << 26, 3,
                                                       mode=emr.EMR_GATED),
                 "c4_round2_hh_d8": streamed_run(emr, torch, c4r2, 1 << 16, 1 << 24, 1 << 26, 3),
                 "c4_round2_hh_d8_backward_config": streamed_run(
                     emr, torch, c4r2, 1 << 16, 1 << 24, 1 << 26, 3,
                     types=emr.substrate_config(emr.SUBSTRATE_BACKWARD)[0], label=c4r2.name + "_backward"),
                 "xor_networks_hh_d5": networks_run(emr, torch, W),
                 "variants_c2_d7": variants_run(emr, torch, W),
                 "configs": config_table(emr, torch, W, sms, probe, flush),
                 "hbm": hbm_rates(emr, torch, W, flush)}
        if not args.no_cpu_baseline:
            extra["oracle_samples"] = oracle_samples(W)

    cpu = parity = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu, ora = oracle_baseline(w, min(args.cpu_genomes, w.P))
        parity = lists_parity(w, dsc, ora, min(args.cpu_genomes, w.P))
        del ora

    kept = int(dsc.offsets[-1])
    if rank == 0:
        print(json.dumps({
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": w.name, "genomes": w.P, "slots": w.S, "depth": w.D, "n_total": g.n_total,
                       "queries_per_step": queries, "theta": w.theta, "band": w.band, "mode": "eager",
                       "l2": "flushed between steps (256 MB write)", "kept_connections": kept,
                       "parallelism": ("one population of %d x %d genomes split by cost into contiguous genome "
                                       "ranges, one per GPU" % (args.pop, ws)) if ws > 1 else "single GPU",
                       "genome_range": list(g_range)},
            "phases": phases, "roofline": roofline, "cpu_baseline": cpu, "parity": parity, "e2e": e2e,
            "gather": gather,
            "extra": extra,
            "gpu_launches": launches_per_step * args.steps, "clocks": clocks,
            "wall_s_timed_region": wall, "gpu": props.name,
        }))
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
