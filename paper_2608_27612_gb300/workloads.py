"""Seeded synthetic inputs: CPPN populations and substrate source lists.

This module only draws inputs. It holds none of the method's arithmetic (no
CPPN evaluation, grid, variance or filtering), so both the CUDA path and the
CPU oracle can be fed from it without sharing any computation.

Genome encoding (flat, CSR over genomes). It follows the NEAT genome of the
paper's background section: nodes carry an activation and a kind, and
connections carry (source id, destination id, weight, enabled).

* node kinds: 0..4 are the CPPN inputs (x1, y1, x2, y2, bias), 5 hidden,
  6 output. The bias input always has the value 1.
* activations: 0 identity, 1 sigmoid, 2 tanh, 3 gauss, 4 sin, 5 abs.
* query sides: 0 = outgoing from a source node (a, b): CPPN(a, b, x, y, 1);
  1 = incoming toward a target node (a, b): CPPN(x, y, a, b, 1).

The five workloads mirror the paper's experiments in shape only (population
sizes, genome sizes, substrate layouts, depths); no task data is involved.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

KIND_X1, KIND_Y1, KIND_X2, KIND_Y2, KIND_BIAS, KIND_HIDDEN, KIND_OUTPUT = range(7)
ACT_IDENTITY, ACT_SIGMOID, ACT_TANH, ACT_GAUSS, ACT_SIN, ACT_ABS = range(6)
N_ACTS = 6
SIDE_OUT, SIDE_IN = 0, 1


@dataclass
class Population:
    """P genomes as flat arrays; genome g owns nodes [node_ptr[g], node_ptr[g+1])."""

    node_ptr: np.ndarray      # int64 [P+1]
    node_id: np.ndarray       # int32 [Nn]
    node_kind: np.ndarray     # int32 [Nn]
    node_act: np.ndarray      # int32 [Nn]
    node_bias: np.ndarray     # float32 [Nn]
    conn_ptr: np.ndarray      # int64 [P+1]
    conn_src: np.ndarray      # int32 [Nc]  (node ids)
    conn_dst: np.ndarray      # int32 [Nc]
    conn_w: np.ndarray        # float32 [Nc]
    conn_enabled: np.ndarray  # uint8 [Nc]

    @property
    def P(self) -> int:
        return len(self.node_ptr) - 1

    def subset(self, genomes) -> "Population":
        """A new population holding the listed genomes, in that order."""
        return population_from_lists([self.genome(int(g)) for g in genomes])

    def genome(self, g: int):
        a, b = self.node_ptr[g], self.node_ptr[g + 1]
        c, d = self.conn_ptr[g], self.conn_ptr[g + 1]
        nodes = [(int(self.node_id[k]), int(self.node_kind[k]), int(self.node_act[k]),
                  float(self.node_bias[k])) for k in range(a, b)]
        conns = [(int(self.conn_src[k]), int(self.conn_dst[k]), float(self.conn_w[k]),
                  bool(self.conn_enabled[k])) for k in range(c, d)]
        return nodes, conns


def population_from_lists(genomes) -> Population:
    """Build a Population from [(nodes, conns)], nodes = [(id, kind, act, bias)],
    conns = [(src_id, dst_id, w, enabled)]."""
    node_ptr = [0]
    conn_ptr = [0]
    nid, nkind, nact, nbias = [], [], [], []
    csrc, cdst, cw, cen = [], [], [], []
    for nodes, conns in genomes:
        for (i, k, a, b) in nodes:
            nid.append(i); nkind.append(k); nact.append(a); nbias.append(b)
        for (s, d, w, e) in conns:
            csrc.append(s); cdst.append(d); cw.append(w); cen.append(1 if e else 0)
        node_ptr.append(len(nid))
        conn_ptr.append(len(csrc))
    return Population(
        node_ptr=np.asarray(node_ptr, np.int64),
        node_id=np.asarray(nid, np.int32),
        node_kind=np.asarray(nkind, np.int32),
        node_act=np.asarray(nact, np.int32),
        node_bias=np.asarray(nbias, np.float32),
        conn_ptr=np.asarray(conn_ptr, np.int64),
        conn_src=np.asarray(csrc, np.int32),
        conn_dst=np.asarray(cdst, np.int32),
        conn_w=np.asarray(cw, np.float32),
        conn_enabled=np.asarray(cen, np.uint8),
    )


@dataclass
class Sources:
    """Query slots. Shared by all genomes ([S]) or per genome ([P, S]).

    a, b: float32 node coordinates; side: int32 (SIDE_OUT / SIDE_IN).
    count: optional int32 [P], number of valid slots per genome (per-genome mode).
    """

    a: np.ndarray
    b: np.ndarray
    side: np.ndarray
    count: np.ndarray | None = None

    @property
    def per_genome(self) -> bool:
        return self.a.ndim == 2

    @property
    def S(self) -> int:
        return self.a.shape[-1]


def shared_sources(points) -> Sources:
    """points = [(a, b, side)] shared by every genome."""
    a = np.asarray([p[0] for p in points], np.float32)
    b = np.asarray([p[1] for p in points], np.float32)
    s = np.asarray([p[2] for p in points], np.int32)
    return Sources(a=a, b=b, side=s)


def evenly_spaced(n: int, y: float, side: int):
    """n substrate nodes evenly spaced on the line y, x from -1 to 1."""
    xs = np.linspace(-1.0, 1.0, n) if n > 1 else np.zeros(1)
    return [(float(np.float32(x)), float(y), side) for x in xs]


def _path_from(conns, start_ids, target):
    adj = {}
    for (s, d, w, e) in conns:
        if e:
            adj.setdefault(s, []).append(d)
    seen = set(start_ids)
    stack = list(start_ids)
    while stack:
        u = stack.pop()
        for v in adj.get(u, []):
            if v not in seen:
                seen.add(v)
                stack.append(v)
    return target in seen


def _random_genome(rng: np.random.Generator, h_lo: int, h_hi: int, e_max: int,
                   p_disabled: float):
    """One feedforward NEAT-style CPPN: ids 0..4 inputs, 5 output, 6.. hidden.

    Hidden nodes take a random topological order; candidate connections are all
    forward pairs in that order; E ~ U{1..min(e_max, #candidates)} are drawn
    without replacement; the output is given at least one in-edge; weights are
    N(0,1) clipped to [-3, 3]; activations are uniform over the six kinds.
    """
    H = int(rng.integers(h_lo, h_hi + 1))
    hidden_ids = [6 + k for k in range(H)]
    order = [hidden_ids[k] for k in rng.permutation(H)]
    nodes = [(k, k, ACT_IDENTITY, 0.0) for k in range(5)]
    nodes.append((5, KIND_OUTPUT, int(rng.integers(0, N_ACTS)), 0.0))
    for hid in hidden_ids:
        nodes.append((hid, KIND_HIDDEN, int(rng.integers(0, N_ACTS)), 0.0))
    cand = []
    for k, h in enumerate(order):
        for s in range(5):
            cand.append((s, h))
        for s in order[:k]:
            cand.append((s, h))
    for s in list(range(5)) + order:
        cand.append((s, 5))
    E = int(rng.integers(1, min(e_max, len(cand)) + 1))
    pick = list(rng.choice(len(cand), size=E, replace=False))
    if not any(cand[i][1] == 5 for i in pick):
        into_out = [i for i, c in enumerate(cand) if c[1] == 5]
        pick[int(rng.integers(0, E))] = int(into_out[int(rng.integers(0, len(into_out)))])
        pick = list(dict.fromkeys(pick))
    w = np.clip(rng.standard_normal(len(pick)), -3.0, 3.0).astype(np.float32)
    en = rng.random(len(pick)) >= p_disabled
    conns = [(cand[i][0], cand[i][1], float(w[k]), bool(en[k])) for k, i in enumerate(pick)]
    return nodes, conns


def random_population(P: int, seed: int, h_lo: int = 0, h_hi: int = 12, e_max: int = 40,
                      p_disabled: float = 0.1) -> Population:
    rng = np.random.default_rng(seed)
    return population_from_lists([_random_genome(rng, h_lo, h_hi, e_max, p_disabled)
                                  for _ in range(P)])


def c1_genome(seed: int = 0) -> Population:
    """The single CPPN of the 1-genome workload: 5 inputs, hidden (sigmoid,
    gauss, sin) in that topological order, tanh output, 10 of the 26 acyclic
    candidate connections with w ~ U(-2, 2). Redrawn (same stream) until the
    output depends on the grid coordinates x2 or y2."""
    rng = np.random.default_rng(seed)
    h = [5, 6, 7]
    out = 8
    nodes = [(k, k, ACT_IDENTITY, 0.0) for k in range(5)]
    nodes += [(5, KIND_HIDDEN, ACT_SIGMOID, 0.0), (6, KIND_HIDDEN, ACT_GAUSS, 0.0),
              (7, KIND_HIDDEN, ACT_SIN, 0.0), (out, KIND_OUTPUT, ACT_TANH, 0.0)]
    cand = [(s, d) for d in h for s in range(5)] + [(s, out) for s in range(5)]
    cand += [(5, 6), (5, 7), (6, 7)] + [(s, out) for s in h]
    assert len(cand) == 26
    while True:
        pick = rng.choice(26, size=10, replace=False)
        w = rng.uniform(-2.0, 2.0, size=10).astype(np.float32)
        conns = [(cand[i][0], cand[i][1], float(w[k]), True) for k, i in enumerate(pick)]
        if _path_from(conns, [KIND_X2, KIND_Y2], out):
            return population_from_lists([(nodes, conns)])


@dataclass
class Workload:
    name: str
    pop: Population
    sources: Sources
    D: int
    theta: float
    band: float
    w_min: float = 0.0
    chunk: int = 0
    notes: str = ""
    extra: dict = field(default_factory=dict)

    @property
    def P(self) -> int:
        return self.pop.P

    @property
    def S(self) -> int:
        return self.sources.S


def c1(D: int = 4) -> Workload:
    """1 genome, 1 outgoing source at (0,-1), depth 4 (341 cells, 1,364 positions)."""
    return Workload("c1_single_d%d" % D, c1_genome(0), shared_sources([(0.0, -1.0, SIDE_OUT)]),
                    D, 0.03, 0.3)


def c2(D: int = 7, P: int = 1000) -> Workload:
    """XOR-shaped population: 1000 genomes with 0-12 hidden nodes and <=40 connections;
    substrate inputs (-1,-1), (1,-1), bias (0,-1) queried outgoing, output (0,1) incoming.
    P > 1000 continues the same generator (the first 1000 genomes are unchanged)."""
    pop = random_population(max(P, 1000), seed=2, h_lo=0, h_hi=12, e_max=40)
    if P != pop.P:
        pop = pop.subset(range(P))
    src = shared_sources([(-1.0, -1.0, SIDE_OUT), (1.0, -1.0, SIDE_OUT), (0.0, -1.0, SIDE_OUT),
                          (0.0, 1.0, SIDE_IN)])
    return Workload("c2_xor_pop%d_d%d" % (P, D), pop, src, D, 0.03, 0.3)


def c3(D: int = 6, P: int = 256) -> Workload:
    """Wide input: 256 genomes, 0-20 hidden, <=64 connections; 32 inputs on y=-1
    (outgoing) plus the output (0,1) (incoming): 33 query slots."""
    pop = random_population(256, seed=3, h_lo=0, h_hi=20, e_max=64)
    if P != 256:
        pop = pop.subset(range(P))
    src = shared_sources(evenly_spaced(32, -1.0, SIDE_OUT) + [(0.0, 1.0, SIDE_IN)])
    return Workload("c3_wide_pop%d_d%d" % (P, D), pop, src, D, 0.03, 0.3)


def c4_round1(D: int = 8, P: int = 150) -> Workload:
    """Full-recurrent substrate, first discovery round: 8 inputs on y=-1 (outgoing)
    and 4 outputs on y=+1 (incoming), depth 8, theta 0.02."""
    pop = random_population(150, seed=4, h_lo=0, h_hi=12, e_max=40)
    if P != 150:
        pop = pop.subset(range(P))
    src = shared_sources(evenly_spaced(8, -1.0, SIDE_OUT) + evenly_spaced(4, 1.0, SIDE_IN))
    return Workload("c4_recurrent_r1_pop%d_d%d" % (P, D), pop, src, D, 0.02, 0.3)


def c4_round2_random(D: int = 8, P: int = 150, S: int = 256, seed: int = 40) -> Workload:
    """Second round with fixed shapes: S hidden-node sources per genome drawn
    U[-1,1]^2 (seeded), queried outgoing (hidden -> hidden)."""
    w1 = c4_round1(D, P)
    rng = np.random.default_rng(seed)
    a = rng.uniform(-1, 1, size=(P, S)).astype(np.float32)
    b = rng.uniform(-1, 1, size=(P, S)).astype(np.float32)
    side = np.zeros((P, S), np.int32)
    return Workload("c4_recurrent_r2_pop%d_d%d_s%d" % (P, D, S), w1.pop,
                    Sources(a=a, b=b, side=side, count=np.full(P, S, np.int32)), D, 0.02, 0.3)


def c5(D: int = 13, P: int = 16, chunk: int = 1 << 26) -> Workload:
    """Deep streamed grid: 16 genomes, 0-16 hidden; 4 outgoing sources on y=-1;
    depth 13 in position chunks of 2^26."""
    pop = random_population(16, seed=5, h_lo=0, h_hi=16, e_max=40)
    if P != 16:
        pop = pop.subset(range(P))
    src = shared_sources(evenly_spaced(4, -1.0, SIDE_OUT))
    return Workload("c5_deep_pop%d_d%d" % (P, D), pop, src, D, 0.03, 0.3, chunk=chunk)

