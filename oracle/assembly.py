"""Substrate network assembly and forward pass, float64 (oracle side).

TEST INFRASTRUCTURE ONLY, like the rest of oracle/: used by the tests and the
smoke check, never by the library. It shares no code with the CUDA path. The
queries go through the oracle's own discovery (`oracle.discover`, fp64); the
graph steps are plain Python on small cases.

The construction (ES-HyperNEAT's, which the paper's Section 2 summarises and
Section 6 configures with connection types):
  Phase 1  an outgoing query from each substrate input keeps positions; each
           kept position becomes a hidden node, connected from that input.
  Phase 2  `rounds` times, an outgoing query from every hidden node found in
           the previous round; kept positions are connected from it and new
           ones become hidden nodes.
  Phase 3  an incoming query toward each substrate output; each kept position
           that is a hidden node is connected to that output.
  Prune    hidden nodes not reachable from an input, or from which no output is
           reachable, are removed with their connections.
Every connection must have an enabled type (Section 6 taxonomy). The network's
nodes are numbered inputs, outputs, then hidden positions ascending; a node's
value is the sigmoid of the weighted sum of its sources' previous values, all
nodes updated at once, inputs fixed to the pattern.

Parity status: pinned (tests/test_assembly_oracle.py) by the linear genome
whose every query keeps exactly Grid_3 (connection counts per configuration in
closed form, weights as closed forms), by a genome whose incoming query keeps
nothing (everything pruned), and by hand-built networks whose outputs after
each step are closed forms.
"""
from __future__ import annotations

import numpy as np

from . import conn_types as _conn_types
from . import discover as _discover

F, B, L, S = 0, 1, 2, 3


def _coords(p):
    d = 0
    while (4 ** (d + 2) - 4) // 3 <= p:
        d += 1
    m = p - (4 ** (d + 1) - 4) // 3
    i = sum(((m >> (2 * k)) & 1) << k for k in range(d + 1))
    j = sum(((m >> (2 * k + 1)) & 1) << k for k in range(d + 1))
    return (2 * i + 1) / 2.0 ** (d + 1) - 1.0, (2 * j + 1) / 2.0 ** (d + 1) - 1.0


class _Sources:
    def __init__(self, a, b, side, count=None):
        self.a = np.asarray(a, np.float32)
        self.b = np.asarray(b, np.float32)
        self.side = np.asarray(side, np.int32)
        self.count = None if count is None else np.asarray(count, np.int32)
        self.per_genome = self.a.ndim == 2
        self.S = self.a.shape[-1]


def _query(pop, src, D, theta, band, w_min, gated, enabled):
    """Kept positions and weights of every (genome, slot): list of lists of (gidx array, w array),
    plus, per genome, the number of uncertain decisions among positions of an enabled type."""
    r = _discover(pop, src, D, theta, band, w_min,
                  fields=("w", "keep_gated" if gated else "keep_eager", "unc_gated" if gated else "unc_eager"))
    keep = r["keep_gated" if gated else "keep_eager"]
    unc = r["unc_gated" if gated else "unc_eager"]
    N = keep.shape[-1]
    out, n_unc = [], np.zeros(pop.P, np.int64)
    for g in range(pop.P):
        row = []
        for s in range(src.S):
            if src.per_genome:
                a, b, side = float(src.a[g, s]), float(src.b[g, s]), int(src.side[g, s])
                if src.count is not None and s >= src.count[g]:
                    row.append((np.zeros(0, np.int64), np.zeros(0)))
                    continue
            else:
                a, b, side = float(src.a[s]), float(src.b[s]), int(src.side[s])
            ok = np.asarray(enabled, bool)[_conn_types(a, b, side, np.arange(N))]
            n_unc[g] += int(np.sum(unc[g, s].astype(bool) & ok))
            p = np.flatnonzero(keep[g, s].astype(bool) & ok)
            row.append((p, r["w"][g, s][p]))
        out.append(row)
    return out, n_unc


def _type(xs, ys, xt, yt):
    if xs == xt and ys == yt:
        return S
    return F if ys < yt else B if ys > yt else L


def assemble(pop, in_xy, out_xy, D, theta, band, w_min=0.0, gated=False, enabled=(1, 1, 1, 1), rounds=1):
    """Per genome: (hidden positions ascending, connections [(src, dst, w, type)] sorted by (dst, src)),
    and per genome the number of uncertain decisions its queries met (a genome's network depends
    on its own queries only, so one with none is fixed exactly)."""
    in_xy = np.asarray(in_xy, np.float32).reshape(-1, 2)
    out_xy = np.asarray(out_xy, np.float32).reshape(-1, 2)
    n_in, n_out = len(in_xy), len(out_xy)
    P = pop.P
    src1 = _Sources(np.r_[in_xy[:, 0], out_xy[:, 0]], np.r_[in_xy[:, 1], out_xy[:, 1]],
                    [0] * n_in + [1] * n_out)
    res, n_unc = _query(pop, src1, D, theta, band, w_min, gated, enabled)
    hidden = [dict() for _ in range(P)]    # position -> discovery order
    conns = [[] for _ in range(P)]         # (src, dst, w, type); src/dst: position or ("in"/"out", k)
    frontier = [[] for _ in range(P)]
    for g in range(P):
        for s in range(n_in):
            for p, w in zip(*res[g][s]):
                p = int(p)
                x, y = _coords(p)
                conns[g].append((("in", s), p, float(w), _type(float(in_xy[s, 0]), float(in_xy[s, 1]), x, y)))
                if p not in hidden[g]:
                    hidden[g][p] = len(hidden[g])
                    frontier[g].append(p)
    for _ in range(rounds):
        S_ = max((len(f) for f in frontier), default=0)
        new = [[] for _ in range(P)]
        if S_ > 0:
            a = np.zeros((P, S_), np.float32); b = np.zeros((P, S_), np.float32)
            for g in range(P):
                for k, p in enumerate(frontier[g]):
                    a[g, k], b[g, k] = _coords(p)
            src = _Sources(a, b, np.zeros((P, S_), np.int32), [len(f) for f in frontier])
            res2, u = _query(pop, src, D, theta, band, w_min, gated, enabled)
            n_unc += u
            for g in range(P):
                for k, sp in enumerate(frontier[g]):
                    xs, ys = _coords(sp)
                    for p, w in zip(*res2[g][k]):
                        p = int(p)
                        x, y = _coords(p)
                        conns[g].append((sp, p, float(w), _type(xs, ys, x, y)))
                        if p not in hidden[g]:
                            hidden[g][p] = len(hidden[g])
                            new[g].append(p)
        frontier = new
    nets = []
    for g in range(P):
        for o in range(n_out):
            for p, w in zip(*res[g][n_in + o]):
                p = int(p)
                if p in hidden[g]:
                    x, y = _coords(p)
                    conns[g].append((p, ("out", o), float(w),
                                     _type(x, y, float(out_xy[o, 0]), float(out_xy[o, 1]))))
        # reachability from the inputs and to the outputs
        succ, pred = {}, {}
        for s_, d_, _, _ in conns[g]:
            succ.setdefault(s_, []).append(d_)
            pred.setdefault(d_, []).append(s_)

        def reach(starts, adj):
            seen, stack = set(starts), list(starts)
            while stack:
                v = stack.pop()
                for u in adj.get(v, []):
                    if u not in seen:
                        seen.add(u)
                        stack.append(u)
            return seen

        fwd = reach([("in", k) for k in range(n_in)], succ)
        bwd = reach([("out", k) for k in range(n_out)], pred)
        kept = sorted(p for p in hidden[g] if p in fwd and p in bwd)
        num = {("in", k): k for k in range(n_in)}
        num.update({("out", k): n_in + k for k in range(n_out)})
        num.update({p: n_in + n_out + k for k, p in enumerate(kept)})
        cs = sorted((num[s_], num[d_], w, t) for s_, d_, w, t in conns[g] if s_ in num and d_ in num)
        cs.sort(key=lambda c: (c[1], c[0]))
        nets.append((np.array(kept, np.int64), cs))
    return nets, n_unc


def forward(n_in, n_out, hidden, conns, patterns, steps):
    """Outputs [K, n_out] of one network after `steps` synchronous updates (float64)."""
    pat = np.asarray(patterns, np.float64).reshape(-1, n_in)
    N = n_in + n_out + len(hidden)
    W = np.zeros((N, N))
    for s_, d_, w, _ in conns:
        W[d_, s_] += w
    v = np.zeros((N, pat.shape[0]))
    v[:n_in] = pat.T
    for _ in range(steps):
        z = W @ v
        with np.errstate(over="ignore"):   # e^-z = inf gives the sigmoid's limit 0 exactly
            nv = 1.0 / (1.0 + np.exp(-z))
        nv[:n_in] = pat.T
        v = nv
    return v[n_in:n_in + n_out].T
