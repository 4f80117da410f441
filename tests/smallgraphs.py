"""Test helpers: seeded random multi-rank graphs, hand-built graphs, and a brute-force
longest-path reference used to pin the oracle.

The random graphs are built in one random issue order: every op is appended to the
timelines it runs on in that order and may only depend on earlier ops, so each graph
is acyclic by construction.  None of this is the method's arithmetic; the brute force
below enumerates paths explicitly and shares nothing with the oracle's event loop.
"""
from __future__ import annotations

import math
from typing import List, Optional

import numpy as np

from paper_2412_12487_gb300 import workloads as W


def graph_from_lists(n_ranks, n_streams, ops, queues, groups, gpus_per_node=8):
    """ops: list of dicts (kind, kclass, group, cc_type, cc_algo, cc_bytes, preds);
    queues: dict (rank, stream) -> list of op ids; groups: list of member lists."""
    V = len(ops)
    kind = np.array([o["kind"] for o in ops], np.uint8).reshape(V)
    kclass = np.array([o.get("kclass", 0) for o in ops], np.uint8).reshape(V)
    group = np.array([o.get("group", -1) for o in ops], np.int32).reshape(V)
    cc_type = np.array([o.get("cc_type", 0) for o in ops], np.uint8).reshape(V)
    cc_algo = np.array([o.get("cc_algo", 0) for o in ops], np.uint8).reshape(V)
    cc_bytes = np.array([o.get("cc_bytes", 0) for o in ops], np.int64).reshape(V)
    pred_off = np.zeros(V + 1, np.int64)
    pred_idx: List[int] = []
    for v, o in enumerate(ops):
        ps = sorted(set(o.get("preds", ())))
        pred_idx += ps
        pred_off[v + 1] = len(pred_idx)
    nq = n_ranks * n_streams
    q_off = np.zeros(nq + 1, np.int64)
    q_ops: List[int] = []
    for q in range(nq):
        q_ops += list(queues.get((q // n_streams, q % n_streams), []))
        q_off[q + 1] = len(q_ops)
    grp_off = np.zeros(len(groups) + 1, np.int64)
    grp_rank: List[int] = []
    for i, m in enumerate(groups):
        grp_rank += list(m)
        grp_off[i + 1] = len(grp_rank)
    return W.Graph(n_ranks, n_streams, gpus_per_node, kind, kclass, group, cc_type, cc_algo,
                   cc_bytes, pred_off, np.array(pred_idx, np.int32), q_off,
                   np.array(q_ops, np.int32), grp_off, np.array(grp_rank, np.int32),
                   np.zeros(V), np.ones(V), name="hand")


def random_graph(rng: np.random.Generator, n_ops: int, max_ranks: int = 3, max_streams: int = 3,
                 gpus_per_node: int = 2, p_edge: float = 0.25, min_streams: int = 2):
    n_ranks = int(rng.integers(1, max_ranks + 1))
    n_streams = int(rng.integers(min_streams, max_streams + 1))
    ops, groups = [], []
    queues = {}
    for v in range(n_ops):
        r = float(rng.random())
        if r < 0.55:
            kind = W.KIND_COMPUTE
        elif r < 0.65:
            kind = W.KIND_MEMCPY
        elif r < 0.85:
            kind = W.KIND_COLL
        else:
            kind = W.KIND_P2P
        o = {"kind": kind, "kclass": int(rng.integers(0, 3))}
        if kind == W.KIND_COMPUTE:
            rank = int(rng.integers(0, n_ranks))
            queues.setdefault((rank, 0), []).append(v)
        elif kind == W.KIND_MEMCPY:
            rank = int(rng.integers(0, n_ranks))
            queues.setdefault((rank, int(rng.integers(1, n_streams))), []).append(v)
        else:
            if kind == W.KIND_P2P:
                size = min(2, n_ranks)
            else:
                size = int(rng.integers(1, n_ranks + 1))
            members = sorted(rng.choice(n_ranks, size=size, replace=False).tolist())
            o["group"] = len(groups)
            groups.append(members)
            o["cc_type"] = W.CC_SENDRECV if kind == W.KIND_P2P else int(rng.integers(0, 3))
            o["cc_algo"] = int(rng.integers(0, 3))
            o["cc_bytes"] = int(rng.integers(0, 1 << 22))
            for m in members:
                queues.setdefault((m, int(rng.integers(1, n_streams))), []).append(v)
        o["preds"] = [u for u in range(v) if rng.random() < p_edge]
        ops.append(o)
    return graph_from_lists(n_ranks, n_streams, ops, queues, groups, gpus_per_node)


def random_scenarios(rng: np.random.Generator, g: W.Graph, S: int, max_dur: int = 40,
                     n_kclass: int = 3) -> W.Scenarios:
    dur = rng.integers(0, max_dur + 1, size=(g.n_ops, S)).astype(np.int64)
    dur[(g.kind == W.KIND_COLL) | (g.kind == W.KIND_P2P)] = 0
    return W.Scenarios(
        dur=dur,
        alpha_ns=rng.integers(0, 30, size=S).astype(np.float64),
        bw_intra=rng.uniform(5e-4, 5e-3, size=S), lat_intra=rng.uniform(0, 5, size=S),
        bw_inter=rng.uniform(1e-4, 1e-3, size=S), lat_inter=rng.uniform(0, 9, size=S),
        delta=rng.uniform(0, 2e-6, size=S),
        slowdown=rng.uniform(1.0, 2.0, size=(n_kclass, S)),
        peak_flop_per_ns=np.ones(S))


# ------------------------------------------------------------------------------------
# brute force
# ------------------------------------------------------------------------------------
def merged_preds(g: W.Graph):
    """Data predecessors plus the op issued just before on each timeline."""
    V = g.n_ops
    preds = [set(g.pred_idx[g.pred_off[v]:g.pred_off[v + 1]].tolist()) for v in range(V)]
    for q in range(len(g.q_off) - 1):
        ops = g.q_ops[g.q_off[q]:g.q_off[q + 1]].tolist()
        for a, b in zip(ops[:-1], ops[1:]):
            preds[b].add(a)
    return [sorted(p) for p in preds]


def all_paths_to(v, preds, memo):
    """Every dependency path that ends at v (as tuples), enumerated explicitly."""
    if v in memo:
        return memo[v]
    out = [(v,)]
    for u in preds[v]:
        for p in all_paths_to(u, preds, memo):
            out.append(p + (v,))
    memo[v] = out
    return out


def brute_finish(g: W.Graph, d: np.ndarray):
    """finish(v) = the largest duration sum over all paths ending at v."""
    preds = merged_preds(g)
    memo = {}
    fin = np.zeros(g.n_ops, np.int64)
    for v in range(g.n_ops):
        fin[v] = max(int(sum(int(d[u]) for u in p)) for p in all_paths_to(v, preds, memo))
    return fin


def group_shape(g: W.Graph, gi: int):
    mem = g.grp_rank[g.grp_off[gi]:g.grp_off[gi + 1]].tolist()
    nodes = [m // g.gpus_per_node for m in mem]
    N, M = len(mem), len(set(nodes))
    K = max(nodes.count(n) for n in set(nodes)) if mem else 0
    return N, M, K, (math.log2(M) if M > 0 else 0.0)


def op_ranks(g: W.Graph):
    """rank(s) each op runs on, read from the timelines."""
    out = [set() for _ in range(g.n_ops)]
    for q in range(len(g.q_off) - 1):
        for v in g.q_ops[g.q_off[q]:g.q_off[q + 1]].tolist():
            out[v].add(q // g.n_streams)
    return out


def launch_preds(g: W.Graph):
    """{(comm op w, member rank r): the ops whose finish rank r waits for before it
    launches w}: the op just before w on r's timeline that holds w, and w's data
    producers that run on r."""
    ranks = op_ranks(g)
    out = {}
    for q in range(len(g.q_off) - 1):
        r = q // g.n_streams
        ops = g.q_ops[g.q_off[q]:g.q_off[q + 1]].tolist()
        for k, w in enumerate(ops):
            if g.kind[w] not in (W.KIND_COLL, W.KIND_P2P):
                continue
            ps = {u for u in g.pred_idx[g.pred_off[w]:g.pred_off[w + 1]].tolist() if r in ranks[u]}
            if k > 0:
                ps.add(ops[k - 1])
            out[(w, r)] = ps
    return out


def covered_length(pieces):
    """Length of the union of half-open intervals, by coordinate compression."""
    xs = sorted({x for p in pieces for x in p})
    return sum(b - a for a, b in zip(xs, xs[1:]) if any(lo <= a and b <= hi for lo, hi in pieces))


def brute_compose(g: W.Graph, sc: W.Scenarios, s: int, refine_passes: int, cc_fn, comm_interval: int = 0,
                  overlap_model: int = 0):
    """Brute-force reference of one scenario: CC durations from ``cc_fn`` (pinned on
    its own), composition by path enumeration, overlap by checking every pair.  A
    comm op's interval on rank r starts at its start (comm_interval 0) or when r
    has launched it (1: the latest finish among ``launch_preds``).  An overlapped
    kernel takes rint(d * f) (overlap_model 0) or rint(d + (f - 1) * covered
    length) (1)."""
    V = g.n_ops
    d0 = np.zeros(V, np.int64)
    for v in range(V):
        if g.kind[v] in (W.KIND_COLL, W.KIND_P2P):
            N, M, K, lg = group_shape(g, int(g.group[v]))
            T = cc_fn(int(g.cc_type[v]), int(g.cc_algo[v]), int(g.cc_bytes[v]), N, M, K, lg,
                      sc.alpha_ns[s], sc.bw_intra[s], sc.lat_intra[s], sc.bw_inter[s],
                      sc.lat_inter[s], sc.delta[s])
            d0[v] = int(np.rint(T))
        else:
            d0[v] = sc.dur[v, s]
    ranks = op_ranks(g)
    lp = launch_preds(g)
    d = d0.copy()
    fin = brute_finish(g, d)
    ov = np.zeros(V, np.uint8)
    for _ in range(refine_passes):
        st = fin - d
        covered = np.zeros(V, np.int64)
        for v in range(V):
            if g.kind[v] != W.KIND_COMPUTE:
                continue
            pieces = []
            for w in range(V):
                for r in ranks[v] & ranks[w] if g.kind[w] in (W.KIND_COLL, W.KIND_P2P) else ():
                    lo = st[w] if comm_interval == 0 else max([0] + [int(fin[u]) for u in lp[(w, r)]])
                    a, b = max(int(st[v]), int(lo)), min(int(fin[v]), int(fin[w]))
                    if a < b:
                        pieces.append((a, b))
            ov[v] = 1 if pieces else 0
            covered[v] = covered_length(pieces)
        d = d0.copy()
        for v in range(V):
            if g.kind[v] == W.KIND_COMPUTE and ov[v]:
                f = float(sc.slowdown[g.kclass[v], s])
                if overlap_model == 1:
                    d[v] = int(np.rint(float(d0[v]) + (f - 1.0) * float(covered[v])))
                else:
                    d[v] = int(np.rint(float(d0[v]) * f))
        fin = brute_finish(g, d)
    return fin - d, fin, ov
